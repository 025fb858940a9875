/*
 * NOBLE linear layer with the CosNet branch: plain fp64 CPU oracle.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may call, link or
 * load this file; only the tests, the smoke check and the CPU-baseline leg of
 * the benchmark do.  It shares no source with the CUDA library.
 *
 * Orientation follows the paper's Eq. 1 (Section 3.1) with row vectors:
 *
 *     y = x W + bias + sigma(x W_down) W_up
 *     W      : [d_in][d_out]
 *     W_down : [d_in][r]
 *     W_up   : [r][d_out]
 *
 * and sigma is CosNet, Eq. 2 (Section 3.2) / Eqs. 5-7 (Appendix A):
 *
 *     h  = x W_down                    (bottleneck input, r wide)
 *     u1 = omega1 * h + phi1           (elementwise)
 *     a  = cos(u1)
 *     b  = a M        b_j = sum_i a_i M[i][j]   (reading of "M . cos(...)")
 *     u2 = omega2 * b + phi2
 *     c  = cos(u2)    = sigma(h)
 *
 * Further sigma modes pin the oracle and are the reference for the GPU's
 * bottleneck variants of the same name:
 *   ORACLE_IDENTITY: sigma(h) = h, where the branch collapses to
 *                    x (W + W_down W_up)   (the LoRA remark in Section 1 and 3.1)
 *   ORACLE_COS1:     sigma(h) = cos(omega1 * h + phi1), the single-cosine
 *                    activation of the ablation in Section 4.4 (Table 5).
 *   ORACLE_{TANH,LEAKY,GELU}{1,2}: the other activations f of that ablation,
 *                    one layer, sigma(h) = f(h), or two layers around the
 *                    mixing matrix, sigma(h) = f(f(h) M).  The paper gives
 *                    frequencies and phases to the cosine only, so these
 *                    have none.  LeakyReLU: f(u) = u for u > 0, 0.01 u
 *                    otherwise (the usual default slope; the paper gives
 *                    none).  GELU: the exact form 0.5 u (1 + erf(u / sqrt 2)).
 *
 * The backward pass is the chain rule applied to the definitions above; the
 * paper trains with autograd and never writes it out.  For a scalar loss
 * L = sum_t sum_o y[t][o] * dy[t][o]:
 *
 *     dc      = dy W_up^T
 *     du2     = -sin(u2) * dc
 *     dphi2   = sum_t du2          domega2 = sum_t du2 * b
 *     db      = omega2 * du2
 *     dM      = sum_t a^T db       (dM[i][j] = sum_t a_i db_j)
 *     da      = db M^T             (da_i = sum_j db_j M[i][j])
 *     du1     = -sin(u1) * da
 *     dphi1   = sum_t du1          domega1 = sum_t du1 * h
 *     dh      = omega1 * du1
 *     dx      = dy W^T + dh W_down^T
 *     dW      = x^T dy     dbias = sum_t dy
 *     dW_up   = c^T dy     dW_down = x^T dh
 *
 * With another activation f (no frequency or phase) the same chain reads
 * du2 = f'(b) dc, db = du2, du1 = f'(h) da, dh = du1 (two layers) or
 * dh = f'(h) dc (one layer).
 *
 * Every sum runs over its index in ascending order.  Rows (tokens) are
 * independent in the forward pass, so the only parallelism is over tokens for
 * per-token outputs and over output rows for weight gradients; neither changes
 * the order of any individual sum.
 *
 * Parity status: pinned (see the oracle tests): W_up = 0 reduction, identity
 * collapse, linear-limit CosNet with random frequencies (fixes the orientation
 * of M and where each omega/phi enters), closed-form cosine values,
 * 2*pi periodicity in the phases, token permutation, and central finite
 * differences for every gradient.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_COSNET 0
#define ORACLE_IDENTITY 1
#define ORACLE_COS1 2
#define ORACLE_TANH1 3
#define ORACLE_TANH2 4
#define ORACLE_LEAKY1 5
#define ORACLE_LEAKY2 6
#define ORACLE_GELU1 7
#define ORACLE_GELU2 8

#define ACT_COS 0
#define ACT_ID 1
#define ACT_TANH 2
#define ACT_LEAKY 3
#define ACT_GELU 4

static int mode_act(int mode)
{
    switch (mode) {
    case ORACLE_IDENTITY: return ACT_ID;
    case ORACLE_TANH1: case ORACLE_TANH2: return ACT_TANH;
    case ORACLE_LEAKY1: case ORACLE_LEAKY2: return ACT_LEAKY;
    case ORACLE_GELU1: case ORACLE_GELU2: return ACT_GELU;
    default: return ACT_COS;
    }
}

/* 2 when sigma has the mixing matrix M (two activation layers), else 1 */
static int mode_layers(int mode)
{
    return (mode == ORACLE_COSNET || mode == ORACLE_TANH2 || mode == ORACLE_LEAKY2 ||
            mode == ORACLE_GELU2) ? 2 : 1;
}

/* activation without frequency or phase, and its derivative */
static double act_f(int act, double u)
{
    switch (act) {
    case ACT_TANH: return tanh(u);
    case ACT_LEAKY: return u > 0.0 ? u : 0.01 * u;
    case ACT_GELU: return 0.5 * u * (1.0 + erf(u / sqrt(2.0)));
    default: return u;
    }
}
static double act_df(int act, double u)
{
    switch (act) {
    case ACT_TANH: { double t = tanh(u); return 1.0 - t * t; }
    case ACT_LEAKY: return u > 0.0 ? 1.0 : 0.01;
    case ACT_GELU:
        return 0.5 * (1.0 + erf(u / sqrt(2.0))) + u * exp(-0.5 * u * u) / sqrt(2.0 * acos(-1.0));
    default: return 1.0;
    }
}

/* sigma for one token, Eq. 2 / Eqs. 5-7.  Writes a, b, c (each [r]).  In the
 * one-layer modes b is set equal to a (there is no M).                       */
static void sigma_token(int mode, int64_t r, const double *h,
                        const double *om1, const double *ph1, const double *M,
                        const double *om2, const double *ph2,
                        double *a, double *b, double *c)
{
    int64_t i, j;
    const int act = mode_act(mode);
    for (i = 0; i < r; ++i) a[i] = act == ACT_COS ? cos(om1[i] * h[i] + ph1[i]) : act_f(act, h[i]);
    if (mode_layers(mode) == 1) {
        for (i = 0; i < r; ++i) { b[i] = a[i]; c[i] = a[i]; }
        return;
    }
    for (j = 0; j < r; ++j) {
        double s = 0.0;
        for (i = 0; i < r; ++i) s += a[i] * M[i * r + j];
        b[j] = s;
    }
    for (j = 0; j < r; ++j) c[j] = act == ACT_COS ? cos(om2[j] * b[j] + ph2[j]) : act_f(act, b[j]);
}

/*
 * Forward pass, Eq. 1 with sigma from Eq. 2.
 * x [T][d_in]; W [d_in][d_out]; bias [d_out] or NULL; W_down [d_in][r];
 * om1, ph1, om2, ph2 [r]; M [r][r]; W_up [r][d_out].
 * Outputs: y [T][d_out]; h, b, c [T][r] each (any may be NULL).
 * r == 0 gives the plain layer x W + bias.
 */
void oracle_fwd(int mode, int64_t T, int64_t d_in, int64_t d_out, int64_t r,
                const double *x, const double *W, const double *bias,
                const double *W_down, const double *om1, const double *ph1,
                const double *M, const double *om2, const double *ph2,
                const double *W_up, double *y, double *h_out, double *b_out,
                double *c_out)
{
    int64_t t;
#pragma omp parallel for schedule(static)
    for (t = 0; t < T; ++t) {
        const double *xt = x + t * d_in;
        double *h = NULL, *a = NULL, *b = NULL, *c = NULL;
        int64_t i, k, o;
        if (r > 0) {
            h = (double *)malloc(sizeof(double) * 4 * r);
            a = h + r; b = a + r; c = b + r;
            /* h = x W_down */
            for (k = 0; k < r; ++k) {
                double s = 0.0;
                for (i = 0; i < d_in; ++i) s += xt[i] * W_down[i * r + k];
                h[k] = s;
            }
            sigma_token(mode, r, h, om1, ph1, M, om2, ph2, a, b, c);
            if (h_out) memcpy(h_out + t * r, h, sizeof(double) * r);
            if (b_out) memcpy(b_out + t * r, b, sizeof(double) * r);
            if (c_out) memcpy(c_out + t * r, c, sizeof(double) * r);
        }
        /* y = x W + bias + c W_up, each term summed in ascending index order */
        for (o = 0; o < d_out; ++o) {
            double s = 0.0, br = 0.0;
            for (i = 0; i < d_in; ++i) s += xt[i] * W[i * d_out + o];
            if (bias) s = s + bias[o];
            for (k = 0; k < r; ++k) br += c[k] * W_up[k * d_out + o];
            y[t * d_out + o] = s + br;
        }
        free(h);
    }
}

/*
 * Backward pass for L = sum(y * dy): the chain rule through Eq. 1 and Eq. 2,
 * recomputing the forward intermediates from the inputs.
 *
 * Outputs (each may be NULL to skip it):
 *   dx [T][d_in], dW [d_in][d_out], dbias [d_out], dW_down [d_in][r],
 *   dM [r][r], dom1/dph1/dom2/dph2 [r], dW_up [r][d_out].
 * Optional intermediates for sampled checks (each may be NULL), all [T][r]:
 *   c_out (= sigma(h)), a_out, db_out, dh_out.
 * In the modes other than CosNet the gradients of parameters that the mode
 * does not use are written as zero.
 */
void oracle_bwd(int mode, int64_t T, int64_t d_in, int64_t d_out, int64_t r,
                const double *x, const double *W, const double *W_down,
                const double *om1, const double *ph1, const double *M,
                const double *om2, const double *ph2, const double *W_up,
                const double *dy, double *dx, double *dW, double *dbias,
                double *dW_down, double *dM, double *dom1, double *dph1,
                double *dom2, double *dph2, double *dW_up, double *c_out,
                double *a_out, double *db_out, double *dh_out)
{
    /* per-token intermediates, [T][r] each */
    size_t n = (size_t)T * (size_t)(r > 0 ? r : 1);
    double *H = (double *)calloc(n, sizeof(double));
    double *U1 = (double *)calloc(n, sizeof(double));
    double *A = (double *)calloc(n, sizeof(double));
    double *B = (double *)calloc(n, sizeof(double));
    double *C = (double *)calloc(n, sizeof(double));
    double *DU1 = (double *)calloc(n, sizeof(double));
    double *DU2 = (double *)calloc(n, sizeof(double));
    double *DB = (double *)calloc(n, sizeof(double));
    double *DH = (double *)calloc(n, sizeof(double));
    int64_t t, i, j, k, o;
    const int act = mode_act(mode);

    if (r > 0) {
#pragma omp parallel for schedule(static) private(i, j, k, o)
        for (t = 0; t < T; ++t) {
            const double *xt = x + t * d_in;
            const double *dyt = dy + t * d_out;
            double *h = H + t * r, *u1 = U1 + t * r, *a = A + t * r;
            double *b = B + t * r, *c = C + t * r;
            double *du1 = DU1 + t * r, *du2 = DU2 + t * r;
            double *db = DB + t * r, *dh = DH + t * r;
            double *dc = (double *)malloc(sizeof(double) * 2 * r);
            double *da = dc + r;
            /* forward intermediates */
            for (k = 0; k < r; ++k) {
                double s = 0.0;
                for (i = 0; i < d_in; ++i) s += xt[i] * W_down[i * r + k];
                h[k] = s;
            }
            sigma_token(mode, r, h, om1, ph1, M, om2, ph2, a, b, c);
            for (k = 0; k < r; ++k) u1[k] = (om1 && act == ACT_COS) ? om1[k] * h[k] + ph1[k] : 0.0;
            /* dc = dy W_up^T */
            for (k = 0; k < r; ++k) {
                double s = 0.0;
                for (o = 0; o < d_out; ++o) s += dyt[o] * W_up[k * d_out + o];
                dc[k] = s;
            }
            if (act != ACT_COS && mode_layers(mode) == 1) {
                /* sigma(h) = f(h): dh = f'(h) dc (identity: dh = dc) */
                for (k = 0; k < r; ++k) dh[k] = act_df(act, h[k]) * dc[k];
            } else if (act != ACT_COS) {
                /* sigma(h) = f(f(h) M) */
                for (j = 0; j < r; ++j) {
                    du2[j] = act_df(act, b[j]) * dc[j];
                    db[j] = du2[j];
                }
                for (i = 0; i < r; ++i) {
                    double s = 0.0;
                    for (j = 0; j < r; ++j) s += db[j] * M[i * r + j];
                    da[i] = s;
                }
                for (i = 0; i < r; ++i) {
                    du1[i] = act_df(act, h[i]) * da[i];
                    dh[i] = du1[i];
                }
            } else if (mode == ORACLE_COS1) {
                /* c = cos(u1): du1 = -sin(u1) dc, dh = omega1 du1 */
                for (k = 0; k < r; ++k) {
                    du1[k] = -sin(u1[k]) * dc[k];
                    dh[k] = om1[k] * du1[k];
                }
            } else {
                for (j = 0; j < r; ++j) {
                    double u2 = om2[j] * b[j] + ph2[j];
                    du2[j] = -sin(u2) * dc[j];
                    db[j] = om2[j] * du2[j];
                }
                for (i = 0; i < r; ++i) {
                    double s = 0.0;
                    for (j = 0; j < r; ++j) s += db[j] * M[i * r + j];
                    da[i] = s;
                }
                for (i = 0; i < r; ++i) {
                    du1[i] = -sin(u1[i]) * da[i];
                    dh[i] = om1[i] * du1[i];
                }
            }
            free(dc);
        }
    }

    /* dx = dy W^T + dh W_down^T */
    if (dx) {
#pragma omp parallel for schedule(static) private(i, k, o)
        for (t = 0; t < T; ++t) {
            for (i = 0; i < d_in; ++i) {
                double s = 0.0, sb = 0.0;
                for (o = 0; o < d_out; ++o) s += dy[t * d_out + o] * W[i * d_out + o];
                for (k = 0; k < r; ++k) sb += DH[t * r + k] * W_down[i * r + k];
                dx[t * d_in + i] = s + sb;
            }
        }
    }
    /* dW = x^T dy: dW[i][o] = sum_t x[t][i] dy[t][o] */
    if (dW) {
#pragma omp parallel for schedule(static) private(t, o)
        for (i = 0; i < d_in; ++i) {
            double *row = dW + i * d_out;
            for (o = 0; o < d_out; ++o) row[o] = 0.0;
            for (t = 0; t < T; ++t) {
                double xv = x[t * d_in + i];
                const double *dyt = dy + t * d_out;
                for (o = 0; o < d_out; ++o) row[o] += xv * dyt[o];
            }
        }
    }
    if (dbias) {
        for (o = 0; o < d_out; ++o) dbias[o] = 0.0;
        for (t = 0; t < T; ++t)
            for (o = 0; o < d_out; ++o) dbias[o] += dy[t * d_out + o];
    }
    /* dW_up = c^T dy */
    if (dW_up && r > 0) {
#pragma omp parallel for schedule(static) private(t, o)
        for (k = 0; k < r; ++k) {
            double *row = dW_up + k * d_out;
            for (o = 0; o < d_out; ++o) row[o] = 0.0;
            for (t = 0; t < T; ++t) {
                double cv = C[t * r + k];
                const double *dyt = dy + t * d_out;
                for (o = 0; o < d_out; ++o) row[o] += cv * dyt[o];
            }
        }
    }
    /* dW_down = x^T dh */
    if (dW_down && r > 0) {
#pragma omp parallel for schedule(static) private(t, k)
        for (i = 0; i < d_in; ++i) {
            double *row = dW_down + i * r;
            for (k = 0; k < r; ++k) row[k] = 0.0;
            for (t = 0; t < T; ++t) {
                double xv = x[t * d_in + i];
                for (k = 0; k < r; ++k) row[k] += xv * DH[t * r + k];
            }
        }
    }
    /* dM = a^T db (zero when the mode has no M) */
    if (dM && r > 0) {
        for (i = 0; i < r * r; ++i) dM[i] = 0.0;
        if (mode_layers(mode) == 2)
            for (t = 0; t < T; ++t)
                for (i = 0; i < r; ++i)
                    for (j = 0; j < r; ++j)
                        dM[i * r + j] += A[t * r + i] * DB[t * r + j];
    }
    /* frequency and phase gradients: sums over tokens */
    if (r > 0) {
        for (k = 0; k < r; ++k) {
            double so1 = 0.0, sp1 = 0.0, so2 = 0.0, sp2 = 0.0;
            if (act == ACT_COS) {
                for (t = 0; t < T; ++t) {
                    so1 += DU1[t * r + k] * H[t * r + k];
                    sp1 += DU1[t * r + k];
                }
            }
            if (mode == ORACLE_COSNET) {
                for (t = 0; t < T; ++t) {
                    so2 += DU2[t * r + k] * B[t * r + k];
                    sp2 += DU2[t * r + k];
                }
            }
            if (dom1) dom1[k] = so1;
            if (dph1) dph1[k] = sp1;
            if (dom2) dom2[k] = so2;
            if (dph2) dph2[k] = sp2;
        }
        if (c_out) memcpy(c_out, C, sizeof(double) * n);
        if (a_out) memcpy(a_out, A, sizeof(double) * n);
        if (db_out) memcpy(db_out, DB, sizeof(double) * n);
        if (dh_out) memcpy(dh_out, DH, sizeof(double) * n);
    }
    free(H); free(U1); free(A); free(B); free(C);
    free(DU1); free(DU2); free(DB); free(DH);
}

/*
 * Three-layer cosine bottleneck, the deepest row of the ablation in
 * Section 4.4 (Table 5): CosNet with a second mixing matrix and a third
 * cosine,
 *     a  = cos(omega1 h + phi1),  b  = a M,
 *     a2 = cos(omega2 b + phi2),  b2 = a2 M2,
 *     c  = cos(omega3 b2 + phi3),  y = x W + bias + c W_up,
 * M2 [r][r] with b2_j = sum_i a2_i M2[i][j], omega3 and phi3 [r].  The
 * backward continues the chain rule of oracle_bwd one layer further:
 *     du3 = -sin(u3) dc,  domega3 = sum_t du3 b2,  dphi3 = sum_t du3,
 *     db2 = omega3 du3,   dM2 = sum_t a2^T db2,   da2 = db2 M2^T,
 *     du2 = -sin(u2) da2, domega2 = sum_t du2 b,   dphi2 = sum_t du2,
 *     db  = omega2 du2,   dM = sum_t a^T db,       da = db M^T,
 *     du1 = -sin(u1) da,  domega1 = sum_t du1 h,   dphi1 = sum_t du1,
 *     dh  = omega1 du1,   and dx, dW, dbias, dW_up, dW_down as in oracle_bwd.
 * Kept apart from oracle_fwd / oracle_bwd (extra parameters); sums run in
 * ascending order.  Any output pointer may be NULL.
 */
static void cos3_token(int64_t r, const double *h, const double *om1, const double *ph1,
                       const double *M, const double *om2, const double *ph2, const double *M2,
                       const double *om3, const double *ph3, double *a, double *b, double *a2,
                       double *b2, double *c)
{
    int64_t i, j;
    for (i = 0; i < r; ++i) a[i] = cos(om1[i] * h[i] + ph1[i]);
    for (j = 0; j < r; ++j) {
        double s = 0.0;
        for (i = 0; i < r; ++i) s += a[i] * M[i * r + j];
        b[j] = s;
    }
    for (i = 0; i < r; ++i) a2[i] = cos(om2[i] * b[i] + ph2[i]);
    for (j = 0; j < r; ++j) {
        double s = 0.0;
        for (i = 0; i < r; ++i) s += a2[i] * M2[i * r + j];
        b2[j] = s;
    }
    for (j = 0; j < r; ++j) c[j] = cos(om3[j] * b2[j] + ph3[j]);
}

void oracle_fwd3(int64_t T, int64_t d_in, int64_t d_out, int64_t r, const double *x, const double *W,
                 const double *bias, const double *W_down, const double *om1, const double *ph1,
                 const double *M, const double *om2, const double *ph2, const double *M2,
                 const double *om3, const double *ph3, const double *W_up, double *y, double *h_out,
                 double *b_out, double *b2_out, double *c_out)
{
    int64_t t;
#pragma omp parallel for schedule(static)
    for (t = 0; t < T; ++t) {
        const double *xt = x + t * d_in;
        double *h = (double *)malloc(sizeof(double) * 6 * r);
        double *a = h + r, *b = a + r, *a2 = b + r, *b2 = a2 + r, *c = b2 + r;
        int64_t i, k, o;
        for (k = 0; k < r; ++k) {
            double s = 0.0;
            for (i = 0; i < d_in; ++i) s += xt[i] * W_down[i * r + k];
            h[k] = s;
        }
        cos3_token(r, h, om1, ph1, M, om2, ph2, M2, om3, ph3, a, b, a2, b2, c);
        if (h_out) memcpy(h_out + t * r, h, sizeof(double) * r);
        if (b_out) memcpy(b_out + t * r, b, sizeof(double) * r);
        if (b2_out) memcpy(b2_out + t * r, b2, sizeof(double) * r);
        if (c_out) memcpy(c_out + t * r, c, sizeof(double) * r);
        for (o = 0; o < d_out; ++o) {
            double s = 0.0, br = 0.0;
            for (i = 0; i < d_in; ++i) s += xt[i] * W[i * d_out + o];
            if (bias) s = s + bias[o];
            for (k = 0; k < r; ++k) br += c[k] * W_up[k * d_out + o];
            y[t * d_out + o] = s + br;
        }
        free(h);
    }
}

void oracle_bwd3(int64_t T, int64_t d_in, int64_t d_out, int64_t r, const double *x, const double *W,
                 const double *W_down, const double *om1, const double *ph1, const double *M,
                 const double *om2, const double *ph2, const double *M2, const double *om3,
                 const double *ph3, const double *W_up, const double *dy, double *dx, double *dW,
                 double *dbias, double *dW_down, double *dM, double *dom1, double *dph1, double *dom2,
                 double *dph2, double *dM2, double *dom3, double *dph3, double *dW_up)
{
    const size_t n = (size_t)T * (size_t)r;
    /* per-token intermediates [T][r] */
    double *H = (double *)calloc(n, sizeof(double)), *A = (double *)calloc(n, sizeof(double));
    double *B = (double *)calloc(n, sizeof(double)), *A2 = (double *)calloc(n, sizeof(double));
    double *B2 = (double *)calloc(n, sizeof(double)), *C = (double *)calloc(n, sizeof(double));
    double *DU1 = (double *)calloc(n, sizeof(double)), *DU2 = (double *)calloc(n, sizeof(double));
    double *DU3 = (double *)calloc(n, sizeof(double)), *DB = (double *)calloc(n, sizeof(double));
    double *DB2 = (double *)calloc(n, sizeof(double)), *DH = (double *)calloc(n, sizeof(double));
    int64_t t, i, j, k, o;
#pragma omp parallel for schedule(static) private(i, j, k, o)
    for (t = 0; t < T; ++t) {
        const double *xt = x + t * d_in, *dyt = dy + t * d_out;
        double *h = H + t * r, *a = A + t * r, *b = B + t * r, *a2 = A2 + t * r, *b2 = B2 + t * r;
        double *c = C + t * r, *du1 = DU1 + t * r, *du2 = DU2 + t * r, *du3 = DU3 + t * r;
        double *db = DB + t * r, *db2 = DB2 + t * r, *dh = DH + t * r;
        double *dc = (double *)malloc(sizeof(double) * 3 * r);
        double *da2 = dc + r, *da = da2 + r;
        for (k = 0; k < r; ++k) {
            double s = 0.0;
            for (i = 0; i < d_in; ++i) s += xt[i] * W_down[i * r + k];
            h[k] = s;
        }
        cos3_token(r, h, om1, ph1, M, om2, ph2, M2, om3, ph3, a, b, a2, b2, c);
        for (k = 0; k < r; ++k) {
            double s = 0.0;
            for (o = 0; o < d_out; ++o) s += dyt[o] * W_up[k * d_out + o];
            dc[k] = s;
        }
        for (j = 0; j < r; ++j) {
            du3[j] = -sin(om3[j] * b2[j] + ph3[j]) * dc[j];
            db2[j] = om3[j] * du3[j];
        }
        for (i = 0; i < r; ++i) {
            double s = 0.0;
            for (j = 0; j < r; ++j) s += db2[j] * M2[i * r + j];
            da2[i] = s;
        }
        for (j = 0; j < r; ++j) {
            du2[j] = -sin(om2[j] * b[j] + ph2[j]) * da2[j];
            db[j] = om2[j] * du2[j];
        }
        for (i = 0; i < r; ++i) {
            double s = 0.0;
            for (j = 0; j < r; ++j) s += db[j] * M[i * r + j];
            da[i] = s;
        }
        for (i = 0; i < r; ++i) {
            du1[i] = -sin(om1[i] * h[i] + ph1[i]) * da[i];
            dh[i] = om1[i] * du1[i];
        }
        free(dc);
    }
    if (dx) {
#pragma omp parallel for schedule(static) private(i, k, o)
        for (t = 0; t < T; ++t)
            for (i = 0; i < d_in; ++i) {
                double s = 0.0, sb = 0.0;
                for (o = 0; o < d_out; ++o) s += dy[t * d_out + o] * W[i * d_out + o];
                for (k = 0; k < r; ++k) sb += DH[t * r + k] * W_down[i * r + k];
                dx[t * d_in + i] = s + sb;
            }
    }
    if (dW) {
#pragma omp parallel for schedule(static) private(t, o)
        for (i = 0; i < d_in; ++i) {
            double *row = dW + i * d_out;
            for (o = 0; o < d_out; ++o) row[o] = 0.0;
            for (t = 0; t < T; ++t)
                for (o = 0; o < d_out; ++o) row[o] += x[t * d_in + i] * dy[t * d_out + o];
        }
    }
    if (dbias) {
        for (o = 0; o < d_out; ++o) dbias[o] = 0.0;
        for (t = 0; t < T; ++t)
            for (o = 0; o < d_out; ++o) dbias[o] += dy[t * d_out + o];
    }
    if (dW_up) {
#pragma omp parallel for schedule(static) private(t, o)
        for (k = 0; k < r; ++k) {
            double *row = dW_up + k * d_out;
            for (o = 0; o < d_out; ++o) row[o] = 0.0;
            for (t = 0; t < T; ++t)
                for (o = 0; o < d_out; ++o) row[o] += C[t * r + k] * dy[t * d_out + o];
        }
    }
    if (dW_down) {
#pragma omp parallel for schedule(static) private(t, k)
        for (i = 0; i < d_in; ++i) {
            double *row = dW_down + i * r;
            for (k = 0; k < r; ++k) row[k] = 0.0;
            for (t = 0; t < T; ++t)
                for (k = 0; k < r; ++k) row[k] += x[t * d_in + i] * DH[t * r + k];
        }
    }
    /* dM = a^T db, dM2 = a2^T db2 */
    for (i = 0; i < r * r; ++i) {
        if (dM) dM[i] = 0.0;
        if (dM2) dM2[i] = 0.0;
    }
    for (t = 0; t < T; ++t)
        for (i = 0; i < r; ++i)
            for (j = 0; j < r; ++j) {
                if (dM) dM[i * r + j] += A[t * r + i] * DB[t * r + j];
                if (dM2) dM2[i * r + j] += A2[t * r + i] * DB2[t * r + j];
            }
    for (k = 0; k < r; ++k) {
        double s[6] = {0.0, 0.0, 0.0, 0.0, 0.0, 0.0};
        for (t = 0; t < T; ++t) {
            s[0] += DU1[t * r + k] * H[t * r + k];
            s[1] += DU1[t * r + k];
            s[2] += DU2[t * r + k] * B[t * r + k];
            s[3] += DU2[t * r + k];
            s[4] += DU3[t * r + k] * B2[t * r + k];
            s[5] += DU3[t * r + k];
        }
        if (dom1) dom1[k] = s[0];
        if (dph1) dph1[k] = s[1];
        if (dom2) dom2[k] = s[2];
        if (dph2) dph2[k] = s[3];
        if (dom3) dom3[k] = s[4];
        if (dph3) dph3[k] = s[5];
    }
    free(H); free(A); free(B); free(A2); free(B2); free(C);
    free(DU1); free(DU2); free(DU3); free(DB); free(DB2); free(DH);
}

/*
 * Selected elements of a token-summed outer product:
 *     out[p] = sum_t P[t][rows[p]] * Q[t][cols[p]]     (ascending t)
 * P is [T][p_ld], Q is [T][q_ld].  This is the definition of one element of a
 * weight gradient (x^T dy, c^T dy, x^T dh, a^T db), used to check sampled
 * elements of large gradients without forming all of them.
 */
void oracle_outer_elems(int64_t T, const double *P, int64_t p_ld,
                        const double *Q, int64_t q_ld, int64_t n,
                        const int64_t *rows, const int64_t *cols, double *out)
{
    int64_t p;
#pragma omp parallel for schedule(static)
    for (p = 0; p < n; ++p) {
        double s = 0.0;
        int64_t t;
        for (t = 0; t < T; ++t) s += P[t * p_ld + rows[p]] * Q[t * q_ld + cols[p]];
        out[p] = s;
    }
}
