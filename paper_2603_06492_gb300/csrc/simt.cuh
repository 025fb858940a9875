// CUDA-core (SIMT) kernels: exact fp32 FMA, no tensor cores.
//
// These carry the fp32 validation mode end to end and every piece of the bf16
// path that has no tensor-core kernel yet.  Every reduction over tokens is
// split into fixed chunks whose partial results are summed in chunk order,
// so results are deterministic.
#pragma once

#include "activations.cuh"

namespace noble {
namespace simt {

// Element (row, k) of an operand lives at p[row * ld_row + k * ld_k].
struct Operand {
    const void *p;
    int64_t ld_row, ld_k;
};
struct Seg {
    Operand A, B;
    int64_t K;
};

constexpr int kBM = 64, kBN = 64, kBK = 16, kThreads = 256;

// C[m][n] = sum_seg sum_k A(m,k) B(n,k) (+ bias[n]), fp32 accumulation.
// With k_chunk > 0 (single segment only) block z sums k in
// [z*k_chunk, (z+1)*k_chunk) and writes to C + z*c_chunk_stride.
template <typename TIn, typename TOut>
__global__ void __launch_bounds__(kThreads)
gemm_kernel(int64_t M, int64_t N, Seg s0, Seg s1, int nseg, const float *bias, TOut *C,
            int64_t ldc, int64_t k_chunk, int64_t c_chunk_stride)
{
    __shared__ float As[kBK][kBM + 1];
    __shared__ float Bs[kBK][kBN + 1];
    const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
    const int64_t m0 = (int64_t)blockIdx.y * kBM, n0 = (int64_t)blockIdx.x * kBN;
    const int64_t z = blockIdx.z;
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

    for (int s = 0; s < nseg; ++s) {
        const Seg &sg = s ? s1 : s0;
        int64_t kb = 0, ke = sg.K;
        if (k_chunk > 0) {
            kb = z * k_chunk;
            ke = min(sg.K, kb + k_chunk);
        }
        const TIn *A = (const TIn *)sg.A.p;
        const TIn *B = (const TIn *)sg.B.p;
        const bool a_kc = sg.A.ld_k == 1, b_kc = sg.B.ld_k == 1;
        for (int64_t k0 = kb; k0 < ke; k0 += kBK) {
#pragma unroll
            for (int i = 0; i < (kBM * kBK) / kThreads; ++i) {
                const int l = tid + i * kThreads;
                int mm, kk;
                if (a_kc) { mm = l / kBK; kk = l % kBK; } else { mm = l % kBM; kk = l / kBM; }
                const int64_t gm = m0 + mm, gk = k0 + kk;
                float v = 0.f;
                if (gm < M && gk < ke) v = Elem<TIn>::load(A + gm * sg.A.ld_row + gk * sg.A.ld_k);
                As[kk][mm] = v;
                int nn;
                if (b_kc) { nn = l / kBK; kk = l % kBK; } else { nn = l % kBN; kk = l / kBN; }
                const int64_t gn = n0 + nn, gk2 = k0 + kk;
                float w = 0.f;
                if (gn < N && gk2 < ke) w = Elem<TIn>::load(B + gn * sg.B.ld_row + gk2 * sg.B.ld_k);
                Bs[kk][nn] = w;
            }
            __syncthreads();
#pragma unroll
            for (int kk = 0; kk < kBK; ++kk) {
                float a[4], b[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
                for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx * 4 + j];
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
            }
            __syncthreads();
        }
    }
    TOut *Cz = C + z * c_chunk_stride;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int64_t gm = m0 + ty * 4 + i;
        if (gm >= M) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int64_t gn = n0 + tx * 4 + j;
            if (gn >= N) continue;
            float v = acc[i][j];
            if (bias) v += bias[gn];
            Elem<TOut>::store(Cz + gm * ldc + gn, v);
        }
    }
}

// CosNet forward on rows (Eq. 2): from h [T][r] (fp32) computes
//   a = cos(omega1 h + phi1), b = a M, c = cos(omega2 b + phi2)
// and writes b (fp32) and c (TOut), each [T][r].  Block: tokens_per_block rows.
// With act != act::kCos the two-layer variant of the ablation (Section 4.4):
// a = f(h), b = a M, c = f(b) (activations.cuh).
template <typename TOut>
__global__ void __launch_bounds__(256)
cosnet_fwd_rows(int64_t T, int r, int act, int tokens_per_block, const float *h, const float *om1,
                const float *ph1, const float *M, const float *om2, const float *ph2,
                float *b_out, TOut *c_out)
{
    extern __shared__ float a_s[];  // [tokens_per_block][r]
    const int64_t t0 = (int64_t)blockIdx.x * tokens_per_block;
    const int n = tokens_per_block * r;
    for (int idx = threadIdx.x; idx < n; idx += blockDim.x) {
        const int tt = idx / r, i = idx % r;
        const int64_t t = t0 + tt;
        if (t >= T)
            a_s[idx] = 0.f;
        else
            a_s[idx] = act == act::kCos ? cosf(fmaf(om1[i], h[t * r + i], ph1[i])) : act::f(act, h[t * r + i]);
    }
    __syncthreads();
    for (int idx = threadIdx.x; idx < n; idx += blockDim.x) {
        const int tt = idx / r, j = idx % r;
        const int64_t t = t0 + tt;
        if (t >= T) continue;
        float s = 0.f;
        for (int i = 0; i < r; ++i) s = fmaf(a_s[tt * r + i], M[i * r + j], s);
        b_out[t * r + j] = s;
        Elem<TOut>::store(c_out + t * r + j, act == act::kCos ? cosf(fmaf(om2[j], s, ph2[j])) : act::f(act, s));
    }
}

// One-layer bottleneck on rows, the variants of the ablation (Section 4.4):
// c = cos(omega1 h + phi1) (act::kCos) or c = f(h) (identity, tanh,
// LeakyReLU, GELU; activations.cuh), elementwise over h [T][r] (n = T r).
template <typename TOut>
__global__ void __launch_bounds__(256)
sigma_fwd_rows(int64_t n, int r, int act, const float *h, const float *om1, const float *ph1, TOut *c_out)
{
    for (int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; idx < n; idx += (int64_t)gridDim.x * blockDim.x) {
        const int i = (int)(idx % r);
        const float v = h[idx];
        Elem<TOut>::store(c_out + idx, act == act::kCos ? cosf(fmaf(om1[i], v, ph1[i])) : act::f(act, v));
    }
}

// Backward of sigma_fwd_rows: cosine: du1 = -sin(omega1 h + phi1) dc,
// dh = omega1 du1; otherwise dh = f'(h) dc.  Per-block column sums over the
// block's tokens in ascending order: part[blk][0:r] = sum du1*h,
// [r:2r] = sum du1 (zero without a phase), [2r:4r] = 0 (no second layer).
template <typename TOut>
__global__ void __launch_bounds__(256)
sigma_bwd_rows(int64_t T, int r, int act, int tokens_per_block, const float *h, const float *dc,
               const float *om1, const float *ph1, TOut *dh_out, float *part)
{
    const int64_t t0 = (int64_t)blockIdx.x * tokens_per_block;
    const int64_t t1 = min(T, t0 + tokens_per_block);
    float *pb = part + (int64_t)blockIdx.x * 4 * r;
    for (int j = threadIdx.x; j < r; j += blockDim.x) {
        float so = 0.f, sp = 0.f;
        for (int64_t t = t0; t < t1; ++t) {
            const float d = dc[t * r + j];
            const float hv = h[t * r + j];
            if (act == act::kCos) {
                const float du1 = -sinf(fmaf(om1[j], hv, ph1[j])) * d;
                Elem<TOut>::store(dh_out + t * r + j, om1[j] * du1);
                so += du1 * hv;
                sp += du1;
            } else {
                Elem<TOut>::store(dh_out + t * r + j, act::df(act, hv) * d);
            }
        }
        pb[j] = so;
        pb[r + j] = sp;
        pb[2 * r + j] = 0.f;
        pb[3 * r + j] = 0.f;
    }
}

// CosNet backward on rows (chain rule through Eq. 2).  From saved h, b (fp32),
// dc = dy W_up (fp32) and Mt = M^T computes per token
//   du2 = -sin(u2) dc, db = omega2 du2, da = db M^T, du1 = -sin(u1) da,
//   dh = omega1 du1, a = cos(u1)
// writing dh (TOut), a and db (fp32) [T][r], and per-block column sums
//   part[blk][0:r] = sum du1*h, [r:2r] = sum du1, [2r:3r] = sum du2*b,
//   [3r:4r] = sum du2      (tokens of the block in ascending order).
// With act != act::kCos (two-layer variant f(f(h) M)): db = f'(b) dc,
// du1 = f'(h) da, dh = du1, a = f(h), and the sums are zero.
template <typename TOut>
__global__ void __launch_bounds__(256)
cosnet_bwd_rows(int64_t T, int r, int act, int tokens_per_block, const float *h, const float *b,
                const float *dc, const float *om1, const float *ph1, const float *Mt,
                const float *om2, const float *ph2, TOut *dh_out, float *a_out, float *db_out,
                float *part)
{
    const bool cosine = act == act::kCos;
    extern __shared__ float sm[];
    const int n = tokens_per_block * r;
    float *db_s = sm, *du2_s = sm + n, *p2_s = sm + 2 * n, *du1_s = sm + 3 * n, *p1_s = sm + 4 * n;
    const int64_t t0 = (int64_t)blockIdx.x * tokens_per_block;
    for (int idx = threadIdx.x; idx < n; idx += blockDim.x) {
        const int tt = idx / r, j = idx % r;
        const int64_t t = t0 + tt;
        float du2 = 0.f, bv = 0.f;
        if (t < T) {
            bv = b[t * r + j];
            du2 = (cosine ? -sinf(fmaf(om2[j], bv, ph2[j])) : act::df(act, bv)) * dc[t * r + j];
        }
        const float dbv = cosine ? om2[j] * du2 : du2;
        db_s[idx] = dbv;
        du2_s[idx] = cosine ? du2 : 0.f;
        p2_s[idx] = cosine ? du2 * bv : 0.f;
        if (t < T) db_out[t * r + j] = dbv;
    }
    __syncthreads();
    for (int idx = threadIdx.x; idx < n; idx += blockDim.x) {
        const int tt = idx / r, i = idx % r;
        const int64_t t = t0 + tt;
        float du1 = 0.f, hv = 0.f;
        if (t < T) {
            float da = 0.f;
            for (int j = 0; j < r; ++j) da = fmaf(db_s[tt * r + j], Mt[j * r + i], da);
            hv = h[t * r + i];
            if (cosine) {
                const float u1 = fmaf(om1[i], hv, ph1[i]);
                float s1, c1;
                sincosf(u1, &s1, &c1);
                du1 = -s1 * da;
                a_out[t * r + i] = c1;
                Elem<TOut>::store(dh_out + t * r + i, om1[i] * du1);
            } else {
                a_out[t * r + i] = act::f(act, hv);
                Elem<TOut>::store(dh_out + t * r + i, act::df(act, hv) * da);
            }
        }
        du1_s[idx] = du1;
        p1_s[idx] = du1 * hv;
    }
    __syncthreads();
    float *pb = part + (int64_t)blockIdx.x * 4 * r;
    for (int j = threadIdx.x; j < r; j += blockDim.x) {
        float so1 = 0.f, sp1 = 0.f, so2 = 0.f, sp2 = 0.f;
        for (int tt = 0; tt < tokens_per_block; ++tt) {
            so1 += p1_s[tt * r + j];
            sp1 += du1_s[tt * r + j];
            so2 += p2_s[tt * r + j];
            sp2 += du2_s[tt * r + j];
        }
        pb[j] = so1;
        pb[r + j] = sp1;
        pb[2 * r + j] = so2;
        pb[3 * r + j] = sp2;
    }
}

// Three-layer cosine (the deepest row of the ablation, Section 4.4, Table 5)
// on rows: from h [T][r] (fp32)
//   a = cos(omega1 h + phi1), b = a M, a2 = cos(omega2 b + phi2), b2 = a2 M2,
//   c = cos(omega3 b2 + phi3)
// writing b, b2 (fp32) and c (TOut), each [T][r].  Block: tokens_per_block
// rows; shared memory 2 tokens_per_block r floats.
template <typename TOut>
__global__ void __launch_bounds__(256)
cosnet3_fwd_rows(int64_t T, int r, int tokens_per_block, const float *h, const float *om1, const float *ph1,
                 const float *M, const float *om2, const float *ph2, const float *M2, const float *om3,
                 const float *ph3, float *b_out, float *b2_out, TOut *c_out)
{
    extern __shared__ float sm3[];
    const int n = tokens_per_block * r;
    float *a_s = sm3, *a2_s = sm3 + n;
    const int64_t t0 = (int64_t)blockIdx.x * tokens_per_block;
    for (int idx = threadIdx.x; idx < n; idx += blockDim.x) {
        const int tt = idx / r, i = idx % r;
        const int64_t t = t0 + tt;
        a_s[idx] = t < T ? cosf(fmaf(om1[i], h[t * r + i], ph1[i])) : 0.f;
    }
    __syncthreads();
    for (int idx = threadIdx.x; idx < n; idx += blockDim.x) {
        const int tt = idx / r, j = idx % r;
        const int64_t t = t0 + tt;
        float s = 0.f;
        for (int i = 0; i < r; ++i) s = fmaf(a_s[tt * r + i], M[i * r + j], s);
        a2_s[idx] = cosf(fmaf(om2[j], s, ph2[j]));
        if (t < T) b_out[t * r + j] = s;
    }
    __syncthreads();
    for (int idx = threadIdx.x; idx < n; idx += blockDim.x) {
        const int tt = idx / r, j = idx % r;
        const int64_t t = t0 + tt;
        if (t >= T) continue;
        float s = 0.f;
        for (int i = 0; i < r; ++i) s = fmaf(a2_s[tt * r + i], M2[i * r + j], s);
        b2_out[t * r + j] = s;
        Elem<TOut>::store(c_out + t * r + j, cosf(fmaf(om3[j], s, ph3[j])));
    }
}

// Backward of cosnet3_fwd_rows (chain rule through the three layers): from
// saved h, b, b2 (fp32) and dc = dy W_up (fp32)
//   du3 = -sin(u3) dc, db2 = omega3 du3, da2 = db2 M2^T,
//   du2 = -sin(u2) da2, db = omega2 du2, da = db M^T,
//   du1 = -sin(u1) da, dh = omega1 du1,  a = cos(u1), a2 = cos(u2)
// writing dh (TDh), a, db, a2, db2 (TAct), each [T][r], and per-block column
// sums over the block's tokens in ascending order, part[blk][q][r] with
// q = 0 sum du1*h, 1 sum du1, 2 sum du2*b, 3 sum du2, 4 sum du3*b2, 5 sum du3.
// Shared memory 8 tokens_per_block r floats.
template <typename TDh, typename TAct>
__global__ void __launch_bounds__(256)
cosnet3_bwd_rows(int64_t T, int r, int tokens_per_block, const float *h, const float *b, const float *b2,
                 const float *dc, const float *om1, const float *ph1, const float *M, const float *om2,
                 const float *ph2, const float *M2, const float *om3, const float *ph3, TDh *dh_out,
                 TAct *a_out, TAct *db_out, TAct *a2_out, TAct *db2_out, float *part)
{
    extern __shared__ float sm3[];
    const int n = tokens_per_block * r;
    float *db2_s = sm3, *db_s = sm3 + n;
    float *q_s = sm3 + 2 * n;  // six [tokens_per_block][r] arrays, in the order of part
    const int64_t t0 = (int64_t)blockIdx.x * tokens_per_block;
    for (int idx = threadIdx.x; idx < n; idx += blockDim.x) {
        const int tt = idx / r, j = idx % r;
        const int64_t t = t0 + tt;
        float du3 = 0.f, bv = 0.f;
        if (t < T) {
            bv = b2[t * r + j];
            du3 = -sinf(fmaf(om3[j], bv, ph3[j])) * dc[t * r + j];
        }
        db2_s[idx] = om3[j] * du3;
        q_s[4 * n + idx] = du3 * bv;
        q_s[5 * n + idx] = du3;
        if (t < T) Elem<TAct>::store(db2_out + t * r + j, om3[j] * du3);
    }
    __syncthreads();
    for (int idx = threadIdx.x; idx < n; idx += blockDim.x) {
        const int tt = idx / r, i = idx % r;
        const int64_t t = t0 + tt;
        float du2 = 0.f, bv = 0.f;
        if (t < T) {
            float da2 = 0.f;
            for (int j = 0; j < r; ++j) da2 = fmaf(db2_s[tt * r + j], M2[i * r + j], da2);
            bv = b[t * r + i];
            float s2, c2;
            sincosf(fmaf(om2[i], bv, ph2[i]), &s2, &c2);
            du2 = -s2 * da2;
            Elem<TAct>::store(a2_out + t * r + i, c2);
            Elem<TAct>::store(db_out + t * r + i, om2[i] * du2);
        }
        db_s[idx] = om2[i] * du2;
        q_s[2 * n + idx] = du2 * bv;
        q_s[3 * n + idx] = du2;
    }
    __syncthreads();
    for (int idx = threadIdx.x; idx < n; idx += blockDim.x) {
        const int tt = idx / r, i = idx % r;
        const int64_t t = t0 + tt;
        float du1 = 0.f, hv = 0.f;
        if (t < T) {
            float da = 0.f;
            for (int j = 0; j < r; ++j) da = fmaf(db_s[tt * r + j], M[i * r + j], da);
            hv = h[t * r + i];
            float s1, c1;
            sincosf(fmaf(om1[i], hv, ph1[i]), &s1, &c1);
            du1 = -s1 * da;
            Elem<TAct>::store(a_out + t * r + i, c1);
            Elem<TDh>::store(dh_out + t * r + i, om1[i] * du1);
        }
        q_s[idx] = du1 * hv;
        q_s[n + idx] = du1;
    }
    __syncthreads();
    float *pb = part + (int64_t)blockIdx.x * 6 * r;
    for (int k = threadIdx.x; k < 6 * r; k += blockDim.x) {
        const int q = k / r, j = k % r;
        float s = 0.f;
        for (int tt = 0; tt < tokens_per_block; ++tt) s += q_s[q * n + tt * r + j];
        pb[k] = s;
    }
}

// part[c][o] = sum over rows t in chunk c (ascending) of X[t][o].
template <typename TIn>
__global__ void colsum_partial(int64_t T, int64_t n, int64_t rows_per_chunk, const TIn *X,
                               float *part)
{
    const int64_t o = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (o >= n) return;
    const int64_t tb = (int64_t)blockIdx.y * rows_per_chunk;
    const int64_t te = min(T, tb + rows_per_chunk);
    float s = 0.f;
    for (int64_t t = tb; t < te; ++t) s += Elem<TIn>::load(X + t * n + o);
    part[(int64_t)blockIdx.y * n + o] = s;
}

// bf16 column sums, 8 columns (16 bytes) per thread and row: part[c][o] =
// sum over rows t in chunk c (ascending) of X[t][o].  n must be a multiple of 8.
__global__ void __launch_bounds__(256) colsum_partial_bf16x8(int64_t T, int64_t n, int64_t rows_per_chunk,
                                                             const __nv_bfloat16 *X, float *part)
{
    const int64_t o = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) * 8;
    if (o >= n) return;
    const int64_t tb = (int64_t)blockIdx.y * rows_per_chunk;
    const int64_t te = min(T, tb + rows_per_chunk);
    float s[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll 4
    for (int64_t t = tb; t < te; ++t) {
        const uint4 q = __ldg(reinterpret_cast<const uint4 *>(X + t * n + o));
        const __nv_bfloat162 *h = reinterpret_cast<const __nv_bfloat162 *>(&q);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 f = __bfloat1622float2(h[i]);
            s[2 * i] += f.x;
            s[2 * i + 1] += f.y;
        }
    }
    float4 *dst = reinterpret_cast<float4 *>(part + (int64_t)blockIdx.y * n + o);
    dst[0] = make_float4(s[0], s[1], s[2], s[3]);
    dst[1] = make_float4(s[4], s[5], s[6], s[7]);
}

// out[k / seg_len][k % seg_len] = sum_p part[p * n + k].
// Block = 8 warps over 32 columns; warp w sums parts [w*P/8, (w+1)*P/8) in
// ascending order, then the 8 warp sums are added in warp order, so the
// result does not depend on scheduling.
struct Outs4 {
    float *p[8];  // up to eight outputs of seg_len elements each
};
__global__ void __launch_bounds__(256) reduce_partials(int64_t nparts, int64_t n, int64_t seg_len,
                                                       const float *part, Outs4 outs)
{
    __shared__ float sm[8][33];
    const int lane = threadIdx.x % 32, w = threadIdx.x / 32;
    const int64_t k = (int64_t)blockIdx.x * 32 + lane;
    const int64_t per = (nparts + 7) / 8;
    const int64_t pb = w * per, pe = min(nparts, pb + per);
    float s = 0.f;
    if (k < n) {
        // eight loads in flight, then added in ascending p
        int64_t p = pb;
        for (; p + 8 <= pe; p += 8) {
            float v[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) v[u] = part[(p + u) * n + k];
#pragma unroll
            for (int u = 0; u < 8; ++u) s += v[u];
        }
        for (; p < pe; ++p) s += part[p * n + k];
    }
    sm[w][lane] = s;
    __syncthreads();
    if (w == 0 && k < n) {
        float t = 0.f;
#pragma unroll
        for (int i = 0; i < 8; ++i) t += sm[i][lane];
        float *dst = outs.p[k / seg_len];
        if (dst) dst[k % seg_len] = t;
    }
}

// Mt[j][i] = M[i][j]
__global__ void transpose_square(int r, const float *M, float *Mt)
{
    const int idx = blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= r * r) return;
    const int i = idx / r, j = idx % r;
    Mt[j * r + i] = M[i * r + j];
}

}  // namespace simt
}  // namespace noble
