/*
 * noble.h -- C ABI of the NOBLE linear layer with the CosNet branch on GB300.
 *
 * The layer (NOBLE, arXiv 2603.06492, Eq. 1 in Section 3.1) is
 *
 *     y = x W^T + bias + sigma(x W_down^T) W_up^T
 *
 * written here with nn.Linear-style "out x in" weight storage, where the paper
 * writes the same thing with row vectors as x W + b + sigma(x W_down) W_up.
 * sigma is CosNet (Eq. 2 in Section 3.2; Eqs. 5-7 in Appendix A), applied per
 * token to h = x W_down^T in R^r:
 *
 *     a = cos(omega1 * h + phi1)           elementwise, learnable omega1, phi1
 *     b = a M          b_j = sum_i a_i M[i][j]
 *     c = cos(omega2 * b + phi2)           elementwise, learnable omega2, phi2
 *     sigma(h) = c
 *
 * Eq. 2 writes M . cos(...) for a column vector; this library reads it with
 * row vectors as b = a M, i.e. M[i][j] couples input channel i to output
 * channel j.  The backward pass is the chain rule through these definitions
 * (the paper trains with autograd and does not write it out).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Every pointer argument is a DEVICE pointer on the current CUDA device,
 *    except `desc`, which is a host pointer read during the call only.
 *  - The caller owns and allocates every buffer; no entry point allocates or
 *    frees device memory.  Cached TMA descriptors live in host memory.
 *  - All tensors are dense, row-major and contiguous:
 *        x [T][d_in]      y, dy [T][d_out]      dx [T][d_in]
 *        W [d_out][d_in]  W_down [r][d_in]      W_up [d_out][r]
 *        M [r][r]         omega1, phi1, omega2, phi2 [r]   bias [d_out]
 *  - Operand dtype (x, W, W_down, W_up, y, dy, dx) is desc->dtype: bf16 or
 *    fp32.  omega, phi, M, bias and every parameter gradient are always fp32.
 *    bf16 operands use tensor cores with fp32 accumulation; fp32 operands use
 *    exact fp32 FMA (no TF32), a validation mode.
 *  - Calls are asynchronous on `stream` (a cudaStream_t; NULL = legacy
 *    default stream).  Outputs are overwritten, never accumulated into.
 *  - Arguments are checked on the host before anything is enqueued.  On an
 *    argument error the call returns a status other than NOBLE_OK, enqueues
 *    nothing and leaves every output untouched; noble_last_error() then
 *    describes it.  NOBLE_ERR_CUDA from a failed launch part-way leaves the
 *    outputs undefined.
 *  - Requirements: T >= 0; d_in, d_out >= 8 and multiples of 8;
 *    r in {0, 16, 32, 64, 128, 256} (r = 0 is the plain layer, and the branch
 *    pointers may then be NULL); every pointer 16-byte aligned.  With T == 0
 *    the per-token pointers (x, y, dy, dx) and `saved` may be NULL; the
 *    forward pass then does nothing and the backward pass writes zero
 *    gradients.
 *  - Kernels never wait without a bound.  A wait that runs out records
 *    NOBLE_ERR_TIMEOUT in a device status word, which
 *    noble_get_device_status() reports.
 */
#ifndef NOBLE_H
#define NOBLE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st *noble_stream; /* same type as cudaStream_t */

typedef enum {
    NOBLE_OK = 0,
    NOBLE_ERR_INVALID_ARG = 1,     /* NULL pointer, negative or bad size      */
    NOBLE_ERR_MISALIGNED = 2,      /* a pointer is not 16-byte aligned         */
    NOBLE_ERR_UNSUPPORTED = 3,     /* r, d_in, d_out or dtype not supported    */
    NOBLE_ERR_BUFFER_TOO_SMALL = 4,/* saved / workspace size below the query   */
    NOBLE_ERR_CUDA = 5,            /* a CUDA runtime or driver call failed     */
    NOBLE_ERR_TIMEOUT = 6,         /* a device-side bounded wait expired       */
    NOBLE_ERR_NO_DEVICE = 7        /* no usable sm_103 device is current       */
} noble_status;

typedef enum { NOBLE_BF16 = 0, NOBLE_FP32 = 1 } noble_dtype;

/* desc->flags bits */
#define NOBLE_FLAG_SIMT_ONLY 1u /* bf16: run every step on CUDA cores (fp32
                                   FMA), not tensor cores; a second path for
                                   cross-checking the tensor-core kernels */
#define NOBLE_FLAG_INFERENCE 2u /* forward only, for inference (the branch
                                   stays in the model at inference, the
                                   Limitations section): on the
                                   tensor-core path h and b are not written
                                   and `saved` holds only c, the second K
                                   segment of the output GEMM (and the ready
                                   flags of a fused launch).  The backward
                                   entry points reject such a descriptor
                                   (NOBLE_ERR_INVALID_ARG).  The CUDA-core
                                   paths (fp32, SIMT_ONLY) use the full saved
                                   layout as scratch. */
#define NOBLE_FLAG_SIGMA_COS1 4u /* bottleneck sigma(h) = cos(omega1 h + phi1),
                                    the single-cosine activation of the
                                    ablation (Section 4.4, Table 5); M,
                                    omega2, phi2 are not used (may be NULL)
                                    and dM, domega2, dphi2 are written as 0 */
#define NOBLE_FLAG_SIGMA_IDENTITY 8u /* bottleneck sigma(h) = h, the linear
                                    collapse to x (W + W_down W_up)
                                    (Sections 1 and 3.1); omega, phi and M are
                                    not used (may be NULL) and their
                                    gradients are written as 0.  Not together
                                    with NOBLE_FLAG_SIGMA_COS1. */
/* The other activations f of the ablation (Section 4.4, Table 5), a 2-bit
 * field: sigma(h) = f(f(h) M) (two layers around the mixing matrix), or with
 * NOBLE_FLAG_SIGMA_SINGLE sigma(h) = f(h).  tanh; LeakyReLU f(u) = u for
 * u > 0, 0.01 u otherwise (the paper gives no slope; 0.01 is the common
 * default); GELU in its exact form u/2 (1 + erf(u / sqrt 2)).  The paper
 * gives frequencies and phases to the cosine only: omega1, phi1, omega2, phi2
 * are not used (may be NULL) and their gradients are written as 0; dM is
 * written as 0 for one layer.  Not together with NOBLE_FLAG_SIGMA_IDENTITY. */
#define NOBLE_FLAG_ACT_TANH 32u
#define NOBLE_FLAG_ACT_LEAKYRELU 64u
#define NOBLE_FLAG_ACT_GELU 96u
#define NOBLE_FLAG_ACT_MASK 96u
/* one activation layer, no mixing matrix: with the cosine (no ACT bits) the
 * same as NOBLE_FLAG_SIGMA_COS1 */
#define NOBLE_FLAG_SIGMA_SINGLE NOBLE_FLAG_SIGMA_COS1
/* The three-layer cosine of the ablation (Section 4.4, Table 5): CosNet with a
 * second mixing matrix and a third cosine,
 *     a2 = cos(omega2 b + phi2), b2 = a2 M2, c = cos(omega3 b2 + phi3),
 * b2_j = sum_i a2_i M2[i][j].  It has parameters the other variants lack, so
 * only noble_linear_fwd_cos3 / noble_linear_bwd_cos3 accept it (and they
 * accept nothing else); saved holds h, b, b2 (fp32) and c.  Not together with
 * another NOBLE_FLAG_SIGMA_* or NOBLE_FLAG_ACT_* bit. */
#define NOBLE_FLAG_SIGMA_COS3 128u
#define NOBLE_FLAG_FUSED_BRANCH 16u /* tensor-core path, CosNet bottleneck,
                                    r in {64, 128}: run the r-wide GEMM and
                                    the CosNet (forward h = x W_down^T and
                                    Eq. 2; backward dc = dy W_up and its chain
                                    rule) as tiles of the output GEMM launch
                                    (y, dx) instead of kernels of their own;
                                    the backward then sums dbias as dy^T 1 in
                                    the weight-gradient launch.  Same results
                                    up to summation order.  Off by default:
                                    slower than the separate kernels at the
                                    measured shapes.  Other shapes and
                                    variants always run separately. */

typedef struct {
    int64_t T;      /* tokens (rows of x)                          */
    int64_t d_in;   /* input features                              */
    int64_t d_out;  /* output features                             */
    int64_t r;      /* bottleneck rank; 0 = plain linear layer     */
    int32_t dtype;  /* noble_dtype of the operands                 */
    uint32_t flags; /* NOBLE_FLAG_* bits; 0 = default              */
} noble_linear_desc;

/*
 * Bytes of the saved-activation buffer that noble_linear_fwd writes and
 * noble_linear_bwd reads (per token: h and b in fp32, c in the operand dtype;
 * only c with NOBLE_FLAG_INFERENCE on the tensor-core path), plus, when the
 * forward runs the bottleneck inside the output GEMM (NOBLE_FLAG_FUSED_BRANCH
 * on the tensor-core path, CosNet, r in {64, 128}), one 32-bit ready flag per
 * 128 tokens that the forward resets itself.  0 when r == 0.
 * Returns 0 for an invalid descriptor as well; the entry points then report
 * why.
 */
size_t noble_linear_saved_bytes(const noble_linear_desc *desc);

/*
 * Bytes of scratch memory noble_linear_bwd needs (dh in the operand dtype,
 * dc and db in fp32, and fixed-size per-block partial sums for dM, domega
 * and dphi).  Nonzero for every valid descriptor.
 */
size_t noble_linear_bwd_workspace_bytes(const noble_linear_desc *desc);

/*
 * Forward pass, Eq. 1 with sigma = CosNet (Eq. 2; Eqs. 5-7).
 *   In : x, W, bias (NULL = no bias), W_down, omega1, phi1, M, omega2,
 *        phi2, W_up.
 *   Out: y [T][d_out] (operand dtype);
 *        saved: `saved_bytes` >= noble_linear_saved_bytes(desc) bytes,
 *        opaque, to be passed unchanged to noble_linear_bwd (may be NULL
 *        when r == 0).  A smaller size returns NOBLE_ERR_BUFFER_TOO_SMALL.
 */
noble_status noble_linear_fwd(const noble_linear_desc *desc,
                              const void *x, const void *W, const float *bias,
                              const void *W_down, const float *omega1,
                              const float *phi1, const float *M,
                              const float *omega2, const float *phi2,
                              const void *W_up, void *y, void *saved,
                              size_t saved_bytes, noble_stream stream);

/*
 * Backward pass: gradients of L = sum(y * dy) by the chain rule through Eq. 1
 * and Eq. 2.
 *   In : dy [T][d_out] (operand dtype), the forward inputs, and `saved` as
 *        written by noble_linear_fwd with the same desc and parameters.
 *   Out: dx [T][d_in] (operand dtype);
 *        dW [d_out][d_in], dbias [d_out] (NULL = skip), dW_down [r][d_in],
 *        dM [r][r], domega1, dphi1, domega2, dphi2 [r], dW_up [d_out][r],
 *        all fp32 (branch gradients may be NULL when r == 0).
 *   workspace: `workspace_bytes` >= noble_linear_bwd_workspace_bytes(desc)
 *        bytes of device scratch, contents undefined on entry and exit.
 *        Smaller saved or workspace sizes return NOBLE_ERR_BUFFER_TOO_SMALL.
 * The fp32 reductions over tokens (dM, domega, dphi, dbias) run in a fixed
 * order, so repeated calls give bit-identical results.
 */
noble_status noble_linear_bwd(const noble_linear_desc *desc, const void *dy,
                              const void *x, const void *W,
                              const void *W_down, const float *omega1,
                              const float *phi1, const float *M,
                              const float *omega2, const float *phi2,
                              const void *W_up, const void *saved,
                              size_t saved_bytes, void *dx,
                              float *dW, float *dbias, float *dW_down,
                              float *dM, float *domega1, float *dphi1,
                              float *domega2, float *dphi2, float *dW_up,
                              void *workspace, size_t workspace_bytes,
                              noble_stream stream);

/*
 * Optimizer step: AdamW with decoupled weight decay (the optimizer of the
 * paper's training runs, Section 4.1: beta1 0.9, beta2 0.98, weight decay
 * 0.01) over a batch of parameter tensors, each with its own learning rate,
 * in one fused pass per 16 tensors.  For step t >= 1, elementwise with the
 * tensor's learning rate a = lr * lr_mult:
 *     p <- p - a * weight_decay * p             (only if `decay`)
 *     m <- beta1 m + (1 - beta1) g,   v <- beta2 v + (1 - beta2) g^2
 *     p <- p - a / (1 - beta1^t) * m / (sqrt(v) / sqrt(1 - beta2^t) + eps)
 * All arrays are device memory, fp32, `n` elements, updated in place (g is
 * read only).  `param_bf16` (optional) receives the new values rounded to
 * bf16, e.g. the operand copy of W, W_down or W_up the layer's kernels read.
 * Pointers must be 16-byte aligned (param_bf16 8-byte aligned).
 * Errors: NOBLE_ERR_INVALID_ARG for NULL pointers, n < 0, t < 1 or bad
 * hyperparameters; NOBLE_ERR_MISALIGNED.  Nothing is enqueued on error.
 */
typedef struct {
    float *param;
    void *param_bf16; /* optional */
    const float *grad;
    float *exp_avg;
    float *exp_avg_sq;
    int64_t n;
    float lr_mult;
    int32_t decay; /* 1: apply weight decay to this tensor */
} noble_adamw_tensor;

typedef struct {
    float lr, beta1, beta2, eps, weight_decay;
    int64_t step; /* t, counted from 1 */
} noble_adamw_hparams;

noble_status noble_adamw_step(const noble_adamw_tensor *tensors, int n_tensors,
                              const noble_adamw_hparams *hp, noble_stream stream);

/*
 * NOBLE's per-group learning-rate multipliers (Section 3.3 and the defaults of
 * Appendix A), with rho = min(d_in, d_out) / r:
 *   out[0] W, bias, W_down: 1      out[1] W_up: rho^(2 gamma)
 *   out[2] M: rho^gamma_M          out[3] omega1, omega2: omega_mult
 *   out[4] phi1, phi2: phi_mult
 * Paper defaults: gamma 0.3, gamma_M 0.45, omega_mult 3, phi_mult 5.
 * Host only.  NOBLE_ERR_INVALID_ARG for r == 0 or a NULL pointer.
 */
noble_status noble_linear_lr_multipliers(const noble_linear_desc *desc, float gamma, float gamma_M,
                                         float omega_mult, float phi_mult, float out[5]);

/*
 * Gradient bucket for data-parallel training (the paper trains on 8 GPUs
 * with data parallelism, Section 4.1.1).  Tokens are split across ranks; the
 * forward needs no exchange, and every parameter gradient is a sum over
 * tokens, so the one exchange of a step is an all-reduce (sum) of the
 * parameter gradients.  This describes one flat fp32 buffer holding all of a
 * layer's parameter gradients, so that noble_linear_bwd writes straight into
 * it (pass bucket + offset[i] as the i-th gradient pointer) and one
 * collective per layer reduces them.
 *
 * Order of the slots (index: gradient, element count):
 *   0 dW [d_out][d_in]   1 dbias [d_out]    2 dW_down [r][d_in]
 *   3 dW_up [d_out][r]   4 dM [r][r]        5 domega1 [r]   6 dphi1 [r]
 *   7 domega2 [r]        8 dphi2 [r]
 *   9 dM2 [r][r]  10 domega3 [r]  11 dphi3 [r]  (NOBLE_FLAG_SIGMA_COS3 only)
 * offset[i] is the byte offset of slot i from the start of the bucket, a
 * multiple of NOBLE_GRAD_ALIGN; count[i] its element count (0 for a slot the
 * descriptor does not have: the branch slots when r == 0, the three-layer
 * slots without NOBLE_FLAG_SIGMA_COS3).  total_bytes is the bucket size, a
 * multiple of NOBLE_GRAD_ALIGN.  Padding between slots is never written.
 * Host only; no CUDA call.  NOBLE_ERR_INVALID_ARG for NULL pointers or an
 * invalid descriptor.
 */
#define NOBLE_GRAD_COUNT 12
#define NOBLE_GRAD_ALIGN 256u
typedef struct {
    size_t offset[NOBLE_GRAD_COUNT];
    size_t count[NOBLE_GRAD_COUNT];
    size_t total_bytes;
} noble_grad_bucket;

noble_status noble_linear_grad_bucket(const noble_linear_desc *desc, noble_grad_bucket *out);

/*
 * Backward pass without a caller workspace, for callers that cannot allocate
 * device memory: code that runs inside a host framework or plugin which owns
 * every device allocation and hands its extensions no allocator, or a
 * real-time loop that forbids allocation once it has started.  The paper has
 * no counterpart; this is an interface convenience.
 *
 * Same arguments, results and errors as noble_linear_bwd, minus `workspace`
 * and `workspace_bytes`: the scratch is a static device array inside the
 * library, NOBLE_NOALLOC_SCRATCH_BYTES (64 MiB) long, which every GPU that
 * loads the library holds until the process exits.  No cudaMalloc, cudaFree
 * or other allocating call is made.
 *  - A shape whose noble_linear_bwd_workspace_bytes() exceeds that size is
 *    rejected with NOBLE_ERR_BUFFER_TOO_SMALL before anything is enqueued.
 *  - The first call in a CUDA context looks up the array's device address
 *    (with that device current) and caches it for that context, so a device
 *    reset, which gives a new context, is followed by a new lookup; make the
 *    first call in a context before any stream capture.
 *  - Every call on a device shares the one array, and it keeps the last
 *    call's contents.  Nothing in it needs to start at zero: each call writes
 *    every scratch value before reading it.  Calls whose work overlaps on the
 *    GPU (other streams, other host threads) race on the array and give wrong
 *    results; the caller must order them, e.g. on a single stream.
 */
#define NOBLE_NOALLOC_SCRATCH_BYTES (64u << 20)
/*
 * Three-layer cosine bottleneck (NOBLE_FLAG_SIGMA_COS3): the extra parameters
 * M2 [r][r], omega3, phi3 [r] (fp32, device) and their gradients.  All are
 * required (not NULL) when r > 0.
 */
typedef struct {
    const float *M2;
    const float *omega3;
    const float *phi3;
} noble_cos3_params;
typedef struct {
    float *dM2;
    float *domega3;
    float *dphi3;
} noble_cos3_grads;

/* noble_linear_fwd for a NOBLE_FLAG_SIGMA_COS3 descriptor; the other
 * arguments as there.  Errors as noble_linear_fwd, and NOBLE_ERR_INVALID_ARG
 * for a descriptor without the flag. */
noble_status noble_linear_fwd_cos3(const noble_linear_desc *desc, const void *x,
                                   const void *W, const float *bias,
                                   const void *W_down, const float *omega1,
                                   const float *phi1, const float *M,
                                   const float *omega2, const float *phi2,
                                   const noble_cos3_params *p3, const void *W_up,
                                   void *y, void *saved, size_t saved_bytes,
                                   noble_stream stream);

/* noble_linear_bwd for a NOBLE_FLAG_SIGMA_COS3 descriptor, also writing
 * g3->dM2 = sum_t a2^T db2, g3->domega3, g3->dphi3 (overwritten).  The
 * workspace size is noble_linear_bwd_workspace_bytes of the same descriptor. */
noble_status noble_linear_bwd_cos3(const noble_linear_desc *desc, const void *dy,
                                   const void *x, const void *W,
                                   const void *W_down, const float *omega1,
                                   const float *phi1, const float *M,
                                   const float *omega2, const float *phi2,
                                   const noble_cos3_params *p3, const void *W_up,
                                   const void *saved, size_t saved_bytes, void *dx,
                                   float *dW, float *dbias, float *dW_down,
                                   float *dM, float *domega1, float *dphi1,
                                   float *domega2, float *dphi2,
                                   const noble_cos3_grads *g3, float *dW_up,
                                   void *workspace, size_t workspace_bytes,
                                   noble_stream stream);

noble_status noble_linear_bwd_noalloc(const noble_linear_desc *desc,
                                      const void *dy, const void *x,
                                      const void *W, const void *W_down,
                                      const float *omega1, const float *phi1,
                                      const float *M, const float *omega2,
                                      const float *phi2, const void *W_up,
                                      const void *saved, size_t saved_bytes,
                                      void *dx, float *dW, float *dbias,
                                      float *dW_down, float *dM,
                                      float *domega1, float *dphi1,
                                      float *domega2, float *dphi2,
                                      float *dW_up, noble_stream stream);

/*
 * Synchronises `stream`, then reads and clears the device status word of the
 * current device.  NOBLE_ERR_TIMEOUT if any kernel gave up a bounded wait
 * since the last call, NOBLE_ERR_CUDA if the stream reported an error,
 * NOBLE_OK otherwise.
 */
noble_status noble_get_device_status(noble_stream stream);

/* Static description of a status code. */
const char *noble_status_string(noble_status s);

/* Description of the last error returned on the calling thread ("" if none). */
const char *noble_last_error(void);

/* Number of kernels this library has launched in the process so far. */
uint64_t noble_kernel_launch_count(void);

/*
 * Test hook: ORs `bits` into the current device's status word (synchronous),
 * so that the reporting path of a device-side timeout can be exercised
 * without making any kernel wait.
 */
noble_status noble_debug_raise_device_status(uint32_t bits);

/*
 * Test hook (no paper counterpart): launches on `stream` one small kernel that
 * waits, through the bounded mbarrier wait every pipeline kernel of this
 * library uses, on an mbarrier that nothing arrives at, for `limit_ns`
 * nanoseconds (0 < limit_ns <= 100 ms).  Nothing else is outstanding in that
 * kernel (no copy, no MMA), so the wait expires: the kernel ORs the timeout
 * flag into the device status word, writes 2 to the device word `*result`
 * (1 if the wait had completed) and exits.  A following
 * noble_get_device_status() then returns NOBLE_ERR_TIMEOUT, and the context
 * stays usable.  NOBLE_ERR_INVALID_ARG for a NULL `result` or a limit out of
 * range.
 */
noble_status noble_debug_wait_expiry(uint64_t limit_ns, uint32_t *result, noble_stream stream);

/*
 * Testing hook (no paper counterpart): the library's tensor-core GEMM alone,
 *     C[z][m][n] = sum_k A0(m,k) B0(n,k) + sum_k A1(m,k) B1(n,k) (+ bias[n])
 * with bf16 operands and fp32 accumulation.  A_s is row-major [M][K_s]
 * (a_mn = 0) or [K_s][M] (a_mn = 1); B_s is [N][K_s] (b_mn = 0) or [K_s][N]
 * (b_mn = 1).  bn selects the N tile (16..256; only the combinations the
 * layer uses exist).  C is fp32 (c_fp32 = 1) or bf16, row-major [M][N] per
 * split; with nsplit > 1 split z sums k-blocks [z*kb_per_split,
 * (z+1)*kb_per_split) of 64 and writes C + z*M*N.  M, N, K_s multiples of 8.
 */
noble_status noble_test_gemm_bf16(int64_t M, int64_t N, int64_t K0, int64_t K1,
                                  int a_mn, int b_mn, int bn, const void *A0,
                                  const void *B0, const void *A1,
                                  const void *B1, const float *bias, void *C,
                                  int c_fp32, int kb_per_split, int nsplit,
                                  noble_stream stream);

/*
 * Instrumentation (no paper counterpart).  When enabled, every kernel the
 * library launches is bracketed by two CUDA events on its own stream and
 * attributed to a kernel class together with its algorithmic FLOPs and DRAM
 * bytes.  noble_profile_count() waits for the recorded events, aggregates
 * them and returns the number of classes; noble_profile_entry() reads class
 * i of that snapshot (bound: 0 tensor pipe, 1 HBM, 2 CUDA-core ALU).
 */
void noble_profile_enable(int on);
void noble_profile_reset(void);
int noble_profile_count(void);
noble_status noble_profile_entry(int i, char *name, size_t name_len,
                                 uint64_t *launches, double *ms,
                                 double *flops, double *bytes, int *bound);

#ifdef __cplusplus
}
#endif

#endif /* NOBLE_H */
