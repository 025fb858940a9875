// C-ABI entry points of the NOBLE linear layer (declared in include/noble.h).
//
// Host side only: argument validation, buffer carving and kernel dispatch.
// Forward = Eq. 1 (Section 3.1) with CosNet (Eq. 2, Section 3.2; Eqs. 5-7,
// Appendix A); backward = the chain rule through the same definitions.
#include <algorithm>
#include <cmath>
#include <atomic>
#include <vector>
#include <mutex>
#include <initializer_list>
#include <type_traits>
#include <cstdarg>
#include <cstdio>
#include <cstring>

#include "../../include/noble.h"
#include "common.cuh"
#include "profile.cuh"
#include "simt.cuh"
#include "adamw.cuh"
#include "tc_gemm.cuh"
#include "tc_persistent.cuh"
#include "tc_cosnet.cuh"
#include "tc_pair.cuh"

namespace noble {

__device__ uint32_t g_device_status = 0;

// Library-owned scratch for noble_linear_bwd_noalloc (see include/noble.h).
// Every GPU that loads this library holds it until the process exits.
constexpr size_t kNoallocScratchBytes = (size_t)NOBLE_NOALLOC_SCRATCH_BYTES;
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocScratchBytes];

namespace {

thread_local char g_last_error[512] = "";
std::atomic<uint64_t> g_launches{0};

noble_status fail(noble_status s, const char *fmt, ...)
{
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_last_error, sizeof(g_last_error), fmt, ap);
    va_end(ap);
    return s;
}

noble_status check_launch(const char *what)
{
    g_launches.fetch_add(1, std::memory_order_relaxed);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return fail(NOBLE_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
    return NOBLE_OK;
}

// Kernels launched so far by the current entry-point call on this thread.
thread_local int g_call_kernels = 0;

// Launch through `f`, bracketed by profiling events when profiling is on.
template <class F>
noble_status run(cudaStream_t st, const KernelInfo &ki, F &&f)
{
    const int slot = Profiler::get().begin(st);
    f();
    Profiler::get().end(slot, st, ki);
    ++g_call_kernels;
    return check_launch(ki.name);
}

// Programmatic dependent launch: the pair GEMMs and the partial-sum
// reductions may start while the previous kernel of the same call still runs,
// on the SMs it leaves free; they wait for it (griddep_wait) before reading
// anything an earlier kernel of the call wrote, and every such grid waits at
// least once, so its completion implies its predecessors'.  The first kernel
// of a call, and the first after a memset, is launched normally and sees all
// prior work in the stream -- except the CosNet kernels, which wait for their
// predecessor grid in every thread before any global read, so that their
// set-up may overlap the previous kernel whatever it is.
constexpr bool kProgrammaticLaunch = true;
bool pdl_ok() { return kProgrammaticLaunch && g_call_kernels > 0; }

template <class... KArgs, class... Args>
void launch_maybe_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, bool pdl,
                      Args &&...args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr.val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = &attr;
    cfg.numAttrs = pdl ? 1 : 0;
    cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

// cudaMemsetAsync on the stream; the next kernel is then launched normally.
cudaError_t memset_async(void *p, int v, size_t n, cudaStream_t st)
{
    g_call_kernels = 0;
    return cudaMemsetAsync(p, v, n, st);
}

#define NOBLE_TRY(expr)                              \
    do {                                             \
        noble_status _s = (expr);                    \
        if (_s != NOBLE_OK) return _s;               \
    } while (0)

constexpr uint32_t kFlagSimtOnly = NOBLE_FLAG_SIMT_ONLY;
constexpr uint32_t kFlagInference = NOBLE_FLAG_INFERENCE;
constexpr uint32_t kFlagSigmaCos1 = NOBLE_FLAG_SIGMA_COS1;
constexpr uint32_t kFlagSigmaIdentity = NOBLE_FLAG_SIGMA_IDENTITY;
constexpr uint32_t kFlagFusedBranch = NOBLE_FLAG_FUSED_BRANCH;
constexpr uint32_t kFlagActMask = NOBLE_FLAG_ACT_MASK;
constexpr uint32_t kFlagSigmaCos3 = NOBLE_FLAG_SIGMA_COS3;

// Three-layer cosine (NOBLE_FLAG_SIGMA_COS3): its extra parameters and
// gradients, threaded through the forward and backward paths (NULL: not a
// three-layer descriptor).
struct Cos3 {
    const float *M2, *om3, *ph3;
    float *dM2, *dom3, *dph3;
};
bool is_cos3(const noble_linear_desc *d) { return (d->flags & kFlagSigmaCos3) != 0 && d->r > 0; }
bool use_tc(const noble_linear_desc *d);
// The three-layer cosine on the tensor-core path runs in the bottleneck
// kernel (both r x r products as tensor-core MMAs) for r <= 128; r = 256 keeps
// the CUDA-core rows (its mixing matrices do not fit shared memory at once).
bool cos3_tc(const noble_linear_desc *d) { return is_cos3(d) && use_tc(d) && d->r <= 128; }

// Bottleneck activation selected by the descriptor: CosNet (Eq. 2), or a
// variant of the ablation (Section 4.4, Table 5): single cosine, identity, or
// another activation with one or two layers (activations.cuh).
struct Sigma {
    int sig;  // tc::kSig*, the CosNet kernels' template parameter
    int act;  // act::k*: the activation of the kSigAct* variants
    bool two_layers() const { return tc::sig_two_layers(sig); }
    bool first_phase() const { return sig == tc::kSigCosnet || sig == tc::kSigCos1; }  // omega1, phi1
    bool second_phase() const { return sig == tc::kSigCosnet; }                         // omega2, phi2
};
Sigma sigma_of(const noble_linear_desc *d)
{
    if (d->flags & kFlagSigmaIdentity) return {tc::kSigIdentity, act::kIdentity};
    const uint32_t a = d->flags & kFlagActMask;
    const bool one = (d->flags & kFlagSigmaCos1) != 0;
    if (a == 0) return {one ? tc::kSigCos1 : tc::kSigCosnet, act::kCos};
    const int f = a == NOBLE_FLAG_ACT_TANH ? act::kTanh : a == NOBLE_FLAG_ACT_LEAKYRELU ? act::kLeaky : act::kGelu;
    return {one ? tc::kSigAct1 : tc::kSigAct2, f};
}

bool rank_supported(int64_t r) { return r == 0 || r == 16 || r == 32 || r == 64 || r == 128 || r == 256; }

noble_status validate_desc(const noble_linear_desc *d)
{
    if (!d) return fail(NOBLE_ERR_INVALID_ARG, "desc is NULL");
    if (d->T < 0 || d->d_in <= 0 || d->d_out <= 0 || d->r < 0)
        return fail(NOBLE_ERR_INVALID_ARG, "negative or zero size (T=%lld d_in=%lld d_out=%lld r=%lld)",
                    (long long)d->T, (long long)d->d_in, (long long)d->d_out, (long long)d->r);
    if (d->T > (int64_t)INT32_MAX || d->d_in > (1 << 20) || d->d_out > (1 << 20))
        return fail(NOBLE_ERR_UNSUPPORTED, "size too large (T <= 2^31-1, d_in/d_out <= 2^20)");
    if (d->d_in < 8 || d->d_out < 8 || d->d_in % 8 || d->d_out % 8)
        return fail(NOBLE_ERR_UNSUPPORTED, "d_in=%lld and d_out=%lld must be multiples of 8 and >= 8",
                    (long long)d->d_in, (long long)d->d_out);
    if (!rank_supported(d->r))
        return fail(NOBLE_ERR_UNSUPPORTED, "r=%lld not in {0,16,32,64,128,256}", (long long)d->r);
    if (d->dtype != NOBLE_BF16 && d->dtype != NOBLE_FP32)
        return fail(NOBLE_ERR_UNSUPPORTED, "dtype %d not supported", (int)d->dtype);
    if (d->flags &
        ~(kFlagSimtOnly | kFlagInference | kFlagSigmaCos1 | kFlagSigmaIdentity | kFlagFusedBranch | kFlagActMask |
          kFlagSigmaCos3))
        return fail(NOBLE_ERR_UNSUPPORTED, "unknown flags 0x%x", d->flags);
    if ((d->flags & kFlagSigmaCos3) && (d->flags & (kFlagSigmaCos1 | kFlagSigmaIdentity | kFlagActMask)))
        return fail(NOBLE_ERR_INVALID_ARG, "NOBLE_FLAG_SIGMA_COS3 with another bottleneck flag");
    if ((d->flags & kFlagSigmaCos1) && (d->flags & kFlagSigmaIdentity))
        return fail(NOBLE_ERR_INVALID_ARG, "NOBLE_FLAG_SIGMA_COS1 and NOBLE_FLAG_SIGMA_IDENTITY together");
    if ((d->flags & kFlagActMask) && (d->flags & kFlagSigmaIdentity))
        return fail(NOBLE_ERR_INVALID_ARG, "NOBLE_FLAG_ACT_* and NOBLE_FLAG_SIGMA_IDENTITY together");
    return NOBLE_OK;
}

noble_status check_ptr(const void *p, const char *name, bool nullable)
{
    if (!p) return nullable ? NOBLE_OK : fail(NOBLE_ERR_INVALID_ARG, "%s is NULL", name);
    if (reinterpret_cast<uintptr_t>(p) % 16) return fail(NOBLE_ERR_MISALIGNED, "%s is not 16-byte aligned", name);
    return NOBLE_OK;
}

noble_status check_device()
{
    static int cached[64];  // 0 unknown, 1 ok, 2 bad
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) {
        cudaGetLastError();
        return fail(NOBLE_ERR_NO_DEVICE, "no current CUDA device");
    }
    if (dev < 64 && cached[dev] == 1) return NOBLE_OK;
    int major = 0, minor = 0;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    cudaGetLastError();
    if (major != 10 || minor != 3) {
        if (dev < 64) cached[dev] = 2;
        return fail(NOBLE_ERR_NO_DEVICE, "device %d is sm_%d%d; this library is built for sm_103a", dev, major, minor);
    }
    if (dev < 64) cached[dev] = 1;
    return NOBLE_OK;
}

size_t esize(const noble_linear_desc *d) { return d->dtype == NOBLE_BF16 ? 2 : 4; }

// True when the bf16 tensor-core path runs (the default for bf16 operands).
bool use_tc(const noble_linear_desc *d) { return d->dtype == NOBLE_BF16 && !(d->flags & kFlagSimtOnly); }

// Tensor-core launches that run the bottleneck inside the output GEMM
// (tc_pair.cuh, FUSE), on request: the CosNet with r in {64, 128}, whose
// leader tiles hold the first r output columns (d_out >= r).  The backward's
// MN-major operands also need d_in a multiple of 64 (4-D TMA layout) and
// d_in >= r.
bool fuse_fwd(const noble_linear_desc *d)
{
    return use_tc(d) && sigma_of(d).sig == tc::kSigCosnet && !is_cos3(d) && (d->r == 64 || d->r == 128) && d->T > 0 &&
           d->d_out >= d->r && (d->flags & kFlagFusedBranch);
}
bool fuse_bwd(const noble_linear_desc *d)
{
    return use_tc(d) && sigma_of(d).sig == tc::kSigCosnet && !is_cos3(d) && (d->r == 64 || d->r == 128) && d->T > 0 &&
           d->d_in >= d->r && d->d_in % 64 == 0 && (d->flags & kFlagFusedBranch);
}
// Output columns of a fused launch after the leader's first r: nfull in
// 256-wide tiles, then a last part of at most 128 columns (if any) in
// 128-wide tiles, so that no tile multiplies more than 128 empty columns.
struct FusedSplit {
    int64_t nfull, ntail;
};
FusedSplit fused_split(int64_t n, int64_t r)
{
    const int64_t rest = n - r, rem = rest % 256;
    if (rem > 0 && rem <= 128) return {rest - rem, rem};
    return {rest, 0};
}
// ready flags of a fused launch: one per 128-row block of whole row pairs
size_t fuse_flag_bytes(const noble_linear_desc *d) { return (size_t)(2 * ((d->T + 255) / 256)) * 4; }

// Saved-activation buffer: h, b (fp32) and c (operand dtype), each [T][r];
// only c for an inference forward on the tensor-core path.
struct SavedLayout {
    size_t h, b, b2, c, flags, total;
    bool only_c;
};
SavedLayout saved_layout(const noble_linear_desc *d)
{
    SavedLayout L{};
    if (d->r == 0 || d->T == 0) return L;
    const size_t tr = (size_t)d->T * (size_t)d->r;
    if (is_cos3(d)) {
        // three-layer cosine: h, b, b2 (fp32) and c, also for inference
        L.h = 0;
        L.b = align_up(tr * 4, 256);
        L.b2 = align_up(L.b + tr * 4, 256);
        L.c = align_up(L.b2 + tr * 4, 256);
        L.total = align_up(L.c + tr * esize(d), 256);
        return L;
    }
    if ((d->flags & kFlagInference) && use_tc(d)) {
        L.only_c = true;
        L.c = 0;
        L.total = align_up(tr * esize(d), 256);
    } else {
        L.h = 0;
        L.b = align_up(L.h + tr * 4, 256);
        L.c = align_up(L.b + tr * 4, 256);
        L.total = align_up(L.c + tr * esize(d), 256);
    }
    if (fuse_fwd(d)) {
        L.flags = L.total;
        L.total = align_up(L.flags + fuse_flag_bytes(d), 256);
    }
    return L;
}

constexpr int64_t kDmChunk = 1024;     // tokens per dM partial (CUDA-core path)
constexpr int64_t kBiasChunk = 128;    // tokens per dbias partial (CUDA-core path)
constexpr int64_t kOnesCols = 64;      // width of the all-ones operand that yields dbias
int cosnet_tokens_per_block(int64_t r) { return (int)(2048 / r); }
int cos3_tokens_per_block(int64_t r) { return (int)(1024 / r); }  // 8 [tokens][r] fp32 arrays in shared memory

// K split of the grouped weight-gradient launch (tensor-core path).  When the
// launch has fewer than two waves of 256 x N tile pairs for a GB300 (74
// resident CTA pairs), K = T is cut into s chunks of at least 16 k-blocks;
// each chunk writes an fp32 partial and one reduction adds them in chunk
// order.  A function of the shape only, so buffer sizes do not depend on the
// device.
constexpr int kAssumedPairs = 74;
int wgrad_tiles(int64_t M, int64_t N, int bn) { return (int)(ceil_div(ceil_div(M, 128), 2) * ceil_div(N, bn)); }
int wgrad_split(const noble_linear_desc *d)
{
    const int64_t T = d->T, di = d->d_in, dout = d->d_out, r = d->r;
    const int rb = r < 128 ? 128 : (int)r;
    int tiles = wgrad_tiles(dout, di, 256) + wgrad_tiles(dout, kOnesCols, 128);
    if (r > 0) tiles += wgrad_tiles(r, di, 256) + wgrad_tiles(dout, r, rb) + wgrad_tiles(r, r, rb);
    if (is_cos3(d)) tiles += wgrad_tiles(r, r, rb);
    const int64_t kb = ceil_div(T, 64);
    int s = (int)ceil_div(2 * kAssumedPairs, tiles);
    if (s > kb / 16) s = (int)(kb / 16);
    return s < 1 ? 1 : s;
}
// Sizes of the token-summed products (M x N), in launch order: dW, dW_down,
// dW_up, dM, dbias, dM2 (three-layer cosine).
constexpr int kWgradKinds = 6;
void wgrad_shapes(const noble_linear_desc *d, int64_t (&mn)[kWgradKinds][2])
{
    const int64_t di = d->d_in, dout = d->d_out, r = d->r;
    const int64_t v[kWgradKinds][2] = {{dout, di}, {r, di}, {dout, r}, {r, r}, {dout, 1}, {r, r}};
    for (int i = 0; i < kWgradKinds; ++i) mn[i][0] = v[i][0], mn[i][1] = v[i][1];
}

// Backward scratch.
//   CUDA-core path: dh (dtype), dc, a, db (fp32) [T][r]; M^T fp32; per-block
//     partials of the CosNet sums, of dM and of dbias.
//   tensor-core path: dh, a, db (bf16) [T][r]; per-CTA CosNet and dbias
//     partials; without a branch, or with the bottleneck fused into the dx
//     launch, an all-ones [T][64] bf16 operand (dbias = dy^T 1); the fused
//     launch's CosNet partials per 32 tokens and its ready flags.
struct WorkLayout {
    size_t dh, dc, a, db, a2, db2, mt, ones, cos_part, dm_part, bias_part, flags, wsplit[kWgradKinds], total;
    int split;
    int64_t n_cos_blocks, n_dm_chunks, n_bias_chunks;
};
WorkLayout work_layout(const noble_linear_desc *d)
{
    WorkLayout L{};
    const int64_t T = d->T, r = d->r;
    const size_t tr = (size_t)T * (size_t)r;
    size_t off = 0;
    auto take = [&](size_t bytes) { size_t o = off; off = align_up(off + bytes, 256); return o; };
    L.dh = take(tr * esize(d));
    if (cos3_tc(d)) {
        // three-layer cosine in the bottleneck kernel: a, db, a2, db2 (bf16),
        // six column sums and the dbias partials per CTA (128-token tile)
        L.a = take(tr * 2);
        L.db = take(tr * 2);
        L.a2 = take(tr * 2);
        L.db2 = take(tr * 2);
        L.n_cos_blocks = ceil_div(T, 128);
        L.cos_part = take((size_t)L.n_cos_blocks * 6 * r * 4);
        L.bias_part = take((size_t)L.n_cos_blocks * d->d_out * 4);
        L.split = wgrad_split(d);
        if (L.split > 1) {
            int64_t mn[kWgradKinds][2];
            wgrad_shapes(d, mn);
            for (int i = 0; i < kWgradKinds; ++i) L.wsplit[i] = take((size_t)L.split * mn[i][0] * mn[i][1] * 4);
        }
    } else if (is_cos3(d)) {
        // three-layer cosine: dc (fp32) from a GEMM, the CUDA-core chain rule
        // writes a, db, a2, db2 (bf16 operands of the tensor-core weight
        // gradients, fp32 on the CUDA-core path) and partials per block
        const size_t act = use_tc(d) ? 2 : 4;
        L.dc = take(tr * 4);
        L.a = take(tr * act);
        L.db = take(tr * act);
        L.a2 = take(tr * act);
        L.db2 = take(tr * act);
        L.n_cos_blocks = ceil_div(T, cos3_tokens_per_block(r));
        L.cos_part = take((size_t)L.n_cos_blocks * 6 * r * 4);
        if (use_tc(d)) {
            L.ones = take((size_t)T * kOnesCols * 2);
            L.split = wgrad_split(d);
            if (L.split > 1) {
                int64_t mn[kWgradKinds][2];
                wgrad_shapes(d, mn);
                for (int i = 0; i < kWgradKinds; ++i) L.wsplit[i] = take((size_t)L.split * mn[i][0] * mn[i][1] * 4);
            }
        } else {
            L.n_dm_chunks = ceil_div(T, kDmChunk);
            L.dm_part = take((size_t)L.n_dm_chunks * r * r * 4);
            L.n_bias_chunks = ceil_div(T, kBiasChunk);
            L.bias_part = take((size_t)L.n_bias_chunks * d->d_out * 4);
        }
    } else if (use_tc(d)) {
        L.a = take(tr * 2);
        L.db = take(tr * 2);
        const bool fused = fuse_bwd(d);
        L.ones = r ? 0 : take((size_t)T * kOnesCols * 2);  // dbias = dy^T 1
        if (fused) {
            // CosNet sums per 32 tokens (an epilogue warp's rows), dbias
            // partials per 128 tokens (a CTA's rows of a leader tile)
            L.n_cos_blocks = ceil_div(T, 32);
            L.cos_part = take((size_t)L.n_cos_blocks * 4 * r * 4);
            L.flags = take(fuse_flag_bytes(d));
            L.n_bias_chunks = ceil_div(T, 128);
            L.bias_part = take((size_t)L.n_bias_chunks * d->d_out * 4);
        } else {
            // one partial per CTA (128-token tile) of the CosNet kernel
            L.n_cos_blocks = r ? ceil_div(T, 128) : 0;
            L.cos_part = take((size_t)L.n_cos_blocks * 4 * r * 4);
            // with a branch, dbias is summed from the dy tiles of the CosNet kernel
            L.bias_part = take((size_t)L.n_cos_blocks * d->d_out * 4);
        }
        L.split = wgrad_split(d);
        if (L.split > 1) {
            int64_t mn[kWgradKinds][2];
            wgrad_shapes(d, mn);
            for (int i = 0; i < 5; ++i) L.wsplit[i] = take((size_t)L.split * mn[i][0] * mn[i][1] * 4);
        }
    } else {
        L.dc = take(tr * 4);
        L.a = take(tr * 4);
        L.db = take(tr * 4);
        L.mt = take((size_t)r * r * 4);
        L.n_cos_blocks = r ? ceil_div(T, cosnet_tokens_per_block(r)) : 0;
        L.cos_part = take((size_t)L.n_cos_blocks * 4 * r * 4);
        L.n_dm_chunks = r ? ceil_div(T, kDmChunk) : 0;
        L.dm_part = take((size_t)L.n_dm_chunks * r * r * 4);
        L.n_bias_chunks = ceil_div(T, kBiasChunk);
        L.bias_part = take((size_t)L.n_bias_chunks * d->d_out * 4);
    }
    L.total = off < 256 ? 256 : off;
    return L;
}

// ------------------------------------------------------------ SIMT dispatch
template <typename TIn, typename TOut>
noble_status simt_gemm(cudaStream_t st, int64_t M, int64_t N, simt::Seg s0, const simt::Seg *s1,
                       const float *bias, TOut *C, int64_t ldc, int64_t k_chunk = 0,
                       int64_t n_chunks = 1, int64_t c_chunk_stride = 0)
{
    if (M == 0 || N == 0) return NOBLE_OK;
    dim3 grid((unsigned)ceil_div(N, simt::kBN), (unsigned)ceil_div(M, simt::kBM), (unsigned)n_chunks);
    simt::Seg empty{};
    const double K = (double)s0.K + (s1 ? (double)s1->K : 0.0);
    const KernelInfo ki{"simt_gemm", kBoundAlu, 2.0 * M * N * K, 0.0};
    return run(st, ki, [&] {
        simt::gemm_kernel<TIn, TOut><<<grid, simt::kThreads, 0, st>>>(
            M, N, s0, s1 ? *s1 : empty, s1 ? 2 : 1, bias, C, ldc, k_chunk, c_chunk_stride);
    });
}

noble_status reduce(cudaStream_t st, int64_t nparts, int64_t n, int64_t seg_len, const float *part,
                    float *o0, float *o1 = nullptr, float *o2 = nullptr, float *o3 = nullptr,
                    float *o4 = nullptr, float *o5 = nullptr)
{
    simt::Outs4 outs{{o0, o1, o2, o3, o4, o5, nullptr, nullptr}};
    const KernelInfo ki{"reduce_partials", kBoundHbm, (double)nparts * n, 4.0 * (nparts + 1) * n};
    return run(st, ki, [&] {
        simt::reduce_partials<<<(unsigned)ceil_div(n, 32), 256, 0, st>>>(nparts, n, seg_len, part, outs);
    });
}

// Three-layer cosine on the CUDA cores, from h (fp32) to b, b2 (saved) and c.
template <typename TOut>
noble_status cos3_fwd_rows(const noble_linear_desc *d, const float *h, const float *om1, const float *ph1,
                           const float *M, const float *om2, const float *ph2, const Cos3 *c3, char *saved,
                           TOut *c, cudaStream_t st)
{
    const int64_t T = d->T, r = d->r;
    const SavedLayout SL = saved_layout(d);
    float *b = (float *)(saved + SL.b), *b2 = (float *)(saved + SL.b2);
    const int tpb = cos3_tokens_per_block(r);
    const KernelInfo ki{"simt_cos3_fwd", kBoundAlu, 4.0 * T * r * r, 0.0};
    return run(st, ki, [&] {
        simt::cosnet3_fwd_rows<TOut><<<(unsigned)ceil_div(T, tpb), 256, 2 * tpb * r * sizeof(float), st>>>(
            T, (int)r, tpb, h, om1, ph1, M, om2, ph2, c3->M2, c3->om3, c3->ph3, b, b2, c);
    });
}

// Three-layer cosine backward on the CUDA cores: dh, a, db, a2, db2 and the
// six frequency/phase gradients (reduced from per-block partials).
template <typename TDh, typename TAct>
noble_status cos3_bwd_rows(const noble_linear_desc *d, const char *saved, const float *dc, const float *om1,
                           const float *ph1, const float *M, const float *om2, const float *ph2, const Cos3 *c3,
                           TDh *dh, TAct *a, TAct *db, TAct *a2, TAct *db2, float *cpart, float *dom1, float *dph1,
                           float *dom2, float *dph2, cudaStream_t st)
{
    const int64_t T = d->T, r = d->r;
    const SavedLayout SL = saved_layout(d);
    const WorkLayout WL = work_layout(d);
    const float *h = (const float *)(saved + SL.h), *b = (const float *)(saved + SL.b);
    const float *b2 = (const float *)(saved + SL.b2);
    const int tpb = cos3_tokens_per_block(r);
    const KernelInfo ki{"simt_cos3_bwd", kBoundAlu, 4.0 * T * r * r, 0.0};
    NOBLE_TRY(run(st, ki, [&] {
        simt::cosnet3_bwd_rows<TDh, TAct><<<(unsigned)WL.n_cos_blocks, 256, 8 * tpb * r * sizeof(float), st>>>(
            T, (int)r, tpb, h, b, b2, dc, om1, ph1, M, om2, ph2, c3->M2, c3->om3, c3->ph3, dh, a, db, a2, db2, cpart);
    }));
    return reduce(st, WL.n_cos_blocks, 6 * r, r, cpart, dom1, dph1, dom2, dph2, c3->dom3, c3->dph3);
}

template <typename TIn>
noble_status fwd_simt(const noble_linear_desc *d, const TIn *x, const TIn *W, const float *bias,
                      const TIn *W_down, const float *om1, const float *ph1, const float *M,
                      const float *om2, const float *ph2, const TIn *W_up, TIn *y, char *saved,
                      cudaStream_t st, const Cos3 *c3 = nullptr)
{
    const int64_t T = d->T, di = d->d_in, dout = d->d_out, r = d->r;
    const SavedLayout SL = saved_layout(d);
    float *h = (float *)(saved + SL.h), *b = (float *)(saved + SL.b);
    TIn *c = (TIn *)(saved + SL.c);
    simt::Seg main{{x, di, 1}, {W, di, 1}, di};
    if (r > 0) {
        simt::Seg down{{x, di, 1}, {W_down, di, 1}, di};
        NOBLE_TRY((simt_gemm<TIn, float>(st, T, r, down, nullptr, nullptr, h, r)));
        const int tpb = cosnet_tokens_per_block(r);
        const Sigma sg = sigma_of(d);
        if (c3) {
            NOBLE_TRY(cos3_fwd_rows<TIn>(d, h, om1, ph1, M, om2, ph2, c3, saved, c, st));
        } else if (sg.two_layers()) {
            const KernelInfo ki{"simt_cosnet_fwd", kBoundAlu, 2.0 * T * r * r, 0.0};
            NOBLE_TRY(run(st, ki, [&] {
                simt::cosnet_fwd_rows<TIn><<<(unsigned)ceil_div(T, tpb), 256, tpb * r * sizeof(float), st>>>(
                    T, (int)r, sg.act, tpb, h, om1, ph1, M, om2, ph2, b, c);
            }));
        } else {
            const KernelInfo ki{"simt_sigma_fwd", kBoundHbm, 0.0, (4.0 + sizeof(TIn)) * T * r};
            NOBLE_TRY(run(st, ki, [&] {
                simt::sigma_fwd_rows<TIn><<<(unsigned)std::min<int64_t>(ceil_div(T * r, 256), 4096), 256, 0, st>>>(
                    T * r, (int)r, sg.act, h, om1, ph1, c);
            }));
        }
        simt::Seg up{{c, r, 1}, {W_up, r, 1}, r};
        return simt_gemm<TIn, TIn>(st, T, dout, main, &up, bias, y, dout);
    }
    return simt_gemm<TIn, TIn>(st, T, dout, main, nullptr, bias, y, dout);
}

template <typename TIn>
noble_status bwd_simt(const noble_linear_desc *d, const TIn *dy, const TIn *x, const TIn *W,
                      const TIn *W_down, const float *om1, const float *ph1, const float *M,
                      const float *om2, const float *ph2, const TIn *W_up, const char *saved,
                      TIn *dx, float *dW, float *dbias, float *dW_down, float *dM, float *dom1,
                      float *dph1, float *dom2, float *dph2, float *dW_up, char *ws, cudaStream_t st,
                      const Cos3 *c3 = nullptr)
{
    const int64_t T = d->T, di = d->d_in, dout = d->d_out, r = d->r;
    const SavedLayout SL = saved_layout(d);
    const WorkLayout WL = work_layout(d);
    const float *h = (const float *)(saved + SL.h), *b = (const float *)(saved + SL.b);
    const TIn *c = (const TIn *)(saved + SL.c);
    TIn *dh = (TIn *)(ws + WL.dh);
    if (r > 0 && c3) {
        float *dc = (float *)(ws + WL.dc), *a = (float *)(ws + WL.a), *db = (float *)(ws + WL.db);
        float *a2 = (float *)(ws + WL.a2), *db2 = (float *)(ws + WL.db2);
        float *cpart = (float *)(ws + WL.cos_part), *dmpart = (float *)(ws + WL.dm_part);
        simt::Seg sdc{{dy, dout, 1}, {W_up, 1, r}, dout};
        NOBLE_TRY((simt_gemm<TIn, float>(st, T, r, sdc, nullptr, nullptr, dc, r)));
        NOBLE_TRY((cos3_bwd_rows<TIn, float>(d, saved, dc, om1, ph1, M, om2, ph2, c3, dh, a, db, a2, db2, cpart,
                                             dom1, dph1, dom2, dph2, st)));
        // dM = a^T db and dM2 = a2^T db2, fixed token chunks, one after the other
        const float *pa[2] = {a, a2}, *pd[2] = {db, db2};
        float *outs[2] = {dM, c3->dM2};
        for (int k = 0; k < 2; ++k) {
            simt::Seg sdm{{pa[k], 1, r}, {pd[k], 1, r}, T};
            NOBLE_TRY((simt_gemm<float, float>(st, r, r, sdm, nullptr, nullptr, dmpart, r, kDmChunk,
                                               WL.n_dm_chunks, r * r)));
            NOBLE_TRY(reduce(st, WL.n_dm_chunks, r * r, r * r, dmpart, outs[k]));
        }
        simt::Seg sup{{dy, 1, dout}, {c, 1, r}, T};
        NOBLE_TRY((simt_gemm<TIn, float>(st, dout, r, sup, nullptr, nullptr, dW_up, r)));
        simt::Seg sdn{{dh, 1, r}, {x, 1, di}, T};
        NOBLE_TRY((simt_gemm<TIn, float>(st, r, di, sdn, nullptr, nullptr, dW_down, di)));
    } else if (r > 0) {
        float *dc = (float *)(ws + WL.dc), *a = (float *)(ws + WL.a), *db = (float *)(ws + WL.db);
        float *Mt = (float *)(ws + WL.mt), *cpart = (float *)(ws + WL.cos_part);
        float *dmpart = (float *)(ws + WL.dm_part);
        const Sigma sg = sigma_of(d);
        if (sg.two_layers()) {
            const KernelInfo kt{"transpose_M", kBoundHbm, 0.0, 8.0 * r * r};
            NOBLE_TRY(run(st, kt, [&] {
                simt::transpose_square<<<(unsigned)ceil_div(r * r, 256), 256, 0, st>>>((int)r, M, Mt);
            }));
        }
        // dc = dy W_up
        simt::Seg sdc{{dy, dout, 1}, {W_up, 1, r}, dout};
        NOBLE_TRY((simt_gemm<TIn, float>(st, T, r, sdc, nullptr, nullptr, dc, r)));
        const int tpb = cosnet_tokens_per_block(r);
        if (sg.two_layers()) {
            const KernelInfo kc{"simt_cosnet_bwd", kBoundAlu, 2.0 * T * r * r, 0.0};
            NOBLE_TRY(run(st, kc, [&] {
                simt::cosnet_bwd_rows<TIn><<<(unsigned)WL.n_cos_blocks, 256, 5 * tpb * r * sizeof(float), st>>>(
                    T, (int)r, sg.act, tpb, h, b, dc, om1, ph1, Mt, om2, ph2, dh, a, db, cpart);
            }));
        } else {
            const KernelInfo kc{"simt_sigma_bwd", kBoundHbm, 0.0, (12.0 + sizeof(TIn)) * T * r};
            NOBLE_TRY(run(st, kc, [&] {
                simt::sigma_bwd_rows<TIn><<<(unsigned)WL.n_cos_blocks, 256, 0, st>>>(T, (int)r, sg.act, tpb, h,
                                                                                    dc, om1, ph1, dh, cpart);
            }));
        }
        NOBLE_TRY(reduce(st, WL.n_cos_blocks, 4 * r, r, cpart, dom1, dph1, dom2, dph2));
        if (sg.two_layers()) {
            // dM = a^T db, fixed token chunks
            simt::Seg sdm{{a, 1, r}, {db, 1, r}, T};
            NOBLE_TRY((simt_gemm<float, float>(st, r, r, sdm, nullptr, nullptr, dmpart, r, kDmChunk,
                                               WL.n_dm_chunks, r * r)));
            NOBLE_TRY(reduce(st, WL.n_dm_chunks, r * r, r * r, dmpart, dM));
        } else if (cudaMemsetAsync(dM, 0, (size_t)r * r * 4, st) != cudaSuccess) {
            return fail(NOBLE_ERR_CUDA, "dM: %s", cudaGetErrorString(cudaGetLastError()));
        }
        // dW_up = dy^T c ; dW_down = dh^T x
        simt::Seg sup{{dy, 1, dout}, {c, 1, r}, T};
        NOBLE_TRY((simt_gemm<TIn, float>(st, dout, r, sup, nullptr, nullptr, dW_up, r)));
        simt::Seg sdn{{dh, 1, r}, {x, 1, di}, T};
        NOBLE_TRY((simt_gemm<TIn, float>(st, r, di, sdn, nullptr, nullptr, dW_down, di)));
    }
    // dx = dy W + dh W_down
    simt::Seg sdx{{dy, dout, 1}, {W, 1, di}, dout};
    simt::Seg sdx2{{dh, r, 1}, {W_down, 1, di}, r};
    NOBLE_TRY((simt_gemm<TIn, TIn>(st, T, di, sdx, r > 0 ? &sdx2 : nullptr, nullptr, dx, di)));
    // dW = dy^T x
    simt::Seg sdw{{dy, 1, dout}, {x, 1, di}, T};
    NOBLE_TRY((simt_gemm<TIn, float>(st, dout, di, sdw, nullptr, nullptr, dW, di)));
    if (dbias) {
        float *bpart = (float *)(ws + WL.bias_part);
        dim3 grid((unsigned)ceil_div(dout, 256), (unsigned)WL.n_bias_chunks);
        const KernelInfo kb{"colsum_dbias", kBoundHbm, (double)T * dout, (double)T * dout * sizeof(TIn)};
        NOBLE_TRY(run(st, kb, [&] {
            simt::colsum_partial<TIn><<<grid, 256, 0, st>>>(T, dout, kBiasChunk, dy, bpart);
        }));
        NOBLE_TRY(reduce(st, WL.n_bias_chunks, dout, dout, bpart, dbias));
    }
    return NOBLE_OK;
}


// ------------------------------------------------------------ tensor-core path
using bf16 = __nv_bfloat16;

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn()
{
    static EncodeTiledFn fn = [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            q != cudaDriverEntryPointSuccess) {
            cudaGetLastError();
            p = nullptr;
        }
        return reinterpret_cast<EncodeTiledFn>(p);
    }();
    return fn;
}

// 2-D TMA map over a row-major bf16 matrix [rows][cols]: box of 64 columns
// (128 bytes) by box_rows rows, 128-byte swizzle, zero fill out of bounds.
// `pitch` is the row pitch in elements (0: cols, a contiguous matrix).
noble_status make_map(CUtensorMap *m, const void *ptr, int64_t rows, int64_t cols, uint32_t box_rows,
                      int64_t pitch = 0)
{
    EncodeTiledFn enc = encode_fn();
    if (!enc) return fail(NOBLE_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)(pitch ? pitch : cols) * 2};
    cuuint32_t box[2] = {64, box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
        return fail(NOBLE_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d): rows=%lld cols=%lld box_rows=%u", (int)r,
                    (long long)rows, (long long)cols, box_rows);
    return NOBLE_OK;
}

// 4-D TMA map over a row-major bf16 matrix [K][MN] (MN contiguous) that loads
// MN-major tiles in the layout [8-row K group][64-wide MN chunk][8 rows][128 B]:
// dimensions (inner first) {64 elements, 8 rows, MN/64 chunks, K/8 groups} with
// strides {P, 128 B, 8 P} for the row pitch P, box {64, 8, nchunks, kgroups}.
// Requires MN % 64 == 0 and K % 8 == 0, so that every in-range coordinate of
// the 4-D description is an element of the matrix.  `pitch` (elements, 0: MN)
// allows a column range of a wider matrix.
noble_status make_map_mn4(CUtensorMap *m, const void *ptr, int64_t K, int64_t MN, uint32_t nchunks,
                          uint32_t kgroups = 8, int64_t pitch = 0)
{
    EncodeTiledFn enc = encode_fn();
    if (!enc) return fail(NOBLE_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
    if (MN % 64 || K % 8) return fail(NOBLE_ERR_INVALID_ARG, "4-D MN-major map needs MN %% 64 == 0 and K %% 8 == 0");
    const cuuint64_t P = (cuuint64_t)(pitch ? pitch : MN) * 2;
    cuuint64_t dims[4] = {64, 8, (cuuint64_t)MN / 64, (cuuint64_t)K / 8};
    cuuint64_t strides[3] = {P, 128, 8 * P};
    cuuint32_t box[4] = {64, 8, nchunks, kgroups};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(ptr), dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
        return fail(NOBLE_ERR_CUDA, "cuTensorMapEncodeTiled (4-D) failed (%d): K=%lld MN=%lld", (int)r, (long long)K,
                    (long long)MN);
    return NOBLE_OK;
}

// 3-D TMA map for the pair kernel's stores into C: dimensions (inner first)
// {N, M, nsplit} with row pitch ldc and split pitch split_stride (elements),
// box {128 bytes of columns, 32 rows, 1}, 128-byte swizzle.
noble_status make_store_map(CUtensorMap *m, void *C, bool fp32, int64_t M, int64_t N, int64_t ldc, int64_t nsplit,
                            int64_t split_stride)
{
    EncodeTiledFn enc = encode_fn();
    if (!enc) return fail(NOBLE_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
    const cuuint64_t es = fp32 ? 4 : 2;
    cuuint64_t dims[3] = {(cuuint64_t)N, (cuuint64_t)M, (cuuint64_t)nsplit};
    cuuint64_t strides[2] = {(cuuint64_t)ldc * es, (cuuint64_t)(nsplit > 1 ? split_stride : M * ldc) * es};
    cuuint32_t box[3] = {(cuuint32_t)(128 / es), 32, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = enc(m, fp32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, C, dims, strides,
                     box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
        return fail(NOBLE_ERR_CUDA, "cuTensorMapEncodeTiled (store) failed (%d): M=%lld N=%lld ldc=%lld", (int)r,
                    (long long)M, (long long)N, (long long)ldc);
    return NOBLE_OK;
}

// 2-D TMA map for the bottleneck kernel's row outputs [T][r] (fp32 or bf16):
// box of 32 columns by 32 rows; 128-byte rows (fp32) with the 128-byte
// swizzle, 64-byte rows (bf16) with the 64-byte swizzle.
noble_status make_rows_map(CUtensorMap *m, void *p, bool fp32, int64_t T, int64_t r)
{
    EncodeTiledFn enc = encode_fn();
    if (!enc) return fail(NOBLE_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
    const cuuint64_t es = fp32 ? 4 : 2;
    cuuint64_t dims[2] = {(cuuint64_t)r, (cuuint64_t)T};
    cuuint64_t strides[1] = {(cuuint64_t)r * es};
    cuuint32_t box[2] = {32, 32};
    cuuint32_t estr[2] = {1, 1};
    CUresult res = enc(m, fp32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, p, dims,
                       strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                       fp32 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                       CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (res != CUDA_SUCCESS)
        return fail(NOBLE_ERR_CUDA, "cuTensorMapEncodeTiled (rows) failed (%d): T=%lld r=%lld", (int)res,
                    (long long)T, (long long)r);
    return NOBLE_OK;
}

// The current CUDA context (NULL if none or the driver call is unavailable).
typedef CUresult (*CtxGetCurrentFn)(CUcontext *);
CUcontext current_context()
{
    static CtxGetCurrentFn fn = [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess) {
            cudaGetLastError();
            p = nullptr;
        }
        return reinterpret_cast<CtxGetCurrentFn>(p);
    }();
    CUcontext c = nullptr;
    if (!fn || fn(&c) != CUDA_SUCCESS) return nullptr;
    return c;
}

// Device address of a __device__ variable in the current context.  The
// host-side name of a __device__ variable is only a stand-in, so the address
// is looked up with the device current; it is cached per context (a new
// context after a device reset loads the module at another address).
template <class T>
void *symbol_address(const T &symbol)
{
    static std::mutex mu;
    static std::vector<std::pair<CUcontext, void *>> cache;
    const CUcontext ctx = current_context();
    std::lock_guard<std::mutex> g(mu);
    if (ctx)
        for (auto &e : cache)
            if (e.first == ctx) return e.second;
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, symbol) != cudaSuccess || !p) {
        cudaGetLastError();
        return nullptr;
    }
    // the lookup may have created the primary context: key on it
    const CUcontext now = ctx ? ctx : current_context();
    if (now) cache.emplace_back(now, p);
    return p;
}

// Device address of this device's status word.
uint32_t *status_ptr() { return static_cast<uint32_t *>(symbol_address(g_device_status)); }

// One K segment of a tensor-core GEMM; A and B are row-major bf16 matrices
// ([M][K] / [N][K] when K-major, [K][M] / [K][N] when MN-major).
struct TcSeg {
    const void *A, *B;
    int64_t K;
    int64_t ldb = 0;  // row pitch of B in elements (0: contiguous); MN-major B only
};

template <int BN> struct StagesFor { static constexpr int value = BN >= 256 ? 4 : BN >= 128 ? 6 : 8; };

template <int BN, bool A_MN, bool B_MN, class Epi>
noble_status tc_gemm(cudaStream_t st, const char *name, int64_t M, int64_t N, TcSeg s0, const TcSeg *s1,
                     int kb_per_split, int nsplit, const typename Epi::Params &ep)
{
    constexpr int STAGES = StagesFor<BN>::value;
    using SM = tc::Smem<BN, STAGES>;
    if (M == 0 || N == 0) return NOBLE_OK;
    CUtensorMap maps[4];
    auto mk = [&](CUtensorMap *m, const void *p, bool mn, int64_t mnrows, int64_t K, uint32_t box_rows) {
        return mn ? make_map(m, p, K, mnrows, 64) : make_map(m, p, mnrows, K, box_rows);
    };
    NOBLE_TRY(mk(&maps[0], s0.A, A_MN, M, s0.K, tc::kBM));
    NOBLE_TRY(mk(&maps[1], s0.B, B_MN, N, s0.K, BN));
    if (s1) {
        NOBLE_TRY(mk(&maps[2], s1->A, A_MN, M, s1->K, tc::kBM));
        NOBLE_TRY(mk(&maps[3], s1->B, B_MN, N, s1->K, BN));
    } else {
        maps[2] = maps[0];
        maps[3] = maps[1];
    }
    const tc::GemmArgs args{M, N, (int)ceil_div(s0.K, tc::kBK), s1 ? (int)ceil_div(s1->K, tc::kBK) : 0,
                            kb_per_split, status_ptr()};
    auto kern = tc::gemm_kernel<BN, A_MN, B_MN, STAGES, Epi>;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, SM::kDynamic) != cudaSuccess)
        return fail(NOBLE_ERR_CUDA, "%s: cudaFuncSetAttribute: %s", name, cudaGetErrorString(cudaGetLastError()));
    const dim3 grid((unsigned)ceil_div(N, BN), (unsigned)ceil_div(M, tc::kBM), (unsigned)nsplit);
    const double K = (double)s0.K + (s1 ? (double)s1->K : 0.0);
    const KernelInfo ki{name, kBoundTensor, 2.0 * M * N * K, 2.0 * (M + N) * K};
    return run(st, ki, [&] {
        kern<<<grid, tc::kThreads, SM::kDynamic, st>>>(maps[0], maps[1], maps[2], maps[3], args, ep);
    });
}


int num_sms()
{
    static int cache[64];
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && cache[dev]) return cache[dev];
    int n = 0;
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    cudaGetLastError();
    if (n <= 0) n = 1;
    if (dev >= 0 && dev < 64) cache[dev] = n;
    return n;
}

// One problem of a grouped persistent GEMM launch.
struct ProbSpec {
    int64_t M, N;
    TcSeg s0;
    const TcSeg *s1;  // nullptr = single segment
    int bn;           // N tile (multiple of 32; of 64 when B is MN-major)
    int nsplit = 1;
    int kb_per_split = 0;
    int dep = 0;         // Problem::dep: segments reading what an earlier kernel of the call wrote
    // fused bottleneck launch, leader problem: segment 0's B operand of CTA
    // rank 1 (the branch weights; N = r rows or columns, like rank 0's)
    const void *B0_rank1 = nullptr;
    int64_t B0_rank1_ld = 0;
};





// Static longest-processing-time-first assignment of the tiles of a grouped
// launch to its clusters.  A tile's cost is its MMA work (N tile x k-blocks).
// When all tiles cost the same, round-robin is already balanced and no
// schedule is built.  Otherwise tiles are taken heaviest first (keeping the
// L2-friendly order among equal costs) and each goes to the least-loaded
// cluster; slot j * clusters + c of the schedule holds cluster c's j-th tile.
template <class GA>
noble_status pair_schedule(GA &g, int clusters)
{
    g.sched_len = 0;
    struct Item {
        int id;
        double cost;
    };
    std::vector<Item> items;
    items.reserve(g.total_tiles);
    for (int p = 0; p < g.nproblems; ++p) {
        const auto &P = g.p[p];
        const int pairs_m = (P.tiles_m + 1) / 2;
        const int per_split = pairs_m * P.tiles_n;
        const int kbt = P.kb0 + P.kb1;
        for (int z = 0; z < P.nsplit; ++z) {
            int kb = kbt;
            if (P.kb_per_split > 0) {
                const int b = z * P.kb_per_split;
                kb = (b + P.kb_per_split < kbt ? b + P.kb_per_split : kbt) - b;
            }
            const double cost = (double)P.bn * kb;
            for (int i = 0; i < per_split; ++i) items.push_back({P.tile_begin + z * per_split + i, cost});
        }
    }
    bool uniform = true;
    for (const Item &it : items) uniform = uniform && it.cost == items[0].cost;
    if (uniform || clusters < 1) return NOBLE_OK;
    std::stable_sort(items.begin(), items.end(), [](const Item &a, const Item &b) { return a.cost > b.cost; });
    std::vector<double> load(clusters, 0.0);
    std::vector<std::vector<int>> lists(clusters);
    for (const Item &it : items) {
        int c = 0;
        for (int k = 1; k < clusters; ++k)
            if (load[k] < load[c]) c = k;
        lists[c].push_back(it.id);
        load[c] += it.cost;
    }
    size_t maxlen = 0;
    for (const auto &l : lists) maxlen = l.size() > maxlen ? l.size() : maxlen;
    if (maxlen * clusters > (size_t)tc::kMaxSched) return NOBLE_OK;  // too long: round-robin
    for (size_t j = 0; j < maxlen; ++j)
        for (int c = 0; c < clusters; ++c)
            g.sched[j * clusters + c] = j < lists[c].size() ? (uint16_t)lists[c][j] : (uint16_t)0xFFFF;
    g.sched_len = (int)(maxlen * clusters);
    return NOBLE_OK;
}

// Grouped GEMM on CTA pairs (tc_pair.cuh): every problem's tile width must be
// 128 or 256.  Tiles are 256 rows (a pair of 128-row halves).
template <bool A_MN, bool B_MN, class Epi, bool MN4 = false, int FUSE = tc::pair::kFuseNone>
noble_status tc_pair_group(cudaStream_t st, const char *name, int n, const ProbSpec *specs,
                           const typename Epi::Params *eps, const tc::pair::FuseArgs *fa = nullptr)
{
    constexpr int STAGES = 6;
    using SM = tc::pair::PairSmem<STAGES>;
    if (n < 1 || n > tc::kMaxProblems) return fail(NOBLE_ERR_INVALID_ARG, "%s: %d problems", name, n);
    tc::GroupMaps maps;
    tc::GroupArgs<typename Epi::Params> g{};
    int tiles = 0, np = 0;
    double flops = 0, bytes = 0;
    for (int i = 0; i < n; ++i) {
        const ProbSpec &P = specs[i];
        if (P.M == 0 || P.N == 0) continue;
        if (P.bn != 128 && P.bn != 256) return fail(NOBLE_ERR_INVALID_ARG, "%s: pair tile width %d", name, P.bn);
        const uint32_t bh = (uint32_t)P.bn / 2;
        auto mk = [&](CUtensorMap *m, const void *p, bool mn, int64_t mnrows, int64_t K, uint32_t box_rows,
                      int64_t ld = 0) {
            if (mn && MN4) return make_map_mn4(m, p, K, mnrows, box_rows / 64, 8, ld);
            return mn ? make_map(m, p, K, mnrows, 64, ld) : make_map(m, p, mnrows, K, box_rows);
        };
        // a fused launch's leader problem multiplies N = 2r columns (r of the
        // output, r of the branch); its output tile is the first r
        const bool lead = FUSE != tc::pair::kFuseNone && i == 0;
        const int64_t nb_rows = lead ? P.bn / 2 : P.N;
        NOBLE_TRY(mk(&maps.m[np][0], P.s0.A, A_MN, P.M, P.s0.K, tc::kBM));
        NOBLE_TRY(mk(&maps.m[np][1], P.s0.B, B_MN, nb_rows, P.s0.K, bh, P.s0.ldb));
        if (P.s1) {
            NOBLE_TRY(mk(&maps.m[np][2], P.s1->A, A_MN, P.M, P.s1->K, tc::kBM));
            NOBLE_TRY(mk(&maps.m[np][3], P.s1->B, B_MN, nb_rows, P.s1->K, bh, P.s1->ldb));
        } else {
            maps.m[np][2] = maps.m[np][0];
            maps.m[np][3] = maps.m[np][1];
        }
        if (lead) {
            if (!P.B0_rank1 || !P.s1 || P.bn != 2 * P.N)
                return fail(NOBLE_ERR_INVALID_ARG, "%s: fused leader problem", name);
            NOBLE_TRY(mk(&maps.m[np][5], P.B0_rank1, B_MN, nb_rows, P.s0.K, bh, P.B0_rank1_ld));
        } else {
            maps.m[np][5] = maps.m[np][1];
        }
        auto &q = g.p[np];
        q.M = P.M;
        q.N = P.N;
        q.kb0 = (int)ceil_div(P.s0.K, tc::kBK);
        q.kb1 = P.s1 ? (int)ceil_div(P.s1->K, tc::kBK) : 0;
        q.bn = P.bn;
        q.tiles_m = (int)ceil_div(P.M, tc::kBM);
        q.tiles_n = (int)ceil_div(P.N, P.bn);
        q.nsplit = P.nsplit;
        q.kb_per_split = P.kb_per_split;
        q.tile_begin = tiles;
        q.dep = P.dep;
        q.ep = eps[i];
        {
            // TMA-store epilogue where C's layout allows it
            using OutT = typename Epi::out_type;
            constexpr int64_t es = sizeof(OutT);
            const auto &e = eps[i];
            // a transposed store writes C with rows n and columns m
            const int64_t outM = e.transpose ? P.N : P.M, outN = e.transpose ? P.M : P.N;
            const bool ok = !e.col0 && reinterpret_cast<uintptr_t>(e.C) % 16 == 0 &&
                            (e.ldc * es) % 16 == 0 && outN % 4 == 0 &&
                            (P.nsplit == 1 || (e.split_stride * es) % 16 == 0);
            q.ep.tma = ok ? 1 : 0;
            if (ok)
                NOBLE_TRY(make_store_map(&maps.m[np][4], e.C, es == 4, outM, outN, e.ldc, P.nsplit, e.split_stride));
        }
        tiles += (int)ceil_div(q.tiles_m, 2) * q.tiles_n * q.nsplit;
        const double K = (double)P.s0.K + (P.s1 ? (double)P.s1->K : 0.0);
        flops += 2.0 * P.M * P.N * K;
        bytes += 2.0 * (P.M + P.N) * K;
        if (lead) {
            // the branch's product in segment 0 and the r x r product (three terms)
            flops += 2.0 * P.M * P.N * (double)P.s0.K + 3.0 * 2.0 * P.M * P.N * P.N;
            bytes += 2.0 * P.N * (double)P.s0.K;
        }
        ++np;
    }
    if (np == 0) return NOBLE_OK;
    g.nproblems = np;
    g.total_tiles = tiles;
    g.status = status_ptr();
    auto kern = tc::pair::gemm_pair<A_MN, B_MN, STAGES, Epi, MN4, FUSE>;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, SM::kDynamic) != cudaSuccess)
        return fail(NOBLE_ERR_CUDA, "%s: cudaFuncSetAttribute: %s", name, cudaGetErrorString(cudaGetLastError()));
    // as many pairs as can be resident at once
    static int max_clusters_cache[64];  // per instantiation
    int dev = 0;
    cudaGetDevice(&dev);
    int max_clusters = (dev >= 0 && dev < 64) ? max_clusters_cache[dev] : 0;
    if (max_clusters <= 0) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(2 * 64, 1, 1);
        cfg.blockDim = dim3(tc::pair::kPairThreads, 1, 1);
        cfg.dynamicSmemBytes = SM::kDynamic;
        cudaLaunchAttribute attr;
        attr.id = cudaLaunchAttributeClusterDimension;
        attr.val.clusterDim.x = 2;
        attr.val.clusterDim.y = 1;
        attr.val.clusterDim.z = 1;
        cfg.attrs = &attr;
        cfg.numAttrs = 1;
        if (cudaOccupancyMaxActiveClusters(&max_clusters, (void *)kern, &cfg) != cudaSuccess || max_clusters <= 0) {
            cudaGetLastError();
            max_clusters = num_sms() / 2;
        }
        if (dev >= 0 && dev < 64) max_clusters_cache[dev] = max_clusters;
    }
    const int clusters = tiles < max_clusters ? tiles : max_clusters;
    // a fused launch walks its own dependency order (tc_pair.cuh: share_tile)
    if (FUSE == tc::pair::kFuseNone) NOBLE_TRY(pair_schedule(g, clusters));
    const tc::pair::FuseArgs fargs = fa ? *fa : tc::pair::FuseArgs{};
    const KernelInfo ki{name, kBoundTensor, flops, bytes};
    // a fused launch waits on flags that assume every cluster resident at once: launched normally
    const bool pdl = FUSE == tc::pair::kFuseNone && pdl_ok();
    return run(st, ki, [&] {
        launch_maybe_pdl(kern, dim3(2 * clusters), dim3(tc::pair::kPairThreads), SM::kDynamic, st, pdl, maps, g,
                         fargs);
    });
}

// Runtime r -> compile-time N tile for the r-wide products.
template <class F>
noble_status with_rank_tile(int64_t r, F &&f)
{
    switch (r) {
    case 16: return f(std::integral_constant<int, 16>{});
    case 32: return f(std::integral_constant<int, 32>{});
    case 64: return f(std::integral_constant<int, 64>{});
    case 128: return f(std::integral_constant<int, 128>{});
    case 256: return f(std::integral_constant<int, 256>{});
    }
    return fail(NOBLE_ERR_UNSUPPORTED, "rank %lld", (long long)r);
}
// The same for r <= 128 (kernels that hold a whole r x r operand in shared memory).
template <class F>
noble_status with_rank_tile_max128(int64_t r, F &&f)
{
    switch (r) {
    case 16: return f(std::integral_constant<int, 16>{});
    case 32: return f(std::integral_constant<int, 32>{});
    case 64: return f(std::integral_constant<int, 64>{});
    case 128: return f(std::integral_constant<int, 128>{});
    }
    return fail(NOBLE_ERR_UNSUPPORTED, "rank %lld", (long long)r);
}

// The all-ones [T][kOnesCols] bf16 operand of the backward without a branch
// (dbias = dy^T 1 as extra weight-gradient columns).
__global__ void fill_ones_kernel(int64_t n, bf16 *ones)
{
    const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx < n) ones[idx] = __float2bfloat16_rn(1.f);
}

noble_status fill_ones(cudaStream_t st, int64_t n, bf16 *ones)
{
    if (n == 0) return NOBLE_OK;
    const KernelInfo ki{"fill_ones", kBoundHbm, 0.0, 2.0 * n};
    return run(st, ki, [&] { fill_ones_kernel<<<(unsigned)ceil_div(n, 256), 256, 0, st>>>(n, ones); });
}

// Fixed-order sums of partial results: out_j[i] = sum_z part_j[z * stride_j + i]
// (z ascending) for up to five outputs in one launch.
struct SplitJobs {
    const float *part[8];
    float *out[8];
    int64_t n[8], stride[8], begin[9];  // stride: elements between consecutive partials
    int nparts;
    int jparts[8];  // partials of job j when non-zero (else nparts; reduce_split_kernel only)
    int njobs;
};
// Block = 8 warps over 32 consecutive outputs: warp w adds partials
// [w P/8, (w+1) P/8) in ascending order for its lane's output, then the eight
// warp sums are added in warp order -- deterministic.
__global__ void __launch_bounds__(256) reduce_split_kernel(SplitJobs J)
{
    ptx::griddep_wait();  // the partials come from the preceding kernel
    ptx::griddep_launch();
    __shared__ float sm[8][33];
    const int lane = threadIdx.x % 32, w = threadIdx.x / 32;
    const int64_t idx = (int64_t)blockIdx.x * 32 + lane;
    const bool in = idx < J.begin[J.njobs];
    int j = 0;
    if (in)
        while (idx >= J.begin[j + 1]) ++j;
    const int64_t i = in ? idx - J.begin[j] : 0;
    const int np = J.jparts[j] ? J.jparts[j] : J.nparts;
    const int per = (np + 7) / 8;
    const int zb = w * per, ze = min(np, zb + per);
    float s = 0.f;
    if (in) {
        // eight loads in flight, then added in ascending z as before
        const float *pp = J.part[j] + i;
        const int64_t st = J.stride[j];
        int z = zb;
        for (; z + 8 <= ze; z += 8) {
            float v[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) v[u] = pp[(int64_t)(z + u) * st];
#pragma unroll
            for (int u = 0; u < 8; ++u) s += v[u];
        }
        for (; z < ze; ++z) s += pp[(int64_t)z * st];
    }
    sm[w][lane] = s;
    __syncthreads();
    if (w == 0 && in) {
        float t = 0.f;
#pragma unroll
        for (int k = 0; k < 8; ++k) t += sm[k][lane];
        J.out[j][i] = t;
    }
}

// Split-K sums (few partials, long outputs): thread q handles outputs
// [4q, 4q + 4) of the concatenated jobs and adds the partials z = 0, 1, ... in
// order -- deterministic, and the same association as reduce_split_kernel
// for up to eight partials.  Every job length and partial stride is a
// multiple of 4 and every pointer 16-byte aligned.
__global__ void __launch_bounds__(256) reduce_split_vec4_kernel(SplitJobs J)
{
    ptx::griddep_wait();  // the partials come from the preceding kernel
    ptx::griddep_launch();
    const int64_t n4 = J.begin[J.njobs] / 4;
    for (int64_t q = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; q < n4; q += (int64_t)gridDim.x * blockDim.x) {
        const int64_t idx = q * 4;
        int j = 0;
        while (idx >= J.begin[j + 1]) ++j;
        const int64_t i = idx - J.begin[j];
        const float4 *p = reinterpret_cast<const float4 *>(J.part[j] + i);
        const int64_t st4 = J.stride[j] / 4;
        float4 s = __ldcs(p);
        for (int z = 1; z < J.nparts; ++z) {
            const float4 v = __ldcs(p + z * st4);
            s.x += v.x, s.y += v.y, s.z += v.z, s.w += v.w;
        }
        *reinterpret_cast<float4 *>(J.out[j] + i) = s;
    }
}

// Fused r-wide GEMM + CosNet launch (forward or backward), one tile per CTA.
template <int R, bool BWD, int SIG>
noble_status cosnet_launch(cudaStream_t st, const char *name, int64_t T, const bf16 *A, int64_t K, const bf16 *B,
                           const tc::CosnetArgs &args_in)
{
    using Cfg = tc::CosnetCfg<R, BWD>;
    CUtensorMap mA, mB;
    NOBLE_TRY(make_map(&mA, A, T, K, tc::kBM));
    if (Cfg::kBInterleaved)  // B = W_up [K = d_out][R], MN-major, all 8 K groups of a k-block
        NOBLE_TRY(make_map_mn4(&mB, B, K, R, (uint32_t)(R / 64), 8));
    else if (BWD)  // B = W_up [K = d_out][R], MN-major, 64 K rows per column chunk
        NOBLE_TRY(make_map(&mB, B, K, R, tc::kBK));
    else  // B = W_down [R][K], K-major, all R rows
        NOBLE_TRY(make_map(&mB, B, R, K, R));
    tc::CosnetArgs args = args_in;
    args.T = T;
    args.kb = (int)ceil_div(K, tc::kBK);
    args.status = status_ptr();
    // the epilogue's row outputs go out through TMA stores (CosNet, r in {64, 128})
    tc::CosnetStoreMaps smaps{};
    if constexpr (SIG == tc::kSigCosnet && Cfg::kStgFits) {
        if (T > 0 && BWD) {
            NOBLE_TRY(make_rows_map(&smaps.m[0], args.db_out, false, T, R));
            NOBLE_TRY(make_rows_map(&smaps.m[1], args.dh_out, false, T, R));
            NOBLE_TRY(make_rows_map(&smaps.m[2], args.a_out, false, T, R));
        } else if (T > 0) {
            if (args.h_out) NOBLE_TRY(make_rows_map(&smaps.m[0], args.h_out, true, T, R));
            if (args.b_out) NOBLE_TRY(make_rows_map(&smaps.m[1], args.b_out, true, T, R));
            NOBLE_TRY(make_rows_map(&smaps.m[2], args.c_out, false, T, R));
        }
    }
    auto kern = tc::cosnet_gemm_kernel<R, BWD, SIG>;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kDynamic) != cudaSuccess)
        return fail(NOBLE_ERR_CUDA, "%s: cudaFuncSetAttribute: %s", name, cudaGetErrorString(cudaGetLastError()));
    const KernelInfo ki{name, kBoundHbm, 2.0 * T * R * (K + R), 2.0 * T * K + 2.0 * R * K + (BWD ? 14.0 : 10.0) * T * R};
    // a programmatic dependent of whatever precedes it in the stream, also as
    // the first kernel of a call: every thread waits for the predecessor grid
    // (griddep_wait) before its first global read
    return run(st, ki, [&] {
        const unsigned grid = (unsigned)ceil_div(T, tc::kBM);
        launch_maybe_pdl(kern, dim3(grid), dim3(Cfg::kThreads), Cfg::kDynamic, st, kProgrammaticLaunch, mA, mB,
                         args, smaps);
    });
}

// MN-major operands can use the 4-D layout when every MN extent tiles by 64
// and every K extent by 8.
bool mn4_ok(std::initializer_list<int64_t> mn_extents, std::initializer_list<int64_t> k_extents)
{
    for (int64_t v : mn_extents)
        if (v % 64) return false;
    for (int64_t v : k_extents)
        if (v % 8) return false;
    return true;
}

noble_status fwd_tc(const noble_linear_desc *d, const bf16 *x, const bf16 *W, const float *bias,
                    const bf16 *W_down, const float *om1, const float *ph1, const float *M, const float *om2,
                    const float *ph2, const bf16 *W_up, bf16 *y, char *saved, cudaStream_t st,
                    const Cos3 *c3 = nullptr)
{
    const int64_t T = d->T, di = d->d_in, dout = d->d_out, r = d->r;
    const TcSeg main{x, W, di};
    const tc::EpiStore<bf16>::Params py{y, dout, bias, 0};
    if (r == 0) {
        const ProbSpec P{T, dout, main, nullptr, 256};
        return tc_pair_group<false, false, tc::EpiStore<bf16>>(st, "tc_main_up_fwd", 1, &P, &py);
    }
    const SavedLayout SL = saved_layout(d);
    float *h = (float *)(saved + SL.h), *b = (float *)(saved + SL.b);
    bf16 *c = (bf16 *)(saved + SL.c);
    if (c3 && cos3_tc(d)) {
        // three-layer cosine in the bottleneck kernel: h, b, b2 (saved) and c
        tc::CosnetArgs a{};
        a.om1 = om1, a.ph1 = ph1, a.om2 = om2, a.ph2 = ph2, a.M = M;
        a.M2 = c3->M2, a.om3 = c3->om3, a.ph3 = c3->ph3;
        a.h_out = h, a.b_out = b, a.b2_out = (float *)(saved + SL.b2), a.c_out = c;
        NOBLE_TRY(with_rank_tile_max128(r, [&](auto bn) {
            constexpr int R = decltype(bn)::value;
            return cosnet_launch<R, false, tc::kSigCos3>(st, "tc_down_cosnet_fwd", T, x, di, W_down, a);
        }));
        const TcSeg up{c, W_up, r};
        ProbSpec P{T, dout, main, &up, 256};
        P.dep = 2;  // c, written by the bottleneck kernel
        return tc_pair_group<false, false, tc::EpiStore<bf16>>(st, "tc_main_up_fwd", 1, &P, &py);
    }
    if (c3) {
        // three-layer cosine, r = 256: h = x W_down^T on the tensor cores (fp32
        // out), the cosines and r x r products on the CUDA cores, then the output GEMM
        const ProbSpec Ph{T, r, TcSeg{x, W_down, di}, nullptr, r <= 128 ? 128 : 256};
        const tc::EpiStore<float>::Params Eh{h, r, nullptr, 0};
        NOBLE_TRY((tc_pair_group<false, false, tc::EpiStore<float>>(st, "tc_h_gemm", 1, &Ph, &Eh)));
        NOBLE_TRY(cos3_fwd_rows<bf16>(d, h, om1, ph1, M, om2, ph2, c3, saved, c, st));
        const TcSeg up{c, W_up, r};
        ProbSpec P{T, dout, main, &up, 256};
        P.dep = 2;  // c, written by the bottleneck kernel
        return tc_pair_group<false, false, tc::EpiStore<bf16>>(st, "tc_main_up_fwd", 1, &P, &py);
    }
    if (fuse_fwd(d)) {
        // one launch: per row pair a leader tile x [W rows 0..r ; W_down]^T (the
        // first r output columns, h beside them; CosNet in its epilogue, then
        // + c W_up^T), and the output tiles of columns [r, d_out)
        uint32_t *flags = (uint32_t *)(saved + SL.flags);
        if (memset_async(flags, 0, fuse_flag_bytes(d), st) != cudaSuccess)
            return fail(NOBLE_ERR_CUDA, "flags: %s", cudaGetErrorString(cudaGetLastError()));
        tc::pair::FuseArgs fa{};
        fa.T = T, fa.r = (int)r;
        fa.om1 = om1, fa.ph1 = ph1, fa.om2 = om2, fa.ph2 = ph2, fa.M = M;
        fa.h_out = SL.only_c ? nullptr : h, fa.b_out = SL.only_c ? nullptr : b, fa.c_out = c;
        fa.flags = flags;
        // columns [r, r + nf) in 256-wide tiles, a last part of at most 128 in 128-wide ones
        const FusedSplit fs = fused_split(dout, r);
        const int64_t o2 = r + fs.nfull;
        const TcSeg up0{c, W_up, r}, up1{c, W_up + r * r, r}, up2{c, W_up + o2 * r, r};
        ProbSpec P[3] = {ProbSpec{T, r, main, &up0, 2 * (int)r},
                         ProbSpec{T, fs.nfull, TcSeg{x, W + r * di, di}, &up1, 256},
                         ProbSpec{T, fs.ntail, TcSeg{x, W + o2 * di, di}, &up2, 128}};
        P[0].B0_rank1 = W_down;
        const tc::EpiStore<bf16>::Params E[3] = {py, {y + r, dout, bias ? bias + r : nullptr, 0},
                                                 {y + o2, dout, bias ? bias + o2 : nullptr, 0}};
        return tc_pair_group<false, false, tc::EpiStore<bf16>, false, tc::pair::kFuseFwd>(st, "tc_main_up_fwd", 3, P,
                                                                                           E, &fa);
    }
    tc::CosnetArgs a{};
    a.om1 = om1, a.ph1 = ph1, a.om2 = om2, a.ph2 = ph2, a.M = M;
    a.h_out = SL.only_c ? nullptr : h, a.b_out = SL.only_c ? nullptr : b, a.c_out = c;
    const Sigma sg = sigma_of(d);
    a.act = sg.act;
    NOBLE_TRY(with_rank_tile(r, [&](auto bn) {
        constexpr int R = decltype(bn)::value;
        const char *nm = "tc_down_cosnet_fwd";
        switch (sg.sig) {
        case tc::kSigCos1: return cosnet_launch<R, false, tc::kSigCos1>(st, nm, T, x, di, W_down, a);
        case tc::kSigIdentity: return cosnet_launch<R, false, tc::kSigIdentity>(st, nm, T, x, di, W_down, a);
        case tc::kSigAct1: return cosnet_launch<R, false, tc::kSigAct1>(st, nm, T, x, di, W_down, a);
        case tc::kSigAct2: return cosnet_launch<R, false, tc::kSigAct2>(st, nm, T, x, di, W_down, a);
        default: return cosnet_launch<R, false, tc::kSigCosnet>(st, nm, T, x, di, W_down, a);
        }
    }));
    const TcSeg up{c, W_up, r};
    ProbSpec P{T, dout, main, &up, 256};
    P.dep = 2;  // c, written by the bottleneck kernel
    return tc_pair_group<false, false, tc::EpiStore<bf16>>(st, "tc_main_up_fwd", 1, &P, &py);
}

noble_status bwd_tc(const noble_linear_desc *d, const bf16 *dy, const bf16 *x, const bf16 *W, const bf16 *W_down,
                    const float *om1, const float *ph1, const float *M, const float *om2, const float *ph2,
                    const bf16 *W_up, const char *saved, bf16 *dx, float *dW, float *dbias, float *dW_down,
                    float *dM, float *dom1, float *dph1, float *dom2, float *dph2, float *dW_up, char *ws,
                    cudaStream_t st, const Cos3 *c3 = nullptr)
{
    const int64_t T = d->T, di = d->d_in, dout = d->d_out, r = d->r;
    const SavedLayout SL = saved_layout(d);
    const WorkLayout WL = work_layout(d);
    bf16 *dh = (bf16 *)(ws + WL.dh), *a = (bf16 *)(ws + WL.a), *db = (bf16 *)(ws + WL.db);
    bf16 *ones = (bf16 *)(ws + WL.ones);
    const bool fused = fuse_bwd(d);
    const bool c3k = c3 && cos3_tc(d);  // three-layer cosine in the bottleneck kernel
    const bool ones_dbias = dbias && (r == 0 || (c3 && !c3k));
    const Sigma sg = sigma_of(d);
    if (ones_dbias) NOBLE_TRY(fill_ones(st, T * kOnesCols, ones));
    // domega1, dphi1, domega2, dphi2 (and dbias) from per-CTA or per-32-token partials
    // (and domega3, dphi3 of the three-layer cosine in the bottleneck kernel)
    auto reduce_cosnet = [&](const float *cpart, const float *bpart) {
        SplitJobs J{};
        float *outs[6] = {dom1, dph1, dom2, dph2, c3k ? c3->dom3 : nullptr, c3k ? c3->dph3 : nullptr};
        const int nq = c3k ? 6 : 4;
        J.nparts = (int)WL.n_cos_blocks;
        J.begin[0] = 0;
        for (int q = 0; q < nq; ++q) {
            J.part[q] = cpart + q * r;
            J.out[q] = outs[q];
            J.n[q] = r;
            J.stride[q] = nq * r;
            J.begin[q + 1] = J.begin[q] + r;
        }
        J.njobs = nq;
        if (bpart) {
            J.part[nq] = bpart;
            J.out[nq] = dbias;
            J.n[nq] = dout;
            J.stride[nq] = dout;
            J.begin[nq + 1] = J.begin[nq] + dout;
            J.njobs = nq + 1;
            // the fused launch keeps dbias partials per 128 tokens
            if (fused) J.jparts[nq] = (int)WL.n_bias_chunks;
        }
        const int64_t total = J.begin[J.njobs];
        const KernelInfo kr{"reduce_partials", kBoundHbm, (double)total * J.nparts, 4.0 * total * (J.nparts + 1)};
        const bool pdl = pdl_ok();
        return run(st, kr, [&] {
            launch_maybe_pdl(reduce_split_kernel, dim3((unsigned)ceil_div(total, 32)), dim3(256), 0, st, pdl, J);
        });
    };
    if (r > 0 && c3k) {
        // three-layer cosine in the bottleneck kernel: dc = dy W_up, the chain
        // rule through the three layers (both r x r products as tensor-core
        // MMAs), dh, a, db, a2, db2 and the six column sums
        float *cpart = (float *)(ws + WL.cos_part);
        float *bpart = (float *)(ws + WL.bias_part);
        tc::CosnetArgs ca{};
        ca.om1 = om1, ca.ph1 = ph1, ca.om2 = om2, ca.ph2 = ph2, ca.M = M;
        ca.M2 = c3->M2, ca.om3 = c3->om3, ca.ph3 = c3->ph3;
        ca.h_in = (const float *)(saved + SL.h), ca.b_in = (const float *)(saved + SL.b);
        ca.b2_in = (const float *)(saved + SL.b2);
        ca.dh_out = dh, ca.a_out = a, ca.db_out = db, ca.part = cpart;
        ca.a2_out = (bf16 *)(ws + WL.a2), ca.db2_out = (bf16 *)(ws + WL.db2);
        ca.bias_part = dbias ? bpart : nullptr;
        ca.kdim = dout;
        NOBLE_TRY(with_rank_tile_max128(r, [&](auto bn) {
            constexpr int R = decltype(bn)::value;
            return cosnet_launch<R, true, tc::kSigCos3>(st, "tc_dc_cosnet_bwd", T, dy, dout, W_up, ca);
        }));
        NOBLE_TRY(reduce_cosnet(cpart, dbias ? bpart : nullptr));
    } else if (r > 0 && c3) {
        // three-layer cosine, r = 256: dc = dy W_up on the tensor cores (fp32 out),
        // the chain rule on the CUDA cores (bf16 a, db, a2, db2 for the weight gradients)
        float *dc = (float *)(ws + WL.dc);
        const ProbSpec Pc{T, r, TcSeg{dy, W_up, dout}, nullptr, r <= 128 ? 128 : 256};
        const tc::EpiStore<float>::Params Ec{dc, r, nullptr, 0};
        if (mn4_ok({r}, {dout}))
            NOBLE_TRY((tc_pair_group<false, true, tc::EpiStore<float>, true>(st, "tc_dc_gemm", 1, &Pc, &Ec)));
        else
            NOBLE_TRY((tc_pair_group<false, true, tc::EpiStore<float>>(st, "tc_dc_gemm", 1, &Pc, &Ec)));
        bf16 *a2 = (bf16 *)(ws + WL.a2), *db2 = (bf16 *)(ws + WL.db2);
        NOBLE_TRY((cos3_bwd_rows<bf16, bf16>(d, saved, dc, om1, ph1, M, om2, ph2, c3, dh, a, db, a2, db2,
                                             (float *)(ws + WL.cos_part), dom1, dph1, dom2, dph2, st)));
    } else if (r > 0 && !fused) {
        float *cpart = (float *)(ws + WL.cos_part);
        tc::CosnetArgs ca{};
        ca.om1 = om1, ca.ph1 = ph1, ca.om2 = om2, ca.ph2 = ph2, ca.M = M;
        ca.h_in = (const float *)(saved + SL.h), ca.b_in = (const float *)(saved + SL.b);
        ca.dh_out = dh, ca.a_out = a, ca.db_out = db, ca.part = cpart;
        float *bpart = (float *)(ws + WL.bias_part);
        ca.bias_part = dbias ? bpart : nullptr;
        ca.kdim = dout;
        ca.act = sg.act;
        NOBLE_TRY(with_rank_tile(r, [&](auto bn) {
            constexpr int R = decltype(bn)::value;
            const char *nm = "tc_dc_cosnet_bwd";
            switch (sg.sig) {
            case tc::kSigCos1: return cosnet_launch<R, true, tc::kSigCos1>(st, nm, T, dy, dout, W_up, ca);
            case tc::kSigIdentity: return cosnet_launch<R, true, tc::kSigIdentity>(st, nm, T, dy, dout, W_up, ca);
            case tc::kSigAct1: return cosnet_launch<R, true, tc::kSigAct1>(st, nm, T, dy, dout, W_up, ca);
            case tc::kSigAct2: return cosnet_launch<R, true, tc::kSigAct2>(st, nm, T, dy, dout, W_up, ca);
            default: return cosnet_launch<R, true, tc::kSigCosnet>(st, nm, T, dy, dout, W_up, ca);
            }
        }));
        NOBLE_TRY(reduce_cosnet(cpart, dbias ? bpart : nullptr));
    }
    // dx = [dy | dh] [W ; W_down]
    if (fused) {
        // one launch: per row pair a leader tile dy [W cols 0..r | W_up] (the
        // first r columns of dx, dc beside them; the CosNet chain rule and the
        // dbias partials in its epilogue, then + dh W_down), and the dx tiles
        // of columns [r, d_in)
        uint32_t *flags = (uint32_t *)(ws + WL.flags);
        if (memset_async(flags, 0, fuse_flag_bytes(d), st) != cudaSuccess)
            return fail(NOBLE_ERR_CUDA, "flags: %s", cudaGetErrorString(cudaGetLastError()));
        float *cpart = (float *)(ws + WL.cos_part);
        float *bpart = (float *)(ws + WL.bias_part);
        tc::pair::FuseArgs fa{};
        fa.T = T, fa.r = (int)r;
        fa.om1 = om1, fa.ph1 = ph1, fa.om2 = om2, fa.ph2 = ph2, fa.M = M;
        fa.h_in = (const float *)(saved + SL.h), fa.b_in = (const float *)(saved + SL.b);
        fa.dh_out = dh, fa.a_out = a, fa.db_out = db, fa.part = cpart, fa.flags = flags;
        fa.bias_part = dbias ? bpart : nullptr;
        fa.kdim = dout;
        const FusedSplit fs = fused_split(di, r);
        const int64_t o2 = r + fs.nfull;
        const tc::EpiStore<bf16>::Params E[3] = {
            {dx, di, nullptr, 0}, {dx + r, di, nullptr, 0}, {dx + o2, di, nullptr, 0}};
        // MN-major B operands: column ranges of W [d_out][d_in] and W_down [r][d_in]
        const TcSeg s0L{dy, W, dout, di}, s1L{dh, W_down, r, di};
        const TcSeg s0O{dy, W + r, dout, di}, s1O{dh, W_down + r, r, di};
        const TcSeg s0T{dy, W + o2, dout, di}, s1T{dh, W_down + o2, r, di};
        ProbSpec P[3] = {ProbSpec{T, r, s0L, &s1L, 2 * (int)r}, ProbSpec{T, fs.nfull, s0O, &s1O, 256},
                         ProbSpec{T, fs.ntail, s0T, &s1T, 128}};
        P[0].B0_rank1 = W_up;
        NOBLE_TRY((tc_pair_group<false, true, tc::EpiStore<bf16>, true, tc::pair::kFuseBwd>(st, "tc_dx", 3, P, E,
                                                                                           &fa)));
        NOBLE_TRY(reduce_cosnet(cpart, dbias ? bpart : nullptr));
    } else {
        const tc::EpiStore<bf16>::Params px{dx, di, nullptr, 0};
        const TcSeg sdx2{dh, W_down, r};
        ProbSpec P{T, di, TcSeg{dy, W, dout}, r > 0 ? &sdx2 : nullptr, 256};
        P.dep = r > 0 ? 2 : 0;  // dh, written by the bottleneck kernel
        if (mn4_ok({di}, {dout, r}))
            NOBLE_TRY((tc_pair_group<false, true, tc::EpiStore<bf16>, true>(st, "tc_dx", 1, &P, &px)));
        else
            NOBLE_TRY((tc_pair_group<false, true, tc::EpiStore<bf16>>(st, "tc_dx", 1, &P, &px)));
    }
    // every token-summed product in one launch: dW_down = dh^T x, dW_up = dy^T c,
    // dM = a^T db, dbias = dy^T 1, dW = dy^T x
    {
        const bf16 *c = r > 0 ? (const bf16 *)(saved + SL.c) : nullptr;
        ProbSpec P[kWgradKinds];
        tc::EpiStore<float>::Params E[kWgradKinds];
        float *final_out[kWgradKinds];
        int64_t mn[kWgradKinds][2];
        wgrad_shapes(d, mn);
        int which[kWgradKinds];
        int n = 0;
        auto add = [&](int k, ProbSpec ps, float *out, int64_t ldc, bool col0, bool transpose = false) {
            // dW_down (dh), dM (a, db), dbias (the ones operand), dM2 (a2, db2) read
            // what earlier kernels of this call wrote; dW and dW_up read the inputs
            ps.dep = (k == 1 || k == 3 || k == 4 || k == 5) ? 1 : 0;
            P[n] = ps;
            E[n] = {out, ldc, nullptr, 0};
            E[n].col0 = col0 ? 1 : 0;
            E[n].transpose = transpose ? 1 : 0;
            final_out[n] = out;
            which[n++] = k;
        };
        // heaviest tiles first: the round-robin tile walk then fills the
        // CTAs that drew fewer full tiles with the small ones
        add(0, ProbSpec{dout, di, TcSeg{dy, x, T}, nullptr, 256}, dW, di, false);
        if (r > 0) {
            // dW_down^T = x^T dh (d_in x r), stored transposed: M = d_in fills
            // whole 256-row pair tiles where M = r would leave half of each empty
            add(1, ProbSpec{di, r, TcSeg{x, dh, T}, nullptr, r < 128 ? 128 : (int)r}, dW_down, di, false, true);
            add(2, ProbSpec{dout, r, TcSeg{dy, c, T}, nullptr, r < 128 ? 128 : (int)r}, dW_up, r, false);
            if (sg.two_layers())
                add(3, ProbSpec{r, r, TcSeg{a, db, T}, nullptr, r < 128 ? 128 : (int)r}, dM, r, false);
            if (c3) {
                const bf16 *a2 = (const bf16 *)(ws + WL.a2), *db2 = (const bf16 *)(ws + WL.db2);
                add(5, ProbSpec{r, r, TcSeg{a2, db2, T}, nullptr, r < 128 ? 128 : (int)r}, c3->dM2, r, false);
            }
            else if (memset_async(dM, 0, (size_t)r * r * 4, st) != cudaSuccess)
                return fail(NOBLE_ERR_CUDA, "dM: %s", cudaGetErrorString(cudaGetLastError()));
        }
        if (ones_dbias) add(4, ProbSpec{dout, kOnesCols, TcSeg{dy, ones, T}, nullptr, 128}, dbias, 1, true);
        const int split = WL.split;
        SplitJobs J{};
        if (split > 1) {
            const int kbt = (int)ceil_div(T, tc::kBK);
            const int per = (int)ceil_div(kbt, split);
            J.nparts = (int)ceil_div(kbt, per);
            J.begin[0] = 0;
            for (int i = 0; i < n; ++i) {
                const int k = which[i];
                float *part = (float *)(ws + WL.wsplit[k]);
                P[i].nsplit = J.nparts;
                P[i].kb_per_split = per;
                E[i].C = part;
                E[i].split_stride = mn[k][0] * mn[k][1];
                J.part[i] = part;
                J.out[i] = final_out[i];
                J.n[i] = mn[k][0] * mn[k][1];
                J.stride[i] = J.n[i];
                J.begin[i + 1] = J.begin[i] + J.n[i];
            }
            J.njobs = n;
        }
        if (mn4_ok({di, dout, r, kOnesCols}, {T}))
            NOBLE_TRY((tc_pair_group<true, true, tc::EpiStore<float>, true>(st, "tc_wgrad", n, P, E)));
        else
            NOBLE_TRY((tc_pair_group<true, true, tc::EpiStore<float>>(st, "tc_wgrad", n, P, E)));
        if (split > 1) {
            const int64_t total = J.begin[J.njobs];
            const KernelInfo kr{"reduce_wgrad_split", kBoundHbm, (double)total * J.nparts,
                                4.0 * total * (J.nparts + 1)};
            bool vec4 = J.nparts <= 8;
            for (int i = 0; i < J.njobs; ++i)
                vec4 = vec4 && J.n[i] % 4 == 0 && J.stride[i] % 4 == 0 &&
                       reinterpret_cast<uintptr_t>(J.out[i]) % 16 == 0 && reinterpret_cast<uintptr_t>(J.part[i]) % 16 == 0;
            const int64_t blocks = std::min<int64_t>(ceil_div(total / 4, 256), 8 * (int64_t)num_sms());
            const bool pdl = pdl_ok();
            NOBLE_TRY(run(st, kr, [&] {
                if (vec4)
                    launch_maybe_pdl(reduce_split_vec4_kernel, dim3((unsigned)blocks), dim3(256), 0, st, pdl, J);
                else
                    launch_maybe_pdl(reduce_split_kernel, dim3((unsigned)ceil_div(total, 32)), dim3(256), 0, st,
                                     pdl, J);
            }));
        }
    }
    return NOBLE_OK;
}

// Test kernel for the device-side expiry of a bounded wait: one thread waits,
// through mbar_wait_limit (the wait every pipeline kernel uses), on an
// mbarrier that nothing arrives at; nothing else is outstanding (no copy, no
// MMA), so the kernel records the timeout in the status word and exits.
__global__ void wait_expiry_kernel(uint64_t limit_ns, uint32_t *status, uint32_t *result)
{
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x != 0) return;
    const uint32_t b = ptx::smem_u32(&bar);
    ptx::mbar_init(b, 1);
    ptx::fence_barrier_init();
    const bool ok = ptx::mbar_wait_limit(b, 0, status, limit_ns);
    *result = ok ? 1u : 2u;
}

noble_status zero_grads(const noble_linear_desc *d, float *dW, float *dbias, float *dW_down, float *dM,
                        float *dom1, float *dph1, float *dom2, float *dph2, float *dW_up,
                        cudaStream_t st)
{
    const size_t di = d->d_in, dout = d->d_out, r = d->r;
    struct { void *p; size_t n; } z[] = {{dW, di * dout}, {dbias, dout}, {dW_down, r * di}, {dM, r * r},
                                        {dom1, r}, {dph1, r}, {dom2, r}, {dph2, r}, {dW_up, dout * r}};
    for (auto &e : z)
        if (e.p && e.n && cudaMemsetAsync(e.p, 0, e.n * 4, st) != cudaSuccess)
            return fail(NOBLE_ERR_CUDA, "cudaMemsetAsync: %s", cudaGetErrorString(cudaGetLastError()));
    return NOBLE_OK;
}

}  // namespace
}  // namespace noble

using namespace noble;

extern "C" {

size_t noble_linear_saved_bytes(const noble_linear_desc *desc)
{
    if (validate_desc(desc) != NOBLE_OK) return 0;
    return saved_layout(desc).total;
}

size_t noble_linear_bwd_workspace_bytes(const noble_linear_desc *desc)
{
    if (validate_desc(desc) != NOBLE_OK) return 0;
    return work_layout(desc).total;
}

// The forward entry point; c3 non-NULL for noble_linear_fwd_cos3.
static noble_status fwd_entry(const noble_linear_desc *desc, const void *x, const void *W, const float *bias,
                              const void *W_down, const float *omega1, const float *phi1, const float *M,
                              const float *omega2, const float *phi2, const void *W_up, void *y, void *saved,
                              size_t saved_bytes, noble_stream stream, const Cos3 *c3)
{
    g_last_error[0] = 0;
    g_call_kernels = 0;
    NOBLE_TRY(validate_desc(desc));
    const bool br = desc->r > 0, empty = desc->T == 0;
    if (((desc->flags & kFlagSigmaCos3) != 0) != (c3 != nullptr))
        return fail(NOBLE_ERR_INVALID_ARG, c3 ? "noble_linear_fwd_cos3 needs NOBLE_FLAG_SIGMA_COS3"
                                              : "a NOBLE_FLAG_SIGMA_COS3 descriptor needs noble_linear_fwd_cos3");
    if (c3) {
        NOBLE_TRY(check_ptr(c3->M2, "M2", !br));
        NOBLE_TRY(check_ptr(c3->om3, "omega3", !br));
        NOBLE_TRY(check_ptr(c3->ph3, "phi3", !br));
    }
    const Cos3 *k3 = is_cos3(desc) ? c3 : nullptr;
    NOBLE_TRY(check_ptr(x, "x", empty));
    NOBLE_TRY(check_ptr(W, "W", false));
    NOBLE_TRY(check_ptr(bias, "bias", true));
    NOBLE_TRY(check_ptr(y, "y", empty));
    // parameters the bottleneck variant does not use may be NULL
    const Sigma sg = sigma_of(desc);
    NOBLE_TRY(check_ptr(W_down, "W_down", !br));
    NOBLE_TRY(check_ptr(omega1, "omega1", !br || !sg.first_phase()));
    NOBLE_TRY(check_ptr(phi1, "phi1", !br || !sg.first_phase()));
    NOBLE_TRY(check_ptr(M, "M", !br || !sg.two_layers()));
    NOBLE_TRY(check_ptr(omega2, "omega2", !br || !sg.second_phase()));
    NOBLE_TRY(check_ptr(phi2, "phi2", !br || !sg.second_phase()));
    NOBLE_TRY(check_ptr(W_up, "W_up", !br));
    NOBLE_TRY(check_ptr(saved, "saved", !br || empty));
    if (saved_bytes < saved_layout(desc).total)
        return fail(NOBLE_ERR_BUFFER_TOO_SMALL, "saved_bytes=%zu < %zu", saved_bytes, saved_layout(desc).total);
    NOBLE_TRY(check_device());
    if (desc->T == 0) return NOBLE_OK;
    cudaStream_t st = (cudaStream_t)stream;
    if (desc->dtype == NOBLE_BF16) {
        using bf = __nv_bfloat16;
        if (!(desc->flags & kFlagSimtOnly))
            return fwd_tc(desc, (const bf *)x, (const bf *)W, bias, (const bf *)W_down, omega1, phi1, M, omega2,
                          phi2, (const bf *)W_up, (bf *)y, (char *)saved, st, k3);
        return fwd_simt<bf>(desc, (const bf *)x, (const bf *)W, bias, (const bf *)W_down, omega1, phi1, M,
                            omega2, phi2, (const bf *)W_up, (bf *)y, (char *)saved, st, k3);
    }
    return fwd_simt<float>(desc, (const float *)x, (const float *)W, bias, (const float *)W_down, omega1,
                           phi1, M, omega2, phi2, (const float *)W_up, (float *)y, (char *)saved, st, k3);
}

noble_status noble_linear_fwd(const noble_linear_desc *desc, const void *x, const void *W,
                              const float *bias, const void *W_down, const float *omega1,
                              const float *phi1, const float *M, const float *omega2,
                              const float *phi2, const void *W_up, void *y, void *saved,
                              size_t saved_bytes, noble_stream stream)
{
    return fwd_entry(desc, x, W, bias, W_down, omega1, phi1, M, omega2, phi2, W_up, y, saved, saved_bytes, stream,
                     nullptr);
}

noble_status noble_linear_fwd_cos3(const noble_linear_desc *desc, const void *x, const void *W,
                                   const float *bias, const void *W_down, const float *omega1,
                                   const float *phi1, const float *M, const float *omega2,
                                   const float *phi2, const noble_cos3_params *p3, const void *W_up,
                                   void *y, void *saved, size_t saved_bytes, noble_stream stream)
{
    g_last_error[0] = 0;
    if (!p3) return fail(NOBLE_ERR_INVALID_ARG, "p3 is NULL");
    const Cos3 c3{p3->M2, p3->omega3, p3->phi3, nullptr, nullptr, nullptr};
    return fwd_entry(desc, x, W, bias, W_down, omega1, phi1, M, omega2, phi2, W_up, y, saved, saved_bytes, stream,
                     &c3);
}

// The backward entry point; c3 non-NULL for noble_linear_bwd_cos3.
static noble_status bwd_entry(const noble_linear_desc *desc, const void *dy, const void *x, const void *W,
                              const void *W_down, const float *omega1, const float *phi1, const float *M,
                              const float *omega2, const float *phi2, const void *W_up, const void *saved,
                              size_t saved_bytes, void *dx, float *dW, float *dbias, float *dW_down, float *dM,
                              float *domega1, float *dphi1, float *domega2, float *dphi2, float *dW_up,
                              void *workspace, size_t workspace_bytes, noble_stream stream, const Cos3 *c3)
{
    g_last_error[0] = 0;
    g_call_kernels = 0;
    NOBLE_TRY(validate_desc(desc));
    if (((desc->flags & kFlagSigmaCos3) != 0) != (c3 != nullptr))
        return fail(NOBLE_ERR_INVALID_ARG, c3 ? "noble_linear_bwd_cos3 needs NOBLE_FLAG_SIGMA_COS3"
                                              : "a NOBLE_FLAG_SIGMA_COS3 descriptor needs noble_linear_bwd_cos3");
    if (c3) {
        const bool br3 = desc->r > 0;
        const char *n3[] = {"M2", "omega3", "phi3", "dM2", "domega3", "dphi3"};
        const void *p3[] = {c3->M2, c3->om3, c3->ph3, c3->dM2, c3->dom3, c3->dph3};
        for (int i = 0; i < 6; ++i) NOBLE_TRY(check_ptr(p3[i], n3[i], !br3));
    }
    const Cos3 *k3 = is_cos3(desc) ? c3 : nullptr;
    if (desc->flags & kFlagInference)
        return fail(NOBLE_ERR_INVALID_ARG, "backward of an inference descriptor (NOBLE_FLAG_INFERENCE)");
    const bool br = desc->r > 0, empty = desc->T == 0;
    const char *names[] = {"dy", "x", "dx", "W", "dW", "workspace"};
    const void *req[] = {dy, x, dx, W, dW, workspace};
    for (int i = 0; i < 6; ++i) NOBLE_TRY(check_ptr(req[i], names[i], empty && i < 3));
    NOBLE_TRY(check_ptr(dbias, "dbias", true));
    const char *bnames[] = {"W_down", "omega1", "phi1", "M", "omega2", "phi2", "W_up", "saved",
                            "dW_down", "dM", "domega1", "dphi1", "domega2", "dphi2", "dW_up"};
    const void *bptr[] = {W_down, omega1, phi1, M, omega2, phi2, W_up, saved,
                          dW_down, dM, domega1, dphi1, domega2, dphi2, dW_up};
    const Sigma sg = sigma_of(desc);
    // inputs the bottleneck variant does not use may be NULL; every gradient
    // output is written (zeros for unused parameters)
    auto unused = [&](int i) {
        return ((i == 1 || i == 2) && !sg.first_phase()) || (i == 3 && !sg.two_layers()) ||
               ((i == 4 || i == 5) && !sg.second_phase());
    };
    for (int i = 0; i < 15; ++i) NOBLE_TRY(check_ptr(bptr[i], bnames[i], !br || (empty && i == 7) || unused(i)));
    if (saved_bytes < saved_layout(desc).total)
        return fail(NOBLE_ERR_BUFFER_TOO_SMALL, "saved_bytes=%zu < %zu", saved_bytes, saved_layout(desc).total);
    if (workspace_bytes < work_layout(desc).total)
        return fail(NOBLE_ERR_BUFFER_TOO_SMALL, "workspace_bytes=%zu < %zu", workspace_bytes,
                    work_layout(desc).total);
    NOBLE_TRY(check_device());
    cudaStream_t st = (cudaStream_t)stream;
    if (desc->T == 0) {
        if (k3) {
            const int64_t r = desc->r;
            if (cudaMemsetAsync(k3->dM2, 0, (size_t)r * r * 4, st) != cudaSuccess ||
                cudaMemsetAsync(k3->dom3, 0, (size_t)r * 4, st) != cudaSuccess ||
                cudaMemsetAsync(k3->dph3, 0, (size_t)r * 4, st) != cudaSuccess)
                return fail(NOBLE_ERR_CUDA, "zero gradients: %s", cudaGetErrorString(cudaGetLastError()));
        }
        return zero_grads(desc, dW, dbias, dW_down, dM, domega1, dphi1, domega2, dphi2, dW_up, st);
    }
    if (desc->dtype == NOBLE_BF16) {
        using bf = __nv_bfloat16;
        if (!(desc->flags & kFlagSimtOnly))
            return bwd_tc(desc, (const bf *)dy, (const bf *)x, (const bf *)W, (const bf *)W_down, omega1, phi1, M,
                          omega2, phi2, (const bf *)W_up, (const char *)saved, (bf *)dx, dW, dbias, dW_down, dM,
                          domega1, dphi1, domega2, dphi2, dW_up, (char *)workspace, st, k3);
        return bwd_simt<bf>(desc, (const bf *)dy, (const bf *)x, (const bf *)W, (const bf *)W_down, omega1,
                            phi1, M, omega2, phi2, (const bf *)W_up, (const char *)saved, (bf *)dx, dW,
                            dbias, dW_down, dM, domega1, dphi1, domega2, dphi2, dW_up, (char *)workspace,
                            st, k3);
    }
    return bwd_simt<float>(desc, (const float *)dy, (const float *)x, (const float *)W, (const float *)W_down,
                           omega1, phi1, M, omega2, phi2, (const float *)W_up, (const char *)saved,
                           (float *)dx, dW, dbias, dW_down, dM, domega1, dphi1, domega2, dphi2, dW_up,
                           (char *)workspace, st, k3);
}

noble_status noble_linear_bwd(const noble_linear_desc *desc, const void *dy, const void *x,
                              const void *W, const void *W_down, const float *omega1,
                              const float *phi1, const float *M, const float *omega2,
                              const float *phi2, const void *W_up, const void *saved,
                              size_t saved_bytes, void *dx,
                              float *dW, float *dbias, float *dW_down, float *dM, float *domega1,
                              float *dphi1, float *domega2, float *dphi2, float *dW_up,
                              void *workspace, size_t workspace_bytes, noble_stream stream)
{
    return bwd_entry(desc, dy, x, W, W_down, omega1, phi1, M, omega2, phi2, W_up, saved, saved_bytes, dx, dW, dbias,
                     dW_down, dM, domega1, dphi1, domega2, dphi2, dW_up, workspace, workspace_bytes, stream, nullptr);
}

noble_status noble_linear_bwd_cos3(const noble_linear_desc *desc, const void *dy, const void *x,
                                   const void *W, const void *W_down, const float *omega1,
                                   const float *phi1, const float *M, const float *omega2,
                                   const float *phi2, const noble_cos3_params *p3, const void *W_up,
                                   const void *saved, size_t saved_bytes, void *dx, float *dW,
                                   float *dbias, float *dW_down, float *dM, float *domega1,
                                   float *dphi1, float *domega2, float *dphi2,
                                   const noble_cos3_grads *g3, float *dW_up, void *workspace,
                                   size_t workspace_bytes, noble_stream stream)
{
    g_last_error[0] = 0;
    if (!p3 || !g3) return fail(NOBLE_ERR_INVALID_ARG, "p3 or g3 is NULL");
    const Cos3 c3{p3->M2, p3->omega3, p3->phi3, g3->dM2, g3->domega3, g3->dphi3};
    return bwd_entry(desc, dy, x, W, W_down, omega1, phi1, M, omega2, phi2, W_up, saved, saved_bytes, dx, dW, dbias,
                     dW_down, dM, domega1, dphi1, domega2, dphi2, dW_up, workspace, workspace_bytes, stream, &c3);
}

noble_status noble_get_device_status(noble_stream stream)
{
    g_last_error[0] = 0;
    cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e != cudaSuccess) return fail(NOBLE_ERR_CUDA, "stream: %s", cudaGetErrorString(e));
    uint32_t v = 0, zero = 0;
    e = cudaMemcpyFromSymbol(&v, g_device_status, sizeof(v));
    if (e == cudaSuccess && v) e = cudaMemcpyToSymbol(g_device_status, &zero, sizeof(zero));
    if (e != cudaSuccess) return fail(NOBLE_ERR_CUDA, "status word: %s", cudaGetErrorString(e));
    if (v & kStatusTimeout) return fail(NOBLE_ERR_TIMEOUT, "a kernel gave up a bounded wait (status 0x%x)", v);
    if (v) return fail(NOBLE_ERR_CUDA, "device status 0x%x", v);
    return NOBLE_OK;
}

noble_status noble_debug_raise_device_status(uint32_t bits)
{
    uint32_t v = 0;
    cudaError_t e = cudaMemcpyFromSymbol(&v, g_device_status, sizeof(v));
    v |= bits;
    if (e == cudaSuccess) e = cudaMemcpyToSymbol(g_device_status, &v, sizeof(v));
    if (e != cudaSuccess) return fail(NOBLE_ERR_CUDA, "status word: %s", cudaGetErrorString(e));
    return NOBLE_OK;
}

noble_status noble_debug_wait_expiry(uint64_t limit_ns, uint32_t *result, noble_stream stream)
{
    g_last_error[0] = 0;
    if (!result) return fail(NOBLE_ERR_INVALID_ARG, "result is NULL");
    if (limit_ns == 0 || limit_ns > 100000000ull)
        return fail(NOBLE_ERR_INVALID_ARG, "limit_ns must be in (0, 100 ms]");
    NOBLE_TRY(check_device());
    uint32_t *status = status_ptr();
    if (!status) return fail(NOBLE_ERR_CUDA, "status word address");
    wait_expiry_kernel<<<1, 32, 0, (cudaStream_t)stream>>>(limit_ns, status, result);
    return check_launch("wait_expiry_kernel");
}

const char *noble_status_string(noble_status s)
{
    switch (s) {
    case NOBLE_OK: return "ok";
    case NOBLE_ERR_INVALID_ARG: return "invalid argument";
    case NOBLE_ERR_MISALIGNED: return "pointer not 16-byte aligned";
    case NOBLE_ERR_UNSUPPORTED: return "unsupported shape, rank, dtype or flag";
    case NOBLE_ERR_BUFFER_TOO_SMALL: return "buffer too small";
    case NOBLE_ERR_CUDA: return "CUDA error";
    case NOBLE_ERR_TIMEOUT: return "device-side wait timed out";
    case NOBLE_ERR_NO_DEVICE: return "no usable sm_103 device";
    }
    return "unknown status";
}

const char *noble_last_error(void) { return g_last_error; }

// Device address of g_noalloc_scratch in the current context.
static noble_status noalloc_scratch_ptr(void **out)
{
    void *p = noble::symbol_address(g_noalloc_scratch);
    if (!p) return fail(NOBLE_ERR_CUDA, "cudaGetSymbolAddress(static scratch) failed");
    *out = p;
    return NOBLE_OK;
}

noble_status noble_linear_bwd_noalloc(const noble_linear_desc *desc, const void *dy, const void *x,
                                      const void *W, const void *W_down, const float *omega1,
                                      const float *phi1, const float *M, const float *omega2,
                                      const float *phi2, const void *W_up, const void *saved,
                                      size_t saved_bytes, void *dx, float *dW, float *dbias,
                                      float *dW_down, float *dM, float *domega1, float *dphi1,
                                      float *domega2, float *dphi2, float *dW_up, noble_stream stream)
{
    g_last_error[0] = 0;
    NOBLE_TRY(validate_desc(desc));
    if (desc->flags & kFlagInference)
        return fail(NOBLE_ERR_INVALID_ARG, "backward of an inference descriptor (NOBLE_FLAG_INFERENCE)");
    const size_t need = work_layout(desc).total;
    if (need > kNoallocScratchBytes)
        return fail(NOBLE_ERR_BUFFER_TOO_SMALL,
                    "this shape needs %zu bytes of backward scratch; the static scratch of "
                    "noble_linear_bwd_noalloc holds %zu (use noble_linear_bwd with a workspace)",
                    need, kNoallocScratchBytes);
    NOBLE_TRY(check_device());
    void *scratch = nullptr;
    NOBLE_TRY(noalloc_scratch_ptr(&scratch));
    return noble_linear_bwd(desc, dy, x, W, W_down, omega1, phi1, M, omega2, phi2, W_up, saved, saved_bytes, dx,
                            dW, dbias, dW_down, dM, domega1, dphi1, domega2, dphi2, dW_up, scratch,
                            kNoallocScratchBytes, stream);
}

noble_status noble_adamw_step(const noble_adamw_tensor *tensors, int n_tensors, const noble_adamw_hparams *hp,
                              noble_stream stream)
{
    g_last_error[0] = 0;
    if (n_tensors < 0 || (n_tensors > 0 && !tensors) || !hp) return fail(NOBLE_ERR_INVALID_ARG, "tensors / hparams");
    if (hp->step < 1 || !(hp->lr >= 0.f) || !(hp->beta1 >= 0.f && hp->beta1 < 1.f) ||
        !(hp->beta2 >= 0.f && hp->beta2 < 1.f) || !(hp->eps > 0.f) || !(hp->weight_decay >= 0.f))
        return fail(NOBLE_ERR_INVALID_ARG, "hyperparameters (step %lld)", (long long)hp->step);
    for (int i = 0; i < n_tensors; ++i) {
        const noble_adamw_tensor &t = tensors[i];
        if (t.n < 0 || !(t.lr_mult >= 0.f)) return fail(NOBLE_ERR_INVALID_ARG, "tensor %d: n or lr_mult", i);
        const bool empty = t.n == 0;
        NOBLE_TRY(check_ptr(t.param, "param", empty));
        NOBLE_TRY(check_ptr(t.grad, "grad", empty));
        NOBLE_TRY(check_ptr(t.exp_avg, "exp_avg", empty));
        NOBLE_TRY(check_ptr(t.exp_avg_sq, "exp_avg_sq", empty));
        if (reinterpret_cast<uintptr_t>(t.param_bf16) % 8)
            return fail(NOBLE_ERR_MISALIGNED, "tensor %d: param_bf16 is not 8-byte aligned", i);
    }
    if (n_tensors == 0) return NOBLE_OK;
    NOBLE_TRY(check_device());
    cudaStream_t st = (cudaStream_t)stream;
    const double bc1 = 1.0 - std::pow((double)hp->beta1, (double)hp->step);
    const double bc2 = 1.0 - std::pow((double)hp->beta2, (double)hp->step);
    for (int i0 = 0; i0 < n_tensors; i0 += opt::kAdamwMaxTensors) {
        const int nt = std::min(opt::kAdamwMaxTensors, n_tensors - i0);
        opt::AdamwBatch b{};
        b.beta1 = hp->beta1, b.beta2 = hp->beta2, b.eps = hp->eps;
        b.inv_bc1 = (float)(1.0 / bc1), b.inv_sqrt_bc2 = (float)(1.0 / std::sqrt(bc2));
        int64_t nmax = 0;
        double bytes = 0;
        for (int j = 0; j < nt; ++j) {
            const noble_adamw_tensor &t = tensors[i0 + j];
            opt::AdamwTensor &d = b.t[j];
            d.p = t.param, d.p_bf16 = (__nv_bfloat16 *)t.param_bf16, d.g = t.grad, d.m = t.exp_avg;
            d.v = t.exp_avg_sq, d.n = t.n;
            d.lr = hp->lr * t.lr_mult;
            d.decay = t.decay ? d.lr * hp->weight_decay : 0.f;
            d.vec4 = t.n % 4 == 0 ? 1 : 0;  // pointers are 16-byte aligned (checked)
            nmax = std::max(nmax, t.n);
            bytes += (28.0 + (t.param_bf16 ? 2.0 : 0.0)) * t.n;
        }
        const unsigned gx = (unsigned)std::max<int64_t>(1, std::min<int64_t>(ceil_div(ceil_div(nmax, 4), 256),
                                                                             4 * (int64_t)num_sms()));
        const KernelInfo ki{"adamw_step", kBoundHbm, 0.0, bytes};
        NOBLE_TRY(run(st, ki, [&] { opt::adamw_kernel<<<dim3(gx, (unsigned)nt), 256, 0, st>>>(b); }));
    }
    return NOBLE_OK;
}

noble_status noble_linear_grad_bucket(const noble_linear_desc *desc, noble_grad_bucket *out)
{
    g_last_error[0] = 0;
    if (!desc || !out) return fail(NOBLE_ERR_INVALID_ARG, "desc / out is NULL");
    NOBLE_TRY(validate_desc(desc));
    const int64_t di = desc->d_in, dout = desc->d_out, r = desc->r;
    const bool cos3 = (desc->flags & kFlagSigmaCos3) != 0 && r > 0;
    // element counts in the documented order; absent gradients take no room
    const int64_t n[NOBLE_GRAD_COUNT] = {dout * di, dout, r * di, dout * r, r * r, r, r, r, r,
                                         cos3 ? r * r : 0, cos3 ? r : 0, cos3 ? r : 0};
    size_t off = 0;
    for (int i = 0; i < NOBLE_GRAD_COUNT; ++i) {
        out->offset[i] = off;
        out->count[i] = (size_t)n[i];
        off += ((size_t)n[i] * sizeof(float) + NOBLE_GRAD_ALIGN - 1) / NOBLE_GRAD_ALIGN * NOBLE_GRAD_ALIGN;
    }
    out->total_bytes = off;
    return NOBLE_OK;
}

noble_status noble_linear_lr_multipliers(const noble_linear_desc *desc, float gamma, float gamma_M, float omega_mult,
                                         float phi_mult, float out[5])
{
    g_last_error[0] = 0;
    if (!desc || !out) return fail(NOBLE_ERR_INVALID_ARG, "desc / out is NULL");
    NOBLE_TRY(validate_desc(desc));
    if (desc->r == 0) return fail(NOBLE_ERR_INVALID_ARG, "r == 0: no branch groups");
    const double rho = (double)std::min(desc->d_in, desc->d_out) / (double)desc->r;
    out[0] = 1.f;
    out[1] = (float)std::pow(rho, 2.0 * gamma);
    out[2] = (float)std::pow(rho, (double)gamma_M);
    out[3] = omega_mult;
    out[4] = phi_mult;
    return NOBLE_OK;
}

noble_status noble_test_gemm_bf16(int64_t M, int64_t N, int64_t K0, int64_t K1, int a_mn, int b_mn, int bn,
                                  const void *A0, const void *B0, const void *A1, const void *B1,
                                  const float *bias, void *C, int c_fp32, int kb_per_split, int nsplit,
                                  noble_stream stream)
{
    g_last_error[0] = 0;
    g_call_kernels = 0;
    // the innermost dimension of every operand must be a multiple of 8 elements (16 bytes)
    if (M <= 0 || N <= 0 || K0 <= 0 || K1 < 0 || nsplit < 1 || N % 8 || (a_mn && M % 8) ||
        (!(a_mn && b_mn) && (K0 % 8 || K1 % 8)))
        return fail(NOBLE_ERR_INVALID_ARG, "bad GEMM sizes");
    const void *ptrs[] = {A0, B0, C};
    for (const void *p : ptrs) NOBLE_TRY(check_ptr(p, "operand", false));
    if (K1 > 0) {
        NOBLE_TRY(check_ptr(A1, "A1", false));
        NOBLE_TRY(check_ptr(B1, "B1", false));
    }
    NOBLE_TRY(check_device());
    cudaStream_t st = (cudaStream_t)stream;
    const TcSeg s0{A0, B0, K0}, s1v{A1, B1, K1};
    const TcSeg *s1 = K1 > 0 ? &s1v : nullptr;
    const int64_t split_stride = nsplit > 1 ? M * N : 0;
    const tc::EpiStore<float>::Params pf{(float *)C, N, bias, split_stride};
    const tc::EpiStore<bf16>::Params pb{(bf16 *)C, N, bias, split_stride};
    // N tiles of 128 and 256 run on CTA pairs (the product path's kernel),
    // narrower ones on the single-CTA one-tile kernel
    if ((bn == 128 || bn == 256) && !(a_mn && !b_mn)) {
        const ProbSpec P{M, N, s0, s1, bn, nsplit, kb_per_split};
        // MN-major operands take the 4-D layout when their extents allow it
        const bool mn4 = mn4_ok({a_mn ? M : 64, b_mn ? N : 64}, {K0, K1});
#define NOBLE_PAIR_CASE(AMN, BMN)                                                                           \
    if (a_mn == AMN && b_mn == BMN) {                                                                       \
        if (mn4 && (AMN || BMN))                                                                            \
            return c_fp32 ? tc_pair_group<AMN, BMN, tc::EpiStore<float>, true>(st, "test", 1, &P, &pf)      \
                          : tc_pair_group<AMN, BMN, tc::EpiStore<bf16>, true>(st, "test", 1, &P, &pb);      \
        return c_fp32 ? tc_pair_group<AMN, BMN, tc::EpiStore<float>>(st, "test", 1, &P, &pf)                \
                      : tc_pair_group<AMN, BMN, tc::EpiStore<bf16>>(st, "test", 1, &P, &pb);                \
    }
        NOBLE_PAIR_CASE(false, false)
        NOBLE_PAIR_CASE(false, true)
        NOBLE_PAIR_CASE(true, true)
#undef NOBLE_PAIR_CASE
    }
#define NOBLE_TEST_CASE(BN_, AMN, BMN)                                                                      \
    if (bn == BN_ && a_mn == AMN && b_mn == BMN)                                                            \
        return c_fp32 ? tc_gemm<BN_, AMN, BMN, tc::EpiStore<float>>(st, "test", M, N, s0, s1, kb_per_split,  \
                                                                     nsplit, pf)                            \
                      : tc_gemm<BN_, AMN, BMN, tc::EpiStore<bf16>>(st, "test", M, N, s0, s1, kb_per_split,   \
                                                                    nsplit, pb);
    NOBLE_TEST_CASE(256, false, false)
    NOBLE_TEST_CASE(128, false, false)
    NOBLE_TEST_CASE(64, false, false)
    NOBLE_TEST_CASE(32, false, false)
    NOBLE_TEST_CASE(16, false, false)
    NOBLE_TEST_CASE(256, false, true)
    NOBLE_TEST_CASE(256, true, true)
    NOBLE_TEST_CASE(128, true, true)
    NOBLE_TEST_CASE(64, true, true)
#undef NOBLE_TEST_CASE
    return fail(NOBLE_ERR_UNSUPPORTED, "no GEMM instance for bn=%d a_mn=%d b_mn=%d", bn, a_mn, b_mn);
}

void noble_profile_enable(int on) { Profiler::get().enable(on != 0); }

void noble_profile_reset(void) { Profiler::get().reset(); }

static std::vector<Profiler::Entry> g_profile_snapshot;

int noble_profile_count(void)
{
    g_profile_snapshot = Profiler::get().read();
    return (int)g_profile_snapshot.size();
}

noble_status noble_profile_entry(int i, char *name, size_t name_len, uint64_t *launches, double *ms,
                                 double *flops, double *bytes, int *bound)
{
    if (i < 0 || i >= (int)g_profile_snapshot.size() || !name || name_len == 0)
        return fail(NOBLE_ERR_INVALID_ARG, "profile entry %d out of range", i);
    const Profiler::Entry &e = g_profile_snapshot[i];
    snprintf(name, name_len, "%s", e.name.c_str());
    if (launches) *launches = e.launches;
    if (ms) *ms = e.ms;
    if (flops) *flops = e.flops;
    if (bytes) *bytes = e.bytes;
    if (bound) *bound = e.bound;
    return NOBLE_OK;
}

uint64_t noble_kernel_launch_count(void) { return g_launches.load(); }

}  // extern "C"
