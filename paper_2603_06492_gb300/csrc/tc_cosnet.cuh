// Fused r-wide GEMM + CosNet kernels (one 128-token tile per CTA, N = r).
// Each CTA loads its whole A and B stages with plain TMA copies (no cluster).
//
// Forward (Eq. 2; Eqs. 5-7):   h = x W_down^T             (tcgen05, TMEM cols [0, r))
//   epilogue: a = cos(omega1 h + phi1) -> bf16 tile in shared memory
//             b = a M                    (second tcgen05 MMA, TMEM cols [R_OFF, R_OFF + r))
//             c = cos(omega2 b + phi2)
//   writes h, b (fp32) and c (bf16), each [T][r].
//
// Backward (chain rule through Eq. 2):   dc = dy W_up         (tcgen05)
//   epilogue: du2 = -sin(omega2 b + phi2) dc,  db = omega2 du2 -> bf16 tile
//             da  = db M^T               (second tcgen05 MMA)
//             du1 = -sin(omega1 h + phi1) da,  dh = omega1 du1,  a = cos(omega1 h + phi1)
//   writes dh, a, db (bf16, [T][r]) and per-CTA column sums
//             part[cta][0] = sum du1*h, [1] = sum du1, [2] = sum du2*b, [3] = sum du2
//   (each [r]), reduced over the 128 tokens of the tile in a fixed order.
//   The saved h and b rows are read straight from memory after the main
//   loop: an L2 prefetch of them during the loop cost the streaming more than
//   it saved the epilogue.
//
// The mixing matrix enters as a bf16 K-major operand that the epilogue
// threads build in shared memory from the fp32 M once the main loop is done:
// Mt[j][i] = M[i][j] for the forward (b_j = sum_i a_i M[i][j]) and M itself
// for the backward (da_i = sum_j db_j M[i][j]).  Both
// the row operand (a or db) and the matrix are split into bf16 high and low
// parts, x = x_hi + x_lo, and the product is formed as
//     x_hi M_hi + x_lo M_hi + x_hi M_lo
// with fp32 accumulation, which keeps it close to fp32 accuracy (the dropped
// x_lo M_lo term is about 2^-16 relative).  A single bf16 product would carry
// the rounding of M as an error shared by every token, which the sums over
// tokens of the frequency and phase gradients do not average away.
#pragma once

#include "activations.cuh"
#include "tc_gemm.cuh"

namespace noble {
namespace tc {

struct CosnetArgs {
    int64_t T;
    int kb;              // k-blocks of the main operand (d_in or d_out)
    const float *om1, *ph1, *om2, *ph2;
    const float *M;      // mixing matrix, fp32 [r][r] (b_j = sum_i a_i M[i][j])
    // forward outputs (h_out, b_out NULL: not saved, inference)
    float *h_out, *b_out;
    __nv_bfloat16 *c_out;
    // backward inputs / outputs
    const float *h_in, *b_in;
    __nv_bfloat16 *dh_out, *a_out, *db_out;
    float *part;         // [gridDim.x][4][r] ([6][r] for the three-layer cosine)
    // backward, optional: column sums of dy over this CTA's tokens,
    // [gridDim.x][kdim], accumulated from the dy tiles of the main loop
    float *bias_part;
    int64_t kdim;
    int act;             // kSigAct1 / kSigAct2: the activation (act::kTanh, kLeaky, kGelu)
    uint32_t *status;
    // three-layer cosine (kSigCos3): the second mixing matrix, the third
    // frequency and phase; the forward also writes b2, the backward reads it
    // and writes a2 = cos(omega2 b + phi2) and db2 (part then holds six sums)
    const float *M2, *om3, *ph3;
    float *b2_out;
    const float *b2_in;
    __nv_bfloat16 *a2_out, *db2_out;
};

// TMA maps for the epilogue's row outputs (CosnetCfg::kStgFits): forward h,
// b (fp32) and c (bf16); backward db, dh and a (bf16).  Each is a 2-D map over
// [T][r] with a box of 32 columns by 32 rows (128-byte rows with the 128-byte
// swizzle for fp32, 64-byte rows with the 64-byte swizzle for bf16).
struct CosnetStoreMaps {
    CUtensorMap m[3];
};

// B_MN: the main loop's B operand is MN-major (W_up [d_out][r] as stored, in
// the backward), loaded as 64-wide column chunks of 64 K rows each; otherwise
// it is K-major with R rows (W_down [r][d_in], in the forward).
template <int R, bool B_MN>
struct CosnetCfg {
    // N of the main MMA: an MN-major B is read in whole 64-wide swizzle atoms,
    // so for r < 64 the MMA runs 64 columns wide (the columns past r are
    // zero-filled by the copy and never read back)
    static constexpr int kMainN = B_MN && R < 64 ? 64 : R;
    static constexpr int kRCols = kMainN < 32 ? 32 : kMainN;  // TMEM columns per accumulator
    static constexpr uint32_t kTmemCols = 2 * kRCols;     // h|dc and b|da
    static constexpr int kBChunks = (R + 63) / 64;         // MN-major B: 64-wide column chunks
    // MN-major B with r a multiple of 64 is copied in the interleaved layout
    // [8-row K group][column chunk][8 rows][128 B] (one 4-D copy per CTA and
    // stage); otherwise as column chunks of 64 K rows.
    static constexpr bool kBInterleaved = B_MN && R % 64 == 0;
    static constexpr uint32_t kChunkBytes = kBK * 128;     // one chunk: 64 K rows of 128 bytes
    static constexpr uint32_t kA = kBM * kBK * 2;
    static constexpr uint32_t kB = B_MN ? kBChunks * kChunkBytes : R * kBK * 2;
    static constexpr uint32_t kStage = kA + kB;
    // Epilogue warps: two per TMEM lane quarter, four for r >= 128 (more warps
    // per scheduler hide the latency of the epilogue's dependent steps); a
    // warp takes the 32-column chunks c with (c / 32) % kColGroups == its group.
    static constexpr int kEpiWarps = R >= 128 ? 16 : 8;
    static constexpr int kEpiThreads = 32 * kEpiWarps;
    static constexpr int kColGroups = kEpiWarps / 4;
    static constexpr int kThreads = 64 + kEpiThreads;
    static constexpr int kMkb = (R + 63) / 64;            // k-blocks of the r x r operand
    static constexpr int kKSteps = R < 64 ? R / 16 : 4;   // MMA K-steps per k-block
    static constexpr uint32_t kMkbBytes = 2 * R * 128;    // one k-block of M_hi and M_lo
    static constexpr uint32_t kTileBytes = kMkb * kBM * 128;  // epilogue row-operand tile, bf16
    // frequencies and phases (up to six vectors), per-quarter column sums (up
    // to six per column), barriers
    static constexpr uint32_t kExtra = 6 * R * 4 + 4 * 6 * R * 4 + 256;
    static constexpr uint32_t kFit = (227u * 1024u - 1024u - kExtra) / kStage;
    static constexpr int kStages = kFit > 8 ? 8 : (int)kFit;
    static_assert(kStages >= 2, "pipeline depth");
    // After the main loop the ring holds the hi and lo row-operand tiles and,
    // behind them, the mixing matrix in passes of kChunkKb k-blocks.
    static constexpr uint32_t kRing = kStages * kStage;
    static constexpr int kFitKb = (int)((kRing - 2 * kTileBytes) / kMkbBytes);
    static constexpr int kChunkKb = kFitKb >= kMkb ? kMkb : kFitKb;
    static_assert(kChunkKb >= 1 && kMkb % kChunkKb == 0, "mixing matrix passes");
    static constexpr int kPasses = kMkb / kChunkKb;
    static constexpr uint32_t kMOff = 2 * kTileBytes;  // 1024-aligned
    static constexpr uint32_t kParamOff = kRing;        // omega/phi copies, 6 x R floats
    static constexpr uint32_t kPartOff = kParamOff + 6 * R * 4;  // [4 quarters][6][R] floats
    static constexpr uint32_t kBarOff = kPartOff + 4 * 6 * R * 4;
    // Epilogue outputs through TMA stores: each epilogue warp stages its 32
    // rows of a 32-column chunk and one lane stores them.  Phase 1 (h, or
    // db) stages behind the mixing matrix, 4 KB per warp; phase 2 (b and c,
    // or dh and a) from the start of the ring, 6 KB per warp, once the r x r
    // product has read the operand tile and the matrix.  The two regions do
    // not overlap, so phase 2 never waits for phase 1's copies.
    static constexpr uint32_t kStg1Off = kMOff + kChunkKb * kMkbBytes;
    static constexpr uint32_t kStg1Bytes = 4096, kStg2Bytes = 6144;
    static constexpr bool kStgFits = kPasses == 1 && (R == 64 || R == 128) &&
                                     kStg1Off + kEpiWarps * kStg1Bytes <= kRing &&
                                     kEpiWarps * kStg2Bytes <= kStg1Off;
    static constexpr uint32_t kBytes = kBarOff + 8 * (2 * kStages + 3) + 16;
    static constexpr uint32_t kDynamic = kBytes + 1024;
};

// Cosine and sine of u for the CosNet epilogues: u is reduced to
// [-pi, pi] by the two-constant Cody-Waite method (W. J. Cody, W. Waite,
// "Software Manual for the Elementary Functions", 1980), with 2 pi split into
// its fp32 rounding C1 = 6.2831854820251465 and the remainder
// C2 = 2 pi - C1 = -1.7484555e-7, then evaluated with the hardware sin/cos
// approximation, whose absolute error on [-pi, pi] is about 2^-21.
// The arguments here are |u| < 100 (|omega h| plus |phi|).
__device__ __forceinline__ float reduce_two_pi(float u)
{
    const float k = rintf(u * 0.159154943091895336f);  // 1 / (2 pi)
    float r = fmaf(-k, 6.28318548202514648f, u);
    return fmaf(-k, -1.74845553e-7f, r);
}
__device__ __forceinline__ float cos_reduced(float u) { return __cosf(reduce_two_pi(u)); }
__device__ __forceinline__ float sin_reduced(float u) { return __sinf(reduce_two_pi(u)); }
__device__ __forceinline__ void sincos_reduced(float u, float *s, float *c) { __sincosf(reduce_two_pi(u), s, c); }

// Sum over the warp's 32 lanes of each of 32 columns: on return lane l holds
// the sum of column l.  Fixed butterfly (recursive halving), deterministic.
__device__ __forceinline__ float warp_colsum32(float (&v)[32])
{
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int w = 16; w >= 1; w >>= 1) {
        const bool upper = (lane & w) != 0;
#pragma unroll
        for (int i = 0; i < w; ++i) {
            const float send = upper ? v[i] : v[i + w];
            const float keep = upper ? v[i + w] : v[i];
            v[i] = keep + __shfl_xor_sync(0xffffffffu, send, w);
        }
    }
    return v[0];
}

// Coalesced row segments for the epilogue.  Lane l of a warp owns row
// t0 + l and holds P 16-byte pieces of it (one segment of P * 16 bytes).
// transpose_pieces swaps the lane and piece index bits within groups of P
// lanes (log2 P xor-shuffle stages): afterwards lane l holds, in slot i,
// piece l % P of row (l & ~(P - 1)) + i, so each memory instruction covers
// 32 / P whole row segments instead of 32 scattered 16-byte pieces.  The
// exchange is its own inverse, which the loads use.
template <int P>
__device__ __forceinline__ void transpose_pieces(uint32_t (&w)[P][4])
{
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int m = P / 2; m >= 1; m >>= 1) {
        const bool hi = (lane & m) != 0;
#pragma unroll
        for (int a = 0; a < P; ++a) {
            if (a & m) continue;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const uint32_t send = hi ? w[a][q] : w[a | m][q];
                const uint32_t recv = __shfl_xor_sync(0xffffffffu, send, m);
                if (hi) w[a][q] = recv;
                else w[a | m][q] = recv;
            }
        }
    }
}
// Store the warp's segments: dst = address of the first piece of row t0;
// rows at or past T are skipped.
template <int P>
__device__ __forceinline__ void store_segments(uint32_t (&w)[P][4], void *dst, int64_t pitch, int64_t t0, int64_t T)
{
    transpose_pieces<P>(w);
    const int lane = threadIdx.x & 31;
    const int gb = lane & ~(P - 1);
    uint8_t *p = reinterpret_cast<uint8_t *>(dst) + (lane & (P - 1)) * 16;
#pragma unroll
    for (int i = 0; i < P; ++i)
        if (t0 + gb + i < T)
            *reinterpret_cast<uint4 *>(p + (int64_t)(gb + i) * pitch) = make_uint4(w[i][0], w[i][1], w[i][2], w[i][3]);
}
// Issue the loads of the warp's segments (zeros for rows at or past T);
// transpose_pieces<P>(w) then gives each lane its own row's pieces.
template <int P>
__device__ __forceinline__ void load_segments_raw(uint32_t (&w)[P][4], const void *src, int64_t pitch, int64_t t0,
                                                  int64_t T)
{
    const int lane = threadIdx.x & 31;
    const int gb = lane & ~(P - 1);
    const uint8_t *p = reinterpret_cast<const uint8_t *>(src) + (lane & (P - 1)) * 16;
#pragma unroll
    for (int i = 0; i < P; ++i) {
        uint4 v = make_uint4(0, 0, 0, 0);
        if (t0 + gb + i < T) v = __ldg(reinterpret_cast<const uint4 *>(p + (int64_t)(gb + i) * pitch));
        w[i][0] = v.x, w[i][1] = v.y, w[i][2] = v.z, w[i][3] = v.w;
    }
}
// Load the warp's segments (zeros for rows at or past T).
template <int P>
__device__ __forceinline__ void load_segments(uint32_t (&w)[P][4], const void *src, int64_t pitch, int64_t t0, int64_t T)
{
    load_segments_raw<P>(w, src, pitch, t0, T);
    transpose_pieces<P>(w);
}

// The warp's rows of a 32-column chunk through a TMA store.  Lane l holds
// row l's P 16-byte pieces (P = 8: fp32, P = 4: bf16) and writes them into
// the warp's slot in the box layout of the map: 128-byte rows with the
// 128-byte swizzle (piece j at j ^ (l & 7)) or 64-byte rows with the 64-byte
// swizzle (piece j at j ^ ((l >> 1) & 3)); eight consecutive lanes then
// cover all 32 banks.  Lane 0 stores the box at (column c, row t0); rows at
// or past the tensor's end are clipped by the copy.  The slot must not be
// written again before this lane's bulk group has read it.
template <int P>
__device__ __forceinline__ void stage_store(const uint32_t (&w)[P][4], uint8_t *slot, const CUtensorMap *map, int c,
                                            int64_t t0)
{
    static_assert(P == 8 || P == 4, "fp32 or bf16 rows of 32 columns");
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int j = 0; j < P; ++j) {
        const int pos = P == 8 ? (j ^ (lane & 7)) : (j ^ ((lane >> 1) & 3));
        *reinterpret_cast<uint4 *>(slot + lane * (P * 16) + pos * 16) = make_uint4(w[j][0], w[j][1], w[j][2], w[j][3]);
    }
    ptx::fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
        ptx::tma_store_2d(map, ptx::smem_u32(slot), c, (int)t0);
        ptx::bulk_commit_group();
    }
}

// Column sums of one A stage (128 rows x 64 bf16 columns, K-major, 128-byte
// swizzle): epilogue warp ew (0..7) takes columns [8 ew, 8 ew + 8), one
// 16-byte piece per row.  Lane l adds rows l, l + 32, l + 64, l + 96 in that
// order (rows l and l + 8 sit in different banks, so each load is four
// conflict-free wavefronts), then the lanes are combined by recursive halving
// (lane bits 4, 3, 2 select the column, bits 1, 0 finish the sum).  Returns
// the sum of column 8 ew + col_of_lane(lane) on every lane; the order of the
// additions is fixed.
__device__ __forceinline__ int stage_colsum_col(int lane) { return ((lane >> 4) & 1) * 4 + ((lane >> 3) & 1) * 2 + ((lane >> 2) & 1); }
__device__ __forceinline__ float stage_colsum8(const uint8_t *sA, int ew, int lane)
{
    float v[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = 0.f;
    const uint32_t piece = ((uint32_t)ew ^ (uint32_t)(lane & 7)) << 4;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int row = lane + 32 * q;
        const uint4 u = *reinterpret_cast<const uint4 *>(sA + row * 128 + piece);
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&w[i]));
            v[2 * i] += f.x;
            v[2 * i + 1] += f.y;
        }
    }
    {
        const bool up = (lane & 16) != 0;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float send = up ? v[i] : v[i + 4], keep = up ? v[i + 4] : v[i];
            v[i] = keep + __shfl_xor_sync(0xffffffffu, send, 16);
        }
    }
    {
        const bool up = (lane & 8) != 0;
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            const float send = up ? v[i] : v[i + 2], keep = up ? v[i + 2] : v[i];
            v[i] = keep + __shfl_xor_sync(0xffffffffu, send, 8);
        }
    }
    {
        const bool up = (lane & 4) != 0;
        const float send = up ? v[0] : v[1], keep = up ? v[1] : v[0];
        v[0] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
    }
    v[0] += __shfl_xor_sync(0xffffffffu, v[0], 2);
    v[0] += __shfl_xor_sync(0xffffffffu, v[0], 1);
    return v[0];
}

// Byte offset of element (row, col) in a 128-row bf16 K-major tile stored as
// 64-column blocks with the 128-byte swizzle (what TMA writes and UMMA reads).
__device__ __forceinline__ uint32_t sw128_offset(int row, int col)
{
    return (uint32_t)(col >> 6) * (kBM * 128) + row * 128 + ((((col & 63) >> 3) ^ (row & 7)) << 4) + (col & 7) * 2;
}

// Row `row`, columns [col, col+8) of the row operand: the bf16 high part goes
// to the first tile, the bf16 rounding of the remainder to the second tile
// (kTileBytes further).  Returns the packed high part.
template <uint32_t kTileBytes>
__device__ __forceinline__ uint4 store_hi_lo_impl(uint8_t *tile, int row, int col, const float (&o)[8])
{
    uint4 hi, lo;
    uint32_t *ph = &hi.x, *pl = &lo.x;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const __nv_bfloat162 h2 = __floats2bfloat162_rn(o[2 * i], o[2 * i + 1]);
        const float2 hf = __bfloat1622float2(h2);
        const __nv_bfloat162 l2 = __floats2bfloat162_rn(o[2 * i] - hf.x, o[2 * i + 1] - hf.y);
        ph[i] = *reinterpret_cast<const uint32_t *>(&h2);
        pl[i] = *reinterpret_cast<const uint32_t *>(&l2);
    }
    const uint32_t off = sw128_offset(row, col);
    *reinterpret_cast<uint4 *>(tile + off) = hi;
    *reinterpret_cast<uint4 *>(tile + kTileBytes + off) = lo;
    return hi;
}

// Warps 0 (TMA) and 1 (MMA, TMEM owner) plus CosnetCfg::kEpiWarps epilogue
// warps, which split the 32-column chunks of their TMEM lane quarter's rows.

// Bottleneck activation of the kernel: the CosNet of Eq. 2 (default), or the
// variants of the ablation in Section 4.4 (Table 5): a single cosine
// sigma(h) = cos(omega1 h + phi1); the identity sigma(h) = h (the linear
// collapse of Sections 1 and 3.1); another activation f (activations.cuh,
// chosen at run time by CosnetArgs::act), one layer sigma(h) = f(h) or two
// layers sigma(h) = f(f(h) M).  The one-layer variants have no mixing matrix,
// so their epilogue ends after the first accumulator; the two-layer ones run
// the CosNet epilogue with f in place of the cosines and no frequencies or
// phases (their partial sums are written as zeros).
//
// kSigCos3, the three-layer cosine of the same ablation, adds a second
// mixing matrix and a third cosine: a2 = cos(omega2 b + phi2), b2 = a2 M2,
// c = cos(omega3 b2 + phi3).  Its epilogue runs a middle phase and a second
// r x r product between the CosNet's two (r <= 128: one pass per matrix).
constexpr int kSigCosnet = 0, kSigCos1 = 1, kSigIdentity = 2, kSigAct1 = 3, kSigAct2 = 4, kSigCos3 = 5;
__host__ __device__ constexpr bool sig_two_layers(int sig)
{
    return sig == kSigCosnet || sig == kSigAct2 || sig == kSigCos3;
}

template <int R, bool BWD, int SIG = kSigCosnet>
__global__ void __launch_bounds__(CosnetCfg<R, BWD>::kThreads, 1)
cosnet_gemm_kernel(const __grid_constant__ CUtensorMap mA, const __grid_constant__ CUtensorMap mB,
                   const CosnetArgs args, const __grid_constant__ CosnetStoreMaps smaps)
{
    using C = CosnetCfg<R, BWD>;
    constexpr int STAGES = C::kStages;
    auto store_hi_lo = [](uint8_t *tile, int row, int col, const float(&o)[8]) {
        return store_hi_lo_impl<C::kTileBytes>(tile, row, col, o);
    };
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = ptx::smem_u32(smem_raw);
    const uint32_t sbase = (raw + 1023u) & ~1023u;
    uint8_t *smem = smem_raw + (sbase - raw);
    const uint32_t bar0 = sbase + C::kBarOff;
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (STAGES + s); };
    const uint32_t tmem_full = bar0 + 8u * (2 * STAGES);
    const uint32_t mma2_done = bar0 + 8u * (2 * STAGES + 1);
    const uint32_t m_empty = bar0 + 8u * (2 * STAGES + 2);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + C::kBarOff + 8 * (2 * STAGES + 3));
    float *prm = reinterpret_cast<float *>(smem + C::kParamOff);  // om1 | ph1 | om2 | ph2
    float *cpart = reinterpret_cast<float *>(smem + C::kPartOff);  // [4][4][R]

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int64_t m0 = (int64_t)blockIdx.x * kBM;

    if (warp == 0 && lane == 0) {
        ptx::griddep_launch();  // the next kernel of the call may take the SMs this grid leaves free
        ptx::tma_prefetch_desc(&mA);
        ptx::tma_prefetch_desc(&mB);
        for (int s = 0; s < STAGES; ++s) {
            ptx::mbar_init(full_bar(s), 1);
            // released by the MMA commit and, when dbias is summed from the dy
            // stages, by the eight epilogue warps
            ptx::mbar_init(empty_bar(s), (BWD && args.bias_part) ? 9 : 1);
        }
        ptx::mbar_init(tmem_full, 1);
        ptx::mbar_init(mma2_done, 1);
        ptx::mbar_init(m_empty, 1);
        ptx::fence_barrier_init();
    }
    if (warp == 1) {
        ptx::tmem_alloc(ptx::smem_u32(tmem_slot), C::kTmemCols);
        ptx::tmem_relinquish();
    }
    // launched as a programmatic dependent: the set-up above overlaps the
    // previous kernel of the stream; nothing it wrote is read before this
    ptx::griddep_wait();
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            int issued = 0;
            for (int i = 0; i < args.kb; ++i) {
                const int s = i % STAGES;
                const uint32_t ph = (i / STAGES) & 1;
                if (!ptx::mbar_wait(empty_bar(s), ph ^ 1, args.status)) break;
                const uint32_t fb = full_bar(s);
                ptx::mbar_arrive_expect_tx(fb, C::kStage);
                const uint32_t sA = sbase + s * C::kStage;
                ptx::tma_load_2d(sA, &mA, fb, i * kBK, (int)m0);
                if constexpr (C::kBInterleaved) {
                    // all eight 8-row K groups across all column chunks, one copy
                    ptx::tma_load_4d(sA + C::kA, &mB, fb, 0, i * 8);
                } else if constexpr (BWD) {
                    // the 64 K rows of every 64-wide column chunk
                    for (int c = 0; c < C::kBChunks; ++c)
                        ptx::tma_load_2d(sA + C::kA + c * C::kChunkBytes, &mB, fb, c * 64, i * kBK);
                } else {
                    // all R rows of W_down for this k-block
                    ptx::tma_load_2d(sA + C::kA, &mB, fb, i * kBK, 0);
                }
                ++issued;
            }
            for (int i = issued > STAGES ? issued - STAGES : 0; i < issued; ++i)
                ptx::mbar_wait(full_bar(i % STAGES), (i / STAGES) & 1, nullptr);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = ptx::idesc_bf16(kBM, C::kMainN, false, BWD);
            for (int i = 0; i < args.kb; ++i) {
                const int s = i % STAGES;
                const uint32_t ph = (i / STAGES) & 1;
                if (!ptx::mbar_wait(full_bar(s), ph, args.status)) break;
                ptx::tc_fence_after();
                const uint32_t sA = sbase + s * C::kStage, sB = sA + C::kA;
#pragma unroll
                for (int kk = 0; kk < kBK / 16; ++kk) {
                    // MN-major B: 16 K rows are two 8-row groups (2048 bytes);
                    // the column chunks are kChunkBytes apart
                    const uint64_t bd =
                        C::kBInterleaved
                            ? ptx::smem_desc_sw128(sB + kk * 2048 * C::kBChunks, 1024, 1024 * C::kBChunks)
                        : BWD ? ptx::smem_desc_sw128(sB + kk * 2048, C::kChunkBytes, 1024)
                              : ptx::smem_desc_sw128(sB + kk * 32, 16, 1024);
                    ptx::mma_bf16(tmem, ptx::smem_desc_sw128(sA + kk * 32, 16, 1024), bd, idesc,
                                  (i > 0 || kk > 0) ? 1u : 0u);
                }
                ptx::mma_commit(empty_bar(s));
            }
            ptx::mma_commit(tmem_full);
            ptx::mbar_wait(tmem_full, 0, nullptr);
        }
    } else {
        // ---------------- epilogue: kEpiWarps warps; a thread owns one token
        // row and the 32-column chunks c with (c / 32) % kColGroups == grp
        constexpr int NE = C::kEpiThreads, CSTEP = 32 * C::kColGroups;
        const int quarter = warp % 4;
        const int grp = (warp - 2) / 4;
        const int row = quarter * 32 + lane;
        const int64_t t = m0 + row;
        const bool live = t < args.T;
        const int64_t t0 = m0 + quarter * 32;  // the warp's first row
        const uint32_t lane_addr = tmem + ((uint32_t)(quarter * 32) << 16);
        const uint32_t acc2 = lane_addr + C::kRCols;
        const float *om1 = prm, *ph1 = prm + R, *om2 = prm + 2 * R, *ph2 = prm + 3 * R;
        const float *om3 = prm + 4 * R, *ph3 = prm + 5 * R;
        // the three-layer cosine: sums per column for three layers, and the
        // outermost layer of the backward's first phase is the third one
        constexpr bool C3 = SIG == kSigCos3;
        static_assert(!C3 || C::kPasses == 1, "three-layer cosine: one pass per mixing matrix (r <= 128)");
        constexpr int NQ = C3 ? 6 : 4;
        const float *omL = C3 ? om3 : om2, *phL = C3 ? ph3 : ph2;  // the last layer's frequency and phase
        // frequencies and phases into shared memory (parameters a variant does
        // not use may be NULL); read after the barrier that follows the main
        // loop, so the copies above start without waiting for these loads
        for (int i = threadIdx.x - 64; i < R; i += NE) {
            prm[i] = args.om1 ? args.om1[i] : 0.f;
            prm[R + i] = args.ph1 ? args.ph1[i] : 0.f;
            prm[2 * R + i] = args.om2 ? args.om2[i] : 0.f;
            prm[3 * R + i] = args.ph2 ? args.ph2[i] : 0.f;
            if constexpr (SIG == kSigCos3) {
                prm[4 * R + i] = args.om3[i];
                prm[5 * R + i] = args.ph3[i];
            }
        }
        uint8_t *tile = smem;  // the ring is free once the main accumulator is complete
        // TMA stores of the row outputs (CosNet, r in {64, 128}): this warp's
        // staging slots for phase 1 and phase 2
        constexpr bool kTma = SIG == kSigCosnet && C::kStgFits;
        uint8_t *stg1 = smem + C::kStg1Off + (warp - 2) * C::kStg1Bytes;
        uint8_t *stg2 = smem + (warp - 2) * C::kStg2Bytes;
        static_assert(!kTma || R == 32 * C::kColGroups, "one 32-column chunk per warp and phase");
        // The mixing matrix, bf16 high and low parts, K-major in the SW128
        // layout: group gi covers operand row n (an output column) and k-columns
        // [c, c + 8) of k-block j of a pass.  n runs fastest, so a warp reads
        // whole 128-byte rows of M in the forward.
        const int et = threadIdx.x - 64;  // 0..NE-1
        constexpr int kGroups = R * 8 * C::kChunkKb;
        constexpr int kIters = (kGroups + NE - 1) / NE;
        float mraw[kIters][8];
        auto m_group = [&](int it, int pass, int &j, int &n, int &cg, int &c) {
            const int gi = et + it * NE;
            j = gi / (R * 8);
            n = gi % R;
            cg = ((gi / R) % 8) * 8;
            c = (pass * C::kChunkKb + j) * 64 + cg;  // k index
            return gi < kGroups && c < R;
        };
        // loads only: the values are first used in m_store, so the loads stay
        // in flight across whatever runs in between
        // the matrices of the r x r products in order: M (forward; the
        // three-layer cosine's backward starts with M2, the forward ends with it)
        const float *mat1 = (C3 && BWD) ? args.M2 : args.M;
        const float *mat2 = (C3 && BWD) ? args.M : args.M2;
        auto m_load = [&](int pass, const float *Mp) {
#pragma unroll
            for (int it = 0; it < kIters; ++it) {
                int j, n, cg, c;
                if (!m_group(it, pass, j, n, cg, c)) continue;
                if constexpr (BWD) {
                    const float4 *src = reinterpret_cast<const float4 *>(Mp + (int64_t)n * R + c);  // M[n][c+q]
                    const float4 u = __ldg(src), w = __ldg(src + 1);
                    mraw[it][0] = u.x, mraw[it][1] = u.y, mraw[it][2] = u.z, mraw[it][3] = u.w;
                    mraw[it][4] = w.x, mraw[it][5] = w.y, mraw[it][6] = w.z, mraw[it][7] = w.w;
                } else {
#pragma unroll
                    for (int q = 0; q < 8; ++q) mraw[it][q] = __ldg(Mp + (int64_t)(c + q) * R + n);  // M[c+q][n]
                }
            }
        };
        auto m_store = [&](int pass) {
#pragma unroll
            for (int it = 0; it < kIters; ++it) {
                int j, n, cg, c;
                if (!m_group(it, pass, j, n, cg, c)) continue;
                uint4 hi, lo;
                uint32_t *ph = &hi.x, *pl = &lo.x;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const __nv_bfloat162 h2 = __floats2bfloat162_rn(mraw[it][2 * q], mraw[it][2 * q + 1]);
                    const float2 hf = __bfloat1622float2(h2);
                    const __nv_bfloat162 l2 =
                        __floats2bfloat162_rn(mraw[it][2 * q] - hf.x, mraw[it][2 * q + 1] - hf.y);
                    ph[q] = *reinterpret_cast<const uint32_t *>(&h2);
                    pl[q] = *reinterpret_cast<const uint32_t *>(&l2);
                }
                const uint32_t off =
                    C::kMOff + j * C::kMkbBytes + n * 128 + ((((uint32_t)cg >> 3) ^ (n & 7)) << 4);
                *reinterpret_cast<uint4 *>(smem + off) = hi;
                *reinterpret_cast<uint4 *>(smem + off + R * 128) = lo;
            }
        };
        // the first pass's part of M is read while the main loop runs
        if constexpr (sig_two_layers(SIG)) m_load(0, mat1);
        bool bias_ok = true;
        if constexpr (BWD) {
            if (args.bias_part) {
                // dbias partials while the main loop runs: epilogue warp ew owns
                // columns [8 ew, 8 ew + 8) of each dy stage and sums all 128 rows
                // (stage_colsum8, a fixed order), so no warp waits for another
                // before the stage goes back to the producer; with sixteen
                // epilogue warps the first eight take part
                const int ew = warp - 2;
                for (int i = 0; ew < 8 && i < args.kb; ++i) {
                    const int s = i % STAGES;
                    const uint32_t ph = (i / STAGES) & 1;
                    bias_ok = __all_sync(0xffffffffu, bias_ok && ptx::mbar_wait(full_bar(s), ph, args.status));
                    if (!bias_ok) break;
                    const float v = stage_colsum8(smem + s * C::kStage, ew, lane);
                    // the stage is refilled by the copy engine (async proxy)
                    // once released: order these generic reads before that
                    ptx::fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) ptx::mbar_arrive(empty_bar(s));
                    const int64_t col = (int64_t)i * kBK + 8 * ew + stage_colsum_col(lane);
                    if ((lane & 3) == 0 && col < args.kdim) args.bias_part[(int64_t)blockIdx.x * args.kdim + col] = v;
                }
            }
        }
        bool ok = bias_ok && ptx::mbar_wait(tmem_full, 0, args.status);
        ok = ptx::named_barrier_and(3, NE, ok);  // uniform over the epilogue warps
        if (ok) {
            // the ring is free once the main accumulator is complete
            if constexpr (sig_two_layers(SIG)) m_store(0);
            ptx::tc_fence_after();
            if constexpr (!sig_two_layers(SIG)) {
                // single-cosine or identity bottleneck: c (forward) or dh
                // (backward) straight from the first accumulator
#pragma unroll 1
                for (int c = 32 * grp; c < R; c += CSTEP) {
                    float v[32];
                    if constexpr (R >= 32) {
                        ptx::tmem_ld_32x32b_x32(lane_addr + c, v);
                    } else {
                        float w[16];
                        ptx::tmem_ld_32x32b_x16(lane_addr + c, w);
#pragma unroll
                        for (int i = 0; i < 16; ++i) v[i] = w[i], v[i + 16] = 0.f;
                    }
                    constexpr int W = R < 32 ? R : 32;
                    if constexpr (!BWD) {
                        // v = h: store h and c = cos(omega1 h + phi1) or c = h
                        {
                            uint32_t w[W / 4][4];
#pragma unroll
                            for (int i = 0; i < W / 4; ++i)
#pragma unroll
                                for (int q = 0; q < 4; ++q) w[i][q] = __float_as_uint(v[4 * i + q]);
                            if (args.h_out)
                                store_segments<W / 4>(w, args.h_out + t0 * R + c, (int64_t)R * 4, t0, args.T);
                        }
                        uint32_t wc[W / 8][4];
#pragma unroll
                        for (int g = 0; g < W / 8; ++g) {
                            float cc[8];
#pragma unroll
                            for (int i = 0; i < 8; ++i) {
                                const int k = c + 8 * g + i;
                                cc[i] = SIG == kSigCos1   ? cos_reduced(fmaf(om1[k], v[8 * g + i], ph1[k]))
                                        : SIG == kSigAct1 ? act::f(args.act, v[8 * g + i])
                                                          : v[8 * g + i];
                            }
#pragma unroll
                            for (int q = 0; q < 4; ++q) wc[g][q] = ptx::pack_bf16x2(cc[2 * q], cc[2 * q + 1]);
                        }
                        store_segments<W / 8>(wc, args.c_out + t0 * R + c, (int64_t)R * 2, t0, args.T);
                    } else {
                        // v = dc; single cosine: du1 = -sin(omega1 h + phi1) dc,
                        // dh = omega1 du1; one-layer f: dh = f'(h) dc; identity: dh = dc
                        float hv[32];
#pragma unroll
                        for (int i = 0; i < 32; ++i) hv[i] = 0.f;
                        if constexpr (SIG == kSigCos1 || SIG == kSigAct1) {
                            uint32_t w[W / 4][4];
                            load_segments<W / 4>(w, args.h_in + t0 * R + c, (int64_t)R * 4, t0, args.T);
#pragma unroll
                            for (int i = 0; i < W / 4; ++i)
#pragma unroll
                                for (int q = 0; q < 4; ++q) hv[4 * i + q] = __uint_as_float(w[i][q]);
                        }
                        float q0[32], q1[32];
                        uint32_t wdh[W / 8][4];
#pragma unroll
                        for (int i = W; i < 32; ++i) q0[i] = 0.f, q1[i] = 0.f;
#pragma unroll
                        for (int g = 0; g < W / 8; ++g) {
                            float dh[8];
#pragma unroll
                            for (int i = 0; i < 8; ++i) {
                                const int k = c + 8 * g + i, j = 8 * g + i;
                                float du1 = 0.f;
                                if constexpr (SIG == kSigCos1) {
                                    du1 = live ? -sin_reduced(fmaf(om1[k], hv[j], ph1[k])) * v[j] : 0.f;
                                    dh[i] = om1[k] * du1;
                                } else if constexpr (SIG == kSigAct1) {
                                    dh[i] = live ? act::df(args.act, hv[j]) * v[j] : 0.f;
                                } else {
                                    dh[i] = live ? v[j] : 0.f;
                                }
                                q0[j] = du1 * hv[j];
                                q1[j] = du1;
                            }
#pragma unroll
                            for (int q = 0; q < 4; ++q) wdh[g][q] = ptx::pack_bf16x2(dh[2 * q], dh[2 * q + 1]);
                        }
                        store_segments<W / 8>(wdh, args.dh_out + t0 * R + c, (int64_t)R * 2, t0, args.T);
                        const float s0 = warp_colsum32(q0);
                        const float s1 = warp_colsum32(q1);
                        if (c + lane < R) {
                            cpart[(quarter * NQ + 0) * R + c + lane] = s0;
                            cpart[(quarter * NQ + 1) * R + c + lane] = s1;
                            cpart[(quarter * NQ + 2) * R + c + lane] = 0.f;  // no second layer
                            cpart[(quarter * NQ + 3) * R + c + lane] = 0.f;
                        }
                    }
                }
            } else {
            // ---- phase 1: first accumulator -> bf16 operand tile (+ outputs)
#pragma unroll 1
            for (int c = 32 * grp; c < R; c += CSTEP) {
                float v[32];
                if constexpr (R >= 32) {
                    ptx::tmem_ld_32x32b_x32(lane_addr + c, v);
                } else {
                    float w[16];
                    ptx::tmem_ld_32x32b_x16(lane_addr + c, w);
#pragma unroll
                    for (int i = 0; i < 16; ++i) v[i] = w[i], v[i + 16] = 0.f;
                }
                constexpr int W = R < 32 ? R : 32;
                if constexpr (!BWD) {
                    // v = h: store h, operand a = cos(omega1 h + phi1)
                    {
                        uint32_t w[W / 4][4];
#pragma unroll
                        for (int i = 0; i < W / 4; ++i)
#pragma unroll
                            for (int q = 0; q < 4; ++q) w[i][q] = __float_as_uint(v[4 * i + q]);
                        if constexpr (kTma) {
                            if (args.h_out) stage_store<W / 4>(w, stg1, &smaps.m[0], c, t0);
                        } else if (args.h_out) {
                            store_segments<W / 4>(w, args.h_out + t0 * R + c, (int64_t)R * 4, t0, args.T);
                        }
                    }
#pragma unroll
                    for (int g = 0; g < W / 8; ++g) {
                        float o[8];
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            const int k = c + 8 * g + i;
                            o[i] = SIG == kSigAct2 ? act::f(args.act, v[8 * g + i])
                                                   : cos_reduced(fmaf(om1[k], v[8 * g + i], ph1[k]));
                        }
                        store_hi_lo(tile, row, c + 8 * g, o);
                    }
                } else {
                    // v = dc; with b of this row: du2, operand db = omega2 du2
                    float bv[32];
#pragma unroll
                    for (int i = 0; i < 32; ++i) bv[i] = 0.f;
                    {
                        uint32_t w[W / 4][4];
                        load_segments<W / 4>(w, (C3 ? args.b2_in : args.b_in) + t0 * R + c, (int64_t)R * 4, t0,
                                             args.T);
#pragma unroll
                        for (int i = 0; i < W / 4; ++i)
#pragma unroll
                            for (int q = 0; q < 4; ++q) bv[4 * i + q] = __uint_as_float(w[i][q]);
                    }
                    // the column-sum operands replace their inputs in place
                    // (bv: du2 b, v: du2), which keeps the register count low;
                    // for the three-layer cosine this is its third layer (b2,
                    // omega3, phi3: du3, db2)
                    uint32_t wdb[W / 8][4];
#pragma unroll
                    for (int i = W; i < 32; ++i) bv[i] = 0.f, v[i] = 0.f;
#pragma unroll
                    for (int g = 0; g < W / 8; ++g) {
                        float o[8];
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            const int k = c + 8 * g + i, j = 8 * g + i;
                            if constexpr (SIG == kSigAct2) {
                                // f(b): db = f'(b) dc, no frequency or phase
                                o[i] = live ? act::df(args.act, bv[j]) * v[j] : 0.f;
                                bv[j] = 0.f;
                                v[j] = 0.f;
                            } else {
                                const float du2 = live ? -sin_reduced(fmaf(omL[k], bv[j], phL[k])) * v[j] : 0.f;
                                o[i] = omL[k] * du2;
                                bv[j] *= du2;
                                v[j] = du2;
                            }
                        }
                        const uint4 q = store_hi_lo(tile, row, c + 8 * g, o);
                        wdb[g][0] = q.x, wdb[g][1] = q.y, wdb[g][2] = q.z, wdb[g][3] = q.w;
                    }
                    if constexpr (kTma)
                        stage_store<W / 8>(wdb, stg1, &smaps.m[0], c, t0);
                    else
                        store_segments<W / 8>(wdb, (C3 ? args.db2_out : args.db_out) + t0 * R + c, (int64_t)R * 2,
                                              t0, args.T);
                    const float s2 = warp_colsum32(bv);
                    const float s3 = warp_colsum32(v);
                    if (c + lane < R) {
                        cpart[(quarter * NQ + (C3 ? 4 : 2)) * R + c + lane] = s2;
                        cpart[(quarter * NQ + (C3 ? 5 : 3)) * R + c + lane] = s3;
                    }
                }
            }
            // ---- second MMA: (128 x r operand tile) x (r x r mixing matrix), the
            // matrix converted to bf16 hi/lo operand blocks by these threads,
            // kChunkKb k-blocks per pass
            constexpr uint32_t idesc = ptx::idesc_bf16(kBM, R, false, false);
            for (int pass = 0; ok && pass < C::kPasses; ++pass) {
                if (pass > 0) {
                    // the previous pass's MMAs have read the operand blocks
                    ok = ptx::mbar_wait(m_empty, (pass - 1) & 1, args.status);
                    ok = ptx::named_barrier_and(3, NE, ok);
                    if (!ok) break;
                    m_load(pass, mat1);
                    m_store(pass);
                }
                ptx::fence_proxy_async_smem();
                ptx::named_barrier_sync(1, NE);
                if (threadIdx.x == 64) {
                    ptx::tc_fence_after();
                    const uint32_t acc = tmem + C::kRCols;
                    for (int j = 0; j < C::kChunkKb; ++j) {
                        const int kb = pass * C::kChunkKb + j;
#pragma unroll
                        for (int kk = 0; kk < C::kKSteps; ++kk) {
                            const uint32_t a_hi = sbase + kb * (kBM * 128) + kk * 32;
                            const uint32_t a_lo = a_hi + C::kTileBytes;
                            const uint32_t m_hi = sbase + C::kMOff + j * C::kMkbBytes + kk * 32;
                            const uint32_t m_lo = m_hi + R * 128;
                            const uint64_t dah = ptx::smem_desc_sw128(a_hi, 16, 1024);
                            const uint64_t dal = ptx::smem_desc_sw128(a_lo, 16, 1024);
                            const uint64_t dmh = ptx::smem_desc_sw128(m_hi, 16, 1024);
                            const uint64_t dml = ptx::smem_desc_sw128(m_lo, 16, 1024);
                            ptx::mma_bf16(acc, dah, dmh, idesc, (kb > 0 || kk > 0) ? 1u : 0u);
                            ptx::mma_bf16(acc, dal, dmh, idesc, 1u);
                            ptx::mma_bf16(acc, dah, dml, idesc, 1u);
                        }
                    }
                    if (pass + 1 < C::kPasses) ptx::mma_commit(m_empty);
                }
            }
            // also after a failed wait: the MMAs already issued finish before
            // the tile and the accumulator are given up
            if (threadIdx.x == 64) ptx::mma_commit(mma2_done);
            const bool done = ptx::mbar_wait(mma2_done, 0, args.status);
            ok = ptx::named_barrier_and(3, NE, ok && done);
            if constexpr (C3) {
                // ---- middle phase (three-layer cosine): the first product's
                // accumulator becomes the second product's row operand; that
                // product (with the other matrix) goes into the first
                // accumulator, whose h or dc phase 1 has consumed
                if (ok) {
                    m_load(0, mat2);
                    m_store(0);
                    ptx::tc_fence_after();
#pragma unroll 1
                    for (int c = 32 * grp; c < R; c += CSTEP) {
                        float v[32];
                        if constexpr (R >= 32) {
                            ptx::tmem_ld_32x32b_x32(acc2 + c, v);
                        } else {
                            float w[16];
                            ptx::tmem_ld_32x32b_x16(acc2 + c, w);
#pragma unroll
                            for (int i = 0; i < 16; ++i) v[i] = w[i], v[i + 16] = 0.f;
                        }
                        constexpr int W = R < 32 ? R : 32;
                        if constexpr (!BWD) {
                            // v = b: store b, operand a2 = cos(omega2 b + phi2)
                            {
                                uint32_t w[W / 4][4];
#pragma unroll
                                for (int i = 0; i < W / 4; ++i)
#pragma unroll
                                    for (int q = 0; q < 4; ++q) w[i][q] = __float_as_uint(v[4 * i + q]);
                                if (args.b_out)
                                    store_segments<W / 4>(w, args.b_out + t0 * R + c, (int64_t)R * 4, t0, args.T);
                            }
#pragma unroll
                            for (int g = 0; g < W / 8; ++g) {
                                float o[8];
#pragma unroll
                                for (int i = 0; i < 8; ++i) {
                                    const int k = c + 8 * g + i;
                                    o[i] = cos_reduced(fmaf(om2[k], v[8 * g + i], ph2[k]));
                                }
                                store_hi_lo(tile, row, c + 8 * g, o);
                            }
                        } else {
                            // v = da2; with b of this row: du2 = -sin(u2) da2,
                            // operand db = omega2 du2, a2 = cos(u2)
                            float bv[32];
#pragma unroll
                            for (int i = 0; i < 32; ++i) bv[i] = 0.f;
                            {
                                uint32_t w[W / 4][4];
                                load_segments<W / 4>(w, args.b_in + t0 * R + c, (int64_t)R * 4, t0, args.T);
#pragma unroll
                                for (int i = 0; i < W / 4; ++i)
#pragma unroll
                                    for (int q = 0; q < 4; ++q) bv[4 * i + q] = __uint_as_float(w[i][q]);
                            }
                            uint32_t wdb[W / 8][4], wa2[W / 8][4];
#pragma unroll
                            for (int i = W; i < 32; ++i) bv[i] = 0.f, v[i] = 0.f;
#pragma unroll
                            for (int g = 0; g < W / 8; ++g) {
                                float o[8], a2v[8];
#pragma unroll
                                for (int i = 0; i < 8; ++i) {
                                    const int k = c + 8 * g + i, j = 8 * g + i;
                                    float s2, c2;
                                    sincos_reduced(fmaf(om2[k], bv[j], ph2[k]), &s2, &c2);
                                    const float du2 = live ? -s2 * v[j] : 0.f;
                                    o[i] = om2[k] * du2;
                                    a2v[i] = c2;
                                    bv[j] *= du2;  // the column-sum operands, in place
                                    v[j] = du2;
                                }
                                const uint4 q = store_hi_lo(tile, row, c + 8 * g, o);
                                wdb[g][0] = q.x, wdb[g][1] = q.y, wdb[g][2] = q.z, wdb[g][3] = q.w;
#pragma unroll
                                for (int q2 = 0; q2 < 4; ++q2) wa2[g][q2] = ptx::pack_bf16x2(a2v[2 * q2], a2v[2 * q2 + 1]);
                            }
                            store_segments<W / 8>(wdb, args.db_out + t0 * R + c, (int64_t)R * 2, t0, args.T);
                            store_segments<W / 8>(wa2, args.a2_out + t0 * R + c, (int64_t)R * 2, t0, args.T);
                            const float s2 = warp_colsum32(bv);
                            const float s3 = warp_colsum32(v);
                            if (c + lane < R) {
                                cpart[(quarter * NQ + 2) * R + c + lane] = s2;
                                cpart[(quarter * NQ + 3) * R + c + lane] = s3;
                            }
                        }
                    }
                    // the first accumulator's loads are complete before the
                    // product overwrites it
                    ptx::tc_fence_before();
                    ptx::fence_proxy_async_smem();
                    ptx::named_barrier_sync(1, NE);
                    if (threadIdx.x == 64) {
                        ptx::tc_fence_after();
#pragma unroll
                        for (int kb = 0; kb < C::kMkb; ++kb) {
#pragma unroll
                            for (int kk = 0; kk < C::kKSteps; ++kk) {
                                const uint32_t a_hi = sbase + kb * (kBM * 128) + kk * 32;
                                const uint32_t a_lo = a_hi + C::kTileBytes;
                                const uint32_t m_hi = sbase + C::kMOff + kb * C::kMkbBytes + kk * 32;
                                const uint32_t m_lo = m_hi + R * 128;
                                const uint64_t dah = ptx::smem_desc_sw128(a_hi, 16, 1024);
                                const uint64_t dal = ptx::smem_desc_sw128(a_lo, 16, 1024);
                                const uint64_t dmh = ptx::smem_desc_sw128(m_hi, 16, 1024);
                                const uint64_t dml = ptx::smem_desc_sw128(m_lo, 16, 1024);
                                ptx::mma_bf16(tmem, dah, dmh, idesc, (kb > 0 || kk > 0) ? 1u : 0u);
                                ptx::mma_bf16(tmem, dal, dmh, idesc, 1u);
                                ptx::mma_bf16(tmem, dah, dml, idesc, 1u);
                            }
                        }
                        ptx::mma_commit(mma2_done);
                    }
                    const bool done2 = ptx::mbar_wait(mma2_done, 1, args.status);
                    ok = ptx::named_barrier_and(3, NE, ok && done2);
                }
            }
            }  // two layers
        }
        if (ok) {
            ptx::tc_fence_after();
            // ---- phase 2: second accumulator
#pragma unroll 1
            // (the three-layer cosine's last product is in the first accumulator)
            const uint32_t accL = C3 ? lane_addr : acc2;
            for (int c = 32 * grp; sig_two_layers(SIG) && c < R; c += CSTEP) {
                float v[32];
                if constexpr (R >= 32) {
                    ptx::tmem_ld_32x32b_x32(accL + c, v);
                } else {
                    float w[16];
                    ptx::tmem_ld_32x32b_x16(accL + c, w);
#pragma unroll
                    for (int i = 0; i < 16; ++i) v[i] = w[i], v[i + 16] = 0.f;
                }
                constexpr int W = R < 32 ? R : 32;
                if constexpr (!BWD) {
                    // v = b (the three-layer cosine: b2, with omega3 and phi3)
                    uint32_t wc[W / 8][4];
#pragma unroll
                    for (int g = 0; g < W / 8; ++g) {
                        float cc[8];
#pragma unroll
                        for (int i = 0; i < 8; ++i)
                            cc[i] = SIG == kSigAct2 ? act::f(args.act, v[8 * g + i])
                                                    : cos_reduced(fmaf(omL[c + 8 * g + i], v[8 * g + i], phL[c + 8 * g + i]));
#pragma unroll
                        for (int q = 0; q < 4; ++q) wc[g][q] = ptx::pack_bf16x2(cc[2 * q], cc[2 * q + 1]);
                    }
                    {
                        uint32_t w[W / 4][4];
#pragma unroll
                        for (int i = 0; i < W / 4; ++i)
#pragma unroll
                            for (int q = 0; q < 4; ++q) w[i][q] = __float_as_uint(v[4 * i + q]);
                        float *bo = C3 ? args.b2_out : args.b_out;
                        if constexpr (kTma) {
                            if (bo) stage_store<W / 4>(w, stg2, &smaps.m[1], c, t0);
                        } else if (bo) {
                            store_segments<W / 4>(w, bo + t0 * R + c, (int64_t)R * 4, t0, args.T);
                        }
                    }
                    if constexpr (kTma)
                        stage_store<W / 8>(wc, stg2 + 4096, &smaps.m[2], c, t0);
                    else
                        store_segments<W / 8>(wc, args.c_out + t0 * R + c, (int64_t)R * 2, t0, args.T);
                } else {
                    // v = da; with h of this row: du1, dh = omega1 du1, a = cos(u1)
                    float hv[32];
#pragma unroll
                    for (int i = 0; i < 32; ++i) hv[i] = 0.f;
                    {
                        uint32_t w[W / 4][4];
                        load_segments<W / 4>(w, args.h_in + t0 * R + c, (int64_t)R * 4, t0, args.T);
#pragma unroll
                        for (int i = 0; i < W / 4; ++i)
#pragma unroll
                            for (int q = 0; q < 4; ++q) hv[4 * i + q] = __uint_as_float(w[i][q]);
                    }
                                        uint32_t wdh[W / 8][4], wa[W / 8][4];
#pragma unroll
                    for (int i = W; i < 32; ++i) hv[i] = 0.f, v[i] = 0.f;
#pragma unroll
                    for (int g = 0; g < W / 8; ++g) {
                        float dh[8], av[8];
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            const int k = c + 8 * g + i, j = 8 * g + i;
                            if constexpr (SIG == kSigAct2) {
                                // f(h): dh = f'(h) da, a = f(h)
                                dh[i] = live ? act::df(args.act, hv[j]) * v[j] : 0.f;
                                av[i] = act::f(args.act, hv[j]);
                                hv[j] = 0.f;
                                v[j] = 0.f;
                            } else {
                                float s1, c1;
                                sincos_reduced(fmaf(om1[k], hv[j], ph1[k]), &s1, &c1);
                                const float du1 = live ? -s1 * v[j] : 0.f;
                                dh[i] = om1[k] * du1;
                                av[i] = c1;
                                hv[j] *= du1;  // the column-sum operands, in place
                                v[j] = du1;
                            }
                        }
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            wdh[g][q] = ptx::pack_bf16x2(dh[2 * q], dh[2 * q + 1]);
                            wa[g][q] = ptx::pack_bf16x2(av[2 * q], av[2 * q + 1]);
                        }
                    }
                    if constexpr (kTma) {
                        stage_store<W / 8>(wdh, stg2, &smaps.m[1], c, t0);
                        stage_store<W / 8>(wa, stg2 + 2048, &smaps.m[2], c, t0);
                    } else {
                        store_segments<W / 8>(wdh, args.dh_out + t0 * R + c, (int64_t)R * 2, t0, args.T);
                        store_segments<W / 8>(wa, args.a_out + t0 * R + c, (int64_t)R * 2, t0, args.T);
                    }
                    const float s0 = warp_colsum32(hv);
                    const float s1 = warp_colsum32(v);
                    if (c + lane < R) {
                        cpart[(quarter * NQ + 0) * R + c + lane] = s0;
                        cpart[(quarter * NQ + 1) * R + c + lane] = s1;
                    }
                }
            }
            if constexpr (BWD) {
                // per-CTA column sums: the four lane quarters added in order
                // (NQ sums per column: four, six for the three-layer cosine)
                ptx::named_barrier_sync(1, NE);
                for (int k = threadIdx.x - 64; k < NQ * R; k += NE) {
                    const int q = k / R, col = k % R;
                    float s = 0.f;
#pragma unroll
                    for (int w = 0; w < 4; ++w) s += cpart[(w * NQ + q) * R + col];
                    args.part[(int64_t)blockIdx.x * NQ * R + k] = s;
                }
            }
        }
    }

    // the epilogue's TMA stores are complete before the shared memory they
    // read goes away
    if constexpr (SIG == kSigCosnet && C::kStgFits)
        if (warp >= 2 && lane == 0) ptx::bulk_wait_all();
    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, C::kTmemCols);
    }
}

}  // namespace tc
}  // namespace noble
