// Persistent grouped GEMM on CTA pairs (tcgen05 .cta_group::2).
//
// A cluster of two CTAs on neighbouring SMs computes one 256 x BN output tile
// with a single M = 256 MMA stream: CTA rank q holds rows [128 q, 128 q + 128)
// of the A tile and columns [q BN/2, (q+1) BN/2) of the B tile in its own
// shared memory and receives those 128 rows of the accumulator in its own
// TMEM.  Per SM this halves the B operand traffic and the shared-memory
// operand reads of a 128 x BN single-CTA tile, for the same MMA rate.
//
// Protocol (both CTAs run the same warp roles):
//   * TMEM: warp 1 of each CTA allocates and frees collectively (cta_group::2).
//   * producer (warp 0 of each CTA): waits its own `empty` slot, loads its A
//     and B halves with TMA into its own ring and signals the LEADER's `full`
//     barrier (rank 0); the leader also posts the expected bytes of both.
//   * MMA (warp 1 of the leader only): waits `full`, issues the pair MMAs,
//     commits to `empty` of both CTAs (multicast) and, per tile, to `tfull`
//     of both CTAs.
//   * epilogue (warps 2-9 of each CTA, two per TMEM lane quarter taking
//     alternate 32-column chunks): reads its own accumulator rows and
//     arrives on the LEADER's `tempty` (16 arrivals: 8 warps x 2 CTAs).
// All waits are bounded as in the single-CTA kernels.
//
// Fused bottleneck (FUSE = kFuseFwd / kFuseBwd, the CosNet with r in {64, 128}):
// the r-wide product of the low-rank branch, h = x W_down^T (forward) or
// dc = dy W_up (backward), shares the A stages of the output GEMM instead of
// streaming x or dy once more.  Problem 0 of the launch holds one "leader"
// tile per row pair, of N = 2r: its B operand is [W rows 0..r ; W_down] (CTA
// rank 0 loads the first r rows, rank 1 the branch's r rows), so one MMA
// stream yields the output columns [0, r) and the branch pre-activation side
// by side in TMEM.  Problem 1 holds the remaining output columns [r, N_out).
// A leader's epilogue, after its first K segment:
//   park      the output columns [0, r) in registers
//   phase 1   a = cos(omega1 h + phi1)      | du2 = -sin(omega2 b + phi2) dc,
//                                           |   db = omega2 du2
//             as bf16 high and low parts written back into TMEM columns [r, 2r)
//   product   b = a M  (or da = db M^T), a second pair MMA with A in TMEM and
//             the mixing matrix (bf16 high/low, this CTA's half of its
//             columns) in the epilogue staging buffer, into columns [0, r)
//   phase 2   c = cos(omega2 b + phi2)      | du1 = -sin(omega1 h + phi1) da,
//                                           |   dh = omega1 du1, a = cos(u1)
//   restore   the parked columns into [0, r)
// then stores c (dh) for its 128 rows and releases a flag per 128-row block.
// Every tile's second K segment (c W_up^T, or dh W_down) waits for that flag
// in the producer.  The MMA warp issues the leader's second segment only
// after the next tile's first segment, so the tensor pipe keeps working while
// the epilogue runs the bottleneck; it issues the second product when the
// epilogue signals its operand ready, polling between k-blocks.  In the
// backward the epilogue warps also sum dy's columns over each leader stage
// (dbias partials per 128 rows) before the stage is released.
// Tiles run in the order of share_tile: waves of leaders, each followed by
// the output tiles of its row pairs, so with all clusters resident every
// flag wait ends.
#pragma once

#include "tc_persistent.cuh"
#include "tc_cosnet.cuh"

namespace noble {
namespace tc {
namespace pair {

__device__ __forceinline__ uint32_t cluster_ctarank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

// Address of the same shared-memory location in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t map_to_rank(uint32_t smem_addr, uint32_t rank)
{
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_addr), "r"(rank));
    return r;
}

__device__ __forceinline__ void cluster_sync()
{
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr)
{
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}

// TMA load into this CTA's shared memory, completing on an mbarrier that may
// live in the peer CTA of the pair (cluster address).
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap *map, uint32_t bar_cluster, int c0,
                                                 int c1)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cta.global.tile.mbarrier::complete_tx::bytes.cta_group::2 [%0], [%1, {%3, "
        "%4}], [%2];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(bar_cluster), "r"(c0), "r"(c1)
        : "memory");
}

// 4-D variant for MN-major operands stored with the 64-wide chunks of each
// 8-row K group side by side (see make_map_mn4 on the host).
__device__ __forceinline__ void tma_load_4d_pair(uint32_t dst, const CUtensorMap *map, uint32_t bar_cluster, int c2,
                                                 int c3)
{
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cta.global.tile.mbarrier::complete_tx::bytes.cta_group::2 [%0], [%1, {%3, "
        "%3, %4, %5}], [%2];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(bar_cluster), "r"(0), "r"(c2), "r"(c3)
        : "memory");
}

__device__ __forceinline__ void tmem_alloc2(uint32_t dst_smem, uint32_t ncols)
{
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tmem_relinquish2()
{
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc2(uint32_t taddr, uint32_t ncols)
{
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

__device__ __forceinline__ void mma2_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Arrive once on `bar` (same offset) in every CTA of `mask` when the MMAs
// issued so far by this thread complete.
__device__ __forceinline__ void mma2_commit_mc(uint32_t bar, uint16_t mask)
{
    asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::
                     "r"(bar),
                 "h"(mask)
                 : "memory");
}

struct PairTile {
    int prob;
    int64_t m0, n0;  // this CTA's first row; the tile's first column
    int z;
    int kb_begin, kb_end;
};

// Tile pairs of a problem: split-major, then groups of 8 row-pair blocks
// with the column index running fastest inside a group.
template <class EpiParams>
__device__ __forceinline__ PairTile locate_pair(const GroupArgs<EpiParams> &g, int t, int rank)
{
    int p = 0;
#pragma unroll 1
    while (p + 1 < g.nproblems && t >= g.p[p + 1].tile_begin) ++p;
    const Problem<EpiParams> &P = g.p[p];
    const int pairs_m = (P.tiles_m + 1) / 2;
    int local = t - P.tile_begin;
    const int per_split = pairs_m * P.tiles_n;
    const int z = local / per_split;
    local -= z * per_split;
    constexpr int G = 8;
    const int group = local / (G * P.tiles_n);
    const int first = group * G;
    const int gm = min(G, pairs_m - first);
    const int in = local - group * G * P.tiles_n;
    const int mp = first + in % gm;
    const int nt = in / gm;
    PairTile r;
    r.prob = p;
    r.m0 = (int64_t)(2 * mp + rank) * kBM;
    r.n0 = (int64_t)nt * P.bn;
    r.z = z;
    const int kbt = P.kb0 + P.kb1;
    if (P.kb_per_split > 0) {
        r.kb_begin = z * P.kb_per_split;
        r.kb_end = min(kbt, r.kb_begin + P.kb_per_split);
    } else {
        r.kb_begin = 0;
        r.kb_end = kbt;
    }
    return r;
}

constexpr int kFuseNone = 0, kFuseFwd = 1, kFuseBwd = 2;

struct FuseArgs {
    int64_t T;
    int r;                       // 64 or 128
    const float *om1, *ph1, *om2, *ph2;
    const float *M;              // fp32 [r][r], b_j = sum_i a_i M[i][j]
    float *h_out, *b_out;        // forward: saved h, b (NULL: not saved)
    __nv_bfloat16 *c_out;        // forward: c
    const float *h_in, *b_in;    // backward: saved h, b
    __nv_bfloat16 *dh_out, *a_out, *db_out;
    float *part;                 // backward: [ceil(T / 32)][4][r] column sums per 32 tokens
    float *bias_part;            // backward: [ceil(T / 128)][kdim] column sums of dy, or NULL
    int64_t kdim;                // backward: columns of dy (d_out)
    uint32_t *flags;             // [2 * row pairs], zero at launch
};

// Fused tile order over `slot` (0 .. total tiles), in chunks of W row pairs,
// W = 8 floor(clusters / 8) (at least 8): the leader tiles (problem 0) of
// chunk 0, then for each chunk k the leaders of chunk k + 1 followed by the
// output tiles of chunk k (problems 1, 2, ..., each in locate_pair's group
// walk, which keeps groups of 8 row pairs together).  Every output tile thus
// comes at least one chunk of leaders after its own leader.
template <class EpiParams>
__device__ __forceinline__ int share_tile(const GroupArgs<EpiParams> &g, int p, int nclusters)
{
    const Problem<EpiParams> &L = g.p[0];
    const int pairs = (L.tiles_m + 1) / 2;
    int tn = 0;
    for (int q = 1; q < g.nproblems; ++q) tn += g.p[q].tiles_n;
    int W = (nclusters / 8) * 8;
    if (W < 8) W = 8;
    const int K = (pairs + W - 1) / W;
    auto nl = [&](int k) { return min(W, pairs - k * W); };
    if (p < nl(0)) return L.tile_begin + p;
    p -= nl(0);
#pragma unroll 1
    for (int k = 0; k < K; ++k) {
        if (k + 1 < K) {
            const int n = nl(k + 1);
            if (p < n) return L.tile_begin + (k + 1) * W + p;
            p -= n;
        }
        const int n = nl(k);
        if (p < n * tn) {
#pragma unroll 1
            for (int q = 1; q < g.nproblems; ++q) {
                const int m = n * g.p[q].tiles_n;
                if (p < m) return g.p[q].tile_begin + k * W * g.p[q].tiles_n + p;
                p -= m;
            }
        }
        p -= n * tn;
    }
    return -1;
}

__device__ __forceinline__ void mma2_bf16_ta(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc,
                                             uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], [%1], %2, %3, p;\n\t}\n" ::"r"(d_tmem),
        "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Tile of the given slot (see GroupArgs::sched); -1 when the slot is empty.
template <class EpiParams>
__device__ __forceinline__ int slot_tile(const GroupArgs<EpiParams> &g, int slot)
{
    if (g.sched_len == 0) return slot;
    const int t = g.sched[slot];
    return t == 0xFFFF ? -1 : t;
}

// Warps 0 (TMA), 1 (MMA, TMEM owner) and eight epilogue warps.
constexpr int kPairThreads = 320;

// Order in which a cluster issues the K segments of its tiles in a fused
// launch (producer and MMA warp alike; the epilogue warps replay it to know
// the ring position of a leader's stages).  Segment 0 of every tile comes in
// tile order.  Segment 1 of a deferred tile -- a leader, or the cluster's
// first tile -- comes only after the next tile's segment 0 (or before it,
// when that tile is deferred too), so that a leader's bottleneck epilogue,
// or the leader a first output tile waits for, overlaps a main loop; segment
// 1 of any other tile comes right after its segment 0.
struct SegOrder {
    bool prev_defer = false;
    // Calls emit(seg, which) for the next tile in order, where which = 0 names
    // this tile and 1 the pending previous deferred tile.
    template <class F>
    __device__ __forceinline__ void tile(bool defer, F &&emit)
    {
        if (prev_defer && defer) emit(1, 1);
        emit(0, 0);
        if (prev_defer && !defer) emit(1, 1);
        if (!defer) emit(1, 0);
        prev_defer = defer;
    }
    template <class F>
    __device__ __forceinline__ void finish(F &&emit)
    {
        if (prev_defer) emit(1, 1);
        prev_defer = false;
    }
};

// ---------------------------------------------------------------- fused bottleneck
// The mixing matrix as the B operand of the second product: this CTA's half of
// its rows n (output columns of b or da), n in [rank R/2, (rank + 1) R/2), all
// K = R, as bf16 high and low parts (x = x_hi + x_lo), K-major with the
// 128-byte swizzle in k-blocks of 64.  Forward B[n][k] = M[k][n]
// (b_j = sum_i a_i M[i][j]); backward B[n][k] = M[n][k] (da_i = sum_j db_j M[i][j]).
// Epilogue thread et (0..255) converts the groups gi = et + 256 it of eight
// consecutive k of one row n.
template <int R>
struct Mix {
    static constexpr int kHr = R / 2;
    static constexpr int kGroups = kHr * (R / 8);
    static constexpr int kIters = (kGroups + 255) / 256;
    static constexpr uint32_t kPartBytes = (uint32_t)(R / 64) * kHr * 128u;  // one of hi / lo
};

template <int R, int FUSE>
__device__ __forceinline__ void mix_load(const FuseArgs &fa, uint32_t rank, int et, float (&mr)[Mix<R>::kIters][8])
{
    using X = Mix<R>;
#pragma unroll
    for (int it = 0; it < X::kIters; ++it) {
        const int gi = et + 256 * it;
        if (gi >= X::kGroups) continue;
        const int n = (int)rank * X::kHr + gi % X::kHr, k = 8 * (gi / X::kHr);
        if constexpr (FUSE == kFuseBwd) {
            const float4 *src = reinterpret_cast<const float4 *>(fa.M + (int64_t)n * R + k);
            const float4 u = __ldg(src), w = __ldg(src + 1);
            mr[it][0] = u.x, mr[it][1] = u.y, mr[it][2] = u.z, mr[it][3] = u.w;
            mr[it][4] = w.x, mr[it][5] = w.y, mr[it][6] = w.z, mr[it][7] = w.w;
        } else {
#pragma unroll
            for (int q = 0; q < 8; ++q) mr[it][q] = __ldg(fa.M + (int64_t)(k + q) * R + n);
        }
    }
}

// x = hi + lo in bf16 for two values: packed high parts and packed low parts.
__device__ __forceinline__ void split_hi_lo(float x0, float x1, uint32_t &hi, uint32_t &lo)
{
    const __nv_bfloat162 h2 = __floats2bfloat162_rn(x0, x1);
    const float2 hf = __bfloat1622float2(h2);
    const __nv_bfloat162 l2 = __floats2bfloat162_rn(x0 - hf.x, x1 - hf.y);
    hi = *reinterpret_cast<const uint32_t *>(&h2);
    lo = *reinterpret_cast<const uint32_t *>(&l2);
}

template <int R>
__device__ __forceinline__ void mix_store(uint8_t *dst, int et, const float (&mr)[Mix<R>::kIters][8])
{
    using X = Mix<R>;
#pragma unroll
    for (int it = 0; it < X::kIters; ++it) {
        const int gi = et + 256 * it;
        if (gi >= X::kGroups) continue;
        const int nl = gi % X::kHr, k = 8 * (gi / X::kHr);
        uint4 hi, lo;
        split_hi_lo(mr[it][0], mr[it][1], hi.x, lo.x);
        split_hi_lo(mr[it][2], mr[it][3], hi.y, lo.y);
        split_hi_lo(mr[it][4], mr[it][5], hi.z, lo.z);
        split_hi_lo(mr[it][6], mr[it][7], hi.w, lo.w);
        const uint32_t off = (uint32_t)(k / 64) * X::kHr * 128u + (uint32_t)nl * 128u +
                             ((((uint32_t)(k % 64) >> 3) ^ ((uint32_t)nl & 7u)) << 4);
        *reinterpret_cast<uint4 *>(dst + off) = hi;
        *reinterpret_cast<uint4 *>(dst + X::kPartBytes + off) = lo;
    }
}

// Bottleneck epilogue of a leader tile (see the header), run by all eight
// epilogue warps of a CTA on its 128 rows.  `acc` is the tile's TMEM
// accumulator after segment 0: columns [0, R) hold the output columns
// [0, R) so far, [R, 2R) the branch pre-activation (h or dc).  A thread owns
// one row and the 32-column chunks c = 32 half + 64 i < R.  On return the
// output columns are back in [0, R) and c (or dh, a, db and the column sums)
// are stored.  Returns false, uniformly over the eight warps, after a
// timed-out wait.
template <int R, int FUSE>
__device__ __noinline__ bool leader_epilogue(const FuseArgs &fa, uint8_t *stg, uint32_t acc, int warp, int lane,
                                             int64_t m0, uint32_t rank, uint32_t a_ready_leader, uint32_t b_full,
                                             uint32_t parity, uint32_t *status)
{
    constexpr int NC = R / 64;  // 32-column chunks per thread
    const int quarter = warp % 4, half = (warp - 2) / 4;
    const int64_t t0 = m0 + quarter * 32;  // the warp's first row
    const bool live = t0 + lane < fa.T;
    const uint32_t lane_addr = acc + ((uint32_t)(quarter * 32) << 16);
    const int et = (warp - 2) * 32 + lane;
    float *part = FUSE == kFuseBwd ? fa.part + (t0 / 32) * 4 * (int64_t)R : nullptr;
    // ---- park the output columns: the second product writes b (da) there
    float park[NC][32];
#pragma unroll
    for (int i = 0; i < NC; ++i) ptx::tmem_ld_32x32b_x32(lane_addr + 32 * half + 64 * i, park[i]);
    // ---- phase 1: h or dc -> the row operand of the second product (a or
    // db), bf16 high parts of a chunk's 32 values in its first 16 columns and
    // low parts in the last 16 (two values per 32-bit column, lower k in the
    // low half), each warp overwriting only columns it has read itself
#pragma unroll
    for (int i = 0; i < NC; ++i) {
        const int c = 32 * half + 64 * i;
        float v[32];
        ptx::tmem_ld_32x32b_x32(lane_addr + R + c, v);
        uint32_t ohi[16], olo[16];
        if constexpr (FUSE == kFuseFwd) {
            if (fa.h_out) {
                uint32_t w[8][4];
#pragma unroll
                for (int g = 0; g < 8; ++g)
#pragma unroll
                    for (int q = 0; q < 4; ++q) w[g][q] = __float_as_uint(v[4 * g + q]);
                store_segments<8>(w, fa.h_out + t0 * R + c, (int64_t)R * 4, t0, fa.T);
            }
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                const int k = c + 2 * e;
                const float a0 = cos_reduced(fmaf(__ldg(fa.om1 + k), v[2 * e], __ldg(fa.ph1 + k)));
                const float a1 = cos_reduced(fmaf(__ldg(fa.om1 + k + 1), v[2 * e + 1], __ldg(fa.ph1 + k + 1)));
                split_hi_lo(a0, a1, ohi[e], olo[e]);
            }
        } else {
            // v = dc; with b of this row: du2 = -sin(omega2 b + phi2) dc (kept
            // in v), db = omega2 du2
            float bv[32];
            {
                uint32_t w[8][4];
                load_segments<8>(w, fa.b_in + t0 * R + c, (int64_t)R * 4, t0, fa.T);
#pragma unroll
                for (int g = 0; g < 8; ++g)
#pragma unroll
                    for (int q = 0; q < 4; ++q) bv[4 * g + q] = __uint_as_float(w[g][q]);
            }
            uint32_t wdb[4][4];
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                const int k = c + 2 * e;
                const float w0 = __ldg(fa.om2 + k), w1 = __ldg(fa.om2 + k + 1);
                const float d0 = live ? -sin_reduced(fmaf(w0, bv[2 * e], __ldg(fa.ph2 + k))) * v[2 * e] : 0.f;
                const float d1 = live ? -sin_reduced(fmaf(w1, bv[2 * e + 1], __ldg(fa.ph2 + k + 1))) * v[2 * e + 1] : 0.f;
                v[2 * e] = d0;
                v[2 * e + 1] = d1;
                split_hi_lo(w0 * d0, w1 * d1, ohi[e], olo[e]);
                wdb[e / 4][e % 4] = ohi[e];
            }
            store_segments<4>(wdb, fa.db_out + t0 * R + c, (int64_t)R * 2, t0, fa.T);
#pragma unroll
            for (int e = 0; e < 32; ++e) bv[e] *= v[e];  // du2 b
            const float s2 = warp_colsum32(bv);
            const float s3 = warp_colsum32(v);
            if (t0 < fa.T) {
                part[2 * R + c + lane] = s2;
                part[3 * R + c + lane] = s3;
            }
        }
        ptx::tmem_st_32x32b_x16(lane_addr + R + c, ohi);
        ptx::tmem_st_32x32b_x16(lane_addr + R + c + 16, olo);
    }
    // ---- the mixing matrix goes into the staging buffer once every warp's
    // TMA stores have left it
    {
        float mr[Mix<R>::kIters][8];
        mix_load<R, FUSE>(fa, rank, et, mr);
        if (lane == 0) ptx::bulk_wait_read_all();
        __syncwarp();
        ptx::tc_fence_before();
        ptx::named_barrier_sync(1, 256);
        ptx::tc_fence_after();
        mix_store<R>(stg, et, mr);
    }
    ptx::fence_proxy_async_smem_cluster();  // generic writes, read by the leader's MMA (async proxy)
    ptx::tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive_cluster(a_ready_leader);
    bool ok = ptx::mbar_wait(b_full, parity, status);
    ok = ptx::named_barrier_and(1, 256, __all_sync(0xffffffffu, ok));
    if (!ok) return false;
    ptx::tc_fence_after();
    // ---- phase 2: b or da in columns [0, R); then the parked columns go back
#pragma unroll
    for (int i = 0; i < NC; ++i) {
        const int c = 32 * half + 64 * i;
        float v[32];
        ptx::tmem_ld_32x32b_x32(lane_addr + c, v);
        if constexpr (FUSE == kFuseFwd) {
            // v = b: c = cos(omega2 b + phi2)
            uint32_t wc[4][4];
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                const int k = c + 2 * e;
                const float c0 = cos_reduced(fmaf(__ldg(fa.om2 + k), v[2 * e], __ldg(fa.ph2 + k)));
                const float c1 = cos_reduced(fmaf(__ldg(fa.om2 + k + 1), v[2 * e + 1], __ldg(fa.ph2 + k + 1)));
                wc[e / 4][e % 4] = ptx::pack_bf16x2(c0, c1);
            }
            if (fa.b_out) {
                uint32_t w[8][4];
#pragma unroll
                for (int g = 0; g < 8; ++g)
#pragma unroll
                    for (int q = 0; q < 4; ++q) w[g][q] = __float_as_uint(v[4 * g + q]);
                store_segments<8>(w, fa.b_out + t0 * R + c, (int64_t)R * 4, t0, fa.T);
            }
            store_segments<4>(wc, fa.c_out + t0 * R + c, (int64_t)R * 2, t0, fa.T);
        } else {
            // v = da; with h of this row: du1 = -sin(u1) da, dh = omega1 du1, a = cos(u1)
            float hv[32];
            {
                uint32_t w[8][4];
                load_segments<8>(w, fa.h_in + t0 * R + c, (int64_t)R * 4, t0, fa.T);
#pragma unroll
                for (int g = 0; g < 8; ++g)
#pragma unroll
                    for (int q = 0; q < 4; ++q) hv[4 * g + q] = __uint_as_float(w[g][q]);
            }
            uint32_t wdh[4][4], wa[4][4];
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                float dh2[2], av2[2];
#pragma unroll
                for (int u = 0; u < 2; ++u) {
                    const int k = c + 2 * e + u;
                    const float w1 = __ldg(fa.om1 + k);
                    float s1, c1;
                    sincos_reduced(fmaf(w1, hv[2 * e + u], __ldg(fa.ph1 + k)), &s1, &c1);
                    const float du1 = live ? -s1 * v[2 * e + u] : 0.f;
                    v[2 * e + u] = du1;
                    dh2[u] = w1 * du1;
                    av2[u] = c1;
                }
                wdh[e / 4][e % 4] = ptx::pack_bf16x2(dh2[0], dh2[1]);
                wa[e / 4][e % 4] = ptx::pack_bf16x2(av2[0], av2[1]);
            }
            store_segments<4>(wdh, fa.dh_out + t0 * R + c, (int64_t)R * 2, t0, fa.T);
            store_segments<4>(wa, fa.a_out + t0 * R + c, (int64_t)R * 2, t0, fa.T);
#pragma unroll
            for (int e = 0; e < 32; ++e) hv[e] *= v[e];  // du1 h
            const float s0 = warp_colsum32(hv);
            const float s1 = warp_colsum32(v);
            if (t0 < fa.T) {
                part[c + lane] = s0;
                part[R + c + lane] = s1;
            }
        }
        ptx::tmem_st_32x32b_x32(lane_addr + c, park[i]);
    }
    return true;
}

// MMA issuer of a fused launch (one thread of the leader CTA).  The k-block
// loop matches the default one: two ring stages per wait, their eight MMAs
// back to back.  Every wait is the suspending try_wait, bounded, and issues
// the pending second product of the last leader as soon as its epilogue has
// the row operand ready.
template <int STAGES, bool B_MN, bool MN4, int FUSE, class EpiParams>
struct FusedIssuer {
    const GroupArgs<EpiParams> &g;
    const FuseArgs &fa;
    uint32_t tmem, sbase, kA, kStage, kStgOff, bar0;
    uint32_t *status;
    int s = 0;
    uint32_t ph = 0;
    bool ok = true;
    bool m2_pending = false;
    uint32_t m2_acc = 0, m2_parity = 0, nlead = 0;

    __device__ __forceinline__ uint32_t full_bar(int i) const { return bar0 + 8u * i; }
    __device__ __forceinline__ uint32_t empty_bar(int i) const { return bar0 + 8u * (STAGES + i); }
    __device__ __forceinline__ uint32_t tfull_bar(int b) const { return bar0 + 8u * (2 * STAGES + b); }
    __device__ __forceinline__ uint32_t a_ready() const { return bar0 + 8u * (2 * STAGES + 5); }
    __device__ __forceinline__ uint32_t b_full() const { return bar0 + 8u * (2 * STAGES + 6); }
    __device__ __forceinline__ uint32_t consumed_bar(int i) const { return bar0 + 8u * (2 * STAGES + 8 + i); }

    // b | da (columns [0, r)) = (a | db in TMEM columns [r, 2r): per 32-column
    // chunk 16 columns of bf16 high parts, then 16 of low parts) x (matrix
    // hi/lo in the staging buffers of both CTAs), as hi*hi + lo*hi + hi*lo
    __device__ __forceinline__ void second_product()
    {
        ptx::tc_fence_after();
        const int r = fa.r;
        const uint32_t idesc2 = ptx::idesc_bf16(2 * kBM, r, false, false);
        const uint32_t mhi = sbase + kStgOff, mlo = mhi + (uint32_t)(r / 64) * (uint32_t)(r / 2) * 128u;
#pragma unroll 1
        for (int kk = 0; kk < r / 16; ++kk) {
            const uint32_t off = (uint32_t)(kk / 4) * (uint32_t)(r / 2) * 128u + (uint32_t)(kk % 4) * 32u;
            const uint64_t dmh = ptx::smem_desc_sw128(mhi + off, 16, 1024);
            const uint64_t dml = ptx::smem_desc_sw128(mlo + off, 16, 1024);
            const uint32_t ahi = m2_acc + (uint32_t)r + (uint32_t)(kk / 2) * 32u + (uint32_t)(kk % 2) * 8u;
            const uint32_t alo = ahi + 16u;
            mma2_bf16_ta(m2_acc, ahi, dmh, idesc2, kk > 0 ? 1u : 0u);
            mma2_bf16_ta(m2_acc, alo, dmh, idesc2, 1u);
            mma2_bf16_ta(m2_acc, ahi, dml, idesc2, 1u);
        }
        mma2_commit_mc(b_full(), 0x3);
        m2_pending = false;
    }

    __device__ __forceinline__ bool wait(uint32_t bar, uint32_t parity)
    {
        if (m2_pending && ptx::mbar_test_wait(a_ready(), m2_parity)) second_product();
        if (ptx::mbar_try_wait(bar, parity)) return true;
        const uint64_t t0 = ptx::globaltimer_ns();
        while (true) {
#pragma unroll 1
            for (int i = 0; i < 64; ++i) {
                if (m2_pending && ptx::mbar_test_wait(a_ready(), m2_parity)) second_product();
                if (ptx::mbar_try_wait(bar, parity)) return true;
            }
            if (ptx::globaltimer_ns() - t0 > ptx::kWaitLimitNs) {
                raise_status(status, kStatusTimeout);
                ok = false;
                return false;
            }
        }
    }

    // a leader's segment 0 is issued: its epilogue starts, its second product is pending
    __device__ __forceinline__ void lead_issued(int buf, uint32_t xfull)
    {
        mma2_commit_mc(xfull, 0x3);
        m2_pending = true;
        m2_acc = tmem + (uint32_t)buf * 256u;
        m2_parity = nlead & 1;
        ++nlead;
    }

    // the k-blocks of segment sg of tile tr into accumulator buffer buf
    __device__ __forceinline__ void seg(const PairTile &tr, int sg, int buf)
    {
        if (!ok) return;
        const auto &P = g.p[tr.prob];
        const bool bias_stage = FUSE == kFuseBwd && tr.prob == 0 && sg == 0 && fa.bias_part != nullptr;
        const uint32_t d_tmem = tmem + (uint32_t)buf * 256u;
        const uint32_t idesc = ptx::idesc_bf16(2 * kBM, P.bn, false, B_MN);
        const uint32_t nchB = (uint32_t)P.bn / 128;  // 64-wide B chunks held per CTA
        const uint64_t a0 = ptx::smem_desc_sw128(sbase, 16, 1024);
        const uint64_t b0 = B_MN ? (MN4 ? ptx::smem_desc_sw128(sbase + kA, 1024, 1024 * nchB)
                                        : ptx::smem_desc_sw128(sbase + kA, kChunkBytes, 1024))
                                 : ptx::smem_desc_sw128(sbase + kA, 16, 1024);
        const uint32_t stepB = B_MN ? (MN4 ? 128u * nchB : 2048u / 16) : 32u / 16;
        const uint32_t kStageUnits = kStage / 16;
        const int nkb = sg ? P.kb1 : P.kb0;
        const uint32_t acc0 = sg ? 1u : 0u;
        for (int i = 0; i < nkb; i += 2) {
            const bool two = i + 1 < nkb;
            int s2 = s + 1;
            uint32_t ph2 = ph;
            if (s2 == STAGES) {
                s2 = 0;
                ph2 ^= 1;
            }
            // the stages are usually full already: look for the epilogue's
            // signal here too, not only while waiting
            if (m2_pending && ptx::mbar_test_wait(a_ready(), m2_parity)) second_product();
            if (!wait(full_bar(s), ph) || (two && !wait(full_bar(s2), ph2))) return;
            const uint64_t so = (uint64_t)((uint32_t)s * kStageUnits);
            const uint64_t ad = a0 + so, bd = b0 + so;
            mma2_bf16(d_tmem, ad, bd, idesc, (i > 0 ? 1u : acc0));
#pragma unroll
            for (int kk = 1; kk < kBK / 16; ++kk) mma2_bf16(d_tmem, ad + kk * 2u, bd + kk * stepB, idesc, 1u);
            mma2_commit_mc(empty_bar(s), 0x3);
            if (bias_stage) mma2_commit_mc(consumed_bar(s), 0x3);
            if (two) {
                const uint64_t so2 = (uint64_t)((uint32_t)s2 * kStageUnits);
                const uint64_t ad2 = a0 + so2, bd2 = b0 + so2;
#pragma unroll
                for (int kk = 0; kk < kBK / 16; ++kk) mma2_bf16(d_tmem, ad2 + kk * 2u, bd2 + kk * stepB, idesc, 1u);
                mma2_commit_mc(empty_bar(s2), 0x3);
                if (bias_stage) mma2_commit_mc(consumed_bar(s2), 0x3);
                s = s2 + 1;
                ph = ph2;
                if (s == STAGES) {
                    s = 0;
                    ph ^= 1;
                }
            } else {
                s = s2;
                ph = ph2;
            }
        }
    }

    // segment 1 of tile tr, which completes its accumulator
    __device__ __forceinline__ void finish_seg(const PairTile &tr, int buf)
    {
        seg(tr, 1, buf);
        if (ok) mma2_commit_mc(tfull_bar(buf), 0x3);
    }
};

template <int STAGES>
struct PairSmem {
    static constexpr uint32_t kA = kBM * kBK * 2;         // 128 rows of A
    static constexpr uint32_t kB = 128 * kBK * 2;         // up to 128 columns of B
    static constexpr uint32_t kStage = kA + kB;
    static constexpr uint32_t kStgOff = STAGES * kStage;  // epilogue staging, 4 KB per epilogue warp
    static constexpr uint32_t kStgBytes = 8 * 4096;
    static constexpr uint32_t kBarOff = kStgOff + kStgBytes;
    // full, empty, tfull[2], tempty[2], mma_done; fused bottleneck: a_ready,
    // b_full, xfull, consumed[STAGES]
    static constexpr uint32_t kNumBars = 3 * STAGES + 8;
    static constexpr uint32_t kBytes = kBarOff + 8 * kNumBars + 16;
    static constexpr uint32_t kDynamic = kBytes + 1024;
};

// Problems of a launch must use bn in {128, 256} (64 or 128 B columns per CTA).
// MN4: MN-major operand tiles are loaded by one 4-D TMA each into the layout
//   [8-row K group][64-wide MN chunk][8 rows][128 B]
// (chunk stride 1 KB, group stride nchunks KB) instead of two or more 2-D
// boxes giving [MN chunk][64 K rows][128 B] (chunk stride 8 KB, group 1 KB).
// FUSE: kFuseNone, or a fused bottleneck launch (problem 0 leader tiles of
// N = 2r, problem 1 the other output tiles, see the header; A K-major).
template <bool A_MN, bool B_MN, int STAGES, class Epi, bool MN4 = false, int FUSE = kFuseNone>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kPairThreads, 1)
gemm_pair(const __grid_constant__ GroupMaps maps, const __grid_constant__ GroupArgs<typename Epi::Params> g,
          const __grid_constant__ FuseArgs fa)
{
    using S = PairSmem<STAGES>;
    constexpr uint32_t kAccCols = 256;
    constexpr uint32_t kCols = 512;

    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = ptx::smem_u32(smem_raw);
    const uint32_t sbase = (raw + 1023u) & ~1023u;
    uint8_t *smem = smem_raw + (sbase - raw);
    const uint32_t bar0 = sbase + S::kBarOff;
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (STAGES + s); };
    auto tfull_bar = [&](int b) { return bar0 + 8u * (2 * STAGES + b); };
    auto tempty_bar = [&](int b) { return bar0 + 8u * (2 * STAGES + 2 + b); };
    const uint32_t mma_done = bar0 + 8u * (2 * STAGES + 4);
    const uint32_t a_ready = bar0 + 8u * (2 * STAGES + 5);  // fused: row operand in TMEM, matrix in smem
    const uint32_t b_full = bar0 + 8u * (2 * STAGES + 6);   // fused: second product complete
    const uint32_t xfull = bar0 + 8u * (2 * STAGES + 7);    // fused: a leader's segment 0 complete
    // fused backward: the MMAs of a leader stage are done (its dy rows are summed for dbias)
    auto consumed_bar = [&](int s) { return bar0 + 8u * (2 * STAGES + 8 + s); };
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + S::kBarOff + 8 * S::kNumBars);

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const uint32_t rank = cluster_ctarank();
    const bool leader = rank == 0;
    const int cluster = blockIdx.x / 2, nclusters = gridDim.x / 2;

    if (warp == 0 && lane == 0) {
        ptx::griddep_launch();  // the next kernel of the call may take SMs as this grid frees them
        for (int p = 0; p < g.nproblems; ++p) {
            ptx::tma_prefetch_desc(&maps.m[p][0]);
            ptx::tma_prefetch_desc(&maps.m[p][1]);
            if (FUSE != kFuseNone) {
                ptx::tma_prefetch_desc(&maps.m[p][2]);
                ptx::tma_prefetch_desc(&maps.m[p][3]);
            }
        }
        if (FUSE != kFuseNone) ptx::tma_prefetch_desc(&maps.m[0][5]);
        for (int s = 0; s < STAGES; ++s) {
            ptx::mbar_init(full_bar(s), 1);
            // fused backward: the MMA commit and eight arrivals, from the
            // epilogue warps after summing a leader stage, else from the producer
            ptx::mbar_init(empty_bar(s), FUSE == kFuseBwd ? 9 : 1);
            ptx::mbar_init(consumed_bar(s), 1);
        }
        for (int b = 0; b < 2; ++b) {
            ptx::mbar_init(tfull_bar(b), 1);
            ptx::mbar_init(tempty_bar(b), 16);  // 8 epilogue warps in each CTA of the pair
        }
        ptx::mbar_init(mma_done, 1);
        ptx::mbar_init(a_ready, 16);  // 8 epilogue warps in each CTA of the pair
        ptx::mbar_init(b_full, 1);
        ptx::mbar_init(xfull, 1);
        ptx::fence_barrier_init();
    }
    if (warp == 1) {
        tmem_alloc2(ptx::smem_u32(tmem_slot), kCols);
        tmem_relinquish2();
    }
    ptx::tc_fence_before();
    __syncthreads();
    cluster_sync();  // the peer's barriers are initialised before any remote use
    ptx::tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if constexpr (FUSE != kFuseNone) {
        // ======================= fused bottleneck launch (see the header)
        const int nslots = g.total_tiles;
        if (warp == 0) {
            if (lane == 0) {
                // ---------------- producer (both CTAs)
                uint32_t it = 0;
                bool ok = true;
                SegOrder order;
                PairTile prev{};
                bool first = true;
                // the k-blocks of segment sg of tile tr into the ring
                auto load_seg = [&](const PairTile &tr, int sg) -> bool {
                    const auto &P = g.p[tr.prob];
                    const bool lead = tr.prob == 0;
                    const int bh = P.bn / 2;  // B columns held by this CTA
                    const int kb_begin = sg ? P.kb0 : 0, kb_end = sg ? P.kb0 + P.kb1 : P.kb0;
                    // the second segment reads c (dh) of this CTA's 128 rows,
                    // stored by the leader of its row pair
                    if (sg == 1 && kb_end > kb_begin && !ptx::flag_wait(fa.flags + tr.m0 / kBM, g.status))
                        return false;
                    const bool bias_stage = FUSE == kFuseBwd && lead && sg == 0 && fa.bias_part != nullptr;
                    const uint32_t b_bytes = (uint32_t)bh * kBK * 2;
                    // a leader's second segment: rank 1 holds no B (its half of
                    // the accumulator columns is not read again)
                    const bool load_b = !(lead && sg == 1 && rank == 1);
                    const uint32_t tx = 2 * S::kA + (lead && sg == 1 ? b_bytes : 2 * b_bytes);
                    const CUtensorMap *mA = &maps.m[tr.prob][sg ? 2 : 0];
                    const CUtensorMap *mB =
                        lead && sg == 0 && rank == 1 ? &maps.m[tr.prob][5] : &maps.m[tr.prob][sg ? 3 : 1];
                    const int nb = lead ? 0 : (int)tr.n0 + (int)rank * bh;
                    for (int kb = kb_begin; kb < kb_end; ++kb, ++it) {
                        const int s = it % STAGES;
                        const uint32_t ph = (it / STAGES) & 1;
                        if (!ptx::mbar_wait(empty_bar(s), ph ^ 1, g.status)) return false;
                        if constexpr (FUSE == kFuseBwd)
                            if (!bias_stage) ptx::mbar_arrive_cnt(empty_bar(s), 8);
                        const uint32_t fb = map_to_rank(full_bar(s), 0);
                        if (leader) ptx::mbar_arrive_expect_tx(full_bar(s), tx);
                        const uint32_t sA = sbase + s * S::kStage, sB = sA + S::kA;
                        const int k = (kb - kb_begin) * kBK;
                        tma_load_2d_pair(sA, mA, fb, k, (int)tr.m0);
                        if (load_b) {
                            if (B_MN && MN4) {
                                tma_load_4d_pair(sB, mB, fb, nb / 64, k / 8);
                            } else if (B_MN) {
                                for (int c = 0; c < bh / 64; ++c)
                                    tma_load_2d_pair(sB + c * kChunkBytes, mB, fb, nb + 64 * c, k);
                            } else {
                                tma_load_2d_pair(sB, mB, fb, k, nb);
                            }
                        }
                    }
                    return true;
                };
                for (int slot = cluster; ok && slot < nslots; slot += nclusters) {
                    const int t = share_tile(g, slot, nclusters);
                    if (t < 0) continue;
                    const PairTile tr = locate_pair(g, t, rank);
                    const bool defer = tr.prob == 0 || first;
                    first = false;
                    order.tile(defer, [&](int sg, int which) {
                        if (ok) ok = load_seg(which ? prev : tr, sg);
                    });
                    if (defer) prev = tr;
                }
                order.finish([&](int sg, int) {
                    if (ok) ok = load_seg(prev, sg);
                });
                // the leader's ring barriers also count the peer's bytes: once
                // they complete, no copy of either CTA is still landing
                if (leader) {
                    const uint32_t first = it > (uint32_t)STAGES ? it - STAGES : 0;
                    for (uint32_t i = first; i < it; ++i)
                        ptx::mbar_wait(full_bar(i % STAGES), (i / STAGES) & 1, nullptr);
                }
            }
        } else if (warp == 1) {
            if (lane == 0 && leader) {
                // ---------------- MMA issuer (leader CTA only)
                FusedIssuer<STAGES, B_MN, MN4, FUSE, typename Epi::Params> is{
                    g, fa, tmem, sbase, S::kA, S::kStage, S::kStgOff, bar0, g.status};
                int j = 0;
                bool prev_defer = false;
                PairTile prev{};
                int prev_buf = 0;
                for (int slot = cluster; is.ok; slot += nclusters) {
                    if (slot >= nslots) {
                        if (prev_defer) is.finish_seg(prev, prev_buf);
                        break;
                    }
                    const int t = share_tile(g, slot, nclusters);
                    if (t < 0) continue;
                    const PairTile tr = locate_pair(g, t, 0);
                    const bool lead = tr.prob == 0;
                    const bool defer = lead || j == 0;
                    const int b = j & 1;
                    const uint32_t use = (uint32_t)(j >> 1);
                    if (prev_defer && defer) is.finish_seg(prev, prev_buf);
                    if (!is.wait(tempty_bar(b), (use & 1) ^ 1)) break;
                    ptx::tc_fence_after();
                    is.seg(tr, 0, b);
                    if (is.ok && lead) is.lead_issued(b, xfull);
                    if (!defer) {
                        if (prev_defer) is.finish_seg(prev, prev_buf);
                        is.finish_seg(tr, b);
                    }
                    if (defer) {
                        prev = tr;
                        prev_buf = b;
                    }
                    prev_defer = defer;
                    ++j;
                }
                mma2_commit_mc(mma_done, 0x1);
                ptx::mbar_wait(mma_done, 0, nullptr);
            }
        } else {
            // ---------------- epilogue (both CTAs): own 128 accumulator rows
            const int quarter = warp % 4;
            const int half = (warp - 2) / 4;  // two warps per TMEM lane quarter split the columns
            const uint32_t leader_tempty0 = map_to_rank(tempty_bar(0), 0);
            const uint32_t leader_tempty1 = map_to_rank(tempty_bar(1), 0);
            const uint32_t leader_a_ready = map_to_rank(a_ready, 0);
            const uint32_t stg = sbase + S::kStgOff + (uint32_t)(warp - 2) * 4096u;
            uint8_t *stg_ptr = smem + S::kStgOff + (warp - 2) * 4096;
            int j = 0;
            uint32_t nlead = 0;
            uint32_t it = 0;    // ring position, replaying the issue order
            uint32_t cons = 0;  // per stage: parity of the next consumed_bar phase
            int prev_kb1 = 0;
            SegOrder order;
            for (int slot = cluster; slot < nslots; slot += nclusters) {
                const int t = share_tile(g, slot, nclusters);
                if (t < 0) continue;
                const PairTile tr = locate_pair(g, t, rank);
                const auto &P = g.p[tr.prob];
                const bool lead = tr.prob == 0;
                const int b = j & 1;
                const uint32_t use = (uint32_t)(j >> 1);
                uint32_t it_x = 0;
                order.tile(lead || j == 0, [&](int sg, int which) {
                    if (which) {
                        it += prev_kb1;
                    } else if (sg == 0) {
                        it_x = it;
                        it += P.kb0;
                    } else {
                        it += P.kb1;
                    }
                });
                if (lead || j == 0) prev_kb1 = P.kb1;
                bool ok = true;
                if (lead) {
                    if constexpr (FUSE == kFuseBwd) {
                        if (fa.bias_part) {
                            // dbias partials: the column sums of this CTA's dy rows,
                            // stage by stage once the MMAs have read it
                            const int ew = warp - 2;
                            for (int i = 0; i < P.kb0; ++i) {
                                const int s = (int)((it_x + i) % STAGES);
                                const uint32_t par = (cons >> s) & 1u;
                                cons ^= 1u << s;
                                ok = __all_sync(0xffffffffu, ptx::mbar_wait(consumed_bar(s), par, g.status));
                                if (!ok) break;
                                const float v = stage_colsum8(smem + s * S::kStage, ew, lane);
                                // the stage is refilled by the copy engine (async
                                // proxy) once released: order these reads before that
                                ptx::fence_proxy_async_smem();
                                __syncwarp();
                                if (lane == 0) ptx::mbar_arrive(empty_bar(s));
                                const int64_t col = (int64_t)i * kBK + 8 * ew + stage_colsum_col(lane);
                                if ((lane & 3) == 0 && tr.m0 < fa.T && col < fa.kdim)
                                    fa.bias_part[(tr.m0 / kBM) * fa.kdim + col] = v;
                            }
                        }
                    }
                    ok = ok && ptx::mbar_wait(xfull, nlead & 1, g.status);
                    ok = ptx::named_barrier_and(1, 256, __all_sync(0xffffffffu, ok));
                    if (!ok) break;
                    ptx::tc_fence_after();
                    const uint32_t acc = tmem + b * kAccCols;
                    ok = fa.r == 128 ? leader_epilogue<128, FUSE>(fa, smem + S::kStgOff, acc, warp, lane, tr.m0, rank,
                                                                  leader_a_ready, b_full, nlead & 1, g.status)
                                     : leader_epilogue<64, FUSE>(fa, smem + S::kStgOff, acc, warp, lane, tr.m0, rank,
                                                                 leader_a_ready, b_full, nlead & 1, g.status);
                    if (!ok) break;
                    // publish this CTA's c (dh) rows and its restored accumulator:
                    // the producers of this row block's second segments wait for it
                    ptx::tc_fence_before();
                    ptx::fence_proxy_async_global();
                    ptx::named_barrier_sync(1, 256);
                    if (warp == 2 && lane == 0) {
                        __threadfence();
                        ptx::fence_proxy_async_global();
                        ptx::st_release_gpu(fa.flags + tr.m0 / kBM, 1u);
                    }
                    ++nlead;
                }
                ok = ptx::mbar_wait(tfull_bar(b), use & 1, g.status);
                // named barriers above: leave together or not at all
                ok = ptx::named_barrier_and(1, 256, __all_sync(0xffffffffu, ok));
                if (!ok) break;
                ptx::tc_fence_after();
                const int bn_out = lead ? fa.r : P.bn;  // a leader stores its first r columns
                if (P.ep.tma)
                    Epi::run_tma(P.ep, &maps.m[tr.prob][4], stg_ptr, stg, tmem + b * kAccCols, bn_out, quarter, lane,
                                 tr.m0, tr.n0, P.N, tr.z, half);
                else
                    Epi::run_dyn(P.ep, tmem + b * kAccCols, bn_out, quarter, lane, tr.m0, tr.n0, P.M, P.N, tr.z,
                                 32 * half, 64);
                ptx::tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive_cluster(b ? leader_tempty1 : leader_tempty0);
                ++j;
            }
            if (lane == 0) ptx::bulk_wait_all();  // stores done before the staging buffer goes away
        }
    } else if (warp == 0) {
        if (lane == 0) {
            // ---------------- producer (both CTAs)
            uint32_t it = 0;
            bool ok = true;
            bool waited = false;  // for the predecessor grid (programmatic launch)
            const int nslots = g.sched_len ? g.sched_len : g.total_tiles;
            for (int slot = cluster; ok && slot < nslots; slot += nclusters) {
                const int t = slot_tile(g, slot);
                if (t < 0) continue;
                const PairTile tr = locate_pair(g, t, rank);
                const auto &P = g.p[tr.prob];
                const int bh = P.bn / 2;  // B columns held by this CTA
                const uint32_t cta_bytes = S::kA + (uint32_t)bh * kBK * 2;
                for (int kb = tr.kb_begin; kb < tr.kb_end; ++kb, ++it) {
                    const int s = it % STAGES;
                    const uint32_t ph = (it / STAGES) & 1;
                    if (!ptx::mbar_wait(empty_bar(s), ph ^ 1, g.status)) {
                        ok = false;
                        break;
                    }
                    const bool seg1 = kb >= P.kb0;
                    if (!waited && (P.dep & (seg1 ? 2 : 1))) {
                        ptx::griddep_wait();
                        waited = true;
                    }
                    const uint32_t fb = map_to_rank(full_bar(s), 0);
                    if (leader) ptx::mbar_arrive_expect_tx(full_bar(s), 2 * cta_bytes);
                    const uint32_t sA = sbase + s * S::kStage, sB = sA + S::kA;
                    const CUtensorMap *mA = &maps.m[tr.prob][seg1 ? 2 : 0];
                    const CUtensorMap *mB = &maps.m[tr.prob][seg1 ? 3 : 1];
                    const int k = (seg1 ? kb - P.kb0 : kb) * kBK;
                    const int nb = (int)tr.n0 + (int)rank * bh;
                    if (A_MN && MN4) {
                        tma_load_4d_pair(sA, mA, fb, (int)(tr.m0 / 64), k / 8);
                    } else if (A_MN) {
                        tma_load_2d_pair(sA, mA, fb, (int)tr.m0, k);
                        tma_load_2d_pair(sA + kChunkBytes, mA, fb, (int)tr.m0 + 64, k);
                    } else {
                        tma_load_2d_pair(sA, mA, fb, k, (int)tr.m0);
                    }
                    if (B_MN && MN4) {
                        tma_load_4d_pair(sB, mB, fb, nb / 64, k / 8);
                    } else if (B_MN) {
                        for (int c = 0; c < bh / 64; ++c) tma_load_2d_pair(sB + c * kChunkBytes, mB, fb, nb + 64 * c, k);
                    } else {
                        tma_load_2d_pair(sB, mB, fb, k, nb);
                    }
                }
            }
            // this grid completes only after its predecessor: what later kernels
            // of the call read through this grid's completion is then complete too
            if (!waited) ptx::griddep_wait();
            // the leader's ring barriers also count the peer's bytes: once they
            // complete, no copy of either CTA is still landing
            if (leader) {
                const uint32_t first = it > (uint32_t)STAGES ? it - STAGES : 0;
                for (uint32_t i = first; i < it; ++i)
                    ptx::mbar_wait(full_bar(i % STAGES), (i / STAGES) & 1, nullptr);
            }
        }
    } else if (warp == 1) {
        if (lane == 0 && leader) {
            // ---------------- MMA issuer (leader CTA only).  The loop keeps the
            // work between consecutive k-blocks small: operand descriptors are
            // a per-tile base plus additive offsets (start addresses are below
            // 256 KB, so the 14-bit address field never carries), and the ring
            // position advances incrementally.
            int s = 0;
            uint32_t ph = 0;
            int j = 0;
            bool ok = true;
            // descriptor address-field steps (16-byte units) per K-step of 16
            constexpr uint32_t kStepA = A_MN ? (MN4 ? 4096 / 16 : 2048 / 16) : 32 / 16;
            constexpr uint32_t kStageUnits = S::kStage / 16;
            const int nslots = g.sched_len ? g.sched_len : g.total_tiles;
            for (int slot = cluster; ok && slot < nslots; slot += nclusters) {
                const int t = slot_tile(g, slot);
                if (t < 0) continue;
                const PairTile tr = locate_pair(g, t, 0);
                const auto &P = g.p[tr.prob];
                const int b = j & 1;
                const uint32_t use = (uint32_t)(j >> 1);
                if (!ptx::mbar_wait(tempty_bar(b), (use & 1) ^ 1, g.status)) break;
                ptx::tc_fence_after();
                const uint32_t d_tmem = tmem + b * kAccCols;
                const uint32_t idesc = ptx::idesc_bf16(2 * kBM, P.bn, A_MN, B_MN);
                const uint32_t nchB = (uint32_t)P.bn / 128;  // 64-wide B chunks held per CTA
                const uint64_t a0 = A_MN ? (MN4 ? ptx::smem_desc_sw128(sbase, 1024, 2048)
                                                : ptx::smem_desc_sw128(sbase, kChunkBytes, 1024))
                                         : ptx::smem_desc_sw128(sbase, 16, 1024);
                const uint64_t b0 = B_MN ? (MN4 ? ptx::smem_desc_sw128(sbase + S::kA, 1024, 1024 * nchB)
                                                : ptx::smem_desc_sw128(sbase + S::kA, kChunkBytes, 1024))
                                         : ptx::smem_desc_sw128(sbase + S::kA, 16, 1024);
                const uint32_t stepB = B_MN ? (MN4 ? 128u * nchB : 2048u / 16) : 32u / 16;
                const int nkb = tr.kb_end - tr.kb_begin;
                for (int i = 0; i < nkb; i += 2) {
                    const bool two = i + 1 < nkb;
                    int s2 = s + 1;
                    uint32_t ph2 = ph;
                    if (s2 == STAGES) {
                        s2 = 0;
                        ph2 ^= 1;
                    }
                    if (!ptx::mbar_wait(full_bar(s), ph, g.status) || (two && !ptx::mbar_wait(full_bar(s2), ph2, g.status))) {
                        ok = false;
                        break;
                    }
                    // no tcgen05 fence here: the stages were written by TMA (the
                    // async proxy, as the MMA) and completed on the barrier waited for
                    const uint64_t so = (uint64_t)((uint32_t)s * kStageUnits);
                    const uint64_t ad = a0 + so, bd = b0 + so;
                    mma2_bf16(d_tmem, ad, bd, idesc, i > 0 ? 1u : 0u);
#pragma unroll
                    for (int kk = 1; kk < kBK / 16; ++kk)
                        mma2_bf16(d_tmem, ad + kk * kStepA, bd + kk * stepB, idesc, 1u);
                    mma2_commit_mc(empty_bar(s), 0x3);
                    if (two) {
                        const uint64_t so2 = (uint64_t)((uint32_t)s2 * kStageUnits);
                        const uint64_t ad2 = a0 + so2, bd2 = b0 + so2;
#pragma unroll
                        for (int kk = 0; kk < kBK / 16; ++kk)
                            mma2_bf16(d_tmem, ad2 + kk * kStepA, bd2 + kk * stepB, idesc, 1u);
                        mma2_commit_mc(empty_bar(s2), 0x3);
                        s = s2 + 1;
                        ph = ph2;
                        if (s == STAGES) {
                            s = 0;
                            ph ^= 1;
                        }
                    } else {
                        s = s2;
                        ph = ph2;
                    }
                }
                mma2_commit_mc(tfull_bar(b), 0x3);
                ++j;
            }
            mma2_commit_mc(mma_done, 0x1);
            ptx::mbar_wait(mma_done, 0, nullptr);
        }
    } else {
        // ---------------- epilogue (both CTAs): own 128 accumulator rows
        const int quarter = warp % 4;
        const int half = (warp - 2) / 4;  // two warps per TMEM lane quarter split the columns
        const uint32_t leader_tempty0 = map_to_rank(tempty_bar(0), 0);
        const uint32_t leader_tempty1 = map_to_rank(tempty_bar(1), 0);
        const uint32_t stg = sbase + S::kStgOff + (uint32_t)(warp - 2) * 4096u;
        uint8_t *stg_ptr = smem + S::kStgOff + (warp - 2) * 4096;
        int j = 0;
        const int nslots = g.sched_len ? g.sched_len : g.total_tiles;
        for (int slot = cluster; slot < nslots; slot += nclusters) {
            const int t = slot_tile(g, slot);
            if (t < 0) continue;
            const PairTile tr = locate_pair(g, t, rank);
            const auto &P = g.p[tr.prob];
            const int b = j & 1;
            const uint32_t use = (uint32_t)(j >> 1);
            bool ok = ptx::mbar_wait(tfull_bar(b), use & 1, g.status);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            ptx::tc_fence_after();
            if (P.ep.tma)
                Epi::run_tma(P.ep, &maps.m[tr.prob][4], stg_ptr, stg, tmem + b * kAccCols, P.bn, quarter, lane, tr.m0,
                             tr.n0, P.N, tr.z, half);
            else
                Epi::run_dyn(P.ep, tmem + b * kAccCols, P.bn, quarter, lane, tr.m0, tr.n0, P.M, P.N, tr.z, 32 * half,
                             64);
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(b ? leader_tempty1 : leader_tempty0);
            ++j;
        }
        if (lane == 0) ptx::bulk_wait_all();  // stores done before the staging buffer goes away
    }

    ptx::tc_fence_before();
    __syncthreads();
    cluster_sync();  // no CTA leaves while its peer may still touch its memory
    if (warp == 1) {
        ptx::tc_fence_after();
        tmem_dealloc2(tmem, kCols);
    }
}

}  // namespace pair
}  // namespace tc
}  // namespace noble
