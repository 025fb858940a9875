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
// Fused bottleneck (FUSE = kFuseFwd / kFuseBwd, on request through
// NOBLE_FLAG_FUSED_BRANCH; the separate kernels of tc_cosnet.cuh are the
// default because they are faster at the measured shapes): problem 0 of the launch is
// the r-wide GEMM of the low-rank branch, h = x W_down^T (forward) or
// dc = dy W_up (backward), one 256 x r tile per row pair, and problem 1 the
// output GEMM whose second K segment reads c = CosNet(h) (forward, Eq. 1-2)
// or dh (backward) of the same rows.  A bottleneck tile's epilogue runs the
// CosNet of Eq. 2 (or its chain rule) on the accumulator:
//   phase 1   a = cos(omega1 h + phi1)      | du2 = -sin(omega2 b + phi2) dc,
//                                           |   db = omega2 du2
//             as bf16 high and low parts written back into TMEM columns [0, r)
//   product   b = a M  (or da = db M^T), a second pair MMA with A in TMEM and
//             the mixing matrix (bf16 high/low, this CTA's half of its
//             columns) in the epilogue staging buffer, into columns
//             [128, 128 + r) of the same accumulator
//   phase 2   c = cos(omega2 b + phi2)      | du1 = -sin(omega1 h + phi1) da,
//                                           |   dh = omega1 du1, a = cos(u1)
// then stores c (dh) for its 128 rows and releases a flag per 128-row block.
// The producer of an output tile polls that flag (bounded) before loading
// its second segment.  Tiles run in the order of fused_tile, which puts
// every bottleneck tile before the output tiles that wait for it, so with all
// clusters resident every wait ends.
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
constexpr uint32_t kR2Col = 128;  // TMEM column of the bottleneck's second accumulator

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
    uint32_t *flags;             // [2 * row pairs], zero at launch
};

// Fused tile order: the bottleneck tiles of row-pair group 0, then for each
// group g the bottleneck tiles of group g + 1 followed by the output tiles of
// group g (groups of 8 row pairs as in locate_pair).
template <class EpiParams>
__device__ __forceinline__ int fused_tile(const GroupArgs<EpiParams> &g, int p)
{
    const Problem<EpiParams> &C = g.p[0], &O = g.p[1];
    const int pairs = (C.tiles_m + 1) / 2;
    const int ng = (pairs + 7) / 8;
    const int tn = O.tiles_n;
    const int c0 = min(8, pairs);
    if (p < c0) return C.tile_begin + p;
    p -= c0;
    // block gi = [C(gi + 1)] [O(gi)]; blocks below ng - 2 are all 8 + 8 tn long
    const int full = 8 + 8 * tn;
    int gi = 0;
    if (ng > 2) {
        gi = min(p / full, ng - 2);
        p -= gi * full;
    }
#pragma unroll 1
    for (; gi < ng; ++gi) {
        const int cn = gi + 1 < ng ? min(8, pairs - 8 * (gi + 1)) : 0;
        const int on = min(8, pairs - 8 * gi) * tn;
        if (p < cn) return C.tile_begin + 8 * (gi + 1) + p;
        p -= cn;
        if (p < on) return O.tile_begin + 8 * gi * tn + p;
        p -= on;
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

// ---------------------------------------------------------------- fused bottleneck
// The mixing matrix as the B operand of the second product: this CTA's half of
// its rows n (output columns of b or da), n in [rank r/2, (rank + 1) r/2), all
// K = r, as bf16 high and low parts (x = x_hi + x_lo), K-major with the
// 128-byte swizzle in k-blocks of 64.  Forward B[n][k] = M[k][n]
// (b_j = sum_i a_i M[i][j]); backward B[n][k] = M[n][k] (da_i = sum_j db_j M[i][j]).
// Epilogue thread et (0..255) converts the groups gi = et + 256 it of eight
// consecutive k of one row n.
template <int FUSE>
__device__ __forceinline__ void mix_load(const FuseArgs &fa, uint32_t rank, int et, float (&mr)[4][8])
{
    const int r = fa.r, hr = r / 2, ngroups = hr * (r / 8);
#pragma unroll
    for (int it = 0; it < 4; ++it) {
        const int gi = et + 256 * it;
        if (gi >= ngroups) continue;
        const int n = (int)rank * hr + gi % hr, k = 8 * (gi / hr);
        if constexpr (FUSE == kFuseBwd) {
            const float4 *src = reinterpret_cast<const float4 *>(fa.M + (int64_t)n * r + k);
            const float4 u = __ldg(src), w = __ldg(src + 1);
            mr[it][0] = u.x, mr[it][1] = u.y, mr[it][2] = u.z, mr[it][3] = u.w;
            mr[it][4] = w.x, mr[it][5] = w.y, mr[it][6] = w.z, mr[it][7] = w.w;
        } else {
#pragma unroll
            for (int q = 0; q < 8; ++q) mr[it][q] = __ldg(fa.M + (int64_t)(k + q) * r + n);
        }
    }
}

__device__ __forceinline__ uint32_t mix_part_bytes(int r) { return (uint32_t)(r / 64) * (uint32_t)(r / 2) * 128u; }

__device__ __forceinline__ void mix_store(int r, uint8_t *dst, int et, const float (&mr)[4][8])
{
    const int hr = r / 2, ngroups = hr * (r / 8);
    const uint32_t part = mix_part_bytes(r);
#pragma unroll
    for (int it = 0; it < 4; ++it) {
        const int gi = et + 256 * it;
        if (gi >= ngroups) continue;
        const int nl = gi % hr, k = 8 * (gi / hr);
        uint4 hi, lo;
        uint32_t *ph = &hi.x, *pl = &lo.x;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const __nv_bfloat162 h2 = __floats2bfloat162_rn(mr[it][2 * q], mr[it][2 * q + 1]);
            const float2 hf = __bfloat1622float2(h2);
            const __nv_bfloat162 l2 = __floats2bfloat162_rn(mr[it][2 * q] - hf.x, mr[it][2 * q + 1] - hf.y);
            ph[q] = *reinterpret_cast<const uint32_t *>(&h2);
            pl[q] = *reinterpret_cast<const uint32_t *>(&l2);
        }
        const uint32_t off = (uint32_t)(k / 64) * hr * 128u + (uint32_t)nl * 128u +
                             ((((uint32_t)(k % 64) >> 3) ^ ((uint32_t)nl & 7u)) << 4);
        *reinterpret_cast<uint4 *>(dst + off) = hi;
        *reinterpret_cast<uint4 *>(dst + part + off) = lo;
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

// Epilogue of a bottleneck tile (see the header), run by all eight epilogue
// warps of a CTA on its 128 rows; `acc` is the tile's TMEM accumulator.  A
// thread owns one row and the 32-column chunks c = 32 half + 64 i < r.
// Returns false, uniformly over the eight warps, after a timed-out wait.
template <int FUSE>
__device__ __noinline__ bool bottleneck_epilogue(const FuseArgs &fa, uint8_t *stg, uint32_t acc, int warp, int lane, int64_t m0,
                                    uint32_t rank, uint32_t a_ready_leader, uint32_t b_full, uint32_t parity,
                                    uint32_t *status)
{
    const int r = fa.r;
    const int quarter = warp % 4, half = (warp - 2) / 4;
    const int64_t t0 = m0 + quarter * 32;  // the warp's first row
    const bool live = t0 + lane < fa.T;
    const uint32_t lane_addr = acc + ((uint32_t)(quarter * 32) << 16);
    const int et = (warp - 2) * 32 + lane;
    float *part = FUSE == kFuseBwd ? fa.part + (t0 / 32) * 4 * (int64_t)r : nullptr;
    // ---- phase 1: first accumulator (h or dc).  The row operand of the
    // second product (a or db) replaces each 32-column chunk it came from:
    // bf16 high parts of its 32 values in the chunk's first 16 columns, low
    // parts in the last 16 (two values per 32-bit column, lower k in the low
    // half), so each warp overwrites only columns it has read itself.
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const int c = 32 * half + 64 * i;
        if (c >= r) continue;
        float v[32];
        ptx::tmem_ld_32x32b_x32(lane_addr + c, v);
        uint32_t ohi[16], olo[16];
        if constexpr (FUSE == kFuseFwd) {
            if (fa.h_out) {
                uint32_t w[8][4];
#pragma unroll
                for (int g = 0; g < 8; ++g)
#pragma unroll
                    for (int q = 0; q < 4; ++q) w[g][q] = __float_as_uint(v[4 * g + q]);
                store_segments<8>(w, fa.h_out + t0 * r + c, (int64_t)r * 4, t0, fa.T);
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
                load_segments<8>(w, fa.b_in + t0 * r + c, (int64_t)r * 4, t0, fa.T);
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
            store_segments<4>(wdb, fa.db_out + t0 * r + c, (int64_t)r * 2, t0, fa.T);
#pragma unroll
            for (int e = 0; e < 32; ++e) bv[e] *= v[e];  // du2 b
            const float s2 = warp_colsum32(bv);
            const float s3 = warp_colsum32(v);
            if (t0 < fa.T) {
                part[2 * r + c + lane] = s2;
                part[3 * r + c + lane] = s3;
            }
        }
        ptx::tmem_st_32x32b_x16(lane_addr + c, ohi);
        ptx::tmem_st_32x32b_x16(lane_addr + c + 16, olo);
    }
    // ---- the mixing matrix goes into the staging buffer once every warp's
    // TMA stores have left it
    {
        float mr[4][8];
        mix_load<FUSE>(fa, rank, et, mr);
        if (lane == 0) ptx::bulk_wait_read_all();
        __syncwarp();
        ptx::tc_fence_before();
        ptx::named_barrier_sync(1, 256);
        ptx::tc_fence_after();
        mix_store(r, stg, et, mr);
    }
    ptx::fence_proxy_async_smem_cluster();  // generic writes, read by the leader's MMA (async proxy)
    ptx::tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive_cluster(a_ready_leader);
    bool ok = ptx::mbar_wait(b_full, parity, status);
    ok = ptx::named_barrier_and(1, 256, __all_sync(0xffffffffu, ok));
    if (!ok) return false;
    ptx::tc_fence_after();
    // ---- phase 2: second accumulator (b or da)
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const int c = 32 * half + 64 * i;
        if (c >= r) continue;
        float v[32];
        ptx::tmem_ld_32x32b_x32(lane_addr + kR2Col + c, v);
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
                store_segments<8>(w, fa.b_out + t0 * r + c, (int64_t)r * 4, t0, fa.T);
            }
            store_segments<4>(wc, fa.c_out + t0 * r + c, (int64_t)r * 2, t0, fa.T);
        } else {
            // v = da; with h of this row: du1 = -sin(u1) da, dh = omega1 du1, a = cos(u1)
            float hv[32];
            {
                uint32_t w[8][4];
                load_segments<8>(w, fa.h_in + t0 * r + c, (int64_t)r * 4, t0, fa.T);
#pragma unroll
                for (int g = 0; g < 8; ++g)
#pragma unroll
                    for (int q = 0; q < 4; ++q) hv[4 * g + q] = __uint_as_float(w[g][q]);
            }
            // du1 kept in v
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
            store_segments<4>(wdh, fa.dh_out + t0 * r + c, (int64_t)r * 2, t0, fa.T);
            store_segments<4>(wa, fa.a_out + t0 * r + c, (int64_t)r * 2, t0, fa.T);
#pragma unroll
            for (int e = 0; e < 32; ++e) hv[e] *= v[e];  // du1 h
            const float s0 = warp_colsum32(hv);
            const float s1 = warp_colsum32(v);
            if (t0 < fa.T) {
                part[c + lane] = s0;
                part[r + c + lane] = s1;
            }
        }
    }
    return true;
}

template <int STAGES>
struct PairSmem {
    static constexpr uint32_t kA = kBM * kBK * 2;         // 128 rows of A
    static constexpr uint32_t kB = 128 * kBK * 2;         // up to 128 columns of B
    static constexpr uint32_t kStage = kA + kB;
    static constexpr uint32_t kStgOff = STAGES * kStage;  // epilogue staging, 4 KB per epilogue warp
    static constexpr uint32_t kStgBytes = 8 * 4096;
    static constexpr uint32_t kBarOff = kStgOff + kStgBytes;
    static constexpr uint32_t kNumBars = 2 * STAGES + 7;  // full, empty, tfull[2], tempty[2], mma_done,
                                                          // a_ready, b_full (fused bottleneck)
    static constexpr uint32_t kBytes = kBarOff + 8 * kNumBars + 16;
    static constexpr uint32_t kDynamic = kBytes + 1024;
};

// Problems of a launch must use bn in {128, 256} (64 or 128 B columns per CTA).
// MN4: MN-major operand tiles are loaded by one 4-D TMA each into the layout
//   [8-row K group][64-wide MN chunk][8 rows][128 B]
// (chunk stride 1 KB, group stride nchunks KB) instead of two or more 2-D
// boxes giving [MN chunk][64 K rows][128 B] (chunk stride 8 KB, group 1 KB).
// FUSE: kFuseNone, or a fused bottleneck launch (problem 0 bottleneck tiles
// of N = r <= 128 with bn = 128, problem 1 output tiles, see the header).
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
    auto tile_of = [&](int slot) { return FUSE != kFuseNone ? fused_tile(g, slot) : slot_tile(g, slot); };
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
        }
        for (int s = 0; s < STAGES; ++s) {
            ptx::mbar_init(full_bar(s), 1);
            ptx::mbar_init(empty_bar(s), 1);
        }
        for (int b = 0; b < 2; ++b) {
            ptx::mbar_init(tfull_bar(b), 1);
            ptx::mbar_init(tempty_bar(b), 16);  // 8 epilogue warps in each CTA of the pair
        }
        ptx::mbar_init(mma_done, 1);
        ptx::mbar_init(a_ready, 16);  // 8 epilogue warps in each CTA of the pair
        ptx::mbar_init(b_full, 1);
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

    if (warp == 0) {
        if (lane == 0) {
            // ---------------- producer (both CTAs)
            uint32_t it = 0;
            bool ok = true;
            bool waited = false;  // for the predecessor grid (programmatic launch)
            const int nslots = g.sched_len ? g.sched_len : g.total_tiles;
            for (int slot = cluster; ok && slot < nslots; slot += nclusters) {
                const int t = tile_of(slot);
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
                    if constexpr (FUSE != kFuseNone) {
                        // the second segment of an output tile reads c (dh) of
                        // this CTA's 128 rows, stored by a bottleneck tile
                        if (tr.prob == 1 && kb == P.kb0 && !ptx::flag_wait(fa.flags + tr.m0 / kBM, g.status)) {
                            ok = false;
                            break;
                        }
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
            uint32_t nc = 0;  // bottleneck tiles so far
            for (int slot = cluster; ok && slot < nslots; slot += nclusters) {
                const int t = tile_of(slot);
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
                if constexpr (FUSE != kFuseNone) {
                    if (ok && tr.prob == 0) {
                        // second product of the bottleneck tile: b | da (cols
                        // kR2Col..) = (a | db in TMEM cols [0, r): per 32-column
                        // chunk 16 columns of bf16 high parts, then 16 of low
                        // parts) x (matrix hi/lo in the staging buffers of both
                        // CTAs), as hi*hi + lo*hi + hi*lo
                        if (!ptx::mbar_wait(a_ready, nc & 1, g.status)) break;
                        ptx::tc_fence_after();
                        const int r = fa.r;
                        const uint32_t acc = tmem + b * kAccCols;
                        const uint32_t idesc2 = ptx::idesc_bf16(2 * kBM, r, false, false);
                        const uint32_t mhi = sbase + S::kStgOff, mlo = mhi + mix_part_bytes(r);
                        for (int kk = 0; kk < r / 16; ++kk) {
                            const uint32_t off = (uint32_t)(kk / 4) * (uint32_t)(r / 2) * 128u + (uint32_t)(kk % 4) * 32u;
                            const uint64_t dmh = ptx::smem_desc_sw128(mhi + off, 16, 1024);
                            const uint64_t dml = ptx::smem_desc_sw128(mlo + off, 16, 1024);
                            const uint32_t ahi = acc + (uint32_t)(kk / 2) * 32u + (uint32_t)(kk % 2) * 8u;
                            const uint32_t alo = ahi + 16u;
                            mma2_bf16_ta(acc + kR2Col, ahi, dmh, idesc2, kk > 0 ? 1u : 0u);
                            mma2_bf16_ta(acc + kR2Col, alo, dmh, idesc2, 1u);
                            mma2_bf16_ta(acc + kR2Col, ahi, dml, idesc2, 1u);
                        }
                        mma2_commit_mc(b_full, 0x3);
                        ++nc;
                    }
                }
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
        uint32_t nc = 0;  // bottleneck tiles so far
        const uint32_t leader_a_ready = map_to_rank(a_ready, 0);
        const int nslots = g.sched_len ? g.sched_len : g.total_tiles;
        for (int slot = cluster; slot < nslots; slot += nclusters) {
            const int t = tile_of(slot);
            if (t < 0) continue;
            const PairTile tr = locate_pair(g, t, rank);
            const auto &P = g.p[tr.prob];
            const int b = j & 1;
            const uint32_t use = (uint32_t)(j >> 1);
            const bool bneck = FUSE != kFuseNone && tr.prob == 0;
            bool ok = ptx::mbar_wait(tfull_bar(b), use & 1, g.status);
            ok = __all_sync(0xffffffffu, ok);
            // fused launches use named barriers below: leave together or not at all
            if constexpr (FUSE != kFuseNone) ok = ptx::named_barrier_and(1, 256, ok);
            if (!ok) break;
            ptx::tc_fence_after();
            if constexpr (FUSE != kFuseNone) {
                if (bneck) {
                    if (!bottleneck_epilogue<FUSE>(fa, smem + S::kStgOff, tmem + b * kAccCols, warp, lane, tr.m0,
                                                   rank, leader_a_ready, b_full, nc & 1, g.status))
                        break;
                    ptx::tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive_cluster(b ? leader_tempty1 : leader_tempty0);
                    // every warp's stores of this CTA's rows are issued: publish them
                    ptx::named_barrier_sync(1, 256);
                    if (warp == 2 && lane == 0) {
                        __threadfence();
                        ptx::fence_proxy_async_global();
                        ptx::st_release_gpu(fa.flags + tr.m0 / kBM, 1u);
                    }
                    ++nc;
                    ++j;
                    continue;
                }
            }
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
