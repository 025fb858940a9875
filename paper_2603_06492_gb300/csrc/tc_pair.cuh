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
#pragma once

#include "tc_persistent.cuh"

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

template <int STAGES>
struct PairSmem {
    static constexpr uint32_t kA = kBM * kBK * 2;         // 128 rows of A
    static constexpr uint32_t kB = 128 * kBK * 2;         // up to 128 columns of B
    static constexpr uint32_t kStage = kA + kB;
    static constexpr uint32_t kStgOff = STAGES * kStage;  // epilogue staging, 4 KB per epilogue warp
    static constexpr uint32_t kStgBytes = 8 * 4096;
    static constexpr uint32_t kBarOff = kStgOff + kStgBytes;
    static constexpr uint32_t kNumBars = 2 * STAGES + 5;  // full, empty, tfull[2], tempty[2], mma_done
    static constexpr uint32_t kBytes = kBarOff + 8 * kNumBars + 16;
    static constexpr uint32_t kDynamic = kBytes + 1024;
};

// Problems of a launch must use bn in {128, 256} (64 or 128 B columns per CTA).
// MN4: MN-major operand tiles are loaded by one 4-D TMA each into the layout
//   [8-row K group][64-wide MN chunk][8 rows][128 B]
// (chunk stride 1 KB, group stride nchunks KB) instead of two or more 2-D
// boxes giving [MN chunk][64 K rows][128 B] (chunk stride 8 KB, group 1 KB).
template <bool A_MN, bool B_MN, int STAGES, class Epi, bool MN4 = false>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kPairThreads, 1)
gemm_pair(const __grid_constant__ GroupMaps maps, const __grid_constant__ GroupArgs<typename Epi::Params> g)
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
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + S::kBarOff + 8 * S::kNumBars);

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const uint32_t rank = cluster_ctarank();
    const bool leader = rank == 0;
    const int cluster = blockIdx.x / 2, nclusters = gridDim.x / 2;

    if (warp == 0 && lane == 0) {
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
                    const uint32_t fb = map_to_rank(full_bar(s), 0);
                    if (leader) ptx::mbar_arrive_expect_tx(full_bar(s), 2 * cta_bytes);
                    const uint32_t sA = sbase + s * S::kStage, sB = sA + S::kA;
                    const bool seg1 = kb >= P.kb0;
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
                    ptx::tc_fence_after();
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
