// Persistent, grouped tcgen05 GEMM: one CTA per SM walks a static
// round-robin list of 128 x BN output tiles drawn from up to kMaxProblems
// independent GEMM problems.  The TMEM accumulator is double-buffered, so the
// epilogue of one tile runs while the MMAs of the next tile are in flight,
// and the TMA producer runs ahead across tile boundaries.
//
// Each problem p computes
//     C_p[z][m][n] = sum_k A0_p(m,k) B0_p(n,k) + sum_k A1_p(m,k) B1_p(n,k)
// with its own N tile bn_p (a multiple of 32 not above BN_MAX; 64-wide
// multiples when B is MN-major), its own operands (TMA maps) and its own
// epilogue parameters; split-K problems write partial tiles per z.
// Operand majorness (A_MN, B_MN) is shared by all problems of a launch.
#pragma once

#include "tc_gemm.cuh"

namespace noble {
namespace tc {

constexpr int kMaxProblems = 6;

template <class EpiParams>
struct Problem {
    int64_t M, N;
    int kb0, kb1;          // k-blocks of segment 0 / 1
    int bn;                // N tile of this problem
    int tiles_m, tiles_n;  // output tiles
    int nsplit, kb_per_split;
    int tile_begin;        // first global tile index of this problem
    EpiParams ep;
};

// Optional explicit schedule (CTA-pair launches): slot j * nclusters + c
// holds the j-th tile of cluster c, 0xFFFF for none.  sched_len = 0 means
// plain round-robin over tile indices.
constexpr int kMaxSched = 2048;

template <class EpiParams>
struct GroupArgs {
    Problem<EpiParams> p[kMaxProblems];
    int nproblems;
    int total_tiles;
    uint32_t *status;
    int sched_len;
    uint16_t sched[kMaxSched];
};

struct GroupMaps {
    CUtensorMap m[kMaxProblems][5];  // A0, B0, A1, B1, C (pair kernel's TMA-store epilogue)
};

struct TileRef {
    int prob;
    int64_t m0, n0;
    int z;
    int kb_begin, kb_end;
};

// Tiles of a problem are ordered split-major, then in groups of 8 row
// blocks with the column index running fastest inside each group, so the
// tiles in flight at one time share A row blocks and B column blocks in L2.
template <class EpiParams>
__device__ __forceinline__ TileRef locate_tile(const GroupArgs<EpiParams> &g, int t)
{
    int p = 0;
#pragma unroll 1
    while (p + 1 < g.nproblems && t >= g.p[p + 1].tile_begin) ++p;
    const Problem<EpiParams> &P = g.p[p];
    int local = t - P.tile_begin;
    const int per_split = P.tiles_m * P.tiles_n;
    const int z = local / per_split;
    local -= z * per_split;
    constexpr int G = 8;
    const int group = local / (G * P.tiles_n);
    const int first_m = group * G;
    const int gm = min(G, P.tiles_m - first_m);
    const int in = local - group * G * P.tiles_n;
    const int mt = first_m + in % gm;
    const int nt = in / gm;
    TileRef r;
    r.prob = p;
    r.m0 = (int64_t)mt * kBM;
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

template <int BN_MAX, int STAGES>
struct PSmem {
    static constexpr uint32_t kA = kBM * kBK * 2;
    static constexpr uint32_t kB = BN_MAX * kBK * 2;
    static constexpr uint32_t kStage = kA + kB;
    static constexpr uint32_t kBarOff = STAGES * kStage;
    // full[S], empty[S], tmem_full[2], tmem_empty[2], mma_done
    static constexpr uint32_t kNumBars = 2 * STAGES + 5;
    static constexpr uint32_t kBytes = kBarOff + 8 * kNumBars + 16;
    static constexpr uint32_t kDynamic = kBytes + 1024;
};

template <int BN_MAX, bool A_MN, bool B_MN, int STAGES, class Epi>
__global__ void __launch_bounds__(kThreads, 1)
gemm_persistent(const __grid_constant__ GroupMaps maps, const __grid_constant__ GroupArgs<typename Epi::Params> g)
{
    using S = PSmem<BN_MAX, STAGES>;
    constexpr uint32_t kAccCols = TmemCols<BN_MAX>::value;  // per accumulator buffer
    constexpr uint32_t kCols = 2 * kAccCols;
    static_assert(kCols <= 512, "two accumulators must fit in TMEM");

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
            ptx::mbar_init(tempty_bar(b), 4);  // one arrive per epilogue warp
        }
        ptx::mbar_init(mma_done, 1);
        ptx::fence_barrier_init();
    }
    if (warp == 1) {
        ptx::tmem_alloc(ptx::smem_u32(tmem_slot), kCols);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            // ---------------- TMA producer: continuous k-block stream over all tiles
            uint32_t it = 0;
            bool ok = true;
            for (int t = blockIdx.x; ok && t < g.total_tiles; t += gridDim.x) {
                const TileRef tr = locate_tile(g, t);
                const auto &P = g.p[tr.prob];
                const uint32_t stage_bytes = S::kA + (uint32_t)P.bn * kBK * 2;
                for (int kb = tr.kb_begin; kb < tr.kb_end; ++kb, ++it) {
                    const int s = it % STAGES;
                    const uint32_t ph = (it / STAGES) & 1;
                    if (!ptx::mbar_wait(empty_bar(s), ph ^ 1, g.status)) {
                        ok = false;
                        break;
                    }
                    const uint32_t fb = full_bar(s);
                    ptx::mbar_arrive_expect_tx(fb, stage_bytes);
                    const uint32_t sA = sbase + s * S::kStage, sB = sA + S::kA;
                    const bool seg1 = kb >= P.kb0;
                    const CUtensorMap *mA = &maps.m[tr.prob][seg1 ? 2 : 0];
                    const CUtensorMap *mB = &maps.m[tr.prob][seg1 ? 3 : 1];
                    const int k = (seg1 ? kb - P.kb0 : kb) * kBK;
                    if (A_MN) {
                        ptx::tma_load_2d(sA, mA, fb, (int)tr.m0, k);
                        ptx::tma_load_2d(sA + kChunkBytes, mA, fb, (int)tr.m0 + 64, k);
                    } else {
                        ptx::tma_load_2d(sA, mA, fb, k, (int)tr.m0);
                    }
                    if (B_MN) {
                        for (int c = 0; c < P.bn / 64; ++c)
                            ptx::tma_load_2d(sB + c * kChunkBytes, mB, fb, (int)tr.n0 + 64 * c, k);
                    } else {
                        ptx::tma_load_2d(sB, mB, fb, k, (int)tr.n0);
                    }
                }
            }
            // no copy may still be landing in shared memory when the CTA exits
            const uint32_t first = it > (uint32_t)STAGES ? it - STAGES : 0;
            for (uint32_t i = first; i < it; ++i) ptx::mbar_wait(full_bar(i % STAGES), (i / STAGES) & 1, nullptr);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ---------------- MMA issuer
            uint32_t it = 0;
            int j = 0;
            bool ok = true;
            for (int t = blockIdx.x; ok && t < g.total_tiles; t += gridDim.x, ++j) {
                const TileRef tr = locate_tile(g, t);
                const auto &P = g.p[tr.prob];
                const int b = j & 1;
                const uint32_t use = (uint32_t)(j >> 1);
                if (!ptx::mbar_wait(tempty_bar(b), (use & 1) ^ 1, g.status)) break;
                ptx::tc_fence_after();
                const uint32_t d_tmem = tmem + b * kAccCols;
                const uint32_t idesc = ptx::idesc_bf16(kBM, P.bn, A_MN, B_MN);
                bool first = true;
                for (int kb = tr.kb_begin; kb < tr.kb_end; ++kb, ++it) {
                    const int s = it % STAGES;
                    const uint32_t ph = (it / STAGES) & 1;
                    if (!ptx::mbar_wait(full_bar(s), ph, g.status)) {
                        ok = false;
                        break;
                    }
                    ptx::tc_fence_after();
                    const uint32_t sA = sbase + s * S::kStage, sB = sA + S::kA;
#pragma unroll
                    for (int kk = 0; kk < kBK / 16; ++kk) {
                        const uint64_t ad = A_MN ? ptx::smem_desc_sw128(sA + kk * 2048, kChunkBytes, 1024)
                                                 : ptx::smem_desc_sw128(sA + kk * 32, 16, 1024);
                        const uint64_t bd = B_MN ? ptx::smem_desc_sw128(sB + kk * 2048, kChunkBytes, 1024)
                                                 : ptx::smem_desc_sw128(sB + kk * 32, 16, 1024);
                        ptx::mma_bf16(d_tmem, ad, bd, idesc, first ? 0u : 1u);
                        first = false;
                    }
                    ptx::mma_commit(empty_bar(s));
                }
                ptx::mma_commit(tfull_bar(b));
            }
            // every issued MMA has completed before TMEM is released
            ptx::mma_commit(mma_done);
            ptx::mbar_wait(mma_done, 0, nullptr);
        }
    } else {
        // ---------------- epilogue warps 2..5 (TMEM lane quarter = warp % 4)
        const int quarter = warp % 4;
        int j = 0;
        for (int t = blockIdx.x; t < g.total_tiles; t += gridDim.x, ++j) {
            const TileRef tr = locate_tile(g, t);
            const auto &P = g.p[tr.prob];
            const int b = j & 1;
            const uint32_t use = (uint32_t)(j >> 1);
            bool ok = ptx::mbar_wait(tfull_bar(b), use & 1, g.status);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            ptx::tc_fence_after();
            Epi::run_dyn(P.ep, tmem + b * kAccCols, P.bn, quarter, lane, tr.m0, tr.n0, P.M, P.N, tr.z);
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(tempty_bar(b));
        }
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, kCols);
    }
}

}  // namespace tc
}  // namespace noble
