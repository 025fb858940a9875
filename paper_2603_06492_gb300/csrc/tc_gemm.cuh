// Warp-specialised tcgen05 GEMM for sm_103a: TMA -> shared memory ring ->
// tcgen05.mma (bf16 in, fp32 accumulate in TMEM) -> epilogue from TMEM.
//
//   C[m][n] = sum over segments s of  sum_k A_s(m, k) * B_s(n, k)
//
// Up to two K segments share one accumulator, so a K-concatenated product
// [A0 | A1] [B0 ; B1]^T runs as one contraction (the main path and the
// low-rank up path of Eq. 1 accumulate into the same tile).  Each operand is
// either K-major (row-major [rows][K]) or MN-major (row-major [K][rows]).
//
// One CTA computes one 128 x BN tile: warp 0 issues TMA loads, warp 1 issues
// MMAs (and owns the TMEM allocation), warps 2-5 run the epilogue.  Every
// mbarrier wait is bounded (ptx::mbar_wait); a wait that expires records
// kStatusTimeout in the status word and the CTA abandons its work, waits
// (bounded) for its own copies and MMAs in flight, frees TMEM and exits.
#pragma once

#include "sm100_ptx.cuh"

namespace noble {
namespace tc {

constexpr int kBM = 128;          // rows of a tile (TMEM lanes)
constexpr int kBK = 64;           // K elements per stage (128 bytes of bf16)
constexpr int kThreads = 192;     // 6 warps
constexpr uint32_t kChunkBytes = 64 * kBK * 2;  // one 64 x 64 bf16 swizzle chunk (8 KB)

struct GemmArgs {
    int64_t M, N;
    int kb0, kb1;       // k-blocks of segment 0 and segment 1
    int kb_per_split;   // k-blocks per blockIdx.z; 0 = no split
    uint32_t *status;   // device status word
};

template <int BN, int STAGES>
struct Smem {
    static constexpr uint32_t kA = kBM * kBK * 2;
    static constexpr uint32_t kB = BN * kBK * 2;
    static constexpr uint32_t kStage = kA + kB;
    static constexpr uint32_t kBarOff = STAGES * kStage;
    static constexpr uint32_t kBytes = kBarOff + 8 * (2 * STAGES + 2) + 16;
    static constexpr uint32_t kDynamic = kBytes + 1024;  // slack to align the base to 1024
};

template <int BN>
struct TmemCols {
    static constexpr uint32_t value = BN <= 32 ? 32 : BN <= 64 ? 64 : BN <= 128 ? 128 : 256;
};

// ---------------------------------------------------------------- epilogues
// Plain store: C[z][m][n] = acc (+ bias[n]) in OutT.  N must be a multiple of 8.
template <typename OutT>
struct EpiStore {
    using out_type = OutT;
    struct Params {
        OutT *C;
        int64_t ldc;
        const float *bias;
        int64_t split_stride;  // elements between blockIdx.z partial outputs
        int col0 = 0;          // store only column 0 of each row, to C[row * ldc]
        int tma = 0;           // pair kernel: store through a 3-D TMA map of C (run_tma)
        int transpose = 0;     // fp32: store the tile transposed, (m, n) to C[n * ldc + m]
    };

    // 32 accumulator columns [c, c+32) of this thread's row -> C (+ bias)
    __device__ static __forceinline__ void store32(const Params &p, OutT *out, const float (&v)[32], int64_t n_base,
                                                   int64_t N)
    {
#pragma unroll
        for (int g = 0; g < 4; ++g) {
            const int64_t n = n_base + g * 8;
            if (n >= N) break;
            float f[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) f[i] = v[g * 8 + i] + (p.bias ? __ldg(p.bias + n + i) : 0.f);
            if constexpr (sizeof(OutT) == 2) {
                uint4 q;
                q.x = ptx::pack_bf16x2(f[0], f[1]);
                q.y = ptx::pack_bf16x2(f[2], f[3]);
                q.z = ptx::pack_bf16x2(f[4], f[5]);
                q.w = ptx::pack_bf16x2(f[6], f[7]);
                // streaming stores: outputs are not read again by this kernel
                // and should not push its operands out of L2
                __stcs(reinterpret_cast<uint4 *>(out + n), q);
            } else {
                __stcs(reinterpret_cast<float4 *>(out + n), make_float4(f[0], f[1], f[2], f[3]));
                __stcs(reinterpret_cast<float4 *>(out + n + 4), make_float4(f[4], f[5], f[6], f[7]));
            }
        }
    }

    // Runtime tile width bn (a multiple of 32), for the persistent kernels.
    // This warp stores the 32-column chunks c0, c0 + cstep, ... of its rows.
    __device__ static void run_dyn(const Params &p, uint32_t tmem, int bn, int quarter, int lane, int64_t m0,
                                   int64_t n0, int64_t M, int64_t N, int z, int c0 = 0, int cstep = 32)
    {
        const int64_t row = m0 + quarter * 32 + lane;
        OutT *out = p.C + (int64_t)z * p.split_stride + row * p.ldc;
        const uint32_t lane_addr = tmem + ((uint32_t)(quarter * 32) << 16);
        if (p.col0) {
            if (c0 != 0) return;
            float v[32];
            ptx::tmem_ld_32x32b_x32(lane_addr, v);
            if (row < M && n0 == 0) *out = (OutT)v[0];
            return;
        }
        if (p.transpose) {
            // column n of the tile is row n of C: for each n the warp's lanes
            // (consecutive m) write one contiguous 128-byte segment
            OutT *outT = p.C + (int64_t)z * p.split_stride + row;
#pragma unroll 1
            for (int c = c0; c < bn; c += cstep) {
                if (n0 + c >= N) break;
                float v[32];
                ptx::tmem_ld_32x32b_x32(lane_addr + c, v);
                if (row < M)
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        if (n0 + c + j < N) __stcs(outT + (n0 + c + j) * p.ldc, (OutT)v[j]);
            }
            return;
        }
#pragma unroll 1
        for (int c = c0; c < bn; c += cstep) {
            if (n0 + c >= N) break;  // warp-uniform: whole chunk past the edge
            float v[32];
            ptx::tmem_ld_32x32b_x32(lane_addr + c, v);
            if (row < M) store32(p, out, v, n0 + c, N);
        }
    }

    // TMA-store epilogue of the pair kernel.  The warp's 32 rows are written
    // in boxes of kBoxCols columns (128 bytes per row): the accumulator chunk
    // (+ bias) is converted into the warp's 4 KB staging buffer in the
    // 128-byte-swizzled layout and stored by one 3-D TMA copy at
    // (column, row, split); rows >= M and columns >= N are clipped by the copy.
    // The warp's boxes start at column half * kBoxCols and step by 2 kBoxCols.
    // Requires N % 4 == 0 (whole float4 groups of bias).
    static constexpr int kBoxCols = 128 / (int)sizeof(OutT);
    __device__ static void run_tma(const Params &p, const CUtensorMap *map, uint8_t *stg_ptr, uint32_t stg,
                                   uint32_t tmem, int bn, int quarter, int lane, int64_t m0, int64_t n0, int64_t N,
                                   int z, int half)
    {
        const uint32_t lane_addr = tmem + ((uint32_t)(quarter * 32) << 16);
        if constexpr (sizeof(OutT) == 4) {
            if (p.transpose) {
                // a 32 x 32 block transposed through the staging buffer: lane
                // (tile row m) writes its column n into staging row n, word m
                // (one 4-byte store per n, 32 distinct banks per store); the
                // map describes C with rows n and columns m
#pragma unroll 1
                for (int c = 32 * half; c < bn; c += 64) {
                    if (n0 + c >= N) break;
                    if (lane == 0) ptx::bulk_wait_read_all();
                    __syncwarp();
                    float v[32];
                    ptx::tmem_ld_32x32b_x32(lane_addr + c, v);
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        *reinterpret_cast<float *>(stg_ptr + j * 128 + ((((lane >> 2) ^ (j & 7))) << 4) + (lane & 3) * 4) =
                            v[j];
                    ptx::fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) {
                        ptx::tma_store_3d_hint(map, stg, (int)(m0 + quarter * 32), (int)(n0 + c), z,
                                               ptx::l2_policy_evict_first());
                        ptx::bulk_commit_group();
                    }
                }
                return;
            }
        }
        uint8_t *my_row = stg_ptr + lane * 128;
#pragma unroll 1
        for (int c = half * kBoxCols; c < bn; c += 2 * kBoxCols) {
            if (n0 + c >= N) break;  // warp-uniform
            if (lane == 0) ptx::bulk_wait_read_all();  // the previous box has left the buffer
            __syncwarp();
#pragma unroll
            for (int h = 0; h < kBoxCols / 32; ++h) {
                float v[32];
                ptx::tmem_ld_32x32b_x32(lane_addr + c + 32 * h, v);
                const int64_t n = n0 + c + 32 * h;
                if (p.bias) {
#pragma unroll
                    for (int q = 0; q < 8; ++q) {
                        if (n + 4 * q < N) {
                            const float4 b = __ldg(reinterpret_cast<const float4 *>(p.bias + n) + q);
                            v[4 * q] += b.x, v[4 * q + 1] += b.y, v[4 * q + 2] += b.z, v[4 * q + 3] += b.w;
                        }
                    }
                }
                if constexpr (sizeof(OutT) == 2) {
#pragma unroll
                    for (int g = 0; g < 4; ++g) {
                        const int j = h * 4 + g;  // 16-byte piece of the 128-byte row
                        uint4 q;
                        q.x = ptx::pack_bf16x2(v[8 * g], v[8 * g + 1]);
                        q.y = ptx::pack_bf16x2(v[8 * g + 2], v[8 * g + 3]);
                        q.z = ptx::pack_bf16x2(v[8 * g + 4], v[8 * g + 5]);
                        q.w = ptx::pack_bf16x2(v[8 * g + 6], v[8 * g + 7]);
                        *reinterpret_cast<uint4 *>(my_row + ((j ^ (lane & 7)) << 4)) = q;
                    }
                } else {
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        *reinterpret_cast<float4 *>(my_row + ((j ^ (lane & 7)) << 4)) =
                            make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
                }
            }
            ptx::fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
                ptx::tma_store_3d_hint(map, stg, (int)(n0 + c), (int)(m0 + quarter * 32), z,
                                       ptx::l2_policy_evict_first());
                ptx::bulk_commit_group();
            }
        }
    }

    template <int BN>
    __device__ static void run(const Params &p, uint32_t tmem, int quarter, int lane, int64_t m0,
                               int64_t n0, int64_t M, int64_t N, int z)
    {
        const int64_t row = m0 + quarter * 32 + lane;
        OutT *out = p.C + (int64_t)z * p.split_stride + row * p.ldc;
        const uint32_t lane_addr = tmem + ((uint32_t)(quarter * 32) << 16);
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
            float v[32];
            if constexpr (BN >= 32) {
                ptx::tmem_ld_32x32b_x32(lane_addr + c, v);
            } else {
                float w[16];
                ptx::tmem_ld_32x32b_x16(lane_addr + c, w);
#pragma unroll
                for (int i = 0; i < 16; ++i) v[i] = w[i];
#pragma unroll
                for (int i = 16; i < 32; ++i) v[i] = 0.f;
            }
            if (row >= M) continue;
#pragma unroll
            for (int g = 0; g < (BN >= 32 ? 4 : 2); ++g) {
                const int64_t n = n0 + c + g * 8;
                if (n >= N) break;
                float f[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) f[i] = v[g * 8 + i] + (p.bias ? __ldg(p.bias + n + i) : 0.f);
                if constexpr (sizeof(OutT) == 2) {
                    uint4 q;
                    q.x = ptx::pack_bf16x2(f[0], f[1]);
                    q.y = ptx::pack_bf16x2(f[2], f[3]);
                    q.z = ptx::pack_bf16x2(f[4], f[5]);
                    q.w = ptx::pack_bf16x2(f[6], f[7]);
                    *reinterpret_cast<uint4 *>(out + n) = q;
                } else {
                    *reinterpret_cast<float4 *>(out + n) = make_float4(f[0], f[1], f[2], f[3]);
                    *reinterpret_cast<float4 *>(out + n + 4) = make_float4(f[4], f[5], f[6], f[7]);
                }
            }
        }
    }
};

// ---------------------------------------------------------------- kernel
template <int BN, bool A_MN, bool B_MN, int STAGES, class Epi>
__global__ void __launch_bounds__(kThreads, 1)
gemm_kernel(const __grid_constant__ CUtensorMap mA0, const __grid_constant__ CUtensorMap mB0,
            const __grid_constant__ CUtensorMap mA1, const __grid_constant__ CUtensorMap mB1,
            const GemmArgs args, const typename Epi::Params ep)
{
    using S = Smem<BN, STAGES>;
    constexpr uint32_t kCols = TmemCols<BN>::value;
    static_assert(BN % 16 == 0 && BN >= 16 && BN <= 256, "MMA N");
    static_assert(!B_MN || BN % 64 == 0, "MN-major B needs whole 64-wide chunks");

    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = ptx::smem_u32(smem_raw);
    const uint32_t sbase = (raw + 1023u) & ~1023u;
    uint8_t *smem = smem_raw + (sbase - raw);
    const uint32_t bar0 = sbase + S::kBarOff;
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (STAGES + s); };
    const uint32_t tmem_full = bar0 + 8u * (2 * STAGES);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + S::kBarOff + 8 * (2 * STAGES + 2));

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int64_t n0 = (int64_t)blockIdx.x * BN, m0 = (int64_t)blockIdx.y * kBM;
    const int z = blockIdx.z;
    int kb_begin = 0, kb_end = args.kb0 + args.kb1;
    if (args.kb_per_split > 0) {
        kb_begin = z * args.kb_per_split;
        kb_end = min(kb_end, kb_begin + args.kb_per_split);
    }
    const int nkb = kb_end - kb_begin;

    if (warp == 0 && lane == 0) {
        ptx::tma_prefetch_desc(&mA0);
        ptx::tma_prefetch_desc(&mB0);
        if (args.kb1 > 0) {
            ptx::tma_prefetch_desc(&mA1);
            ptx::tma_prefetch_desc(&mB1);
        }
        for (int s = 0; s < STAGES; ++s) {
            ptx::mbar_init(full_bar(s), 1);
            ptx::mbar_init(empty_bar(s), 1);
        }
        ptx::mbar_init(tmem_full, 1);
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
            // ---------------- TMA producer
            int issued = 0;
            for (int i = 0; i < nkb; ++i) {
                const int s = i % STAGES;
                const uint32_t ph = (i / STAGES) & 1;
                if (!ptx::mbar_wait(empty_bar(s), ph ^ 1, args.status)) break;
                const uint32_t fb = full_bar(s);
                ptx::mbar_arrive_expect_tx(fb, S::kStage);
                const uint32_t sA = sbase + s * S::kStage, sB = sA + S::kA;
                const int kb = kb_begin + i;
                const bool seg1 = kb >= args.kb0;
                const CUtensorMap *mA = seg1 ? &mA1 : &mA0;
                const CUtensorMap *mB = seg1 ? &mB1 : &mB0;
                const int k = (seg1 ? kb - args.kb0 : kb) * kBK;
                if (A_MN) {
                    ptx::tma_load_2d(sA, mA, fb, (int)m0, k);
                    ptx::tma_load_2d(sA + kChunkBytes, mA, fb, (int)m0 + 64, k);
                } else {
                    ptx::tma_load_2d(sA, mA, fb, k, (int)m0);
                }
                if (B_MN) {
#pragma unroll
                    for (int c = 0; c < BN / 64; ++c)
                        ptx::tma_load_2d(sB + c * kChunkBytes, mB, fb, (int)n0 + 64 * c, k);
                } else {
                    ptx::tma_load_2d(sB, mB, fb, k, (int)n0);
                }
                ++issued;
            }
            // no copy may still be landing in shared memory when the CTA exits
            for (int i = issued > STAGES ? issued - STAGES : 0; i < issued; ++i)
                ptx::mbar_wait(full_bar(i % STAGES), (i / STAGES) & 1, nullptr);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ---------------- MMA issuer (single thread)
            constexpr uint32_t idesc = ptx::idesc_bf16(kBM, BN, A_MN, B_MN);
            for (int i = 0; i < nkb; ++i) {
                const int s = i % STAGES;
                const uint32_t ph = (i / STAGES) & 1;
                if (!ptx::mbar_wait(full_bar(s), ph, args.status)) break;
                ptx::tc_fence_after();
                const uint32_t sA = sbase + s * S::kStage, sB = sA + S::kA;
#pragma unroll
                for (int kk = 0; kk < kBK / 16; ++kk) {
                    const uint64_t ad = A_MN ? ptx::smem_desc_sw128(sA + kk * 2048, kChunkBytes, 1024)
                                             : ptx::smem_desc_sw128(sA + kk * 32, 16, 1024);
                    const uint64_t bd = B_MN ? ptx::smem_desc_sw128(sB + kk * 2048, kChunkBytes, 1024)
                                             : ptx::smem_desc_sw128(sB + kk * 32, 16, 1024);
                    ptx::mma_bf16(tmem, ad, bd, idesc, (i > 0 || kk > 0) ? 1u : 0u);
                }
                ptx::mma_commit(empty_bar(s));
            }
            ptx::mma_commit(tmem_full);
            // every MMA has finished before TMEM is released below
            ptx::mbar_wait(tmem_full, 0, nullptr);
        }
    } else {
        // ---------------- epilogue: warps 2..5, TMEM lane quarter = warp % 4
        bool ok = ptx::mbar_wait(tmem_full, 0, args.status);
        ok = __all_sync(0xffffffffu, ok);
        if (ok) {
            ptx::tc_fence_after();
            Epi::template run<BN>(ep, tmem, warp % 4, lane, m0, n0, args.M, args.N, z);
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
