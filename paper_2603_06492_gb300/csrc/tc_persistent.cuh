// Grouped GEMM launches (used by the CTA-pair kernel in tc_pair.cuh): up to
// kMaxProblems independent problems in one persistent launch.
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
    int dep;               // bit s: segment s reads what an earlier kernel of the same call wrote
                           // (the producer waits for the predecessor grid before loading it)
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
    // A0, B0, A1, B1, C (pair kernel's TMA-store epilogue), and for a fused
    // launch's leader problem the B0 of CTA rank 1 (the branch weights)
    CUtensorMap m[kMaxProblems][6];
};

}  // namespace tc
}  // namespace noble
