// Tensor-core (tcgen05 / TMEM / TMA) path for bf16 operands.  Placeholder:
// no shape is routed here yet.
#pragma once

#include <atomic>

#include "../../include/noble.h"
#include "common.cuh"

namespace noble {
namespace tc {

inline bool fwd_supported(const noble_linear_desc *) { return false; }
inline bool bwd_supported(const noble_linear_desc *) { return false; }

inline noble_status fwd(const noble_linear_desc *, const __nv_bfloat16 *, const __nv_bfloat16 *,
                        const float *, const __nv_bfloat16 *, const float *, const float *,
                        const float *, const float *, const float *, const __nv_bfloat16 *,
                        __nv_bfloat16 *, char *, cudaStream_t, std::atomic<uint64_t> &)
{
    return NOBLE_ERR_UNSUPPORTED;
}

inline noble_status bwd(const noble_linear_desc *, const __nv_bfloat16 *, const __nv_bfloat16 *,
                        const __nv_bfloat16 *, const __nv_bfloat16 *, const float *, const float *,
                        const float *, const float *, const float *, const __nv_bfloat16 *,
                        const char *, __nv_bfloat16 *, float *, float *, float *, float *, float *,
                        float *, float *, float *, float *, char *, cudaStream_t,
                        std::atomic<uint64_t> &)
{
    return NOBLE_ERR_UNSUPPORTED;
}

}  // namespace tc
}  // namespace noble
