// Shared device/host helpers of the NOBLE library (not part of the C ABI).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace noble {

// Bit flags of the per-device status word (see noble_get_device_status).
enum : uint32_t {
    kStatusTimeout = 1u,   // a bounded mbarrier / flag wait gave up
    kStatusBadShape = 2u,  // a kernel saw a shape it cannot handle and skipped work
};

// Kernels that can give up a bounded wait receive a pointer to the
// per-device status word and OR flags into it; they never trap.
__device__ __forceinline__ void raise_status(uint32_t *status, uint32_t bits)
{
    if (status) atomicOr(status, bits);
}

template <typename T> struct Elem;
template <> struct Elem<float> {
    static __device__ __forceinline__ float load(const float *p) { return *p; }
    static __device__ __forceinline__ void store(float *p, float v) { *p = v; }
};
template <> struct Elem<__nv_bfloat16> {
    static __device__ __forceinline__ float load(const __nv_bfloat16 *p) { return __bfloat162float(*p); }
    static __device__ __forceinline__ void store(__nv_bfloat16 *p, float v) { *p = __float2bfloat16_rn(v); }
};

__host__ __device__ constexpr inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }
__host__ __device__ constexpr inline size_t align_up(size_t a, size_t b) { return (a + b - 1) / b * b; }

}  // namespace noble
