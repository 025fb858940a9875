// Fused AdamW step over a batch of parameter tensors (decoupled weight decay;
// the optimizer of the paper's training runs, Section 4.1), each tensor with
// its own learning rate (NOBLE's per-group scaling, Section 3.3).  One launch
// covers up to kAdamwMaxTensors tensors: blockIdx.y selects the tensor, the
// blocks along x stride over its elements, four at a time where the tensor's
// arrays are 16-byte aligned and its length a multiple of four.
#pragma once

#include <cstdint>
#include <cuda_bf16.h>

namespace noble {
namespace opt {

constexpr int kAdamwMaxTensors = 16;

struct AdamwTensor {
    float *p;               // fp32 values, updated in place
    __nv_bfloat16 *p_bf16;  // optional bf16 copy of the new values
    const float *g;
    float *m, *v;
    int64_t n;
    float lr;               // this tensor's learning rate
    float decay;            // lr * weight_decay, or 0
    int vec4;               // 1: process in float4 groups
};

struct AdamwBatch {
    AdamwTensor t[kAdamwMaxTensors];
    float beta1, beta2, eps;
    float inv_bc1, inv_sqrt_bc2;  // 1 / (1 - beta1^t), 1 / sqrt(1 - beta2^t)
};

__device__ __forceinline__ float adamw_elem(float p, float g, float &m, float &v, const AdamwBatch &b, float lr,
                                            float decay)
{
    p -= decay * p;
    m = fmaf(b.beta1, m, (1.f - b.beta1) * g);
    v = fmaf(b.beta2, v, (1.f - b.beta2) * g * g);
    const float denom = sqrtf(v) * b.inv_sqrt_bc2 + b.eps;
    return p - (lr * b.inv_bc1) * (m / denom);
}

__global__ void __launch_bounds__(256) adamw_kernel(const __grid_constant__ AdamwBatch b)
{
    const AdamwTensor &T = b.t[blockIdx.y];
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t first = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (T.vec4) {
        const int64_t n4 = T.n / 4;
        for (int64_t i = first; i < n4; i += stride) {
            float4 p = reinterpret_cast<float4 *>(T.p)[i];
            const float4 g = __ldcs(reinterpret_cast<const float4 *>(T.g) + i);
            float4 m = reinterpret_cast<float4 *>(T.m)[i];
            float4 v = reinterpret_cast<float4 *>(T.v)[i];
            p.x = adamw_elem(p.x, g.x, m.x, v.x, b, T.lr, T.decay);
            p.y = adamw_elem(p.y, g.y, m.y, v.y, b, T.lr, T.decay);
            p.z = adamw_elem(p.z, g.z, m.z, v.z, b, T.lr, T.decay);
            p.w = adamw_elem(p.w, g.w, m.w, v.w, b, T.lr, T.decay);
            reinterpret_cast<float4 *>(T.p)[i] = p;
            reinterpret_cast<float4 *>(T.m)[i] = m;
            reinterpret_cast<float4 *>(T.v)[i] = v;
            if (T.p_bf16) {
                __nv_bfloat162 lo = __floats2bfloat162_rn(p.x, p.y), hi = __floats2bfloat162_rn(p.z, p.w);
                uint2 q;
                q.x = *reinterpret_cast<uint32_t *>(&lo);
                q.y = *reinterpret_cast<uint32_t *>(&hi);
                reinterpret_cast<uint2 *>(T.p_bf16)[i] = q;
            }
        }
    } else {
        for (int64_t i = first; i < T.n; i += stride) {
            float m = T.m[i], v = T.v[i];
            const float p = adamw_elem(T.p[i], T.g[i], m, v, b, T.lr, T.decay);
            T.p[i] = p;
            T.m[i] = m;
            T.v[i] = v;
            if (T.p_bf16) T.p_bf16[i] = __float2bfloat16_rn(p);
        }
    }
}

}  // namespace opt
}  // namespace noble
