// Bottleneck activations other than the cosine, for the variants of the
// ablation in Section 4.4 (Table 5): sigma(h) = f(h) (one layer) or
// sigma(h) = f(f(h) M) (two layers around the mixing matrix).  The paper
// gives frequencies and phases to the cosine only; these take the
// pre-activation as it is.
//   tanh       f(u) = tanh(u)                    f'(u) = 1 - tanh(u)^2
//   LeakyReLU  f(u) = u (u > 0), 0.01 u          f'(u) = 1 (u > 0), 0.01
//              (the common default slope; the paper gives none)
//   GELU       f(u) = u Phi(u) = u/2 (1 + erf(u / sqrt 2))
//              f'(u) = Phi(u) + u phi(u),  phi(u) = exp(-u^2 / 2) / sqrt(2 pi)
// tanh, erf and exp are CUDA's own functions (tanhf, erff, expf).
#pragma once

#include "common.cuh"

namespace noble {
namespace act {

constexpr int kCos = 0, kIdentity = 1, kTanh = 2, kLeaky = 3, kGelu = 4;

constexpr float kLeakySlope = 0.01f;
constexpr float kInvSqrt2 = 0.70710678118654752f;    // 1 / sqrt(2)
constexpr float kInvSqrt2Pi = 0.39894228040143268f;  // 1 / sqrt(2 pi)

__device__ __forceinline__ float f(int a, float u)
{
    switch (a) {
    case kTanh: return tanhf(u);
    case kLeaky: return u > 0.f ? u : kLeakySlope * u;
    case kGelu: return 0.5f * u * (1.f + erff(u * kInvSqrt2));
    default: return u;
    }
}

__device__ __forceinline__ float df(int a, float u)
{
    switch (a) {
    case kTanh: {
        const float t = tanhf(u);
        return 1.f - t * t;
    }
    case kLeaky: return u > 0.f ? 1.f : kLeakySlope;
    case kGelu: return 0.5f * (1.f + erff(u * kInvSqrt2)) + u * kInvSqrt2Pi * expf(-0.5f * u * u);
    default: return 1.f;
    }
}

}  // namespace act
}  // namespace noble
