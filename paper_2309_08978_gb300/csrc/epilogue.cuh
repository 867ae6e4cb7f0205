// The elementwise activation a kernel applies to each output after the bias
// (nnjit_epilogue).  `act` is uniform across a launch, so the switch costs one predictable
// branch per element.
//
// The epilogue runs on the 4 warps that drain TMEM, so a long per-element computation is
// on the critical path of every tile; both transcendental activations therefore use a
// short form built on the hardware exp2/reciprocal approximations:
//   * GELU(x) = 0.5 x (1 + erf(x / sqrt 2)) with erf from Abramowitz & Stegun, Handbook of
//     Mathematical Functions, formula 7.1.26: for z >= 0,
//         erf(z) = 1 - (a1 t + a2 t^2 + a3 t^3 + a4 t^4 + a5 t^5) exp(-z^2),  t = 1 / (1 + p z),
//     with |error| <= 1.5e-7.  Writing q = 0.5 P(t) exp(-x^2 / 2) (z = |x| / sqrt 2):
//     GELU(x) = x (1 - q) for x >= 0 and x q for x < 0.
//   * SiLU(x) = x sigmoid(x), with sigmoid from e = exp(-|x|) in (0, 1] (no overflow):
//     sigmoid(x) = 1 / (1 + e) for x >= 0 and e / (1 + e) for x < 0.
#pragma once

#include "../../include/nnjit.h"

namespace nnjit {

__device__ __forceinline__ float gelu_as7126(float x) {
    constexpr float kP = 0.3275911f * 0.70710678118654752f;  // p / sqrt(2): t = 1 / (1 + p |x| / sqrt 2)
    constexpr float a1 = 0.254829592f, a2 = -0.284496736f, a3 = 1.421413741f, a4 = -1.453152027f,
                    a5 = 1.061405429f;
    const float ax = fabsf(x);
    const float t = __fdividef(1.0f, fmaf(kP, ax, 1.0f));
    const float poly = t * fmaf(fmaf(fmaf(fmaf(a5, t, a4), t, a3), t, a2), t, a1);
    const float q = 0.5f * poly * __expf(-0.5f * x * x);
    return x * (x >= 0.0f ? 1.0f - q : q);
}

__device__ __forceinline__ float silu_fast(float x) {
    const float e = __expf(-fabsf(x));
    const float r = __fdividef(1.0f, 1.0f + e);
    return x * (x >= 0.0f ? r : e * r);
}

// A chunk of 32 outputs of one thread: one switch per chunk, then 32 independent
// evaluations the compiler can interleave (a switch per element serialises them).
__device__ __forceinline__ void apply_act32(float (&v)[32], int act) {
    switch (act) {
        case NNJIT_EPI_RELU:
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = fmaxf(v[j], 0.0f);
            break;
        case NNJIT_EPI_GELU:
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = gelu_as7126(v[j]);
            break;
        case NNJIT_EPI_SILU:
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = silu_fast(v[j]);
            break;
        default:
            break;
    }
}

// The activation over a thread's 32 outputs after they have been staged: a 128-byte row
// of shared memory (any order within it: the 128-byte swizzle only permutes a row), or
// n <= 32 consecutive floats in global memory that this thread has just written.  The
// loops stay rolled, so a kernel carries one short copy of each activation: inlined
// 32-wide bodies (twice per tile loop) added registers and instruction-cache footprint
// that slowed plans without an activation by 0.2-0.7 us per product.
__device__ __forceinline__ void act_row128(void* row128, int act) {
    float4* r = static_cast<float4*>(row128);
    switch (act) {
        case NNJIT_EPI_RELU:
#pragma unroll 1
            for (int u = 0; u < 8; ++u) {
                float4 x = r[u];
                r[u] = make_float4(fmaxf(x.x, 0.0f), fmaxf(x.y, 0.0f), fmaxf(x.z, 0.0f), fmaxf(x.w, 0.0f));
            }
            break;
        case NNJIT_EPI_GELU:
#pragma unroll 1
            for (int u = 0; u < 8; ++u) {
                float4 x = r[u];
                r[u] = make_float4(gelu_as7126(x.x), gelu_as7126(x.y), gelu_as7126(x.z), gelu_as7126(x.w));
            }
            break;
        case NNJIT_EPI_SILU:
#pragma unroll 1
            for (int u = 0; u < 8; ++u) {
                float4 x = r[u];
                r[u] = make_float4(silu_fast(x.x), silu_fast(x.y), silu_fast(x.z), silu_fast(x.w));
            }
            break;
        default:
            break;
    }
}

__device__ __forceinline__ void act_written(float* dst, int n, int act) {
#pragma unroll 1
    for (int j = 0; j < n; ++j) {
        const float x = dst[j];
        dst[j] = act == NNJIT_EPI_RELU ? fmaxf(x, 0.0f) : act == NNJIT_EPI_GELU ? gelu_as7126(x) : silu_fast(x);
    }
}

__device__ __forceinline__ float apply_act(float v, int act) {
    switch (act) {
        case NNJIT_EPI_RELU: return fmaxf(v, 0.0f);
        case NNJIT_EPI_GELU: return gelu_as7126(v);
        case NNJIT_EPI_SILU: return silu_fast(v);
        default: return v;
    }
}

}  // namespace nnjit
