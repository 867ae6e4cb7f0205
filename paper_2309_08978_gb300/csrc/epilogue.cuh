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

__device__ __forceinline__ float apply_act(float v, int act) {
    switch (act) {
        case NNJIT_EPI_RELU: return fmaxf(v, 0.0f);
        case NNJIT_EPI_GELU: return gelu_as7126(v);
        case NNJIT_EPI_SILU: return silu_fast(v);
        default: return v;
    }
}

}  // namespace nnjit
