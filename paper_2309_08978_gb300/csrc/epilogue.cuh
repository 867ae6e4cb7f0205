// The elementwise activation a kernel applies to each output after the bias
// (nnjit_epilogue).  Kernels receive the epilogue code: the activation in bits 0-3 and
// NNJIT_EPI_RESIDUAL (add the output's prior value after the activation).  The code is
// uniform across a launch, so each switch costs one predictable branch.
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
    switch (act & 15) {
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
    switch (act & 15) {
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

// The epilogue of a staged row (plain order, n <= 32 values) written element by element to
// dst: activation, then with NNJIT_EPI_RESIDUAL the value dst held before.
__device__ __forceinline__ void epi_store_row(const float* row, int code, float* dst, int n) {
    const int act = code & 15;
    const bool res = (code & NNJIT_EPI_RESIDUAL) != 0;
#pragma unroll 1
    for (int j = 0; j < n; ++j) {
        const float x = row[j];
        float y = act == NNJIT_EPI_RELU ? fmaxf(x, 0.0f)
                  : act == NNJIT_EPI_GELU ? gelu_as7126(x)
                  : act == NNJIT_EPI_SILU ? silu_fast(x) : x;
        if (res) y += dst[j];
        dst[j] = y;
    }
}

// With NNJIT_EPI_RESIDUAL: add the prior content of a thread's output segment (n <= 32
// columns at dst, 16-byte aligned) to its staged 128-byte row, whose logical 16-byte unit j
// sits at unit j ^ swz (the 128-byte swizzle of the TMA-store staging).
__device__ __forceinline__ void residual_row128(void* row128, int swz, const float* dst, int n) {
    float4* r = static_cast<float4*>(row128);
    if (n >= 32) {
#pragma unroll 1
        for (int j = 0; j < 8; ++j) {
            const float4 o = *reinterpret_cast<const float4*>(dst + 4 * j);
            float4& s = r[j ^ swz];
            s.x += o.x; s.y += o.y; s.z += o.z; s.w += o.w;
        }
    } else {
#pragma unroll 1
        for (int j = 0; j < n; ++j) reinterpret_cast<float*>(&r[(j >> 2) ^ swz])[j & 3] += dst[j];
    }
}

__device__ __forceinline__ float apply_act(float v, int act) {
    switch (act & 15) {
        case NNJIT_EPI_RELU: return fmaxf(v, 0.0f);
        case NNJIT_EPI_GELU: return gelu_as7126(v);
        case NNJIT_EPI_SILU: return silu_fast(v);
        default: return v;
    }
}

// One output element: act(v), plus the element's prior value *c with NNJIT_EPI_RESIDUAL.
__device__ __forceinline__ float epi_out(float v, int code, const float* c) {
    const float y = apply_act(v, code);
    return (code & NNJIT_EPI_RESIDUAL) ? y + *c : y;
}

}  // namespace nnjit
