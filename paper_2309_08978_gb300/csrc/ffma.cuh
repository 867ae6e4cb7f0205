// Register-tiled FP32 FFMA GEMM: the CUDA form of the paper's tile template (Table 2):
// a CTA loads the (x1 x r1) A tile and (r1 x y1) B tile into shared memory
// ("cache_read"), each thread keeps an x0 x y0 tile of C in registers and walks k one
// step at a time (r0 = 1), multiplying a column of x0 A values by a row of y0 B values.
// Exact FP32: every update is one fmaf, in ascending k within the CTA's K slice.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>

#include "epilogue.cuh"

namespace nnjit {

struct FfmaParams {
    const float* A;
    const float* B;
    const float* bias;  // applied only when split == 1
    float* C;
    float* ws;
    int M, N, K, batch, split, kper;
    int act;            // nnjit_epilogue, applied when split == 1
    long long lda, ldb, ldc, stride_a, stride_b, stride_c;
};

// grid: (tiles_n, tiles_m, batch * split); block: (BM/TM)*(BN/TN) threads.
template <int BM, int BN, int BK, int TM, int TN, bool kNK>
__global__ void __launch_bounds__((BM / TM) * (BN / TN))
    ffma_gemm_kernel(const FfmaParams p) {
    constexpr int T = (BM / TM) * (BN / TN);
    constexpr int TX = BN / TN;
    constexpr int A_PER = (BM * BK) / T;  // A elements each thread moves per k-tile
    constexpr int B_PER = (BK * BN) / T;
    static_assert((BM * BK) % T == 0 && (BK * BN) % T == 0, "tile not divisible by threads");
    __shared__ __align__(16) float As[2][BK][BM + 4];
    __shared__ __align__(16) float Bs[2][BK][BN + 4];

    asm volatile("griddepcontrol.wait;" ::: "memory");
    if (threadIdx.x == 0) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int tid = threadIdx.x;
    const int ty = tid / TX, tx = tid % TX;
    const int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN;
    const int b = blockIdx.z / p.split, s = blockIdx.z % p.split;
    const int kbeg = s * p.kper;
    const int kend = min(p.K, kbeg + p.kper);
    const float* A = p.A + (long long)b * p.stride_a;
    const float* B = p.B + (long long)b * p.stride_b;

    float ra[A_PER], rb[B_PER];
    auto load_tile = [&](int k0) {
#pragma unroll
        for (int i = 0; i < A_PER; ++i) {
            const int e = tid + i * T;
            const int m = e / BK, k = e % BK;
            const int gm = m0 + m, gk = k0 + k;
            ra[i] = (gm < p.M && gk < kend) ? __ldg(A + (long long)gm * p.lda + gk) : 0.0f;
        }
#pragma unroll
        for (int i = 0; i < B_PER; ++i) {
            const int e = tid + i * T;
            int k, n;
            if constexpr (kNK) { n = e / BK; k = e % BK; } else { k = e / BN; n = e % BN; }
            const int gn = n0 + n, gk = k0 + k;
            float v = 0.0f;
            if (gn < p.N && gk < kend)
                v = kNK ? __ldg(B + (long long)gn * p.ldb + gk) : __ldg(B + (long long)gk * p.ldb + gn);
            rb[i] = v;
        }
    };
    auto store_tile = [&](int buf) {
#pragma unroll
        for (int i = 0; i < A_PER; ++i) {
            const int e = tid + i * T;
            As[buf][e % BK][e / BK] = ra[i];
        }
#pragma unroll
        for (int i = 0; i < B_PER; ++i) {
            const int e = tid + i * T;
            if constexpr (kNK) Bs[buf][e % BK][e / BK] = rb[i];
            else Bs[buf][e / BN][e % BN] = rb[i];
        }
    };

    float acc[TM][TN];
#pragma unroll
    for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < TN; ++j) acc[i][j] = 0.0f;

    int buf = 0;
    if (kbeg < kend) {
        load_tile(kbeg);
        store_tile(0);
    }
    __syncthreads();
    for (int k0 = kbeg; k0 < kend; k0 += BK) {
        const bool more = k0 + BK < kend;
        if (more) load_tile(k0 + BK);  // global loads in flight during the FMAs below
#pragma unroll
        for (int kk = 0; kk < BK; ++kk) {
            float a[TM], bv[TN];
#pragma unroll
            for (int i = 0; i < TM; i += 4) {
                const float4 t4 = *reinterpret_cast<const float4*>(&As[buf][kk][ty * TM + i]);
                a[i] = t4.x; a[i + 1] = t4.y; a[i + 2] = t4.z; a[i + 3] = t4.w;
            }
#pragma unroll
            for (int j = 0; j < TN; j += 4) {
                const float4 t4 = *reinterpret_cast<const float4*>(&Bs[buf][kk][tx * TN + j]);
                bv[j] = t4.x; bv[j + 1] = t4.y; bv[j + 2] = t4.z; bv[j + 3] = t4.w;
            }
#pragma unroll
            for (int i = 0; i < TM; ++i)
#pragma unroll
                for (int j = 0; j < TN; ++j) acc[i][j] = fmaf(a[i], bv[j], acc[i][j]);
        }
        if (more) {
            store_tile(buf ^ 1);
            __syncthreads();
            buf ^= 1;
        }
    }

    const long long MN = (long long)p.M * p.N;
#pragma unroll
    for (int i = 0; i < TM; ++i) {
        const int gm = m0 + ty * TM + i;
        if (gm >= p.M) continue;
        float* dst;
        const float* bias = nullptr;
        if (p.split == 1) {
            dst = p.C + (long long)b * p.stride_c + (long long)gm * p.ldc;
            bias = p.bias;
        } else {
            dst = p.ws + ((long long)s * p.batch + b) * MN + (long long)gm * p.N;
        }
#pragma unroll
        for (int j = 0; j < TN; ++j) {
            const int gn = n0 + tx * TN + j;
            if (gn < p.N) {
                const float v = bias ? acc[i][j] + __ldg(bias + gn) : acc[i][j];
                dst[gn] = p.split == 1 ? epi_out(v, p.act, dst + gn) : v;
            }
        }
    }
}

}  // namespace nnjit
