// Decode-sized products (M <= 8) with bf16 weights, the fixed-order split-K reduction,
// and small utility kernels.
//
// GEMV, B stored [N][K] (Linear weights): each warp owns R consecutive output columns
// (weight rows) and one K slice; lanes stream the rows with 16-byte non-allocating loads
// (U loads per row in flight per lane), multiply by x held in shared memory, and reduce
// across the warp with a butterfly of shuffles.  Weights are read exactly once.
// GEMV, B stored [K][N]: each lane owns 8 consecutive columns, the CTA's warps split the
// K slice, and partial sums are added across warps in shared memory in a fixed order.
#include <cuda_runtime.h>

#include <cstdint>
#include <algorithm>

#include "epilogue.cuh"
#include "launch.h"
#include "ptx.cuh"

namespace nnjit {

namespace {

constexpr int kMaxM = 8;

struct GemvParams {
    const uint16_t* x;   // [M][lda] bf16
    const uint16_t* W;   // NK: [N][ldb]; KN: [K][ldb]
    const float* bias;   // split == 1 only
    float* C;            // [M][ldc]
    float* ws;           // [split][M][N]
    int M, N, K, split, kper;
    int vec_ok;          // KN: rows of W are 16-byte aligned (ldb % 8 == 0)
    int b_const;         // W is not written by kernels launched before this one
    int act;             // nnjit_epilogue, applied when split == 1
    long long lda, ldb, ldc;
};

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__device__ __forceinline__ float dot8(const uint4& w, const uint4& x, float acc) {
    acc = fmaf(bf_lo(w.x), bf_lo(x.x), acc);
    acc = fmaf(bf_hi(w.x), bf_hi(x.x), acc);
    acc = fmaf(bf_lo(w.y), bf_lo(x.y), acc);
    acc = fmaf(bf_hi(w.y), bf_hi(x.y), acc);
    acc = fmaf(bf_lo(w.z), bf_lo(x.z), acc);
    acc = fmaf(bf_hi(w.z), bf_hi(x.z), acc);
    acc = fmaf(bf_lo(w.w), bf_lo(x.w), acc);
    acc = fmaf(bf_hi(w.w), bf_hi(x.w), acc);
    return acc;
}

__device__ __forceinline__ float bf16_to_f(uint16_t h) { return __uint_as_float((uint32_t)h << 16); }

// grid: (CTAs, split) with CTAs <= ceil(N / (warps * R)); dynamic smem: M * kper bf16.
// Each warp streams R weight rows in batches of U 16-byte loads per lane and row; the
// other warps of the SM hide each batch's latency.
template <int R, int U>
__global__ void __launch_bounds__(256) gemv_nk_kernel(const GemvParams p) {
    extern __shared__ __align__(16) uint16_t xs[];
    const int warps = blockDim.x >> 5;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int s = blockIdx.y;
    const int k0 = s * p.kper;
    const int klen = max(0, min(p.K, k0 + p.kper) - k0);
    const int M = p.M;
    const int nvec = klen >> 3;  // full 16-byte chunks in this slice
    // Row groups of R weight rows are dealt to warps round-robin over the whole grid.
    const int groups = (p.N + R - 1) / R;
    const int g_first = blockIdx.x * warps + warp;

    auto row_ptrs = [&](int g, const uint16_t* (&wrow)[R]) {
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const int n = min(g * R + r, p.N - 1);  // rows past N repeat the last row, unused
            wrow[r] = p.W + (long long)n * p.ldb + k0;
        }
    };
    auto load_batch = [&](const uint16_t* const (&wrow)[R], int c0, uint4 (&w)[U][R]) {
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int c = c0 + u * 32 + lane;
#pragma unroll
            for (int r = 0; r < R; ++r)
                w[u][r] = c < nvec ? ptx::ld_stream_v4(wrow[r] + c * 8) : make_uint4(0, 0, 0, 0);
        }
    };

    // With constant weights the first batch is requested before the dependency wait, so
    // the weight stream overlaps the previous kernel's tail; x is read only after it.
    uint4 w[U][R];
    const uint16_t* wrow[R];
    bool have_first = false;
    if (g_first < groups) {
        row_ptrs(g_first, wrow);
        if (p.b_const && nvec > 0) {
            load_batch(wrow, 0, w);
            have_first = true;
        }
    }
    ptx::griddep_wait();
    if (threadIdx.x == 0) ptx::griddep_launch_dependents();

    // x slice -> shared memory (16-byte copies when the slice allows, else scalar)
    const int kl8 = klen & ~7;
    for (int m = 0; m < M; ++m) {
        const uint16_t* src = p.x + (long long)m * p.lda + k0;
        uint16_t* dst = xs + (long long)m * p.kper;
        for (int i = threadIdx.x * 8; i < kl8; i += blockDim.x * 8)
            *reinterpret_cast<uint4*>(dst + i) = *reinterpret_cast<const uint4*>(src + i);
        for (int i = kl8 + threadIdx.x; i < klen; i += blockDim.x) dst[i] = src[i];
    }
    __syncthreads();

    for (int g = g_first; g < groups; g += gridDim.x * warps) {
        const int n_base = g * R;
        if (g != g_first) row_ptrs(g, wrow);
        float acc[R][kMaxM];
#pragma unroll
        for (int r = 0; r < R; ++r)
#pragma unroll
            for (int m = 0; m < kMaxM; ++m) acc[r][m] = 0.0f;
        for (int c0 = 0; c0 < nvec; c0 += 32 * U) {
            if (!(c0 == 0 && g == g_first && have_first)) load_batch(wrow, c0, w);
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int c = c0 + u * 32 + lane;
                if (c < nvec) {
#pragma unroll
                    for (int m = 0; m < kMaxM; ++m) {
                        if (m < M) {
                            const uint4 xv = *reinterpret_cast<const uint4*>(xs + (long long)m * p.kper + c * 8);
#pragma unroll
                            for (int r = 0; r < R; ++r) acc[r][m] = dot8(w[u][r], xv, acc[r][m]);
                        }
                    }
                }
            }
        }
        // ragged K tail (fewer than 8 elements)
        for (int k = (nvec << 3) + lane; k < klen; k += 32) {
#pragma unroll
            for (int r = 0; r < R; ++r) {
                const float wv = bf16_to_f(wrow[r][k]);
#pragma unroll
                for (int m = 0; m < kMaxM; ++m)
                    if (m < M) acc[r][m] = fmaf(wv, bf16_to_f(xs[(long long)m * p.kper + k]), acc[r][m]);
            }
        }
        // butterfly reduction over the warp
#pragma unroll
        for (int r = 0; r < R; ++r)
#pragma unroll
            for (int m = 0; m < kMaxM; ++m) {
                if (m < M) {
                    float v = acc[r][m];
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
                    acc[r][m] = v;
                }
            }
        if (lane == 0) {
#pragma unroll
            for (int r = 0; r < R; ++r) {
                const int n = n_base + r;
                if (n >= p.N) continue;
#pragma unroll
                for (int m = 0; m < kMaxM; ++m) {
                    if (m >= M) continue;
                    if (p.split == 1)
                        p.C[(long long)m * p.ldc + n] = epi_out(p.bias ? acc[r][m] + p.bias[n] : acc[r][m], p.act,
                                                                p.C + (long long)m * p.ldc + n);
                    else
                        p.ws[((long long)s * M + m) * p.N + n] = acc[r][m];
                }
            }
        }
    }
}

// grid: (ceil(N / 256), split); dynamic smem: warps * M * 256 floats.
template <int U>
__global__ void __launch_bounds__(256) gemv_kn_kernel(const GemvParams p) {
    extern __shared__ __align__(16) float red[];
    ptx::griddep_wait();
    if (threadIdx.x == 0) ptx::griddep_launch_dependents();
    const int warps = blockDim.x >> 5;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int s = blockIdx.y;
    const int k0 = s * p.kper;
    const int k1 = min(p.K, k0 + p.kper);
    const int M = p.M;
    const int n0 = blockIdx.x * 256 + lane * 8;
    const bool vec = p.vec_ok && n0 + 8 <= p.N;
    float acc[kMaxM][8];
#pragma unroll
    for (int m = 0; m < kMaxM; ++m)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[m][j] = 0.0f;
    for (int kb = k0 + warp; kb < k1; kb += warps * U) {
        uint4 w[U];
        float xv[U][kMaxM];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int k = kb + u * warps;
            w[u] = make_uint4(0, 0, 0, 0);
            if (k < k1) {
                const uint16_t* src = p.W + (long long)k * p.ldb + n0;
                if (vec) {
                    w[u] = ptx::ld_stream_v4(src);
                } else {
                    uint16_t t[8] = {0, 0, 0, 0, 0, 0, 0, 0};
                    for (int j = 0; j < 8; ++j)
                        if (n0 + j < p.N) t[j] = src[j];
                    w[u] = make_uint4(t[0] | (uint32_t)t[1] << 16, t[2] | (uint32_t)t[3] << 16,
                                      t[4] | (uint32_t)t[5] << 16, t[6] | (uint32_t)t[7] << 16);
                }
            }
#pragma unroll
            for (int m = 0; m < kMaxM; ++m)
                xv[u][m] = (m < M && k < k1) ? bf16_to_f(p.x[(long long)m * p.lda + k]) : 0.0f;
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const float wf[8] = {bf_lo(w[u].x), bf_hi(w[u].x), bf_lo(w[u].y), bf_hi(w[u].y),
                                 bf_lo(w[u].z), bf_hi(w[u].z), bf_lo(w[u].w), bf_hi(w[u].w)};
#pragma unroll
            for (int m = 0; m < kMaxM; ++m)
                if (m < M)
#pragma unroll
                    for (int j = 0; j < 8; ++j) acc[m][j] = fmaf(xv[u][m], wf[j], acc[m][j]);
        }
    }
#pragma unroll
    for (int m = 0; m < kMaxM; ++m)
        if (m < M)
#pragma unroll
            for (int j = 0; j < 8; ++j) red[((long long)warp * M + m) * 256 + lane * 8 + j] = acc[m][j];
    __syncthreads();
    for (int e = threadIdx.x; e < M * 256; e += blockDim.x) {
        const int m = e / 256, col = e % 256;
        const int n = blockIdx.x * 256 + col;
        if (n >= p.N) continue;
        float v = 0.0f;
        for (int w = 0; w < warps; ++w) v += red[((long long)w * M + m) * 256 + col];
        if (p.split == 1)
            p.C[(long long)m * p.ldc + n] = epi_out(p.bias ? v + p.bias[n] : v, p.act, p.C + (long long)m * p.ldc + n);
        else
            p.ws[((long long)s * M + m) * p.N + n] = v;
    }
}

using GemvKernel = void (*)(GemvParams);
// Instance table, indexed as gemv_instance(): NK (R, U) pairs, then KN U = 2, 4.
const GemvKernel kGemvKernels[8] = {
    gemv_nk_kernel<1, 2>, gemv_nk_kernel<1, 4>, gemv_nk_kernel<2, 2>, gemv_nk_kernel<2, 4>,
    gemv_nk_kernel<4, 2>, gemv_nk_kernel<4, 4>, gemv_kn_kernel<2>,    gemv_kn_kernel<4>,
};


// Fixed-order sum of the split-K partials (s = 0, 1, ... per element; + bias, activation)
// into C.  With vec4, four consecutive columns per thread in 16-byte accesses (N, ldc and
// stride_c multiples of 4; C, bias and the workspace 16-byte aligned).
__global__ void splitk_reduce_kernel(const float* __restrict__ ws, int split, long long batch_mn,
                                     int M, int N, long long ldc, long long stride_c,
                                     const float* __restrict__ bias, int act, int vec4, float* __restrict__ C) {
    ptx::griddep_wait();
    if (threadIdx.x == 0) ptx::griddep_launch_dependents();
    const long long step = (long long)gridDim.x * blockDim.x;
    if (vec4) {
        const int n4 = N >> 2;
        const long long total = batch_mn >> 2;
        for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total; i += step) {
            const long long row = i / n4;  // batch item * M + m
            const int c = (int)(i - row * n4) << 2;
            const long long e = row * N + c;
            float4 v = *reinterpret_cast<const float4*>(ws + e);
            for (int s = 1; s < split; ++s) {
                const float4 w = *reinterpret_cast<const float4*>(ws + (long long)s * batch_mn + e);
                v.x += w.x; v.y += w.y; v.z += w.z; v.w += w.w;
            }
            if (bias) {
                const float4 b4 = *reinterpret_cast<const float4*>(bias + c);
                v.x += b4.x; v.y += b4.y; v.z += b4.z; v.w += b4.w;
            }
            if ((act & 15) != NNJIT_EPI_NONE) {
                v.x = apply_act(v.x, act); v.y = apply_act(v.y, act);
                v.z = apply_act(v.z, act); v.w = apply_act(v.w, act);
            }
            const long long b = row / M;
            const int m = (int)(row - b * M);
            float4* out = reinterpret_cast<float4*>(C + b * stride_c + (long long)m * ldc + c);
            if (act & NNJIT_EPI_RESIDUAL) {
                const float4 o = *out;
                v.x += o.x; v.y += o.y; v.z += o.z; v.w += o.w;
            }
            *out = v;
        }
        return;
    }
    const long long mn = (long long)M * N;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < batch_mn; i += step) {
        float v = ws[i];
        for (int s = 1; s < split; ++s) v += ws[(long long)s * batch_mn + i];
        const long long b = i / mn;
        const long long r = i % mn;
        const int m = (int)(r / N), n = (int)(r % N);
        if (bias) v += bias[n];
        float* out = C + b * stride_c + (long long)m * ldc + n;
        *out = act != NNJIT_EPI_NONE ? epi_out(v, act, out) : v;
    }
}

__global__ void fill_bias_kernel(long long total, int M, int N, long long ldc, long long stride_c,
                                 const float* __restrict__ bias, int act, float* __restrict__ C) {
    ptx::griddep_wait();
    if (threadIdx.x == 0) ptx::griddep_launch_dependents();
    const long long mn = (long long)M * N;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        const long long b = i / mn, r = i % mn;
        const int m = (int)(r / N), n = (int)(r % N);
        float* out = C + b * stride_c + (long long)m * ldc + n;
        *out = epi_out(bias ? bias[n] : 0.0f, act, out);
    }
}

__device__ __forceinline__ uint32_t hash32(uint32_t x) {
    x ^= x >> 16; x *= 0x7feb352dU; x ^= x >> 15; x *= 0x846ca68bU; x ^= x >> 16;
    return x;
}

// Values in [-1, 1) with 8 significant bits, as f32 or bf16 bit patterns.
__global__ void fill_scratch_kernel(void* dst, long long n, int elem_bytes, uint32_t seed) {
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
         i += (long long)gridDim.x * blockDim.x) {
        const uint32_t h = hash32((uint32_t)i * 2654435761u ^ seed ^ (uint32_t)(i >> 32));
        const float v = ((int)(h >> 24) - 128) * (1.0f / 128.0f);
        if (elem_bytes == 2)
            static_cast<uint16_t*>(dst)[i] = (uint16_t)(__float_as_uint(v) >> 16);
        else
            static_cast<float*>(dst)[i] = v;
    }
}

__global__ void l2_flush_kernel(uint4* buf, long long n16) {
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n16;
         i += (long long)gridDim.x * blockDim.x)
        buf[i] = make_uint4((uint32_t)i, 0, 0, 0);
}

int grid_for(long long n, int threads) {
    long long g = (n + threads - 1) / threads;
    if (g > 152 * 16) g = 152 * 16;
    return (int)(g < 1 ? 1 : g);
}

}  // namespace

cudaError_t prepare_gemv_instance(int instance, int smem_bytes) {
    if (instance < 0 || instance >= 8) return cudaErrorInvalidValue;
    if (smem_bytes <= 48 * 1024) return cudaSuccess;
    return ensure_dynamic_smem(reinterpret_cast<const void*>(kGemvKernels[instance]), smem_bytes);
}

cudaError_t launch_gemv(const LaunchArgs& a) {
    const Problem& p = *a.p;
    const nnjit_candidate& c = *a.c;
    if (gemv_uses_tma(c)) return launch_gemv_tma(a);
    if (gemv_uses_w4(c)) return launch_gemv_w4(a);
    if (c.instance < 0 || c.instance >= 8 || p.M > kMaxM) return cudaErrorInvalidValue;
    const bool kn_inst = c.instance >= 6;
    if (kn_inst != (p.b_layout == NNJIT_B_KN)) return cudaErrorInvalidValue;
    GemvParams prm;
    prm.x = static_cast<const uint16_t*>(a.A);
    prm.W = static_cast<const uint16_t*>(a.B);
    prm.bias = a.bias;
    prm.C = a.C;
    prm.ws = a.ws;
    prm.M = (int)p.M; prm.N = (int)p.N; prm.K = (int)p.K;
    prm.split = c.split_k;
    prm.lda = p.lda; prm.ldb = p.ldb; prm.ldc = p.ldc;
    prm.vec_ok = (p.ldb % 8 == 0 && (reinterpret_cast<uintptr_t>(a.B) & 15) == 0) ? 1 : 0;
    prm.b_const = (p.flags & NNJIT_PLAN_B_CONSTANT) ? 1 : 0;
    prm.act = prm.split == 1 ? p.epilogue : NNJIT_EPI_NONE;
    const int warps = c.threads / 32;
    dim3 grid;
    int smem;
    if (!kn_inst) {
        // K slice: a multiple of 8 elements so every slice starts 16-byte aligned
        prm.kper = (int)((((p.K + c.split_k - 1) / c.split_k) + 7) / 8 * 8);
        grid = dim3((unsigned)std::max(1, c.grid / c.split_k), (unsigned)c.split_k);
        smem = (int)((p.M * (long long)prm.kper * 2 + 15) / 16 * 16);
    } else {
        prm.kper = (int)((p.K + c.split_k - 1) / c.split_k);
        grid = dim3((unsigned)((p.N + 255) / 256), (unsigned)c.split_k);
        smem = warps * (int)p.M * 256 * 4;
    }
    cudaError_t e = prepare_gemv_instance(c.instance, smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(kGemvKernels[c.instance], grid, dim3(c.threads), smem, a.stream, prm);
}

cudaError_t launch_splitk_reduce(const float* ws, int split, const Problem& p, const float* bias,
                                 float* C, cudaStream_t s) {
    const long long n = p.batch * p.M * p.N;
    if (n == 0) return cudaSuccess;
    auto a16 = [](const void* q) { return (reinterpret_cast<uintptr_t>(q) & 15) == 0; };
    const int vec4 = (p.N % 4 == 0 && p.ldc % 4 == 0 && p.stride_c % 4 == 0 && a16(C) && a16(ws) &&
                      (!bias || a16(bias))) ? 1 : 0;
    return launch_pdl(splitk_reduce_kernel, dim3(grid_for(vec4 ? n / 4 : n, 256)), dim3(256), 0, s, ws, split,
                      n, (int)p.M, (int)p.N, p.ldc, p.stride_c, bias, p.epilogue, vec4, C);
}

cudaError_t launch_fill_bias(const Problem& p, const float* bias, float* C, cudaStream_t s) {
    const long long n = p.batch * p.M * p.N;
    if (n == 0) return cudaSuccess;
    return launch_pdl(fill_bias_kernel, dim3(grid_for(n, 256)), dim3(256), 0, s, n, (int)p.M,
                      (int)p.N, p.ldc, p.stride_c, bias, p.epilogue, C);
}

cudaError_t launch_fill_scratch(void* dst, int64_t n_elems, int elem_bytes, uint32_t seed,
                                cudaStream_t s) {
    if (n_elems <= 0) return cudaSuccess;
    fill_scratch_kernel<<<grid_for(n_elems, 256), 256, 0, s>>>(dst, n_elems, elem_bytes, seed);
    return cudaGetLastError();
}

cudaError_t launch_l2_flush(void* buf, int64_t bytes, cudaStream_t s) {
    const long long n16 = bytes / 16;
    if (n16 <= 0) return cudaSuccess;
    l2_flush_kernel<<<grid_for(n16, 256), 256, 0, s>>>(static_cast<uint4*>(buf), n16);
    return cudaGetLastError();
}

}  // namespace nnjit
