// Launch of the FP32-FFMA family: picks the precompiled instance and the grid.
#include "ffma.cuh"
#include "launch.h"

namespace nnjit {

using FfmaKernel = void (*)(FfmaParams);
FfmaKernel ffma_kernel_kn(int i);
FfmaKernel ffma_kernel_nk(int i);

cudaError_t launch_ffma(const LaunchArgs& a) {
    const Problem& p = *a.p;
    const nnjit_candidate& c = *a.c;
    if (c.instance < 0 || c.instance >= 24) return cudaErrorInvalidValue;
    const bool nk = (c.instance & 1) != 0;
    FfmaKernel k = nk ? ffma_kernel_nk(c.instance >> 1) : ffma_kernel_kn(c.instance >> 1);
    if (!k || nk != (p.b_layout == NNJIT_B_NK)) return cudaErrorInvalidValue;
    FfmaParams prm;
    prm.A = static_cast<const float*>(a.A);
    prm.B = static_cast<const float*>(a.B);
    prm.bias = a.bias;
    prm.act = p.epilogue;
    prm.C = a.C;
    prm.ws = a.ws;
    prm.M = (int)p.M; prm.N = (int)p.N; prm.K = (int)p.K; prm.batch = (int)p.batch;
    prm.split = c.split_k;
    // K slice per split: a whole number of BK steps so every slice but the last is full
    const long long steps = (p.K + c.bk - 1) / c.bk;
    prm.kper = (int)(((steps + c.split_k - 1) / c.split_k) * c.bk);
    prm.lda = p.lda; prm.ldb = p.ldb; prm.ldc = p.ldc;
    prm.stride_a = p.stride_a; prm.stride_b = p.stride_b; prm.stride_c = p.stride_c;
    const long long gz = p.batch * (long long)c.split_k;
    if (gz > 65535) return cudaErrorInvalidValue;
    dim3 grid((unsigned)((p.N + c.bn - 1) / c.bn), (unsigned)((p.M + c.bm - 1) / c.bm), (unsigned)gz);
    if (grid.y > 65535) return cudaErrorInvalidValue;
    return launch_pdl(k, grid, dim3(c.threads), 0, a.stream, prm);
}

}  // namespace nnjit
