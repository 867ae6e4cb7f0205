// Split-K GEMV entry point that allocates nothing.
//
// Some callers cannot allocate device memory when they run a product: a process whose
// device memory has already been reserved by a framework's caching allocator (a side
// cudaMalloc can fail or fragment it), or a latency-critical decode loop that must not
// pay for cudaMalloc / cudaFree, which may synchronise the device.  Plans allocate their
// split-K workspace when they are made; this entry point needs no plan: its split-K
// partial sums go to a fixed-size array that lives in the library's device image, so it
// exists on every GPU that loads the library, from module load until process exit.
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "../../include/nnjit.h"
#include "launch.h"
#include "space.h"

namespace nnjit {

// Shared split-K scratch of every call of nnjit_gemv_bf16_noalloc on a device.
static __device__ __align__(256) float g_noalloc_scratch[NNJIT_NOALLOC_SCRATCH_FLOATS];

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
float* g_noalloc_ptr[kMaxDevices] = {nullptr};

// Device address of the scratch array on the current device.  In host code the array's
// name is only a host-side stand-in, so the address is looked up once per device (with
// that device current) and passed to the kernels.
cudaError_t noalloc_scratch(int dev, float** out) {
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
        void* p = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        g_noalloc_ptr[dev] = static_cast<float*>(p);
    }
    *out = g_noalloc_ptr[dev];
    return cudaSuccess;
}

}  // namespace
}  // namespace nnjit

using namespace nnjit;

extern "C" nnjit_status nnjit_gemv_bf16_noalloc(int64_t M, int64_t N, int64_t K, const void* x,
                                                const void* W, const float* bias, float* C,
                                                int32_t split_k, void* stream) {
    // Problem checks: the fixed configuration below streams W with 16-byte loads.
    if (M < 1 || M > ModelConstants::kGemvMaxM || N < 1 || K < 1 || K >= ((int64_t)1 << 31) ||
        N >= ((int64_t)1 << 31)) {
        set_last_error("nnjit_gemv_bf16_noalloc: needs 1 <= M <= 8, N >= 1, K >= 1 (< 2^31)");
        return NNJIT_ERR_INVALID_ARG;
    }
    if (split_k < 1 || split_k > 64) {
        set_last_error("nnjit_gemv_bf16_noalloc: split_k must be in 1..64");
        return NNJIT_ERR_INVALID_ARG;
    }
    if (!x || !W || !C) {
        set_last_error("nnjit_gemv_bf16_noalloc: x, W and C must not be NULL");
        return NNJIT_ERR_INVALID_ARG;
    }
    if (K % 8 != 0 || (reinterpret_cast<uintptr_t>(x) & 15) || (reinterpret_cast<uintptr_t>(W) & 15) ||
        (reinterpret_cast<uintptr_t>(C) & 3) || (bias && (reinterpret_cast<uintptr_t>(bias) & 3))) {
        set_last_error("nnjit_gemv_bf16_noalloc: needs K % 8 == 0, x and W 16-byte aligned, "
                       "C and bias 4-byte aligned");
        return NNJIT_ERR_UNSUPPORTED;
    }
    // The partials of all K slices must fit the library's scratch array.
    if (split_k > 1 && (int64_t)split_k * M * N > (int64_t)NNJIT_NOALLOC_SCRATCH_FLOATS) {
        set_last_error("nnjit_gemv_bf16_noalloc: split_k * M * N exceeds the library's scratch "
                       "(NNJIT_NOALLOC_SCRATCH_FLOATS = 1048576 floats); lower split_k or use a plan");
        return NNJIT_ERR_UNSUPPORTED;
    }
    // x slice held in shared memory: M * (K / split, rounded up to 8) bf16 values
    const int64_t kper = ((K + split_k - 1) / split_k + 7) / 8 * 8;
    if (M * kper * 2 > 96 * 1024) {
        set_last_error("nnjit_gemv_bf16_noalloc: M * ceil(K / split_k) bf16 values exceed 96 KiB "
                       "of shared memory; raise split_k");
        return NNJIT_ERR_UNSUPPORTED;
    }

    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
        set_last_error("nnjit_gemv_bf16_noalloc: no usable current CUDA device");
        return NNJIT_ERR_CUDA;
    }
    float* scratch = nullptr;
    if (split_k > 1 && noalloc_scratch(dev, &scratch) != cudaSuccess) {
        set_last_error("nnjit_gemv_bf16_noalloc: cudaGetSymbolAddress of the scratch array failed");
        return NNJIT_ERR_CUDA;
    }

    Problem p;
    p.M = M; p.N = N; p.K = K; p.batch = 1;
    p.dtype = NNJIT_BF16;
    p.b_layout = NNJIT_B_NK;
    p.lda = K; p.ldb = K; p.ldc = N;
    p.stride_a = M * K; p.stride_b = N * K; p.stride_c = M * N;
    p.has_bias = bias ? 1 : 0;
    // One fixed GEMV configuration: 8 warps per CTA, 2 weight rows per warp, 4 16-byte
    // loads in flight per row and lane.
    nnjit_candidate c{};
    c.family = NNJIT_FAMILY_GEMV;
    c.bm = (int32_t)M;
    c.tm = 2;
    c.tn = 1;
    c.stages = 4;
    c.split_k = split_k;
    c.threads = 256;
    c.bn = 8 * 2;
    c.grid = (int32_t)(((N + c.bn - 1) / c.bn) * split_k);  // one CTA per 16-row block
    c.instance = gemv_instance(NNJIT_B_NK, 2, 4);

    LaunchArgs la;
    la.p = &p;
    la.c = &c;
    la.A = x;
    la.B = W;
    la.bias = split_k > 1 ? nullptr : bias;
    la.C = C;
    la.ws = scratch;
    la.stream = static_cast<cudaStream_t>(stream);
    if (launch_gemv(la) != cudaSuccess) {
        set_last_error("nnjit_gemv_bf16_noalloc: GEMV launch failed");
        return NNJIT_ERR_CUDA;
    }
    if (split_k > 1 &&
        launch_splitk_reduce(scratch, split_k, p, bias, C, static_cast<cudaStream_t>(stream)) != cudaSuccess) {
        set_last_error("nnjit_gemv_bf16_noalloc: split-K reduce launch failed");
        return NNJIT_ERR_CUDA;
    }
    return NNJIT_OK;
}
