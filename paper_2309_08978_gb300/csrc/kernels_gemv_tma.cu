// Decode-sized products (M <= 8, bf16, B stored [N][K]) fed by the tensor memory
// accelerator.
//
// Warp 0 (one lane) streams ring stages into shared memory: ROWS weight rows x 256 K
// elements (512-byte rows, one 2-D TMA box) plus the matching 256-element slice of every
// row of x (a second box).  Warps 1..4 each own ROWS / 4 rows of a stage and read them
// with 16-byte shared loads (lane l takes bytes 16l..16l+15 of a row, so a warp's read
// of one row is conflict-free); each lane keeps partial dot products over the stages of
// a work item, reduced across the warp when the item ends.  A work item is one group of
// ROWS output columns and one K slice; CTAs take items round-robin and the ring runs on
// across item boundaries, so a CTA keeps up to `stages` boxes in flight from start to
// finish.  Elements past K or N are zero-filled by the copy engine and contribute
// nothing.  The weights are read from HBM exactly once.
//
// Every wait is bounded (ptx::mbar_wait): an expired wait records an error code in the
// plan's watchdog word, the CTA stops, the producer drains its copies still in flight
// (bounded), and the kernel returns.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>

#include "epilogue.cuh"
#include "launch.h"
#include "ptx.cuh"

namespace nnjit {

namespace {

constexpr int kKc = 256;              // K elements per stage
constexpr int kRowBytes = kKc * 2;    // bytes of one row of one stage
constexpr int kThreads = 160;         // producer warp + 4 consumer warps
constexpr int kMaxStages = 8;
constexpr long long kPrefetchBytes = 48ll << 20;
constexpr int kErrGemvEmpty = 0x201;
constexpr int kErrGemvFull = 0x202;
constexpr int kErrGemvDrain = 0x203;

struct GemvTmaParams {
    CUtensorMap tmap_w;  // W [N][ldb] bf16: dims {K, N}, box {256, ROWS}
    CUtensorMap tmap_x;  // x [M][lda] bf16: dims {K, M}, box {256, M}
    const float* bias;   // split == 1 only
    float* C;            // [M][ldc]
    float* ws;           // [split][M][N]
    int* err;
    int M, N, split;
    int chunks;          // ceil(K / 256)
    int cps;             // chunks per K slice
    int groups;          // ceil(N / ROWS)
    int items;           // groups * split
    int stages;
    int b_const;         // W is not written by kernels launched earlier in the stream
    int pf_chunks;       // b_const: chunks of the first item past the ring to prefetch into L2
    int act;             // nnjit_epilogue, applied when split == 1
    long long ldc;
};

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__device__ __forceinline__ void unpack8(const uint4& v, float (&f)[8]) {
    f[0] = bf_lo(v.x); f[1] = bf_hi(v.x); f[2] = bf_lo(v.y); f[3] = bf_hi(v.y);
    f[4] = bf_lo(v.z); f[5] = bf_hi(v.z); f[6] = bf_lo(v.w); f[7] = bf_hi(v.w);
}

// Chunk range [c0, c1) of the K slice of item `it`; the item's row group is it % groups.
struct Item {
    int g, s, c0, c1;
};
__device__ __forceinline__ Item item_of(int it, const GemvTmaParams& p) {
    Item r;
    r.g = it % p.groups;
    r.s = it / p.groups;
    r.c0 = r.s * p.cps;
    r.c1 = min(p.chunks, r.c0 + p.cps);
    if (r.c1 < r.c0) r.c1 = r.c0;
    return r;
}

// grid: persistent CTAs (<= items); block: 160 threads; dynamic smem: 128 (alignment)
// + stages * (ROWS + M) * 512 bytes.
template <int ROWS, int MAXM>
__global__ void __launch_bounds__(kThreads, 1) gemv_tma_kernel(const __grid_constant__ GemvTmaParams p) {
    constexpr int RW = ROWS / 4;  // rows per consumer warp
    constexpr uint32_t kWBytes = ROWS * kRowBytes;
    static_assert(ROWS % 4 == 0 && ROWS <= 256, "rows per stage");
    extern __shared__ uint8_t gsm_raw[];
    __shared__ __align__(8) uint64_t bars[2 * kMaxStages];
    __shared__ int abort_word;
    volatile int* abort_flag = &abort_word;

    const int S = p.stages, M = p.M;
    const uint32_t xbytes = (uint32_t)M * kRowBytes;
    const uint32_t w_base = (ptx::smem_u32(gsm_raw) + 127u) & ~127u;
    const uint32_t x_base = w_base + (uint32_t)S * kWBytes;
    auto full_bar = [&](int s) { return ptx::smem_u32(bars + s); };
    auto empty_bar = [&](int s) { return ptx::smem_u32(bars + kMaxStages + s); };
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            ptx::mbar_init(full_bar(s), 1);
            ptx::mbar_init(empty_bar(s), 4);  // one arrival per consumer warp
        }
        abort_word = 0;
        ptx::fence_barrier_init();
    }
    __syncthreads();

    if (warp == 0) {
        // ------------------------------------------------------------------ producer
        if (lane == 0) {
            ptx::prefetch_tmap(&p.tmap_w);
            ptx::prefetch_tmap(&p.tmap_x);
            int stage = 0;
            uint32_t phase = 0;
            uint32_t armed = 0, armed_parity = 0;
            // With constant weights the first ring's worth of weight boxes is requested
            // before the dependency wait; their x boxes follow once the previous kernel
            // (which may produce x) has finished.
            // Weights are read once: their lines go first when L2 needs room, so they do
            // not evict what the next kernel has prefetched.
            const uint64_t pol = ptx::l2_policy_evict_first();
            int pre = 0;
            int pre_chunk[kMaxStages];
            Item first{};
            if (p.b_const && (int)blockIdx.x < p.items) {
                first = item_of(blockIdx.x, p);
                for (int c = first.c0; c < first.c1 && pre < S; ++c, ++pre) {
                    ptx::mbar_arrive_expect_tx(full_bar(pre), kWBytes + xbytes);
                    ptx::tma_load_2d_hint(w_base + pre * kWBytes, &p.tmap_w, c * kKc, first.g * ROWS,
                                          full_bar(pre), pol);
                    pre_chunk[pre] = c;
                }
                // ... and the next part of the first item is brought into L2, so the
                // weight stream keeps HBM busy while the previous kernel drains.
                const int pf_end = min(first.c1, first.c0 + pre + p.pf_chunks);
                for (int c = first.c0 + pre; c < pf_end; ++c)
                    ptx::tma_prefetch_l2_2d(&p.tmap_w, c * kKc, first.g * ROWS);
            }
            ptx::griddep_wait();
            ptx::griddep_launch_dependents();
            for (int q = 0; q < pre; ++q) {
                ptx::tma_load_2d(x_base + q * xbytes, &p.tmap_x, pre_chunk[q] * kKc, 0, full_bar(q));
                armed |= 1u << q;
            }
            stage = pre == S ? 0 : pre;
            phase = pre == S ? 1u : 0u;
            bool ok = true;
            for (int it = blockIdx.x; ok && it < p.items; it += gridDim.x) {
                const Item w = item_of(it, p);
                const int cbeg = (it == (int)blockIdx.x) ? w.c0 + pre : w.c0;
                for (int c = cbeg; c < w.c1; ++c) {
                    if (!ptx::mbar_wait(empty_bar(stage), phase ^ 1u, abort_flag, p.err, kErrGemvEmpty)) {
                        ok = false;
                        break;
                    }
                    ptx::mbar_arrive_expect_tx(full_bar(stage), kWBytes + xbytes);
                    ptx::tma_load_2d_hint(w_base + stage * kWBytes, &p.tmap_w, c * kKc, w.g * ROWS,
                                          full_bar(stage), pol);
                    ptx::tma_load_2d(x_base + stage * xbytes, &p.tmap_x, c * kKc, 0, full_bar(stage));
                    armed |= 1u << stage;
                    armed_parity = (armed_parity & ~(1u << stage)) | (phase << stage);
                    if (++stage == S) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            // Drain: every copy issued has landed before the CTA may exit.
            for (int s = 0; s < S; ++s) {
                if (armed & (1u << s)) {
                    volatile int no_abort = 0;
                    ptx::mbar_wait(full_bar(s), (armed_parity >> s) & 1u, &no_abort, p.err, kErrGemvDrain,
                                   ptx::kWaitLimitNs / 4);
                }
            }
        }
        return;
    }

    // ---------------------------------------------------------------------- consumers
    ptx::griddep_wait();
    const int cw = warp - 1;
    int stage = 0;
    uint32_t phase = 0;
    for (int it = blockIdx.x; it < p.items; it += gridDim.x) {
        const Item w = item_of(it, p);
        float acc[RW][MAXM];
#pragma unroll
        for (int r = 0; r < RW; ++r)
#pragma unroll
            for (int m = 0; m < MAXM; ++m) acc[r][m] = 0.0f;
        bool ok = true;
        for (int c = w.c0; c < w.c1; ++c) {
            // the warp's lanes agree on the outcome, so the warp stays converged
            if (!__all_sync(0xffffffffu, ptx::mbar_wait(full_bar(stage), phase, abort_flag, p.err, kErrGemvFull))) {
                ok = false;
                break;
            }
            float xf[MAXM][8];
#pragma unroll
            for (int m = 0; m < MAXM; ++m) {
                if (m < M) {
                    unpack8(ptx::ld_shared_v4(x_base + stage * xbytes + m * kRowBytes + lane * 16), xf[m]);
                } else {
#pragma unroll
                    for (int j = 0; j < 8; ++j) xf[m][j] = 0.0f;
                }
            }
            const uint32_t wrow = w_base + stage * kWBytes + (cw * RW) * kRowBytes + lane * 16;
#pragma unroll
            for (int r = 0; r < RW; ++r) {
                float wf[8];
                unpack8(ptx::ld_shared_v4(wrow + r * kRowBytes), wf);
#pragma unroll
                for (int m = 0; m < MAXM; ++m) {
                    if (m < M) {
#pragma unroll
                        for (int j = 0; j < 8; ++j) acc[r][m] = fmaf(wf[j], xf[m][j], acc[r][m]);
                    }
                }
            }
            ptx::mbar_arrive_elect(empty_bar(stage));  // after every lane's reads of the stage
            if (++stage == S) {
                stage = 0;
                phase ^= 1u;
            }
        }
        if (!ok) break;
        // butterfly reduction over the warp, then lane 0 writes the warp's rows
#pragma unroll
        for (int r = 0; r < RW; ++r)
#pragma unroll
            for (int m = 0; m < MAXM; ++m) {
                if (m < M) {
                    float v = acc[r][m];
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
                    acc[r][m] = v;
                }
            }
        if (lane == 0) {
#pragma unroll
            for (int r = 0; r < RW; ++r) {
                const int n = w.g * ROWS + cw * RW + r;
                if (n >= p.N) continue;
#pragma unroll
                for (int m = 0; m < MAXM; ++m) {
                    if (m >= M) continue;
                    if (p.split == 1)
                        p.C[(long long)m * p.ldc + n] = epi_out(p.bias ? acc[r][m] + p.bias[n] : acc[r][m], p.act,
                                                                p.C + (long long)m * p.ldc + n);
                    else
                        p.ws[((long long)w.s * M + m) * p.N + n] = acc[r][m];
                }
            }
        }
    }
}

using GemvTmaKernel = void (*)(GemvTmaParams);
// Instance table, indexed as gemv_tma_instance() - kGemvTmaFirstInstance:
// (ROWS 8, 16, 32) x (MAXM 1, 8).
const GemvTmaKernel kKernels[6] = {
    gemv_tma_kernel<8, 1>,  gemv_tma_kernel<8, 8>,  gemv_tma_kernel<16, 1>,
    gemv_tma_kernel<16, 8>, gemv_tma_kernel<32, 1>, gemv_tma_kernel<32, 8>,
};
const int kRowsOf[6] = {8, 8, 16, 16, 32, 32};
const int kMaxMOf[6] = {1, 8, 1, 8, 1, 8};


}  // namespace

bool gemv_uses_tma(const nnjit_candidate& c) {
    return c.family == NNJIT_FAMILY_GEMV && c.instance >= kGemvTmaFirstInstance &&
           c.instance < kGemvTmaFirstInstance + 6;
}

cudaError_t encode_gemv_tensor_maps(const Problem& p, const nnjit_candidate& c, const void* A,
                                    const void* B, CUtensorMap* tx, CUtensorMap* tw,
                                    const char** why) {
    EncodeTiledFn enc = get_encode_fn();
    if (!enc) {
        *why = "cuTensorMapEncodeTiled entry point unavailable";
        return cudaErrorNotSupported;
    }
    const int i = c.instance - kGemvTmaFirstInstance;
    if (i < 0 || i >= 6 || p.M < 1 || p.M > 8) {
        *why = "not a TMA GEMV candidate";
        return cudaErrorInvalidValue;
    }
    const cuuint32_t estr[2] = {1, 1};
    {
        const cuuint64_t dims[2] = {(cuuint64_t)p.K, (cuuint64_t)p.N};
        const cuuint64_t strides[1] = {(cuuint64_t)(p.ldb * 2)};
        const cuuint32_t box[2] = {(cuuint32_t)kKc, (cuuint32_t)kRowsOf[i]};
        CUresult r = enc(tw, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(B), dims, strides, box,
                         estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                         CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) {
            *why = "cuTensorMapEncodeTiled failed for the GEMV weights";
            return cudaErrorInvalidValue;
        }
    }
    {
        const cuuint64_t dims[2] = {(cuuint64_t)p.K, (cuuint64_t)p.M};
        const cuuint64_t strides[1] = {(cuuint64_t)(p.lda * 2)};
        const cuuint32_t box[2] = {(cuuint32_t)kKc, (cuuint32_t)p.M};
        CUresult r = enc(tx, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(A), dims, strides, box,
                         estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                         CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) {
            *why = "cuTensorMapEncodeTiled failed for the GEMV activations";
            return cudaErrorInvalidValue;
        }
    }
    return cudaSuccess;
}

cudaError_t launch_gemv_tma(const LaunchArgs& a) {
    const Problem& p = *a.p;
    const nnjit_candidate& c = *a.c;
    const int i = c.instance - kGemvTmaFirstInstance;
    if (i < 0 || i >= 6 || !a.tmap_a || !a.tmap_b || p.b_layout != NNJIT_B_NK) return cudaErrorInvalidValue;
    if (p.M < 1 || p.M > kMaxMOf[i] || c.bn != kRowsOf[i] || c.stages < 2 || c.stages > kMaxStages ||
        c.split_k < 1 || c.threads != kThreads)
        return cudaErrorInvalidValue;
    GemvTmaParams prm;
    prm.tmap_x = *a.tmap_a;
    prm.tmap_w = *a.tmap_b;
    prm.bias = a.bias;
    prm.C = a.C;
    prm.ws = a.ws;
    prm.err = a.err;
    prm.M = (int)p.M;
    prm.N = (int)p.N;
    prm.split = c.split_k;
    prm.chunks = (int)((p.K + kKc - 1) / kKc);
    prm.cps = (prm.chunks + c.split_k - 1) / c.split_k;
    prm.groups = (int)((p.N + kRowsOf[i] - 1) / kRowsOf[i]);
    const long long items = (long long)prm.groups * c.split_k;
    if (items >= (1LL << 31)) return cudaErrorInvalidValue;
    prm.items = (int)items;
    prm.stages = c.stages;
    prm.b_const = (p.flags & NNJIT_PLAN_B_CONSTANT) ? 1 : 0;
    prm.ldc = p.ldc;
    prm.act = c.split_k == 1 ? p.epilogue : NNJIT_EPI_NONE;
    const int grid = (int)std::min<long long>(items, std::max(1, c.grid));
    // L2 prefetch ahead of the dependency wait: at most kPrefetchBytes over the grid
    // (well under the 129 MB L2, which the previous kernel is also streaming through).
    prm.pf_chunks = 0;
    if (prm.b_const) {
        const long long per_cta = kPrefetchBytes / grid / ((long long)kRowsOf[i] * kRowBytes);
        prm.pf_chunks = (int)std::min<long long>(per_cta, prm.cps);
    }
    const int smem = 128 + c.stages * (kRowsOf[i] + (int)p.M) * kRowBytes;
    cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void*>(kKernels[i]), smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(kKernels[i], dim3(grid), dim3(kThreads), smem, a.stream, prm);
}

}  // namespace nnjit
