// Decode-sized products over 4-bit weights (NNJIT_W4_BF16): C[m][n] = sum_k x[m][k] *
// (q[n][k] - 8) * s[k / 128][n] (+ bias[n]), M <= 8, fed by the tensor memory accelerator.
//
// The structure is that of the bf16 TMA-fed GEMV: warp 0 (one lane) streams ring stages
// of ROWS weight rows x 1024 codes (512 bytes a row, one 2-D box of 32-bit words), the 8
// group scales of those rows (a second box, group-major) and the matching 1024-element
// slice of every row of x (four boxes of 256); warps 1..4 each own ROWS / 4 rows of a
// stage.  Lane l takes 8 consecutive codes at k = 8l + 256i for i = 0..3 (a 4-byte word
// of codes at byte 4l + 128i, 16 bytes of x at 16l + 512i: both conflict-free), whose
// group is 2i + l / 16.
//
// Dequantisation costs one logic operation per weight and one packed add and one packed
// FMA (f32x2) per two weights.  Masking a code in place (nibble t of a 16-bit half at
// bits 4t) and or-ing the exponent of 2^23 gives the float 2^23 + c 16^t exactly;
// subtracting 2^23 + 8 16^t leaves (c - 8) 16^t exactly, and x, pre-scaled once per
// stage by 16^-t, turns the FMA into (c - 8) x.  Nibble t of the low and of the high half
// share the constant and the scale, so they travel as one f32x2 pair.  Every product is
// exact in float32 (a 4-bit integer times a bfloat16); the 8 products of a group slice
// are summed in a pair, which is multiplied by the group scale into the pair
// accumulator of its row; the pair's two halves are added when the work item ends.
//
// Codes past K are zero-filled by the copy engine, and so are the scales of groups past
// K and the x elements: nothing past K contributes.  Every wait is bounded.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>
#include <mutex>

#include "epilogue.cuh"
#include "launch.h"
#include "ptx.cuh"

namespace nnjit {

namespace {

constexpr int kKc = 1024;             // codes per stage and row
constexpr int kWRowBytes = kKc / 2;   // 512
constexpr int kGroupsPerStage = kKc / 128;
constexpr int kXBox = 256;            // x elements per TMA box
constexpr int kThreads = 160;
constexpr int kMaxStages = 8;
constexpr long long kPrefetchBytes = 48ll << 20;
constexpr int kErrEmpty = 0x211;
constexpr int kErrFull = 0x212;
constexpr int kErrDrain = 0x213;

struct GemvW4Params {
    CUtensorMap tmap_w;  // codes as 32-bit words: dims {ceil(K/8), N}, box {128, ROWS}
    CUtensorMap tmap_s;  // scales bf16, group-major: dims {N, groups}, box {ROWS, 8}
    CUtensorMap tmap_x;  // x bf16: dims {K, M}, box {256, M}
    const float* bias;
    float* C;
    float* ws;
    int* err;
    int M, N, split, chunks, cps, groups, items, stages, b_const, pf_chunks, act;
    long long ldc;
};

struct Item {
    int g, s, c0, c1;
};
__device__ __forceinline__ Item item_of(int it, const GemvW4Params& p) {
    Item r;
    r.g = it % p.groups;
    r.s = it / p.groups;
    r.c0 = r.s * p.cps;
    r.c1 = min(p.chunks, r.c0 + p.cps);
    if (r.c1 < r.c0) r.c1 = r.c0;
    return r;
}

// Packed float32 pairs (f32x2 arithmetic of sm_10x).
__device__ __forceinline__ uint64_t pk2(float a, float b) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
    return r;
}
__device__ __forceinline__ void unpk2(uint64_t v, float& a, float& b) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(v));
}
__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ uint64_t mul2(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
    uint64_t r;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
    return r;
}

// The 8 codes of one 32-bit word w (code t of the word at bits 4t) as pairs (code t of the
// low half, code t of the high half) minus 8, times xs[t] = (x[t], x[t + 4]) * 16^-t,
// summed over t: the pair (sum over the low codes, sum over the high codes).
__device__ __forceinline__ uint64_t dot8_w4(uint32_t w, const uint64_t (&xs)[4]) {
    const uint32_t lo = w, hi = w >> 16;
    const uint64_t c0 = pk2(-8388616.0f, -8388616.0f), c1 = pk2(-8388736.0f, -8388736.0f),
                   c2 = pk2(-8390656.0f, -8390656.0f), c3 = pk2(-8421376.0f, -8421376.0f);
    auto code2 = [&](uint32_t mask) {
        return pk2(__uint_as_float((lo & mask) | 0x4B000000u), __uint_as_float((hi & mask) | 0x4B000000u));
    };
    uint64_t s = mul2(add2(code2(0x000Fu), c0), xs[0]);
    s = fma2(add2(code2(0x00F0u), c1), xs[1], s);
    s = fma2(add2(code2(0x0F00u), c2), xs[2], s);
    s = fma2(add2(code2(0xF000u), c3), xs[3], s);
    return s;
}

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

template <int ROWS, int MAXM>
__global__ void __launch_bounds__(kThreads, 1) gemv_w4_kernel(const __grid_constant__ GemvW4Params p) {
    constexpr int RW = ROWS / 4;
    constexpr uint32_t kWBytes = ROWS * kWRowBytes;
    constexpr uint32_t kSBytes = ROWS * kGroupsPerStage * 2;
    static_assert(ROWS % 8 == 0 && ROWS <= 256, "rows per stage");
    extern __shared__ uint8_t gsm_raw[];
    __shared__ __align__(8) uint64_t bars[2 * kMaxStages];
    __shared__ int abort_word;
    volatile int* abort_flag = &abort_word;

    const int S = p.stages, M = p.M;
    const uint32_t xbytes = (uint32_t)M * kKc * 2;  // four boxes of [M][256]
    const uint32_t stage_bytes = kWBytes + kSBytes + xbytes;
    const uint32_t base = (ptx::smem_u32(gsm_raw) + 127u) & ~127u;
    const uint8_t* gbase = gsm_raw + (base - ptx::smem_u32(gsm_raw));  // generic address of `base`
    auto w_at = [&](int s) { return base + (uint32_t)s * stage_bytes; };
    auto s_at = [&](int s) { return w_at(s) + kWBytes; };
    auto x_at = [&](int s) { return w_at(s) + kWBytes + kSBytes; };
    auto full_bar = [&](int s) { return ptx::smem_u32(bars + s); };
    auto empty_bar = [&](int s) { return ptx::smem_u32(bars + kMaxStages + s); };
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            ptx::mbar_init(full_bar(s), 1);
            ptx::mbar_init(empty_bar(s), 4);
        }
        abort_word = 0;
        ptx::fence_barrier_init();
    }
    __syncthreads();

    if (warp == 0) {
        // ------------------------------------------------------------------ producer
        if (lane == 0) {
            ptx::prefetch_tmap(&p.tmap_w);
            ptx::prefetch_tmap(&p.tmap_s);
            ptx::prefetch_tmap(&p.tmap_x);
            const uint64_t pol = ptx::l2_policy_evict_first();
            auto load_w = [&](int st, int c, int g) {  // codes and scales of chunk c, row group g
                ptx::tma_load_2d_hint(w_at(st), &p.tmap_w, c * (kKc / 8), g * ROWS, full_bar(st), pol);
                ptx::tma_load_2d_hint(s_at(st), &p.tmap_s, g * ROWS, c * kGroupsPerStage, full_bar(st), pol);
            };
            auto load_x = [&](int st, int c) {
#pragma unroll
                for (int j = 0; j < kKc / kXBox; ++j)
                    ptx::tma_load_2d(x_at(st) + j * M * kXBox * 2, &p.tmap_x, c * kKc + j * kXBox, 0, full_bar(st));
            };
            int stage = 0;
            uint32_t phase = 0;
            uint32_t armed = 0, armed_parity = 0;
            int pre = 0;
            int pre_chunk[kMaxStages];
            if (p.b_const && (int)blockIdx.x < p.items) {
                const Item first = item_of(blockIdx.x, p);
                for (int c = first.c0; c < first.c1 && pre < S; ++c, ++pre) {
                    ptx::mbar_arrive_expect_tx(full_bar(pre), stage_bytes);
                    load_w(pre, c, first.g);
                    pre_chunk[pre] = c;
                }
                const int pf_end = min(first.c1, first.c0 + pre + p.pf_chunks);
                for (int c = first.c0 + pre; c < pf_end; ++c)
                    ptx::tma_prefetch_l2_2d(&p.tmap_w, c * (kKc / 8), first.g * ROWS);
            }
            ptx::griddep_wait();
            ptx::griddep_launch_dependents();
            for (int q = 0; q < pre; ++q) {
                load_x(q, pre_chunk[q]);
                armed |= 1u << q;
            }
            stage = pre == S ? 0 : pre;
            phase = pre == S ? 1u : 0u;
            bool ok = true;
            for (int it = blockIdx.x; ok && it < p.items; it += gridDim.x) {
                const Item w = item_of(it, p);
                const int cbeg = (it == (int)blockIdx.x) ? w.c0 + pre : w.c0;
                for (int c = cbeg; c < w.c1; ++c) {
                    if (!ptx::mbar_wait(empty_bar(stage), phase ^ 1u, abort_flag, p.err, kErrEmpty)) {
                        ok = false;
                        break;
                    }
                    ptx::mbar_arrive_expect_tx(full_bar(stage), stage_bytes);
                    load_w(stage, c, w.g);
                    load_x(stage, c);
                    armed |= 1u << stage;
                    armed_parity = (armed_parity & ~(1u << stage)) | (phase << stage);
                    if (++stage == S) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            for (int s = 0; s < S; ++s) {
                if (armed & (1u << s)) {
                    volatile int no_abort = 0;
                    ptx::mbar_wait(full_bar(s), (armed_parity >> s) & 1u, &no_abort, p.err, kErrDrain,
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
        uint64_t acc2[RW][MAXM];
#pragma unroll
        for (int r = 0; r < RW; ++r)
#pragma unroll
            for (int m = 0; m < MAXM; ++m) acc2[r][m] = 0ull;  // (+0.0f, +0.0f)
        bool ok = true;
        for (int c = w.c0; c < w.c1; ++c) {
            if (!ptx::mbar_wait(full_bar(stage), phase, abort_flag, p.err, kErrFull)) {
                ok = false;
                break;
            }
            const uint8_t* wst = gbase + (w_at(stage) - base);
            const uint32_t* codes = reinterpret_cast<const uint32_t*>(wst) + lane;
            const uint16_t* sc = reinterpret_cast<const uint16_t*>(wst + kWBytes);
            const uint8_t* xst = wst + kWBytes + kSBytes;
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                // (x[m][8l + 256i + t], x[m][8l + 256i + t + 4]) * 16^-t, t = 0..3
                uint64_t xs[MAXM][4];
#pragma unroll
                for (int m = 0; m < MAXM; ++m) {
                    if (m < M) {
                        const uint4 v = *reinterpret_cast<const uint4*>(xst + (i * M + m) * kXBox * 2 + lane * 16);
                        xs[m][0] = pk2(bf_lo(v.x), bf_lo(v.z));
                        xs[m][1] = mul2(pk2(bf_hi(v.x), bf_hi(v.z)), pk2(0.0625f, 0.0625f));
                        xs[m][2] = mul2(pk2(bf_lo(v.y), bf_lo(v.w)), pk2(0.00390625f, 0.00390625f));
                        xs[m][3] = mul2(pk2(bf_hi(v.y), bf_hi(v.w)), pk2(0.000244140625f, 0.000244140625f));
                    } else {
#pragma unroll
                        for (int t = 0; t < 4; ++t) xs[m][t] = 0ull;
                    }
                }
                const int grp = 2 * i + (lane >> 4);
#pragma unroll
                for (int r = 0; r < RW; ++r) {
                    const int row = cw * RW + r;
                    const uint32_t code = codes[row * (kWRowBytes / 4) + i * 32];
                    const float scale = __uint_as_float((uint32_t)sc[grp * ROWS + row] << 16);
                    const uint64_t scale2 = pk2(scale, scale);
#pragma unroll
                    for (int m = 0; m < MAXM; ++m)
                        if (m < M) acc2[r][m] = fma2(scale2, dot8_w4(code, xs[m]), acc2[r][m]);
                }
            }
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(empty_bar(stage));
            if (++stage == S) {
                stage = 0;
                phase ^= 1u;
            }
        }
        if (!ok) break;
        float acc[RW][MAXM];
#pragma unroll
        for (int r = 0; r < RW; ++r)
#pragma unroll
            for (int m = 0; m < MAXM; ++m) {
                float a, b;
                unpk2(acc2[r][m], a, b);
                acc[r][m] = a + b;
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
                        p.C[(long long)m * p.ldc + n] = apply_act(p.bias ? acc[r][m] + p.bias[n] : acc[r][m], p.act);
                    else
                        p.ws[((long long)w.s * M + m) * p.N + n] = acc[r][m];
                }
            }
        }
    }
}

using GemvW4Kernel = void (*)(GemvW4Params);
// Instance table, indexed as gemv_w4_instance() - kGemvW4FirstInstance:
// (ROWS 8, 16, 32) x (MAXM 1, 8).
const GemvW4Kernel kKernels[6] = {
    gemv_w4_kernel<8, 1>,  gemv_w4_kernel<8, 8>,  gemv_w4_kernel<16, 1>,
    gemv_w4_kernel<16, 8>, gemv_w4_kernel<32, 1>, gemv_w4_kernel<32, 8>,
};
const int kRowsOf[6] = {8, 8, 16, 16, 32, 32};
const int kMaxMOf[6] = {1, 8, 1, 8, 1, 8};

std::mutex g_mu;
int g_smem[6] = {0};

}  // namespace

bool gemv_uses_w4(const nnjit_candidate& c) {
    return c.family == NNJIT_FAMILY_GEMV && c.instance >= kGemvW4FirstInstance &&
           c.instance < kGemvW4FirstInstance + 6;
}

cudaError_t encode_gemv_w4_maps(const Problem& p, const nnjit_candidate& c, const void* A, const void* B,
                                CUtensorMap* tx, CUtensorMap* tw, CUtensorMap* ts, const char** why) {
    EncodeTiledFn enc = get_encode_fn();
    if (!enc) {
        *why = "cuTensorMapEncodeTiled entry point unavailable";
        return cudaErrorNotSupported;
    }
    const int i = c.instance - kGemvW4FirstInstance;
    if (i < 0 || i >= 6 || p.M < 1 || p.M > 8) {
        *why = "not a 4-bit GEMV candidate";
        return cudaErrorInvalidValue;
    }
    const cuuint32_t estr[2] = {1, 1};
    const char* blob = static_cast<const char*>(B);
    {
        const cuuint64_t dims[2] = {(cuuint64_t)((p.K + 7) / 8), (cuuint64_t)p.N};
        const cuuint64_t strides[1] = {(cuuint64_t)(p.ldb / 2)};
        const cuuint32_t box[2] = {(cuuint32_t)(kKc / 8), (cuuint32_t)kRowsOf[i]};
        if (enc(tw, CU_TENSOR_MAP_DATA_TYPE_UINT32, 2, const_cast<char*>(blob), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS) {
            *why = "cuTensorMapEncodeTiled failed for the 4-bit codes";
            return cudaErrorInvalidValue;
        }
    }
    {
        const cuuint64_t dims[2] = {(cuuint64_t)p.N, (cuuint64_t)p.w4_groups()};
        const cuuint64_t strides[1] = {(cuuint64_t)(p.N * 2)};
        const cuuint32_t box[2] = {(cuuint32_t)kRowsOf[i], (cuuint32_t)kGroupsPerStage};
        if (enc(ts, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<char*>(blob + p.w4_scale_offset()), dims,
                strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS) {
            *why = "cuTensorMapEncodeTiled failed for the group scales";
            return cudaErrorInvalidValue;
        }
    }
    {
        const cuuint64_t dims[2] = {(cuuint64_t)p.K, (cuuint64_t)p.M};
        const cuuint64_t strides[1] = {(cuuint64_t)(p.lda * 2)};
        const cuuint32_t box[2] = {(cuuint32_t)kXBox, (cuuint32_t)p.M};
        if (enc(tx, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(A), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS) {
            *why = "cuTensorMapEncodeTiled failed for the activations";
            return cudaErrorInvalidValue;
        }
    }
    return cudaSuccess;
}

cudaError_t launch_gemv_w4(const LaunchArgs& a) {
    const Problem& p = *a.p;
    const nnjit_candidate& c = *a.c;
    const int i = c.instance - kGemvW4FirstInstance;
    if (i < 0 || i >= 6 || !a.tmap_a || !a.tmap_b || !a.tmap_c || p.dtype != NNJIT_W4_BF16 ||
        p.b_layout != NNJIT_B_NK)
        return cudaErrorInvalidValue;
    if (p.M < 1 || p.M > kMaxMOf[i] || c.bn != kRowsOf[i] || c.stages < 2 || c.stages > kMaxStages ||
        c.split_k < 1 || c.threads != kThreads || c.bk != kKc)
        return cudaErrorInvalidValue;
    GemvW4Params prm;
    prm.tmap_x = *a.tmap_a;
    prm.tmap_w = *a.tmap_b;
    prm.tmap_s = *a.tmap_c;
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
    prm.act = c.split_k == 1 ? p.epilogue : NNJIT_EPI_NONE;
    prm.ldc = p.ldc;
    const int grid = (int)std::min<long long>(items, std::max(1, c.grid));
    prm.pf_chunks = 0;
    if (prm.b_const) {
        const long long per_cta = kPrefetchBytes / grid / ((long long)kRowsOf[i] * kWRowBytes);
        prm.pf_chunks = (int)std::min<long long>(per_cta, prm.cps);
    }
    const int stage_bytes = kRowsOf[i] * (kWRowBytes + kGroupsPerStage * 2) + (int)p.M * kKc * 2;
    const int smem = 128 + c.stages * stage_bytes;
    {
        std::lock_guard<std::mutex> lk(g_mu);
        if (g_smem[i] < smem) {
            cudaError_t e = cudaFuncSetAttribute(kKernels[i], cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
            if (e != cudaSuccess) return e;
            g_smem[i] = smem;
        }
    }
    return launch_pdl(kKernels[i], dim3(grid), dim3(kThreads), smem, a.stream, prm);
}

}  // namespace nnjit
