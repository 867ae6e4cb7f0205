// Decode-sized products over 4-bit weights (NNJIT_W4_BF16): C[m][n] = sum_k x[m][k] *
// (q[n][k] - 8) * s[k / 128][n] (+ bias[n]), M <= 8.  The weight rows are the M dimension
// of warp-level tensor-core MMAs (mma.sync m16n8k16, bf16 x bf16 -> f32) and the (up to 8)
// rows of x are their N dimension, so the CUDA cores only dequantise.
//
// Ring (one producer lane, TMA): a stage holds ROWS weight rows x 1024 codes as four
// 128-byte-swizzled boxes of 256 codes (box b = K quarter b), the 8 group scales of those
// rows, and the matching 1024 elements of every row of x (four boxes of 256).  Consumer
// warp w takes K quarter w of every stage for all ROWS rows (16-row MMA tiles); the four
// warps' partial sums meet in shared memory at the end of a work item (ROWS output
// columns x one K slice), in a fixed order.
//
// Fragments (m16n8k16; lane = 4 g + t): A rows g and g + 8, B column (token) g.  Within a
// block of 128 codes (one scale group) thread t loads 32 consecutive codes of each of its
// rows (a conflict-free 16-byte read of the swizzled box) and, for its token, the 32
// matching x.  The k order inside an MMA is free as long as A and B agree, so each 8-code
// word feeds two MMAs in the order the bit tricks produce: with (c0 .. c7) the codes of
// the word, or-ing the exponent of 128 onto the masked nibbles of the word shifted by 0,
// 4, 8 and 12 bits gives the bf16 pairs (128 + c0, 128 + c4), (128 + c1, 128 + c5),
// (128 + c2, 128 + c6) and (128 + c3, 128 + c7); one packed subtract leaves (c - 8) exactly.
// MMA 1 takes the pairs (c0, c4), (c1, c5) and x pairs (x0, x4), (x1, x5); MMA 2 the rest.
// Two shared-memory bank conflicts are taken out by choices the MMA does not see: MMA row
// g reads stage row ((g & 1) << 2 | g >> 1) (a row permutation undone at the output), and
// thread t walks its 4 words in the order pp ^ (t & 2).
// The 8 MMAs of a scale group accumulate from zero; the group sum is then scaled per row
// and added to the thread's float32 accumulators.  Products are exact ((c - 8) times a
// bf16 value); only the float32 accumulation rounds.
//
// Codes past K are zero-filled, and so are the scales of groups past K and x: nothing
// past K contributes.  Every wait is bounded; an expired wait raises the CTA's abort
// flag, and every consumer warp still meets the others at the item-end barriers before
// all leave together.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>

#include "epilogue.cuh"
#include "launch.h"
#include "ptx.cuh"

namespace nnjit {

namespace {

constexpr int kKc = 1024;             // codes per stage and row
constexpr int kQuarter = 256;         // codes per box (one consumer warp's K share)
constexpr int kGroupsPerStage = kKc / 128;
constexpr int kThreads = 160;         // producer warp + 4 consumer warps
constexpr int kMaxStages = 8;
constexpr long long kPrefetchBytes = 48ll << 20;
constexpr int kErrEmpty = 0x211;
constexpr int kErrFull = 0x212;
constexpr int kErrDrain = 0x213;

struct GemvW4Params {
    CUtensorMap tmap_w;  // codes as 32-bit words: dims {ceil(K/8), N}, box {32, ROWS}, 128B swizzle
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

__device__ __forceinline__ uint32_t lop_or(uint32_t a, uint32_t mask, uint32_t bits) {
    return (a & mask) | bits;
}
// bf16x2 a - b
__device__ __forceinline__ uint32_t sub_bf2(uint32_t a, uint32_t b) {
    uint32_t r;
    asm("sub.rn.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
    return r;
}
__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t r;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(r) : "r"(a), "r"(b), "r"(sel));
    return r;
}

// The 8 codes of word q as four bf16 pairs (c - 8): P[0] = (c0, c4), P[1] = (c1, c5),
// P[2] = (c2, c6), P[3] = (c3, c7) (low half first).  A nibble or-ed into the low mantissa
// bits of bf16 128 (exponent 134, mantissa unit 1) reads 128 + c; bf16 has 7 mantissa
// bits, so each nibble is first shifted down to bits 0-3 (at bits 4-7 it would reach the
// exponent).
__device__ __forceinline__ void dequant8(uint32_t q, uint32_t (&P)[4]) {
    constexpr uint32_t kE128 = 0x43004300u;  // bf16 (128, 128)
    constexpr uint32_t k136 = 0x43084308u;   // bf16 (136, 136)
    P[0] = sub_bf2(lop_or(q, 0x000F000Fu, kE128), k136);
    P[1] = sub_bf2(lop_or(q >> 4, 0x000F000Fu, kE128), k136);
    P[2] = sub_bf2(lop_or(q >> 8, 0x000F000Fu, kE128), k136);
    P[3] = sub_bf2(lop_or(q >> 12, 0x000F000Fu, kE128), k136);
}

__device__ __forceinline__ void mma_bf16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
    asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
        "{%8, %9}, {%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Named barrier 1 over the 4 consumer warps; the second form also returns whether any of
// their threads passed v = true (the same answer in all of them).
__device__ __forceinline__ void consumers_sync() {
    asm volatile("bar.sync 1, 128;" ::: "memory");
}
__device__ __forceinline__ bool consumers_sync_any(bool v) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "barrier.cta.red.or.pred q, 1, 128, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"((uint32_t)v)
        : "memory");
    return r != 0;
}

template <int ROWS>
__global__ void __launch_bounds__(kThreads, 1) gemv_w4_kernel(const __grid_constant__ GemvW4Params p) {
    constexpr int kTiles = ROWS / 16;                 // 16-row MMA tiles per stage
    constexpr uint32_t kBoxBytes = ROWS * 128;        // one 256-code quarter of ROWS rows
    constexpr uint32_t kWBytes = 4 * kBoxBytes;
    constexpr uint32_t kSBytes = ROWS * kGroupsPerStage * 2;
    static_assert(ROWS == 16 || ROWS == 32, "rows per stage");
    extern __shared__ uint8_t gsm_raw[];
    __shared__ __align__(8) uint64_t bars[2 * kMaxStages];
    __shared__ int abort_word;
    __shared__ float red[4][ROWS][8];                 // per-warp partial sums of an item
    volatile int* abort_flag = &abort_word;

    const int S = p.stages, M = p.M;
    const uint32_t xbytes = (uint32_t)M * kKc * 2;
    const uint32_t stride = (kWBytes + xbytes + kSBytes + 1023u) & ~1023u;
    const uint32_t base = (ptx::smem_u32(gsm_raw) + 1023u) & ~1023u;
    const uint8_t* gbase = gsm_raw + (base - ptx::smem_u32(gsm_raw));
    auto w_at = [&](int s) { return base + (uint32_t)s * stride; };
    auto x_at = [&](int s) { return w_at(s) + kWBytes; };
    auto s_at = [&](int s) { return w_at(s) + kWBytes + xbytes; };
    auto full_bar = [&](int s) { return ptx::smem_u32(bars + s); };
    auto empty_bar = [&](int s) { return ptx::smem_u32(bars + kMaxStages + s); };
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t tx_bytes = kWBytes + kSBytes + xbytes;

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
#pragma unroll
                for (int b = 0; b < 4; ++b)
                    ptx::tma_load_2d_hint(w_at(st) + b * kBoxBytes, &p.tmap_w, c * (kKc / 8) + b * (kQuarter / 8),
                                          g * ROWS, full_bar(st), pol);
                ptx::tma_load_2d_hint(s_at(st), &p.tmap_s, g * ROWS, c * kGroupsPerStage, full_bar(st), pol);
            };
            auto load_x = [&](int st, int c) {
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    ptx::tma_load_2d(x_at(st) + j * M * kQuarter * 2, &p.tmap_x, c * kKc + j * kQuarter, 0,
                                     full_bar(st));
            };
            int stage = 0;
            uint32_t phase = 0;
            uint32_t armed = 0, armed_parity = 0;
            int pre = 0;
            int pre_chunk[kMaxStages];
            if (p.b_const && (int)blockIdx.x < p.items) {
                const Item first = item_of(blockIdx.x, p);
                for (int c = first.c0; c < first.c1 && pre < S; ++c, ++pre) {
                    ptx::mbar_arrive_expect_tx(full_bar(pre), tx_bytes);
                    load_w(pre, c, first.g);
                    pre_chunk[pre] = c;
                }
                const int pf_end = min(first.c1, first.c0 + pre + p.pf_chunks);
                for (int c = first.c0 + pre; c < pf_end; ++c)
#pragma unroll
                    for (int b = 0; b < 4; ++b)
                        ptx::tma_prefetch_l2_2d(&p.tmap_w, c * (kKc / 8) + b * (kQuarter / 8), first.g * ROWS);
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
                    ptx::mbar_arrive_expect_tx(full_bar(stage), tx_bytes);
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
    const int cw = warp - 1;          // K quarter of every stage
    const int g = lane >> 2, t = lane & 3;
    const bool tok = g < M;           // this lane's B column is a real row of x
    // MMA row g of a tile is stage row sg (and g + 8 is sg + 8): g = 2i and 2i + 1 land
    // in different halves of the 128-byte swizzle, so the 8 lanes of a 16-byte load phase
    // read 8 distinct bank quads.
    const int sg = ((g & 1) << 2) | (g >> 1);
    // Thread t takes the 4 words of its 16-byte unit in the order pp ^ rot: the x reads of
    // t and t + 2 (64 bytes apart) then hit different bank quads.
    const int rot = t & 2;
    int stage = 0;
    uint32_t phase = 0;
    for (int it = blockIdx.x; it < p.items; it += gridDim.x) {
        const Item w = item_of(it, p);
        float acc[kTiles][4];
#pragma unroll
        for (int r = 0; r < kTiles; ++r)
#pragma unroll
            for (int j = 0; j < 4; ++j) acc[r][j] = 0.0f;
        for (int c = w.c0; c < w.c1; ++c) {
            // one answer for the whole warp: mma.sync needs all 32 lanes
            const bool ready = ptx::mbar_wait(full_bar(stage), phase, abort_flag, p.err, kErrFull);
            if (!__all_sync(0xffffffffu, ready)) break;
            const uint8_t* wst = gbase + (w_at(stage) - base);
            const uint8_t* box = wst + cw * kBoxBytes;
            const uint8_t* xq = wst + kWBytes + (cw * M + (tok ? g : 0)) * kQuarter * 2;
            const uint16_t* sc = reinterpret_cast<const uint16_t*>(wst + kWBytes + xbytes);
#pragma unroll
            for (int h = 0; h < 2; ++h) {  // scale group 2 cw + h of the stage
                // x[g][128h + 32t + 8(pp ^ rot) .. +7], as the B pairs of MMA 1 and 2
                uint32_t B[4][4];
#pragma unroll
                for (int pp = 0; pp < 4; ++pp) {
                    uint4 v = make_uint4(0, 0, 0, 0);
                    if (tok) v = *reinterpret_cast<const uint4*>(xq + (128 * h + 32 * t + 8 * (pp ^ rot)) * 2);
                    B[pp][0] = prmt(v.x, v.z, 0x5410u);  // (x0, x4)
                    B[pp][1] = prmt(v.x, v.z, 0x7632u);  // (x1, x5)
                    B[pp][2] = prmt(v.y, v.w, 0x5410u);  // (x2, x6)
                    B[pp][3] = prmt(v.y, v.w, 0x7632u);  // (x3, x7)
                }
                const int grp = 2 * cw + h;
                // 16-byte unit 4h + t of a row, at (4h + t) ^ (row % 8) under the swizzle
                const uint32_t u = (uint32_t)(4 * h + t) ^ (uint32_t)sg;
#pragma unroll
                for (int r = 0; r < kTiles; ++r) {
                    const int r0 = 16 * r + sg, r1 = r0 + 8;
                    uint4 q0 = *reinterpret_cast<const uint4*>(box + r0 * 128 + u * 16);
                    uint4 q1 = *reinterpret_cast<const uint4*>(box + r1 * 128 + u * 16);
                    if (rot) {
                        q0 = make_uint4(q0.z, q0.w, q0.x, q0.y);
                        q1 = make_uint4(q1.z, q1.w, q1.x, q1.y);
                    }
                    const uint32_t w0[4] = {q0.x, q0.y, q0.z, q0.w}, w1[4] = {q1.x, q1.y, q1.z, q1.w};
                    // two accumulation chains (codes (c0, c4, c1, c5) and (c2, c6, c3, c7))
                    float d[4] = {0.0f, 0.0f, 0.0f, 0.0f}, e[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
                    for (int pp = 0; pp < 4; ++pp) {
                        uint32_t P0[4], P1[4];
                        dequant8(w0[pp], P0);
                        dequant8(w1[pp], P1);
                        mma_bf16(d, P0[0], P1[0], P0[1], P1[1], B[pp][0], B[pp][1]);
                        mma_bf16(e, P0[2], P1[2], P0[3], P1[3], B[pp][2], B[pp][3]);
                    }
                    const float s0 = __uint_as_float((uint32_t)sc[grp * ROWS + r0] << 16);
                    const float s1 = __uint_as_float((uint32_t)sc[grp * ROWS + r1] << 16);
                    acc[r][0] = fmaf(s0, d[0] + e[0], acc[r][0]);
                    acc[r][1] = fmaf(s0, d[1] + e[1], acc[r][1]);
                    acc[r][2] = fmaf(s1, d[2] + e[2], acc[r][2]);
                    acc[r][3] = fmaf(s1, d[3] + e[3], acc[r][3]);
                }
            }
            ptx::mbar_arrive_elect(empty_bar(stage));  // after every lane's reads of the stage
            if (++stage == S) {
                stage = 0;
                phase ^= 1u;
            }
        }
        // the four K quarters meet: D element (row, token 2t + j) of tile r
#pragma unroll
        for (int r = 0; r < kTiles; ++r) {
            red[cw][16 * r + sg][2 * t] = acc[r][0];
            red[cw][16 * r + sg][2 * t + 1] = acc[r][1];
            red[cw][16 * r + sg + 8][2 * t] = acc[r][2];
            red[cw][16 * r + sg + 8][2 * t + 1] = acc[r][3];
        }
        // one vote for all four warps, so that they leave the item loop together
        const bool aborted = consumers_sync_any(*abort_flag != 0);
        if (!aborted) {
            for (int o = threadIdx.x - 32; o < ROWS * M; o += 128) {
                const int row = o / M, m = o % M;
                const int n = w.g * ROWS + row;
                if (n >= p.N) continue;
                const float v = ((red[0][row][m] + red[1][row][m]) + red[2][row][m]) + red[3][row][m];
                if (p.split == 1)
                    p.C[(long long)m * p.ldc + n] = epi_out(p.bias ? v + p.bias[n] : v, p.act, p.C + (long long)m * p.ldc + n);
                else
                    p.ws[((long long)w.s * M + m) * p.N + n] = v;
            }
        }
        consumers_sync();
        if (aborted) break;
    }
}

using GemvW4Kernel = void (*)(GemvW4Params);
// Instance table, indexed as gemv_w4_instance() - kGemvW4FirstInstance: ROWS 16, 32.
const GemvW4Kernel kKernels[2] = {gemv_w4_kernel<16>, gemv_w4_kernel<32>};
const int kRowsOf[2] = {16, 32};


}  // namespace

bool gemv_uses_w4(const nnjit_candidate& c) {
    return c.family == NNJIT_FAMILY_GEMV && c.instance >= kGemvW4FirstInstance &&
           c.instance < kGemvW4FirstInstance + 2;
}

cudaError_t encode_gemv_w4_maps(const Problem& p, const nnjit_candidate& c, const void* A, const void* B,
                                CUtensorMap* tx, CUtensorMap* tw, CUtensorMap* ts, const char** why) {
    EncodeTiledFn enc = get_encode_fn();
    if (!enc) {
        *why = "cuTensorMapEncodeTiled entry point unavailable";
        return cudaErrorNotSupported;
    }
    const int i = c.instance - kGemvW4FirstInstance;
    if (i < 0 || i >= 2 || p.M < 1 || p.M > 8) {
        *why = "not a 4-bit GEMV candidate";
        return cudaErrorInvalidValue;
    }
    const cuuint32_t estr[2] = {1, 1};
    const char* blob = static_cast<const char*>(B);
    {
        const cuuint64_t dims[2] = {(cuuint64_t)((p.K + 7) / 8), (cuuint64_t)p.N};
        const cuuint64_t strides[1] = {(cuuint64_t)(p.ldb / 2)};
        const cuuint32_t box[2] = {(cuuint32_t)(kQuarter / 8), (cuuint32_t)kRowsOf[i]};
        if (enc(tw, CU_TENSOR_MAP_DATA_TYPE_UINT32, 2, const_cast<char*>(blob), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
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
        const cuuint32_t box[2] = {(cuuint32_t)kQuarter, (cuuint32_t)p.M};
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
    if (i < 0 || i >= 2 || !a.tmap_a || !a.tmap_b || !a.tmap_c || p.dtype != NNJIT_W4_BF16 ||
        p.b_layout != NNJIT_B_NK)
        return cudaErrorInvalidValue;
    if (p.M < 1 || p.M > 8 || c.bn != kRowsOf[i] || c.stages < 2 || c.stages > kMaxStages || c.split_k < 1 ||
        c.threads != kThreads || c.bk != kKc)
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
        const long long per_cta = kPrefetchBytes / grid / ((long long)kRowsOf[i] * (kKc / 2));
        prm.pf_chunks = (int)std::min<long long>(per_cta, prm.cps);
    }
    const int stride = (kRowsOf[i] * (kKc / 2) + (int)p.M * kKc * 2 + kRowsOf[i] * kGroupsPerStage * 2 + 1023) / 1024 * 1024;
    const int smem = 1024 + c.stages * stride;
    cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void*>(kKernels[i]), smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(kKernels[i], dim3(grid), dim3(kThreads), smem, a.stream, prm);
}

}  // namespace nnjit
