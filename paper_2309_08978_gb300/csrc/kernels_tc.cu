// Tensor-core GEMM for sm_103a: TMA -> shared-memory ring -> tcgen05.mma (cta_group::1,
// M = 128) -> TMEM f32 accumulators -> tcgen05.ld epilogue (+ bias) -> f32 global stores.
//
// This is the tensor-core member of the kernel family the JIT tunes (the MatMul and
// BatchMatMul operators of Table 3).  One CTA per SM runs persistently over output tiles
// of BM x BN = 128 x BN; per tile it streams K in blocks of 128 bytes (64 bf16 / 32 tf32
// elements), so every shared-memory row is one 128-byte swizzle row.
//
// Warp roles (192 threads):
//   warp 0      TMA producer: waits "empty[s]", arms "full[s]" with the stage bytes and
//               issues the A and B tile loads.
//   warp 1      TMEM owner and MMA issuer (the whole warp waits and stays converged;
//               one lane elected by elect.sync issues): waits "full[s]", issues BK/UMMA_K MMAs into
//               accumulator buffer (tile & 1), commits to "empty[s]"; after the last
//               k-block commits to "tmem_full[acc]".
//   warps 2..5  epilogue: wait "tmem_full[acc]", tcgen05.ld 32 columns at a time, add
//               bias, store f32; then arrive on "tmem_empty[acc]" (128 arrivals).
// Two accumulator buffers let the epilogue of one tile overlap the mainloop of the next.
// Every wait is bounded (ptx::mbar_wait); an expired wait records an error code in the
// plan's watchdog word, all roles leave their loops, in-flight copies and MMAs are
// drained (bounded), TMEM is freed and the CTA exits.
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

constexpr int kThreads = 192;
constexpr int kMaxStages = 8;
constexpr int kEpiStageBytes = 4 * 2 * 4096;  // 4 epilogue warps x 2 buffers x (32 x 32 f32)

struct TcParams {
    CUtensorMap tmap_a;  // A [batch][M][K]: dims {K, M, batch}, box {BK, 128, 1}
    CUtensorMap tmap_b;  // NK: dims {K, N, batch}, box {BK, BN, 1}; KN: dims {N, K, batch}, box {atom, BK, 1}
    CUtensorMap tmap_c;  // output (C, or the split-K partials): dims {N, M, z}, box {32, 32, 1}
    int tma_store;       // 1: epilogue stores through tmap_c; 0: direct global stores
    int b_const;         // B is not written by kernels launched earlier in the stream
    float* C;
    const float* bias;
    float* ws;
    int* err;
    int M, N, K, batch;
    long long ldc, stride_c;
    int num_kb, split, tiles_m, tiles_n, total_tiles, stages, raster;
    int act;             // nnjit_epilogue, applied where C is written (not to partials)
};

struct TileCoord {
    int b, s, tm, tn;
};

// Kernel modes: persistent CTAs (slices of a tile are separate work items) and cluster
// split-K (the split_k consecutive CTAs of a cluster share one output tile, CTA rank =
// K slice).
constexpr int kModePersistent = 0;
constexpr int kModeClusterSplitK = 1;

// Work item t -> (batch, K slice, tile row, tile column).
template <int kMode>
__device__ __forceinline__ TileCoord decode_tile(int t, const TcParams& p) {
    TileCoord c;
    const int rows = p.tiles_m;
    const int per = rows * p.tiles_n;
    int r, q;
    if constexpr (kMode == kModeClusterSplitK) {
        c.s = t % p.split;
        const int ot = t / p.split;
        r = ot % per;
        c.b = ot / per;
    } else {
        r = t % per;
        q = t / per;
        c.s = q % p.split;
        c.b = q / p.split;
    }
    if (p.raster == 0) {
        c.tm = r % rows;
        c.tn = r / rows;
    } else {
        c.tn = r % p.tiles_n;
        c.tm = r / p.tiles_n;
    }
    return c;
}

// Error codes written to the watchdog word: 0x100 | role << 4 | which wait.
constexpr int kErrProducerEmpty = 0x101;
constexpr int kErrMmaTmemEmpty = 0x111;
constexpr int kErrMmaFull = 0x112;
constexpr int kErrEpiTmemFull = 0x121;
constexpr int kErrDrain = 0x131;

// KG: k-blocks per ring slot.  Each slot is guarded by one pair of barriers, so the MMA
// issuer pays one barrier wait and one commit per KG k-blocks (4 * KG instructions);
// with N <= 128 the issue path, not the tensor pipe, sets the pace, and KG = 2 shortens it.
template <int kKind, bool kBMn, int BN, int kMode, int BM, int KG>
__global__ void __launch_bounds__(kThreads, 1) tc_gemm_kernel(const __grid_constant__ TcParams p) {
    constexpr bool kCluster = kMode == kModeClusterSplitK;
    static_assert(BM == 128 || (BM == 64 && kMode == kModePersistent), "BM 64 tiles run persistent only");
    static_assert(KG == 1 || (KG == 2 && kMode == kModePersistent && BN <= 128),
                  "k-block groups: persistent tiles with BN <= 128");
    // Rows of the accumulator per epilogue warp.  An M = 128 MMA puts row r in TMEM lane
    // r; an M = 64 MMA puts rows 16q .. 16q+15 in lanes 32q .. 32q+15 of sub-partition q.
    constexpr int kRowsPerWarp = BM / 4;
    constexpr int kElem = kKind == 0 ? 2 : 4;
    constexpr int BK = 128 / kElem;                     // K elements per stage (one swizzle row)
    constexpr int kUmmaK = 32 / kElem;                  // K per MMA instruction (32 bytes)
    constexpr int kKSteps = BK / kUmmaK;                // 4
    constexpr int kAtom = 128 / kElem;                  // MN-major swizzle atom width (elements)
    constexpr uint32_t kABytes = BM * 128;              // 16 KB (BM 128) or 8 KB
    constexpr uint32_t kBBytes = BN * 128;
    constexpr uint32_t kStageBytes = kABytes + kBBytes;  // one k-block
    constexpr uint32_t kGroupBytes = KG * kStageBytes;   // one ring slot
    constexpr uint32_t kTmemCols = 2 * BN < 32 ? 32 : 2 * BN;
    constexpr uint32_t kIdesc = ptx::instr_desc(kKind == 0 ? 1u : 2u, kBMn, BM, BN);
    // MN-major 32-bit (tf32) operands use the 32-byte-atom variant of the 128-byte swizzle
    // (the TMA load writes the matching CU_TENSOR_MAP_SWIZZLE_128B_ATOM_32B pattern).
    constexpr uint32_t kBLayout = (kKind == 1 && kBMn) ? ptx::kLayoutSw128Atom32 : ptx::kLayoutSw128;
    // In that layout the MMA walks K in groups of 4 rows of 128 bytes, so consecutive
    // K groups sit 512 bytes apart (8-row groups, 1024 bytes, for the other layouts).
    constexpr uint32_t kBSbo = (kKind == 1 && kBMn) ? 512u : 1024u;

    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~static_cast<uintptr_t>(1023));
    const int S = p.stages;
    uint8_t* epi_smem = smem + (size_t)S * kGroupBytes;  // 1024-aligned (stage bytes are)
    uint64_t* bars = reinterpret_cast<uint64_t*>(epi_smem + kEpiStageBytes);
    // bars[0..S): full, [S..2S): empty, 2S..2S+1: tmem_full, 2S+2..2S+3: tmem_empty,
    // 2S+4: drain
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * kMaxStages + 5);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t smem_base = ptx::smem_u32(smem);
    auto full_bar = [&](int s) { return ptx::smem_u32(bars + s); };
    auto empty_bar = [&](int s) { return ptx::smem_u32(bars + S + s); };
    auto tfull_bar = [&](int a) { return ptx::smem_u32(bars + 2 * S + a); };
    auto tempty_bar = [&](int a) { return ptx::smem_u32(bars + 2 * S + 2 + a); };
    const uint32_t drain_bar = ptx::smem_u32(bars + 2 * S + 4);
    // k-blocks [kb0, kb1) of a work item
    auto kb_range = [&](const TileCoord& tc, int& kb0, int& kb1) {
        kb0 = (int)((long long)tc.s * p.num_kb / p.split);
        kb1 = (int)((long long)(tc.s + 1) * p.num_kb / p.split);
    };
    const int t_begin = (int)blockIdx.x;
    const int t_step = (int)gridDim.x;
    // B tile of k-block kb into the ring slot at `sb`.
    auto load_b = [&](uint32_t sb, const TileCoord& tc, int kb, uint32_t bar) {
        if constexpr (!kBMn) {
            ptx::tma_load_3d(sb, &p.tmap_b, kb * BK, tc.tn * BN, tc.b, bar);
        } else {
            constexpr int kBoxes = BN / kAtom;
#pragma unroll
            for (int j = 0; j < kBoxes; ++j)
                ptx::tma_load_3d(sb + j * (BK * 128), &p.tmap_b, tc.tn * BN + j * kAtom, kb * BK, tc.b, bar);
        }
    };

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            ptx::mbar_init(full_bar(s), 1);
            ptx::mbar_init(empty_bar(s), 1);
        }
        for (int a = 0; a < 2; ++a) {
            ptx::mbar_init(tfull_bar(a), 1);
            ptx::mbar_init(tempty_bar(a), 4 * 32);
        }
        ptx::mbar_init(drain_bar, 1);
        *abort_flag = 0;
        ptx::fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        ptx::prefetch_tmap(&p.tmap_a);
        ptx::prefetch_tmap(&p.tmap_b);
        if (p.tma_store) ptx::prefetch_tmap(&p.tmap_c);
        // Warm L2 with the first ring's worth of this CTA's operand tiles while the
        // previous kernel may still be running: an L2 prefetch writes nothing, and L2 is
        // where the previous kernel's stores land, so no stale copy can result.
        if (t_begin < p.total_tiles) {
            const TileCoord tc = decode_tile<kMode>(t_begin, p);
            int kb0, kb1;
            kb_range(tc, kb0, kb1);
            for (int kb = kb0; kb < kb1 && kb < kb0 + S * KG; ++kb) {
                ptx::tma_prefetch_l2_3d(&p.tmap_a, kb * BK, tc.tm * BM, tc.b);
                if constexpr (!kBMn) {
                    ptx::tma_prefetch_l2_3d(&p.tmap_b, kb * BK, tc.tn * BN, tc.b);
                } else {
                    for (int j = 0; j < BN / kAtom; ++j)
                        ptx::tma_prefetch_l2_3d(&p.tmap_b, tc.tn * BN + j * kAtom, kb * BK, tc.b);
                }
            }
        }
    }
    if (warp == 1) {
        ptx::tmem_alloc(ptx::smem_u32(tmem_slot), kTmemCols);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    // With a constant B the producer arms the first ring and starts its B tiles before
    // the dependency wait (the ring is empty, so no "empty" wait is needed); the loop
    // below then only adds the A tiles of those stages.
    int b_preloaded = 0;  // ring slots whose B tiles are already requested
    if (p.b_const && warp == 0 && t_begin < p.total_tiles) {
        const TileCoord tc = decode_tile<kMode>(t_begin, p);
        int kb0, kb1;
        kb_range(tc, kb0, kb1);
        b_preloaded = min(S, (kb1 - kb0 + KG - 1) / KG);
        if (lane == 0) {
            for (int i = 0; i < b_preloaded; ++i) {
                const int g0 = kb0 + i * KG;
                const int nk = min(KG, kb1 - g0);
                ptx::mbar_arrive_expect_tx(full_bar(i), nk * kStageBytes);
                for (int j = 0; j < nk; ++j)
                    load_b(smem_base + i * kGroupBytes + j * kStageBytes + kABytes, tc, g0 + j, full_bar(i));
            }
        }
        __syncwarp();
    }
    // Global memory that earlier kernels may write is touched only from here.
    ptx::griddep_wait();
    if (threadIdx.x == 0) ptx::griddep_launch_dependents();

    if (warp == 0) {
        // ---------------------------------------------------------------- TMA producer
        int stage = 0;
        uint32_t phase = 0;
        uint32_t armed = 0, armed_parity = 0;
        bool ok = true;
        int issued = 0;  // ring slots filled so far by this CTA
        for (int t = t_begin; ok && t < p.total_tiles; t += t_step) {
            const TileCoord tc = decode_tile<kMode>(t, p);
            int kb0, kb1;
            kb_range(tc, kb0, kb1);
            for (int g0 = kb0; g0 < kb1; g0 += KG) {
                const int nk = min(KG, kb1 - g0);
                if (!ptx::mbar_wait(empty_bar(stage), phase ^ 1u, abort_flag, p.err,
                                    kErrProducerEmpty)) {
                    ok = false;
                    break;
                }
                const bool pre = issued < b_preloaded;  // B of this slot already on its way
                ++issued;
                if (lane == 0) {
                    if (!pre) ptx::mbar_arrive_expect_tx(full_bar(stage), nk * kStageBytes);
                    for (int j = 0; j < nk; ++j) {
                        const uint32_t sa = smem_base + stage * kGroupBytes + j * kStageBytes;
                        ptx::tma_load_3d(sa, &p.tmap_a, (g0 + j) * BK, tc.tm * BM, tc.b, full_bar(stage));
                        if (!pre) load_b(sa + kABytes, tc, g0 + j, full_bar(stage));
                    }
                }
                __syncwarp();
                armed |= 1u << stage;
                armed_parity = (armed_parity & ~(1u << stage)) | (phase << stage);
                if (++stage == S) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
        }
        // Drain: every load this warp issued has landed before the CTA may exit.
        for (int s = 0; s < S; ++s) {
            if (armed & (1u << s)) {
                volatile int no_abort = 0;
                ptx::mbar_wait(full_bar(s), (armed_parity >> s) & 1u, &no_abort, p.err, kErrDrain,
                               ptx::kWaitLimitNs / 4);
            }
        }
    } else if (warp == 1) {
        // ---------------------------------------------------------------- MMA issuer
        int stage = 0;
        uint32_t phase = 0;
        uint32_t iter = 0;
        bool ok = true;
        // Descriptors of ring slot 0; a slot's are these plus its byte offset >> 4 (the
        // start-address field holds shared addresses >> 4, below 2^14, so no carry).
        const uint64_t a_desc0 = ptx::smem_desc(smem_base, 16, 1024);
        const uint64_t b_desc0 = kBMn ? ptx::smem_desc(smem_base + kABytes, BK * 128, kBSbo, kBLayout)
                                      : ptx::smem_desc(smem_base + kABytes, 16, 1024);
        constexpr uint32_t kBStep = kBMn ? (kUmmaK * 128) >> 4 : 32 >> 4;  // per MMA along K
        for (int t = t_begin; ok && t < p.total_tiles; t += t_step, ++iter) {
            const TileCoord tc = decode_tile<kMode>(t, p);
            int kb0, kb1;
            kb_range(tc, kb0, kb1);
            const uint32_t acc = iter & 1u;
            const uint32_t acc_phase = (iter >> 1) & 1u;
            // every lane waits; the warp leaves together if any lane's wait expired
            if (!__all_sync(0xffffffffu,
                            ptx::mbar_wait(tempty_bar(acc), acc_phase ^ 1u, abort_flag, p.err, kErrMmaTmemEmpty))) {
                ok = false;
                break;
            }
            ptx::tc_fence_after();
            const uint32_t d_tmem = tmem_base + acc * BN;
            for (int g0 = kb0; g0 < kb1; g0 += KG) {
                const int nk = min(KG, kb1 - g0);
                if (!__all_sync(0xffffffffu, ptx::mbar_wait(full_bar(stage), phase, abort_flag, p.err, kErrMmaFull))) {
                    ok = false;
                    break;
                }
                ptx::tc_fence_after();
                // the whole warp issues (one elected lane), so it stays converged
#pragma unroll
                for (int j = 0; j < KG; ++j) {
                    if (j < nk) {
                        const uint64_t off = (uint64_t)((stage * kGroupBytes + j * kStageBytes) >> 4);
                        const uint64_t ad = a_desc0 + off, bd = b_desc0 + off;
#pragma unroll
                        for (int kk = 0; kk < kKSteps; ++kk)
                            ptx::mma_ss_elect<kKind>(d_tmem, ad + 2 * kk, bd + kBStep * kk, kIdesc,
                                                     (g0 > kb0 || j > 0 || kk > 0) ? 1u : 0u);
                    }
                }
                ptx::tc_commit_elect(empty_bar(stage));
                if (++stage == S) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (!ok) break;
            ptx::tc_commit_elect(tfull_bar(acc));
        }
        // Drain: all MMAs the warp issued have completed before TMEM is released.
        __syncwarp();
        ptx::tc_commit_elect(drain_bar);
        volatile int no_abort = 0;
        ptx::mbar_wait(drain_bar, 0, &no_abort, p.err, kErrDrain, ptx::kWaitLimitNs / 4);
    } else {
        // ---------------------------------------------------------------- epilogue
        // Warp (2 + e) owns TMEM sub-partition q = warp % 4, i.e. tile rows 32q .. 32q+31;
        // thread `lane` holds one row.  Each 32 x 32 chunk goes either through a 128B-
        // swizzled shared-memory buffer and a TMA store (coalesced, bounds-clipped), or,
        // when the output's strides do not allow TMA, straight to global memory.
        const int q = warp & 3;
        const int row_in_tile = q * kRowsPerWarp + lane;   // valid for lane < kRowsPerWarp
        const bool row_lane = lane < kRowsPerWarp;
        uint8_t* stage_buf = epi_smem + (warp - 2) * 8192;
        uint32_t chunk_ctr = 0;
        uint32_t iter = 0;
        const long long MN = (long long)p.M * p.N;
        for (int t = t_begin; t < p.total_tiles; t += t_step, ++iter) {
            const TileCoord tc = decode_tile<kMode>(t, p);
            const uint32_t acc = iter & 1u;
            const uint32_t acc_phase = (iter >> 1) & 1u;
            if (!ptx::mbar_wait(tfull_bar(acc), acc_phase, abort_flag, p.err, kErrEpiTmemFull)) break;
            ptx::tc_fence_after();
            if constexpr (kCluster) {
                // The partial stays in TMEM until every CTA of the cluster has finished
                // its main loop (see the reduction after the role branches).
                continue;
            }
            const int row = tc.tm * BM + row_in_tile;
            const float* bias = p.split == 1 ? p.bias : nullptr;
            const int act = p.split == 1 ? p.act : NNJIT_EPI_NONE;  // partials stay raw
            float* dst_row = p.split == 1
                                 ? p.C + (long long)tc.b * p.stride_c + (long long)row * p.ldc
                                 : p.ws + ((long long)tc.s * p.batch + tc.b) * MN + (long long)row * p.N;
            const int zc = p.split == 1 ? tc.b : tc.s * p.batch + tc.b;
            const uint32_t tbase = tmem_base + ((uint32_t)(q * 32) << 16) + acc * BN;
            constexpr int kChunks = BN / 32;
            static_assert(kChunks % 2 == 0, "chunks are processed in pairs");
            // The CTA's last tile: its MMAs have completed and no load follows, so the ring
            // is idle and each warp stages every chunk in its own part of it, with no wait
            // for earlier stores (the tail of the launch is bound by stores in flight).
            const bool ring_out = p.tma_store && t + t_step >= p.total_tiles &&
                                  S * (int)kGroupBytes >= 4 * kChunks * 4096;
            // One 32-column chunk: bias (lane j fetched column j; broadcast by shuffles),
            // then the staged TMA store or the direct stores.
            auto emit = [&](const uint32_t (&r)[32], float bl, int c) {
                const int col0 = tc.tn * BN + c * 32;
                float v[32];
#pragma unroll
                for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
                if (bias) {
#pragma unroll
                    for (int j = 0; j < 32; ++j) v[j] += __shfl_sync(0xffffffffu, bl, j);
                }
                if (p.tma_store) {
                    uint8_t* buf = ring_out ? smem + ((warp - 2) * kChunks + c) * 4096
                                            : stage_buf + (chunk_ctr & 1u) * 4096;
                    if (!ring_out && lane == 0) ptx::bulk_wait_read<1>();  // the store that used buf is done
                    __syncwarp();
                    if (row_lane) {
#pragma unroll
                        for (int j = 0; j < 8; ++j)
                            *reinterpret_cast<float4*>(buf + lane * 128 + ((j ^ (lane & 7)) << 4)) =
                                make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
                        if ((act & 15) != NNJIT_EPI_NONE) act_row128(buf + lane * 128, act);
                        if ((act & NNJIT_EPI_RESIDUAL) && row < p.M && col0 < p.N)
                            residual_row128(buf + lane * 128, lane & 7, dst_row + col0, p.N - col0);
                    }
                    ptx::fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) {
                        ptx::tma_store_3d(&p.tmap_c, ptx::smem_u32(buf), col0, tc.tm * BM + q * kRowsPerWarp, zc);
                        ptx::bulk_commit();
                    }
                    if (!ring_out) ++chunk_ctr;
                } else if (row_lane && row < p.M) {
                    float* dst = dst_row + col0;
                    if (act != NNJIT_EPI_NONE) {
                        // stage the row (this thread's own 128 bytes of the idle staging
                        // buffer), then activation and residual element by element
                        if (col0 < p.N) {
                            float* srow = reinterpret_cast<float*>(stage_buf + lane * 128);
#pragma unroll
                            for (int j = 0; j < 32; j += 4)
                                *reinterpret_cast<float4*>(srow + j) = make_float4(v[j], v[j + 1], v[j + 2], v[j + 3]);
                            epi_store_row(srow, act, dst, min(32, p.N - col0));
                        }
                    } else if (col0 + 32 <= p.N && (reinterpret_cast<uintptr_t>(dst) & 15) == 0) {
#pragma unroll
                        for (int j = 0; j < 32; j += 4)
                            *reinterpret_cast<float4*>(dst + j) = make_float4(v[j], v[j + 1], v[j + 2], v[j + 3]);
                    } else {
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            if (col0 + j < p.N) dst[j] = v[j];
                    }
                }
            };
            auto bias_of = [&](int c) {
                const int col = tc.tn * BN + c * 32 + lane;
                return (bias && col < p.N) ? __ldg(bias + col) : 0.0f;
            };
            // The load of chunk c + 1 (TMEM and bias) is in flight while chunk c is stored;
            // TMEM goes back to the MMA warp as soon as its last chunk is in registers.
            auto release = [&]() {
                ptx::tc_fence_before();
                ptx::mbar_arrive(tempty_bar(acc));
            };
            uint32_t ra[32], rb[32];
            ptx::tmem_ld32(tbase, ra);
            float ba = bias_of(0), bb = 0.0f;
            ptx::tmem_wait_ld(ra);
#pragma unroll 1
            for (int c = 0; c < kChunks; c += 2) {
                ptx::tmem_ld32(tbase + (c + 1) * 32, rb);
                bb = bias_of(c + 1);
                emit(ra, ba, c);
                ptx::tmem_wait_ld(rb);
                if (c + 2 == kChunks) release();
                if (c + 2 < kChunks) {
                    ptx::tmem_ld32(tbase + (c + 2) * 32, ra);
                    ba = bias_of(c + 2);
                }
                emit(rb, bb, c + 1);
                if (c + 2 < kChunks) ptx::tmem_wait_ld(ra);
            }
        }
        // the shared-memory sources must outlive the stores; the global writes complete
        // with the kernel
        if (p.tma_store && lane == 0) ptx::bulk_wait_all_read();
        __syncwarp();
    }

    if constexpr (kCluster) {
        // Cluster split-K reduction.  CTA rank r owns rows [r*R, (r+1)*R) of the tile
        // (R = 128 / split).  (1) A cluster barrier: every CTA's main loop is over, so every
        // ring is idle.  (2) Each CTA streams its partial rows from TMEM straight into the
        // owning CTA's ring, slot [its rank][row][BN + 4] (fire-and-forget remote stores).
        // (3) A second barrier publishes them.  (4) Each owner adds its rows over the
        // slices in slice order (deterministic), adds bias, and stores them.  No CTA
        // touches another's shared memory after the second barrier.
        const int R = BM / p.split;
        const uint32_t my_rank = ptx::cluster_ctarank();
        ptx::tc_fence_before();
        ptx::cluster_sync();
        ptx::tc_fence_after();
        if (warp >= 2) {
            const int q = warp & 3;
            const int row = q * 32 + lane;
            const uint32_t owner = (uint32_t)(row / R);
            const uint32_t dst_row = ptx::map_shared_rank(smem_base, owner) +
                                     (uint32_t)(((int)my_rank * R + row % R) * (BN + 4)) * 4u;
#pragma unroll 1
            for (int c = 0; c < BN / 32; ++c) {
                uint32_t r[32];
                ptx::tmem_ld32(tmem_base + ((uint32_t)(q * 32) << 16) + c * 32, r);
                ptx::tmem_wait_ld(r);
#pragma unroll
                for (int j = 0; j < 32; j += 4)
                    ptx::st_shared_cluster_v4(dst_row + (uint32_t)(c * 32 + j) * 4u, __uint_as_float(r[j]),
                                              __uint_as_float(r[j + 1]), __uint_as_float(r[j + 2]),
                                              __uint_as_float(r[j + 3]));
            }
        }
        ptx::cluster_sync();
        const TileCoord tc = decode_tile<kModeClusterSplitK>(blockIdx.x, p);
        constexpr int kVec = BN / 4;
        const float* recv = reinterpret_cast<const float*>(smem);
        float* Cb = p.C + (long long)tc.b * p.stride_c;
        const int row0 = (int)my_rank * R;
        for (int e = threadIdx.x; e < R * kVec; e += kThreads) {
            const int lr = e / kVec;
            const int cv = e % kVec;
            const int row = tc.tm * BM + row0 + lr;
            const int col = tc.tn * BN + cv * 4;
            if (row >= p.M || col >= p.N) continue;
            float4 a = *reinterpret_cast<const float4*>(recv + (size_t)lr * (BN + 4) + cv * 4);
            for (int s = 1; s < p.split; ++s) {
                const float4 v = *reinterpret_cast<const float4*>(recv + (size_t)(s * R + lr) * (BN + 4) + cv * 4);
                a.x += v.x; a.y += v.y; a.z += v.z; a.w += v.w;
            }
            float o[4] = {a.x, a.y, a.z, a.w};
            float* dst = Cb + (long long)row * p.ldc + col;
            if (col + 4 <= p.N && (reinterpret_cast<uintptr_t>(dst) & 15) == 0) {
#pragma unroll
                for (int j = 0; j < 4; ++j) o[j] = epi_out(p.bias ? o[j] + __ldg(p.bias + col + j) : o[j], p.act, dst + j);
                *reinterpret_cast<float4*>(dst) = make_float4(o[0], o[1], o[2], o[3]);
            } else {
                for (int j = 0; j < 4 && col + j < p.N; ++j)
                    dst[j] = epi_out(p.bias ? o[j] + __ldg(p.bias + col + j) : o[j], p.act, dst + j);
            }
        }
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (warp == 1) ptx::tmem_dealloc(tmem_base, kTmemCols);
}

using TcKernel = void (*)(TcParams);

// Instance table, indexed as tc_instance(): variant * 12 + (dtype_i * 2 + kn) * 3 + bn_i
// for variant 0 = 128-row persistent, 1 = 128-row cluster split-K, 2 = 64-row persistent;
// then 36 + (dtype_i * 2 + kn) * 2 + bn_i for 128-row persistent tiles with BN = 64, 128
// and two k-blocks per ring slot.  (With BN = 256 the tensor pipe, not the issue path,
// sets the pace, and halving the number of slots only shortens the lookahead.)
constexpr int kNumTcInstances = 44;
#define NNJIT_TC_ROW(K, MN, MODE, BM)                                                  \
    tc_gemm_kernel<K, MN, 64, MODE, BM, 1>, tc_gemm_kernel<K, MN, 128, MODE, BM, 1>, \
        tc_gemm_kernel<K, MN, 256, MODE, BM, 1>
#define NNJIT_TC_KG2(K, MN) tc_gemm_kernel<K, MN, 64, 0, 128, 2>, tc_gemm_kernel<K, MN, 128, 0, 128, 2>
const TcKernel kTcKernels[kNumTcInstances] = {
    NNJIT_TC_ROW(0, false, 0, 128), NNJIT_TC_ROW(0, true, 0, 128),
    NNJIT_TC_ROW(1, false, 0, 128), NNJIT_TC_ROW(1, true, 0, 128),
    NNJIT_TC_ROW(0, false, 1, 128), NNJIT_TC_ROW(0, true, 1, 128),
    NNJIT_TC_ROW(1, false, 1, 128), NNJIT_TC_ROW(1, true, 1, 128),
    NNJIT_TC_ROW(0, false, 0, 64),  NNJIT_TC_ROW(0, true, 0, 64),
    NNJIT_TC_ROW(1, false, 0, 64),  NNJIT_TC_ROW(1, true, 0, 64),
    NNJIT_TC_KG2(0, false), NNJIT_TC_KG2(0, true), NNJIT_TC_KG2(1, false), NNJIT_TC_KG2(1, true),
};
#undef NNJIT_TC_ROW
#undef NNJIT_TC_KG2

}  // namespace

EncodeTiledFn get_encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPoint("cuTensorMapEncodeTiled", &ptr, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(ptr);
    });
    return fn;
}

cudaError_t prepare_tc_instance(int instance, int smem_bytes) {
    if (instance < 0 || instance >= kNumTcInstances) return cudaErrorInvalidValue;
    return ensure_dynamic_smem(reinterpret_cast<const void*>(kTcKernels[instance]), smem_bytes);
}

cudaError_t encode_tc_tensor_maps(const Problem& p, const nnjit_candidate& c, const void* A,
                                  const void* B, CUtensorMap* ta, CUtensorMap* tb,
                                  const char** why) {
    EncodeTiledFn enc = get_encode_fn();
    if (!enc) {
        *why = "cuTensorMapEncodeTiled entry point unavailable";
        return cudaErrorNotSupported;
    }
    const int e = p.elem_bytes();
    const CUtensorMapDataType dt =
        p.dtype == NNJIT_BF16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32;
    const cuuint32_t bk = 128 / e;
    const cuuint32_t estr[3] = {1, 1, 1};
    {
        const cuuint64_t dims[3] = {(cuuint64_t)p.K, (cuuint64_t)p.M, (cuuint64_t)p.batch};
        const cuuint64_t strides[2] = {(cuuint64_t)(p.lda * e), (cuuint64_t)(p.stride_a * e)};
        // a CTA of a pair tile loads its own 128 rows
        const cuuint32_t box[3] = {bk, (cuuint32_t)std::min(c.bm, 128), 1};
        CUresult r = enc(ta, dt, 3, const_cast<void*>(A), dims, strides, box, estr,
                         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                         CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) {
            *why = "cuTensorMapEncodeTiled failed for A";
            return cudaErrorInvalidValue;
        }
    }
    {
        cuuint64_t dims[3];
        cuuint32_t box[3];
        if (p.b_layout == NNJIT_B_NK) {
            dims[0] = (cuuint64_t)p.K; dims[1] = (cuuint64_t)p.N;
            // each CTA of a pair tile (bm = 256) loads its own half of the B tile
            box[0] = bk; box[1] = (cuuint32_t)(c.bm == 256 ? c.bn / 2 : c.bn);
        } else {
            dims[0] = (cuuint64_t)p.N; dims[1] = (cuuint64_t)p.K;
            box[0] = 128 / e; box[1] = bk;
        }
        dims[2] = (cuuint64_t)p.batch;
        box[2] = 1;
        const cuuint64_t strides[2] = {(cuuint64_t)(p.ldb * e), (cuuint64_t)(p.stride_b * e)};
        const CUtensorMapSwizzle swz = (p.dtype != NNJIT_BF16 && p.b_layout == NNJIT_B_KN)
                                           ? CU_TENSOR_MAP_SWIZZLE_128B_ATOM_32B
                                           : CU_TENSOR_MAP_SWIZZLE_128B;
        CUresult r = enc(tb, dt, 3, const_cast<void*>(B), dims, strides, box, estr,
                         CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
                         CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) {
            *why = "cuTensorMapEncodeTiled failed for B";
            return cudaErrorInvalidValue;
        }
    }
    return cudaSuccess;
}

cudaError_t encode_tc_output_map(const Problem& p, const nnjit_candidate& c, float* out,
                                 bool partials, CUtensorMap* tc_map, bool* ok) {
    *ok = false;
    EncodeTiledFn enc = get_encode_fn();
    if (!enc || !out) return cudaSuccess;
    const long long ld = partials ? p.N : p.ldc;
    const long long zs = partials ? p.M * p.N : p.stride_c;
    const long long nz = partials ? p.batch * c.split_k : p.batch;
    if ((reinterpret_cast<uintptr_t>(out) & 15) || (ld * 4) % 16 || (zs * 4) % 16) return cudaSuccess;
    const cuuint64_t dims[3] = {(cuuint64_t)p.N, (cuuint64_t)p.M, (cuuint64_t)nz};
    const cuuint64_t strides[2] = {(cuuint64_t)(ld * 4), (cuuint64_t)(zs * 4)};
    const cuuint32_t box[3] = {32, (cuuint32_t)(std::min(c.bm, 128) / 4), 1};  // one epilogue warp's rows
    const cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = enc(tc_map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, out, dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    *ok = (r == CUDA_SUCCESS);
    return cudaSuccess;
}

cudaError_t launch_tc(const LaunchArgs& a) {
    const Problem& p = *a.p;
    const nnjit_candidate& c = *a.c;
    if (c.instance >= kTcPairFirstInstance && c.instance < kTcPairFirstInstance + 2) return launch_tc_pair(a);
    if (c.instance < 0 || c.instance >= kNumTcInstances || !a.tmap_a || !a.tmap_b)
        return cudaErrorInvalidValue;
    const bool cluster = c.instance >= 12 && c.instance < 24;
    const int kg = c.instance >= 36 ? 2 : 1;  // k-blocks per ring slot
    const int bk = 128 / p.elem_bytes();      // K elements per k-block
    if ((c.instance >= 24 && c.instance < 36) != (c.bm == 64) || (c.bm != 64 && c.bm != 128))
        return cudaErrorInvalidValue;
    if (c.bk != bk * kg || (kg == 2 && (c.bm != 128 || c.bn > 128 || c.reduce != 0)))
        return cudaErrorInvalidValue;
    if (c.cluster_m != 1) return cudaErrorInvalidValue;
    if (cluster != (c.reduce == 1)) return cudaErrorInvalidValue;
    if (cluster && (c.split_k < 2 || c.split_k > 8 || (c.split_k & (c.split_k - 1)) != 0))
        return cudaErrorInvalidValue;
    if (c.stages < 2 || c.stages > kMaxStages) return cudaErrorInvalidValue;
    TcParams prm;
    prm.tmap_a = *a.tmap_a;
    prm.tmap_b = *a.tmap_b;
    prm.tma_store = a.tmap_c ? 1 : 0;
    prm.b_const = (p.flags & NNJIT_PLAN_B_CONSTANT) ? 1 : 0;
    if (a.tmap_c) prm.tmap_c = *a.tmap_c;
    prm.C = a.C;
    prm.bias = a.bias;
    prm.act = p.epilogue;
    prm.ws = a.ws;
    prm.err = a.err;
    prm.M = (int)p.M;
    prm.N = (int)p.N;
    prm.K = (int)p.K;
    prm.batch = (int)p.batch;
    prm.ldc = p.ldc;
    prm.stride_c = p.stride_c;
    prm.num_kb = (int)((p.K + bk - 1) / bk);
    prm.split = c.split_k;
    prm.tiles_m = (int)((p.M + c.bm - 1) / c.bm);
    prm.tiles_n = (int)((p.N + c.bn - 1) / c.bn);
    // work items: tiles x K slices
    const long long total = (long long)p.batch * c.split_k * prm.tiles_m * prm.tiles_n;
    if (total >= (1LL << 31)) return cudaErrorInvalidValue;
    if (c.split_k > prm.num_kb) return cudaErrorInvalidValue;  // every split owns >= 1 k-block
    prm.total_tiles = (int)total;
    prm.stages = c.stages;
    prm.raster = c.raster;
    // persistent: at most the candidate's grid; cluster mode: one CTA per (tile, slice)
    const int grid = cluster ? (int)total : (int)std::min<long long>(total, c.grid > 0 ? c.grid : total);
    // ring + alignment slack + barriers/TMEM slot/abort flag
    const int stage_bytes = kg * (c.bm + c.bn) * 128;
    const int smem = c.stages * stage_bytes + kEpiStageBytes + 1024 + 256;
    cudaError_t e = prepare_tc_instance(c.instance, smem);
    if (e != cudaSuccess) return e;
    if (!cluster)
        return launch_pdl(kTcKernels[c.instance], dim3(grid), dim3(kThreads), smem, a.stream, prm);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = a.stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = (unsigned)c.split_k;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, kTcKernels[c.instance], prm);
}

}  // namespace nnjit
