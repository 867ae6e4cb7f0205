// Tensor-core GEMM on CTA pairs (tcgen05 .cta_group::2): a cluster of two CTAs on two
// SMs computes one 256 x BN output tile with M = 256 MMAs issued by the even CTA.
//
// Each CTA of the pair loads its own 128 rows of A and its own half (BN / 2 rows of the
// [N][K] operand) of B into the same ring offsets; the tensor cores of both SMs read
// both halves of B, so an SM receives (128 + BN / 2) x 128 bytes per k-block instead of
// (128 + BN) x 128 for a 128 x BN tile of its own: a third less L2 -> SM traffic for the
// same MMA work, and one issuing thread drives two SMs' tensor cores.  B is K-major
// ([N][K], Linear weights); split-K is not used (the pair tiles are for large products).
//
// Roles (192 threads per CTA, as in the single-CTA kernel):
//   warp 0      TMA producer of each CTA.  Loads complete on the EVEN CTA's "full[s]"
//               barrier (whose producer arms it with both CTAs' bytes); a slot is
//               refilled once the MMA has released it in this CTA ("empty[s]").
//   warp 1      TMEM owner in each CTA (the pair allocation is done by one warp of each
//               CTA); in the even CTA also the MMA issuer (the whole warp, converged; one
//               lane elected by elect.sync issues): waits "full[s]", issues 4 MMAs
//               per k-block, commits to "empty[s]" of both CTAs, and per tile to
//               "tmem_full[acc]" of both CTAs.
//   warps 2..5  epilogue of each CTA on its own 128 accumulator rows; each warp releases
//               the accumulator on the even CTA's "tmem_empty[acc]" (8 arrivals).
// Every wait is bounded; on expiry the error word is set and the roles fall through to
// the teardown (the producers wait, bounded, for their ring slots to drain first).
//
// Stream-K over the last waves (candidate reduce = 2).  The pairs are persistent and
// take tiles round-robin, so when the pair tiles are not a whole number of waves of the
// P resident pairs the last wave runs a few tiles while the other pairs idle.  Then only
// the first (waves - 1) * P tiles run whole ("dp" tiles, round-robin); the k-blocks of
// the remaining tiles ("sk" tiles, between 1 and 2 waves' worth) are laid end to end and
// cut into P equal ranges, pair p taking range p after its dp tiles.  A range may start
// inside a tile (its first segment), hold whole tiles, and end inside a tile (its last
// segment).  A segment that starts inside a tile writes its raw sum to the pair's slot
// of the workspace and raises a flag per (CTA, epilogue warp) with release semantics: so
// a pair writes at most one partial.  The segment that starts a tile's k-blocks but does
// not reach their end finishes the tile: it waits (bounded) for the flags of the pairs
// that cover the rest, adds their partials to its own sum in pair order (identical bits
// on every run), applies bias, activation and residual, stores C and lowers the flags
// for the next launch.  A finishing segment is the last of its pair and waits only for
// first segments of later pairs, which never wait, so every wait ends.

#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>

#include "epilogue.cuh"
#include "launch.h"
#include "ptx.cuh"

namespace nnjit {

namespace {

constexpr int kThreads = 192;
constexpr int kMaxStages = 8;
constexpr int kEpiStageBytes = 4 * 2 * 4096;  // 4 epilogue warps x 2 buffers x (32 x 32 f32)

constexpr int kPairAccBuffers = ModelConstants::kTcPairAccCols / 256;
constexpr int kErrProducerEmpty = 0x141;
constexpr int kErrMmaTmemEmpty = 0x142;
constexpr int kErrMmaFull = 0x143;
constexpr int kErrEpiTmemFull = 0x144;
constexpr int kErrDrain = 0x145;
constexpr int kErrSkWait = 0x146;

struct Tc2Params {
    CUtensorMap tmap_a;  // A: dims {K, M, batch}, box {BK, 128, 1}
    CUtensorMap tmap_b;  // B [N][K]: dims {K, N, batch}, box {BK, BN / 2, 1}
    CUtensorMap tmap_c;  // C: dims {N, M, batch}, box {32, 32, 1}
    int tma_store;
    int b_const;
    float* C;
    const float* bias;
    int* err;
    int M, N, K, batch;
    long long ldc, stride_c;
    int num_kb, tiles2_m, tiles_n, total, stages, raster;
    int act;  // nnjit_epilogue
    // stream-K: tiles [0, dp) whole and round-robin; the k-blocks of tiles [dp, total)
    // split evenly over the pairs (dp = total: no stream-K)
    int dp, pairs;
    long long sk_iters;  // (total - dp) * num_kb
    float* part;         // [pairs][2 CTAs][BN / 32 chunks][4 warps][8][32 lanes] float4 partials
    unsigned* flag;      // [pairs][2 CTAs][4 epilogue warps], zero between launches
};

struct PairTile {
    int b, tm2, tn;
};

__device__ __forceinline__ PairTile decode(int t, const Tc2Params& p) {
    PairTile c;
    const int per = p.tiles2_m * p.tiles_n;
    const int r = t % per;
    c.b = t / per;
    if (p.raster == 0) {
        c.tm2 = r % p.tiles2_m;
        c.tn = r / p.tiles2_m;
    } else {
        c.tn = r % p.tiles_n;
        c.tm2 = r / p.tiles_n;
    }
    return c;
}

// One segment of a pair's work: k-blocks [kb0, kb1) of tile `tile`.  role 0: the whole
// tile; 1: a partial sum for another pair to finish (the pair's first stream-K segment,
// starting inside the tile); 2: finish the tile, adding the partials of pairs
// [p_lo, p_hi].
struct Seg {
    int tile, kb0, kb1, role, p_lo, p_hi;
};
struct SegIter {
    int dp_next;
    long long i, end;
};

__device__ __forceinline__ SegIter seg_begin(int pc, const Tc2Params& p) {
    SegIter st;
    st.dp_next = pc;
    st.i = (long long)pc * p.sk_iters / p.pairs;
    st.end = (long long)(pc + 1) * p.sk_iters / p.pairs;
    return st;
}

// The pair whose stream-K range holds k-block iteration i: the largest q with
// floor(q * T / P) <= i (only called with T = sk_iters > 0).
__device__ __forceinline__ int sk_pair_of(long long i, const Tc2Params& p) {
    return (int)(((i + 1) * p.pairs - 1) / p.sk_iters);
}

__device__ __forceinline__ bool seg_next(SegIter& st, Seg& sg, const Tc2Params& p) {
    if (st.dp_next < p.dp) {
        sg.tile = st.dp_next; sg.kb0 = 0; sg.kb1 = p.num_kb; sg.role = 0; sg.p_lo = sg.p_hi = 0;
        st.dp_next += p.pairs;
        return true;
    }
    if (st.i >= st.end) return false;
    const long long t = st.i / p.num_kb;
    sg.tile = p.dp + (int)t;
    sg.kb0 = (int)(st.i - t * p.num_kb);
    sg.kb1 = (int)min((long long)p.num_kb, sg.kb0 + (st.end - st.i));
    sg.p_lo = sg.p_hi = 0;
    if (sg.kb0 > 0) {
        sg.role = 1;
    } else if (sg.kb1 == p.num_kb) {
        sg.role = 0;
    } else {
        sg.role = 2;
        sg.p_lo = sk_pair_of(t * p.num_kb + sg.kb1, p);
        sg.p_hi = sk_pair_of(t * p.num_kb + p.num_kb - 1, p);
    }
    st.i = t * p.num_kb + sg.kb1;
    return true;
}

// NB: accumulator buffers in TMEM (2: the epilogue of one tile overlaps the mainloop of
// the next; 1: half the columns).
template <int kKind, int BN, int NB>
__global__ void __launch_bounds__(kThreads, 1) tc2_gemm_kernel(const __grid_constant__ Tc2Params p) {
    constexpr int kElem = kKind == 0 ? 2 : 4;
    constexpr int BK = 128 / kElem;          // K elements per k-block (one 128-byte row)
    constexpr int kKSteps = 4;               // 32 bytes of K per MMA
    constexpr int kHalfN = BN / 2;           // B rows held by each CTA
    constexpr uint32_t kABytes = 128 * 128;
    constexpr uint32_t kBBytes = kHalfN * 128;
    constexpr uint32_t kStageBytes = kABytes + kBBytes;
    constexpr uint32_t kTmemCols = NB * BN;
    constexpr uint32_t kIdesc = ptx::instr_desc(kKind == 0 ? 1u : 2u, false, 256, BN);
    static_assert(kTmemCols <= 512 && BN % 64 == 0 && (NB == 1 || NB == 2), "pair tile");

    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~static_cast<uintptr_t>(1023));
    const int S = p.stages;
    uint8_t* epi_smem = smem + (size_t)S * kStageBytes;
    uint64_t* bars = reinterpret_cast<uint64_t*>(epi_smem + kEpiStageBytes);
    // bars[0..S): full (used in the even CTA), [S..2S): empty, 2S..2S+1: tmem_full,
    // 2S+2..2S+3: tmem_empty (even CTA), 2S+4: drain (even CTA)
    // bars[2 kMaxStages + 5 + q]: partial-tile copy of epilogue warp q (stream-K finisher)
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * kMaxStages + 9);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t rank = ptx::cluster_ctarank();
    const bool leader = rank == 0;
    const uint32_t smem_base = ptx::smem_u32(smem);
    auto full_bar = [&](int s) { return ptx::smem_u32(bars + s); };
    auto empty_bar = [&](int s) { return ptx::smem_u32(bars + S + s); };
    auto tfull_bar = [&](int a) { return ptx::smem_u32(bars + 2 * S + a); };
    auto tempty_bar = [&](int a) { return ptx::smem_u32(bars + 2 * S + 2 + a); };
    const uint32_t drain_bar = ptx::smem_u32(bars + 2 * S + 4);
    auto pcopy_bar = [&](int q) { return ptx::smem_u32(bars + 2 * kMaxStages + 5 + q); };
    const int t_begin = (int)(blockIdx.x >> 1);

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            ptx::mbar_init(full_bar(s), 1);   // the even CTA's producer arms it
            ptx::mbar_init(empty_bar(s), 1);  // one commit of the pair MMAs
        }
        for (int a = 0; a < 2; ++a) {
            ptx::mbar_init(tfull_bar(a), 1);
            ptx::mbar_init(tempty_bar(a), 8);  // 4 epilogue warps of each CTA
        }
        ptx::mbar_init(drain_bar, 1);
        for (int q = 0; q < 4; ++q) ptx::mbar_init(pcopy_bar(q), 1);
        *abort_flag = 0;
        ptx::fence_barrier_init();
    }
    const int row_off = (int)rank * 128;      // this CTA's rows within the pair tile
    const int bcol_off = (int)rank * kHalfN;  // this CTA's half of the tile's columns
    if (warp == 0 && lane == 0) {
        ptx::prefetch_tmap(&p.tmap_a);
        ptx::prefetch_tmap(&p.tmap_b);
        if (p.tma_store) ptx::prefetch_tmap(&p.tmap_c);
        SegIter st0 = seg_begin(t_begin, p);
        Seg it;
        if (seg_next(st0, it, p)) {
            const PairTile tc = decode(it.tile, p);
            for (int kb = it.kb0; kb < it.kb1 && kb < it.kb0 + S; ++kb) {
                ptx::tma_prefetch_l2_3d(&p.tmap_a, kb * BK, tc.tm2 * 256 + row_off, tc.b);
                ptx::tma_prefetch_l2_3d(&p.tmap_b, kb * BK, tc.tn * BN + bcol_off, tc.b);
            }
        }
    }
    if (warp == 1) {
        ptx::tmem_alloc_pair(ptx::smem_u32(tmem_slot), kTmemCols);
        ptx::tmem_relinquish_pair();
    }
    ptx::tc_fence_before();
    __syncthreads();
    // both CTAs' barriers exist and TMEM is allocated before any cross-CTA signal
    ptx::cluster_sync();
    ptx::tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    auto leader_full = [&](int s) { return ptx::map_shared_rank(full_bar(s), 0); };

    // With a constant B the first ring's B halves are requested before the dependency
    // wait; the even CTA arms those slots with the bytes of both CTAs' A and B.
    int b_preloaded = 0;
    SegIter st_first = seg_begin(t_begin, p);
    Seg first;
    if (p.b_const && warp == 0 && seg_next(st_first, first, p)) {
        const Seg& it = first;
        const PairTile tc = decode(it.tile, p);
        b_preloaded = min(S, it.kb1 - it.kb0);
        if (lane == 0) {
            for (int i = 0; i < b_preloaded; ++i) {
                if (leader) ptx::mbar_arrive_expect_tx(full_bar(i), 2 * kStageBytes);
                ptx::tma_load_3d_pair(smem_base + i * kStageBytes + kABytes, &p.tmap_b, (it.kb0 + i) * BK,
                                      tc.tn * BN + bcol_off, tc.b, leader_full(i));
            }
        }
        __syncwarp();
    }
    ptx::griddep_wait();
    if (threadIdx.x == 0) ptx::griddep_launch_dependents();

    if (warp == 0) {
        // ---------------------------------------------------------------- TMA producer
        int stage = 0;
        uint32_t phase = 0;
        bool ok = true;
        int issued = 0;
        SegIter st = seg_begin(t_begin, p);
        Seg it;
        while (ok && seg_next(st, it, p)) {
            const PairTile tc = decode(it.tile, p);
            for (int kb = it.kb0; kb < it.kb1; ++kb) {
                if (!ptx::mbar_wait(empty_bar(stage), phase ^ 1u, abort_flag, p.err, kErrProducerEmpty)) {
                    ok = false;
                    break;
                }
                const bool pre = issued < b_preloaded;
                ++issued;
                if (lane == 0) {
                    const uint32_t sa = smem_base + stage * kStageBytes;
                    const uint32_t fb = leader_full(stage);
                    if (!pre && leader) ptx::mbar_arrive_expect_tx(full_bar(stage), 2 * kStageBytes);
                    ptx::tma_load_3d_pair(sa, &p.tmap_a, kb * BK, tc.tm2 * 256 + row_off, tc.b, fb);
                    if (!pre) ptx::tma_load_3d_pair(sa + kABytes, &p.tmap_b, kb * BK, tc.tn * BN + bcol_off, tc.b, fb);
                }
                __syncwarp();
                if (++stage == S) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
        }
        // Tail: every slot this CTA filled has been consumed by the pair MMAs (so every
        // copy into this CTA has landed) before the CTA may leave.
        for (int i = 0; i < S; ++i) {
            volatile int no_abort = 0;
            ptx::mbar_wait(empty_bar(stage), phase ^ 1u, &no_abort, p.err, kErrDrain, ptx::kWaitLimitNs / 4);
            if (++stage == S) {
                stage = 0;
                phase ^= 1u;
            }
        }
    } else if (warp == 1) {
        // ---------------------------------------------------------------- MMA issuer
        if (leader) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t iter = 0;
            bool ok = true;
            const uint64_t a_desc0 = ptx::smem_desc(smem_base, 16, 1024);
            const uint64_t b_desc0 = ptx::smem_desc(smem_base + kABytes, 16, 1024);
            SegIter st = seg_begin(t_begin, p);
            Seg it;
            for (; ok && seg_next(st, it, p); ++iter) {
                const uint32_t acc = NB == 2 ? (iter & 1u) : 0u;
                const uint32_t acc_phase = NB == 2 ? ((iter >> 1) & 1u) : (iter & 1u);
                // every lane waits; the warp leaves together if any lane's wait expired
                if (!__all_sync(0xffffffffu, ptx::mbar_wait_cluster(tempty_bar(acc), acc_phase ^ 1u, abort_flag,
                                                                    p.err, kErrMmaTmemEmpty))) {
                    ok = false;
                    break;
                }
                ptx::tc_fence_after();
                const uint32_t d_tmem = tmem_base + acc * BN;
                for (int kb = it.kb0; kb < it.kb1; ++kb) {
                    if (!__all_sync(0xffffffffu, ptx::mbar_wait(full_bar(stage), phase, abort_flag, p.err, kErrMmaFull))) {
                        ok = false;
                        break;
                    }
                    ptx::tc_fence_after();
                    // the whole warp issues (one elected lane), so it stays converged
                    const uint64_t off = (uint64_t)((stage * kStageBytes) >> 4);
                    const uint64_t ad = a_desc0 + off, bd = b_desc0 + off;
#pragma unroll
                    for (int kk = 0; kk < kKSteps; ++kk)
                        ptx::mma_pair_elect<kKind>(d_tmem, ad + 2 * kk, bd + 2 * kk, kIdesc,
                                                   (kb > it.kb0 || kk > 0) ? 1u : 0u);
                    ptx::tc_commit_pair_elect(empty_bar(stage), 0x3);  // frees the slot in both CTAs
                    if (++stage == S) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                if (!ok) break;
                ptx::tc_commit_pair_elect(tfull_bar(acc), 0x3);
            }
            // Drain: all pair MMAs the warp issued have completed before TMEM is freed.
            __syncwarp();
            ptx::tc_commit_pair_elect(drain_bar, 0x1);
            volatile int no_abort = 0;
            ptx::mbar_wait(drain_bar, 0, &no_abort, p.err, kErrDrain, ptx::kWaitLimitNs / 4);
        }
    } else {
        // ---------------------------------------------------------------- epilogue
        // Warp (2 + e) reads TMEM sub-partition q = warp % 4: rows 32q .. 32q+31 of this
        // CTA's 128 rows; thread `lane` holds one row.
        const int q = warp & 3;
        uint8_t* stage_buf = epi_smem + (warp - 2) * 8192;
        uint32_t chunk_ctr = 0;
        uint32_t iter = 0;
        const uint32_t leader_tempty0 = ptx::map_shared_rank(tempty_bar(0), 0);
        const uint32_t leader_tempty1 = ptx::map_shared_rank(tempty_bar(1), 0);
        constexpr int kChunks = BN / 32;
        static_assert(kChunks % 2 == 0, "chunks are processed in pairs");
        // Pair pr's partial in the workspace, for this CTA and warp: kChunks blocks of 8 x 32
        // float4 (32 KB, contiguous), element [c][i][lane] = columns 32c + 4i .. 32c + 4i + 3
        // of the lane's row, so that each warp-wide access covers 512 contiguous bytes.
        auto part_block = [&](int pr) {
            return reinterpret_cast<float4*>(p.part) + (((long long)pr * 2 + rank) * 4 + q) * (kChunks * 256);
        };
        auto part_chunk = [&](int pr, int c) { return part_block(pr) + c * 256 + lane; };
        // A finisher reads the partials from shared memory: the ring is idle once its last
        // segment's MMAs have completed, and warp q stages them in its quarter of the ring,
        // `cpr` chunks (4 KB each) of every partial per round.
        const int stage_slots = S * (int)kStageBytes / 4 / 4096;
        const uint32_t stage_u32 = ptx::smem_u32(smem) + (uint32_t)(q * stage_slots * 4096);
        const float4* stage_f4 = reinterpret_cast<const float4*>(smem + q * stage_slots * 4096) + lane;
        auto flag_of = [&](int pr) { return p.flag + ((pr * 2 + (int)rank) * 4 + q); };
        const int pc = t_begin;  // this pair
        SegIter st = seg_begin(pc, p);
        Seg it;
        for (; seg_next(st, it, p); ++iter) {
            const PairTile tc = decode(it.tile, p);
            const bool partial = it.role == 1;  // hand the sum over to the tile's finisher
            const bool last = it.role == 2;     // finish the tile with the other pairs' sums
            const uint32_t acc = NB == 2 ? (iter & 1u) : 0u;
            const uint32_t acc_phase = NB == 2 ? ((iter >> 1) & 1u) : (iter & 1u);
            if (!ptx::mbar_wait(tfull_bar(acc), acc_phase, abort_flag, p.err, kErrEpiTmemFull)) break;
            ptx::tc_fence_after();
            if (last) {
                bool ok = true;
                if (lane == 0)
                    for (int pr = it.p_lo; ok && pr <= it.p_hi; ++pr)
                        ok = ptx::wait_counter(flag_of(pr), 1u, abort_flag, p.err, kErrSkWait);
                if (!__shfl_sync(0xffffffffu, ok ? 1 : 0, 0)) break;
                for (int pr = it.p_lo; pr <= it.p_hi; ++pr)
                    (void)ptx::ld_acquire_gpu(flag_of(pr));  // every lane orders its partial reads
                if (lane == 0) ptx::fence_proxy_async_global();  // the copies read what the flags released
            }
            // partials to stage per round: all chunks, half, or a quarter, as the ring allows
            const int n_part = last ? it.p_hi - it.p_lo + 1 : 0;
            const int cpr = !last ? 0 : n_part * kChunks <= stage_slots ? kChunks
                                  : n_part * (kChunks / 2) <= stage_slots ? kChunks / 2
                                  : n_part * 2 <= stage_slots ? 2 : 0;
            uint32_t stage_phase = 0;
            bool stage_ok = true;
            // The pair's last segment (not a stream-K one): its MMAs have completed and no
            // load follows, so the ring is idle and each warp stages every chunk in its own
            // part of it, with no wait for earlier stores.
            SegIter peek = st;
            Seg after;
            const bool ring_out = p.tma_store && !partial && !last && !seg_next(peek, after, p) &&
                                  S * (int)kStageBytes >= 4 * kChunks * 4096;
            const int row_base = tc.tm2 * 256 + row_off + q * 32;
            const int row = row_base + lane;
            const float* bias = p.bias;
            float* dst_row = p.C + (long long)tc.b * p.stride_c + (long long)row * p.ldc;
            const uint32_t tbase = tmem_base + ((uint32_t)(q * 32) << 16) + acc * BN;
            auto emit = [&](const uint32_t (&r)[32], float bl, int c) {
                const int col0 = tc.tn * BN + c * 32;
                float v[32];
#pragma unroll
                for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
                if (partial) {  // raw sum of this segment's k-blocks to the pair's slot
                    float4* dst = part_chunk(pc, c);
#pragma unroll
                    for (int j = 0; j < 8; ++j) dst[32 * j] = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
                    return;
                }
                if (last && cpr > 0) {  // ((own sum + staged partial of p_lo) + ...) + p_hi
                    for (int k = 0; k < n_part; ++k) {
                        const float4* src = stage_f4 + (k * cpr + c % cpr) * 256;
#pragma unroll
                        for (int j = 0; j < 8; ++j) {
                            const float4 x = src[32 * j];
                            v[4 * j] += x.x; v[4 * j + 1] += x.y; v[4 * j + 2] += x.z; v[4 * j + 3] += x.w;
                        }
                    }
                } else if (last) {  // ((own sum + partial of pair p_lo) + ...) + partial of pair p_hi
                    for (int pr = it.p_lo; pr <= it.p_hi; ++pr) {
                        const float4* src = part_chunk(pr, c);
#pragma unroll
                        for (int j = 0; j < 8; ++j) {
                            const float4 x = __ldcg(src + 32 * j);
                            v[4 * j] += x.x; v[4 * j + 1] += x.y; v[4 * j + 2] += x.z; v[4 * j + 3] += x.w;
                        }
                    }
                }
                if (bias) {
#pragma unroll
                    for (int j = 0; j < 32; ++j) v[j] += __shfl_sync(0xffffffffu, bl, j);
                }
                if (p.tma_store) {
                    uint8_t* buf = ring_out ? smem + (q * kChunks + c) * 4096 : stage_buf + (chunk_ctr & 1u) * 4096;
                    if (!ring_out && lane == 0) ptx::bulk_wait_read<1>();
                    __syncwarp();
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        *reinterpret_cast<float4*>(buf + lane * 128 + ((j ^ (lane & 7)) << 4)) =
                            make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
                    if ((p.act & 15) != NNJIT_EPI_NONE) act_row128(buf + lane * 128, p.act);
                    if ((p.act & NNJIT_EPI_RESIDUAL) && row < p.M && col0 < p.N)
                        residual_row128(buf + lane * 128, lane & 7, dst_row + col0, p.N - col0);
                    ptx::fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) {
                        ptx::tma_store_3d(&p.tmap_c, ptx::smem_u32(buf), col0, row_base, tc.b);
                        ptx::bulk_commit();
                    }
                    if (!ring_out) ++chunk_ctr;
                } else if (row < p.M) {
                    float* dst = dst_row + col0;
                    if (p.act != NNJIT_EPI_NONE) {
                        // stage the row (this thread's own 128 bytes of the idle staging
                        // buffer), then activation and residual element by element
                        if (col0 < p.N) {
                            float* srow = reinterpret_cast<float*>(stage_buf + lane * 128);
#pragma unroll
                            for (int j = 0; j < 32; j += 4)
                                *reinterpret_cast<float4*>(srow + j) = make_float4(v[j], v[j + 1], v[j + 2], v[j + 3]);
                            epi_store_row(srow, p.act, dst, min(32, p.N - col0));
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
            // The accumulator goes back to the MMA issuer (in the even CTA) once this
            // warp's last chunk is in registers.
            auto release = [&]() {
                ptx::tc_fence_before();
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive_cluster(acc ? leader_tempty1 : leader_tempty0);
            };
            uint32_t ra[32], rb[32];
            ptx::tmem_ld32(tbase, ra);
            float ba = bias_of(0), bb = 0.0f;
            ptx::tmem_wait_ld(ra);
#pragma unroll 1
            for (int c = 0; c < kChunks; c += 2) {
                if (cpr > 0 && c % cpr == 0) {
                    // stage chunks [c, c + cpr) of every partial: one bulk copy per partial
                    __syncwarp();  // this warp's reads of the previous round are done
                    if (lane == 0) {
                        ptx::fence_proxy_async_smem();
                        ptx::mbar_arrive_expect_tx(pcopy_bar(q), (uint32_t)(n_part * cpr * 4096));
                        for (int k = 0; k < n_part; ++k)
                            ptx::bulk_copy_g2s(stage_u32 + (uint32_t)(k * cpr * 4096), part_block(it.p_lo + k) + c * 256,
                                               (uint32_t)(cpr * 4096), pcopy_bar(q));
                    }
                    __syncwarp();
                    const bool landed = ptx::mbar_wait(pcopy_bar(q), stage_phase, abort_flag, p.err, kErrSkWait);
                    stage_phase ^= 1u;
                    if (!__all_sync(0xffffffffu, landed)) {
                        stage_ok = false;
                        break;
                    }
                }
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
            if (!stage_ok) break;
            if (partial) {  // publish this warp's rows of the partial
                __threadfence();
                __syncwarp();
                if (lane == 0) ptx::red_release_add_gpu(flag_of(pc), 1u);
            }
            if (last) {  // every partial has been read: ready for the next launch
                __syncwarp();
                if (lane == 0)
                    for (int pr = it.p_lo; pr <= it.p_hi; ++pr) *flag_of(pr) = 0u;
            }
        }
        if (p.tma_store && lane == 0) ptx::bulk_wait_all_read();
        __syncwarp();
    }

    ptx::tc_fence_before();
    __syncthreads();
    // neither CTA frees TMEM or leaves while its partner may still address it
    ptx::cluster_sync();
    ptx::tc_fence_after();
    if (warp == 1) ptx::tmem_dealloc_pair(tmem_base, kTmemCols);
}

using Tc2Kernel = void (*)(Tc2Params);
// Instance table, indexed as instance - kTcPairFirstInstance: dtype_i (bf16, tf32).
const Tc2Kernel kKernels[2] = {tc2_gemm_kernel<0, 256, kPairAccBuffers>, tc2_gemm_kernel<1, 256, kPairAccBuffers>};


}  // namespace

cudaError_t launch_tc_pair(const LaunchArgs& a) {
    const Problem& p = *a.p;
    const nnjit_candidate& c = *a.c;
    const int i = c.instance - kTcPairFirstInstance;
    const int di = p.dtype == NNJIT_BF16 ? 0 : 1;
    if (i != di || !a.tmap_a || !a.tmap_b || p.b_layout != NNJIT_B_NK) return cudaErrorInvalidValue;
    if (c.bm != 256 || c.bn != 256 || c.cluster_m != 2 || c.stages < 2 || c.stages > kMaxStages ||
        c.bk != 128 / p.elem_bytes())
        return cudaErrorInvalidValue;
    // unsplit (reduce 0) or stream-K over the last waves (reduce 2); split_k is 1
    const bool stream_k = c.reduce == 2;
    if (c.split_k != 1 || (c.reduce != 0 && !stream_k) || (stream_k && !a.ws)) return cudaErrorInvalidValue;
    // a stream-K finisher stages a partial (4 warps x 32 KB) in the idle ring
    if (stream_k && c.stages * (128 + 128) * 128 < 4 * 32768) return cudaErrorInvalidValue;
    Tc2Params prm;
    prm.tmap_a = *a.tmap_a;
    prm.tmap_b = *a.tmap_b;
    prm.tma_store = a.tmap_c ? 1 : 0;
    if (a.tmap_c) prm.tmap_c = *a.tmap_c;
    prm.b_const = (p.flags & NNJIT_PLAN_B_CONSTANT) ? 1 : 0;
    prm.C = a.C;
    prm.bias = a.bias;
    prm.act = p.epilogue;
    prm.err = a.err;
    prm.M = (int)p.M;
    prm.N = (int)p.N;
    prm.K = (int)p.K;
    prm.batch = (int)p.batch;
    prm.ldc = p.ldc;
    prm.stride_c = p.stride_c;
    prm.num_kb = (int)((p.K + c.bk - 1) / c.bk);
    prm.tiles2_m = (int)((p.M + 255) / 256);
    prm.tiles_n = (int)((p.N + 255) / 256);
    const long long total = (long long)p.batch * prm.tiles2_m * prm.tiles_n;
    if (total >= (1LL << 30) || c.grid < 2 || (c.grid & 1)) return cudaErrorInvalidValue;
    prm.total = (int)total;
    prm.stages = c.stages;
    prm.raster = c.raster;
    // unsplit: at most one pair per tile; stream-K: every pair of the candidate's grid
    const int grid = stream_k ? c.grid : (int)std::min<long long>(2 * total, c.grid);
    prm.pairs = grid / 2;
    prm.dp = prm.total;
    prm.sk_iters = 0;  // no stream-K region: every pair's range is empty
    prm.part = nullptr;
    prm.flag = nullptr;
    if (stream_k) {
        // whole waves but the last run as whole tiles; the rest (1 to 2 waves) stream-K
        const int P = prm.pairs;
        const int waves = prm.total / P;
        if (prm.total % P == 0) return cudaErrorInvalidValue;
        prm.dp = waves >= 1 ? (waves - 1) * P : 0;
        prm.sk_iters = (long long)(prm.total - prm.dp) * prm.num_kb;
        if (prm.sk_iters < (long long)P) return cudaErrorInvalidValue;
        // workspace: the flags, then one partial tile per pair (tc2_sk_ws_bytes)
        prm.flag = reinterpret_cast<unsigned*>(a.ws);
        prm.part = a.ws + tc2_sk_flag_floats(P);
    }
    const int stage_bytes = (128 + 128) * 128;
    const int smem = c.stages * stage_bytes + kEpiStageBytes + 1024 + 256;
    {
        cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void*>(kKernels[i]), smem);
        if (e != cudaSuccess) return e;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = a.stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = 2;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, kKernels[i], prm);
}

}  // namespace nnjit
