// Lite kernel-configuration space: descriptor resolution, family choice, enumeration,
// pruning by hardware-usage formulas and ordering (Sec. 5.2, Table 1, Table 2).
#include "space.h"

#include <algorithm>
#include <cstdio>

namespace nnjit {

namespace {

int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

int64_t pow2_ceil(int64_t x) {
    int64_t p = 1;
    while (p < x) p <<= 1;
    return p;
}

int min4(int a, int b, int c, int d) { return std::min(std::min(a, b), std::min(c, d)); }

// Block_core of Table 1 generalised: the number of CTAs one SM can hold is the smallest
// of the per-resource limits (registers, shared memory = L1Limit, warps, TMEM, blocks).
int blocks_per_core(const nnjit_device_limits& L, int regs, int threads, int smem, int tmem) {
    const int reg_lim = L.regs_per_sm / std::max(1, regs * threads);
    // every resident CTA also holds the per-block reservation of the SM's shared memory
    // (the difference between the SM's shared memory and the largest opt-in per block)
    const int reserved = std::max(0, L.smem_per_sm - L.smem_per_block_optin);
    const int smem_lim = smem > 0 ? L.smem_per_sm / (smem + reserved) : L.max_blocks_per_sm;
    const int warp_lim = (L.max_threads_per_sm / 32) / std::max(1, threads / 32);
    const int tmem_lim = tmem > 0 ? L.tmem_cols_per_sm / tmem : L.max_blocks_per_sm;
    return std::min(min4(reg_lim, smem_lim, warp_lim, tmem_lim), L.max_blocks_per_sm);
}

nnjit_candidate blank() {
    nnjit_candidate c{};
    c.split_k = 1;
    c.instance = -1;
    c.cluster_m = 1;
    return c;
}

// ---------------------------------------------------------------------------------
// tcgen05 tensor-core family.  The CTA tile is BM x BN with BM = 128, or BM = 64 when the
// 128-row tiles leave SMs idle (an M = 64 MMA costs about half as long, so 64-row tiles
// double the CTAs without split-K partial traffic).  BK is fixed at one 128-byte swizzle
// row of K (64 bf16,
// 32 tf32): the Blackwell counterpart of the paper's "consistent" primitive settings
// (Sec. 5.1), fixed once instead of searched.  The searched axes are BN, split-K and
// the tile raster order; the stage count is derived, not searched: the ring fills the
// shared memory a CTA may opt in to (the counterpart of heuristic 7, "use all of the
// fastest storage").
// ---------------------------------------------------------------------------------
void tc_space(const Problem& p, const nnjit_device_limits& L, std::vector<nnjit_candidate>& v,
              int64_t* naive) {
    using MC = ModelConstants;
    const int e = p.elem_bytes();
    const int BK = 128 / e;
    const int64_t M = std::max<int64_t>(p.M, 1), N = std::max<int64_t>(p.N, 1);
    const int64_t K = std::max<int64_t>(p.K, 1);
    const int64_t num_kb = ceil_div(K, BK);
    const int bns[3] = {64, 128, 256};
    const int splits[4] = {1, 2, 4, 8};
    // BM x BN x stages x split x raster x reduce x CTA pair x k-blocks per ring slot
    *naive = 2 * 3 * (MC::kTcMaxStages - 1) * 4 * 2 * 2 * 2 * 2;
    for (int BM : {MC::kTcBM, 64})
    for (int bn : bns)
    for (int kg : {1, 2}) {
        if (bn > 64 && bn > pow2_ceil(N)) continue;  // no tile wider than the padded N
        if (BM == 64 && p.batch * ceil_div(M, MC::kTcBM) * ceil_div(N, bn) >= L.sm_count) continue;
        // two k-blocks per ring slot where the MMA issue path, not the tensor pipe, sets
        // the pace: 128-row tiles with BN <= 128
        if (kg == 2 && (BM != MC::kTcBM || bn > 128)) continue;
        const int kb_bytes = (BM + bn) * 128;
        const int stage_bytes = kg * kb_bytes;
        const int stages = std::min(MC::kTcMaxStages,
                                    (L.smem_per_block_optin - MC::kTcFixedSmem) / stage_bytes);
        if (stages < 2) continue;
        const int smem = stages * stage_bytes + MC::kTcFixedSmem;
        const int tmem = (int)pow2_ceil(std::max(32, 2 * bn));  // two accumulator buffers
        if (tmem > L.tmem_cols_per_sm) continue;
        const int threads = MC::kTcThreads, regs = MC::kTcRegsPerThread;
        const int blk = blocks_per_core(L, regs, threads, smem, tmem);
        if (blk < 1) continue;
        const int64_t tiles_m = ceil_div(M, BM), tiles_n = ceil_div(N, bn);
        const int64_t tiles = p.batch * tiles_m * tiles_n;
        for (int split : splits) {
            // split only while the previous split count still leaves SMs idle
            if (split > 1 && (tiles * (split / 2) >= L.sm_count || num_kb < 4 * split)) continue;
            // split-K partials: summed by a second kernel (reduce 0) or, one output tile
            // per thread-block cluster of `split` CTAs, through distributed shared memory
            // (reduce 1; the partial tile reuses the idle ring)
            for (int reduce = 0; reduce < (split > 1 && kg == 1 ? 2 : 1); ++reduce)
            for (int raster = 0; raster < 2; ++raster) {
                if (raster == 1 && (tiles_m == 1 || tiles_n == 1)) continue;
                if (reduce == 1 && (BM != MC::kTcBM || raster == 1 || stages * stage_bytes < 128 * (bn + 4) * 4))
                    continue;
                nnjit_candidate c = blank();
                c.family = NNJIT_FAMILY_TC;
                c.bm = BM; c.bn = bn; c.bk = BK * kg;
                c.tm = 0; c.tn = 0;
                c.stages = stages;
                c.split_k = split;
                c.raster = raster;
                c.threads = threads;
                c.smem_bytes = smem;
                c.tmem_cols = tmem;
                c.regs_per_thread = regs;
                c.blocks_per_sm = blk;
                c.reduce = reduce;
                const int64_t work = tiles * split;
                const int64_t slots = (int64_t)L.sm_count * blk;
                // persistent grid; cluster mode launches one CTA per (tile, slice)
                const int64_t grid = reduce ? work : std::min(work, slots);
                const int64_t waves = ceil_div(work, std::min(work, slots));
                c.grid = (int32_t)grid;
                c.wave_eff_ppm = (int32_t)(work * 1000000 / (waves * std::min(work, slots)));
                // per k-block (4 MMA instructions): the slowest of the tensor pipe (an
                // instruction takes kMmaN256Clk * N / 256, at least a quarter of that),
                // the issuing thread (kMmaIssueClk per instruction plus one barrier wait
                // and commit per ring slot) and the operand feed (bytes over the per-SM
                // L2 feed), plus the share of the issue path that the feed does not hide
                const int64_t t_tensor = 4LL * std::max(MC::kMmaN256Clk / 4, MC::kMmaN256Clk * bn / 256);
                const int64_t t_issue = 4LL * MC::kMmaIssueClk + MC::kSlotSyncClk / kg;
                const int64_t t_kb = std::max(std::max(t_tensor, t_issue),
                                              ceil_div(kb_bytes, MC::kFeedBytesPerClk)) +
                                     t_issue / MC::kIssueShowDiv;
                int64_t cost = waves * t_kb * ceil_div(num_kb, split);
                if (split > 1 && reduce == 0)
                    cost += MC::kLaunchClk +
                            ceil_div(2LL * split * p.batch * M * N * 4, MC::kHbmBytesPerClk);
                if (split > 1 && reduce == 1)  // DSMEM reduction of the partial tiles
                    cost += waves * (128LL * bn * 4 / MC::kDsmemReduceBytesPerClk);
                c.predicted_cost = cost;
                c.instance = tc_instance(p.dtype, p.b_layout, bn, reduce, BM, kg);
                v.push_back(c);
            }
        }
    }
    // 256 x 256 tiles on CTA pairs (tcgen05 cta_group::2), B as [N][K]: an SM receives its
    // 128 rows of A and half of the B tile per k-block (32 KB), one thread issues the MMAs
    // of both SMs.  Unsplit, persistent over pair tiles.
    if (p.b_layout == NNJIT_B_NK && M > MC::kTcBM && L.sm_count >= 2) {
        const int kb_bytes = (MC::kTcBM + 128) * 128;
        const int stages = std::min(MC::kTcMaxStages, (L.smem_per_block_optin - MC::kTcFixedSmem) / kb_bytes);
        const int smem = stages * kb_bytes + MC::kTcFixedSmem;
        const int tmem = MC::kTcPairAccCols;
        const int blk = blocks_per_core(L, MC::kTcRegsPerThread, MC::kTcThreads, smem, tmem);
        const int64_t tiles2_m = ceil_div(M, 256), tiles_n = ceil_div(N, 256);
        const int64_t pairs = p.batch * tiles2_m * tiles_n;
        if (stages >= 2 && blk >= 1 && tmem <= L.tmem_cols_per_sm) {
            for (int raster = 0; raster < 2; ++raster) {
                if (raster == 1 && (tiles2_m == 1 || tiles_n == 1)) continue;
                nnjit_candidate c = blank();
                c.family = NNJIT_FAMILY_TC;
                c.bm = 256; c.bn = 256; c.bk = BK;
                c.stages = stages;
                c.raster = raster;
                c.threads = MC::kTcThreads;
                c.smem_bytes = smem;
                c.tmem_cols = tmem;
                c.regs_per_thread = MC::kTcRegsPerThread;
                c.blocks_per_sm = blk;
                c.cluster_m = 2;
                const int64_t pair_slots = std::max<int64_t>(1, (int64_t)L.sm_count * blk / 2);
                const int64_t live = std::min(pairs, pair_slots);
                const int64_t waves = ceil_div(pairs, live);
                c.grid = (int32_t)(2 * live);
                c.wave_eff_ppm = (int32_t)(pairs * 1000000 / (waves * live));
                const int64_t t_tensor = 4LL * MC::kMmaN256Clk;
                const int64_t t_issue = 4LL * MC::kMmaIssueClk + MC::kSlotSyncClk;
                const int64_t t_kb = std::max(std::max(t_tensor, t_issue), ceil_div(kb_bytes, MC::kFeedBytesPerClk)) +
                                     t_issue / MC::kIssueShowDiv;
                c.predicted_cost = waves * t_kb * num_kb;
                c.instance = kTcPairFirstInstance + (p.dtype == NNJIT_BF16 ? 0 : 1);
                v.push_back(c);
                // Stream-K over the last waves: the whole waves but the last run as whole
                // tiles, the k-blocks of the remaining tiles are shared evenly by all pairs;
                // each pair hands at most one partial tile over, and a tile's finisher reads
                // the partials of the pairs covering the rest of it (one 128-row x 256-column
                // f32 partial per CTA each, at the per-SM feed rate).
                // Only from two whole waves on.  With fewer tiles every tile is stream-K and
                // the hand-offs sit on the critical path: a per-CTA timeline of T5-large wo
                // (32 tiles) showed the MMAs done at 15 us against 22.5 us for whole tiles,
                // but 2.5 us to publish a partial, 1.8 us to see its flag and 8 us to add two
                // partials and store, so the launch ended later than with whole tiles.
                if (pairs % pair_slots != 0 && pairs / pair_slots >= 2) {
                    const int64_t waves_sk = pairs / pair_slots;
                    const int64_t dp = (waves_sk - 1) * pair_slots;
                    const int64_t iters = (pairs - dp) * num_kb;
                    const int64_t share = iters / pair_slots;
                    if (share >= 4) {
                        nnjit_candidate t = c;
                        t.reduce = 2;
                        t.grid = (int32_t)(2 * pair_slots);
                        const int64_t per_pair = ceil_div(iters, pair_slots);
                        t.wave_eff_ppm = (int32_t)(pairs * num_kb * 1000000 / (dp * num_kb + pair_slots * per_pair));
                        t.predicted_cost = (dp / pair_slots) * t_kb * num_kb + t_kb * per_pair +
                                           (1 + ceil_div(num_kb, share)) * (128LL * 256 * 4 / MC::kFeedBytesPerClk);
                        v.push_back(t);
                    }
                }
            }
        }
    }
}

// ---------------------------------------------------------------------------------
// FP32-FFMA SIMT family: the direct descendant of the paper's WebGPU tile template
// (Table 2): thread tile x0 = y0 in {4, 8} (inner range [4..32]), block tile x1, y1 in
// {32, 64, 128} (range [32..256]), r1 = BK = 16, r0 = 1.  Table 1's usage formulas
// are applied as written; heuristic 5 (Thread_block <= 256) is kept, the WebGPU 16 KB
// limit of heuristic 6 becomes the CTA's shared-memory limit.
// ---------------------------------------------------------------------------------
void ffma_space(const Problem& p, const nnjit_device_limits& L, std::vector<nnjit_candidate>& v,
                int64_t* naive) {
    using MC = ModelConstants;
    const int64_t M = std::max<int64_t>(p.M, 1), N = std::max<int64_t>(p.N, 1);
    const int64_t K = std::max<int64_t>(p.K, 1);
    const int tiles_x[3] = {32, 64, 128};
    const int bks[1] = {16};
    const int splits[4] = {1, 2, 4, 8};
    *naive = 2 * 3 * 3 * 2 * 4;  // thread tile x block tile x BK {8, 16} x split
    for (int t0 : {4, 8}) {
        for (int bm : tiles_x) {
            for (int bn : tiles_x) {
                const int threads = (bm / t0) * (bn / t0);       // Thread_block
                if (threads < 64 || threads > 256) continue;     // >= 2 warps; heuristic 5
                if ((bm > 32 && bm > pow2_ceil(M)) || (bn > 32 && bn > pow2_ceil(N))) continue;
                for (int bk : bks) {
                    // Table 1: Reg_thread = x0 r0 + r0 y0 + x0 y0 (r0 = 1), divided by the
                    // relaxation share for the kernel's other variables.
                    const int reg_paper = t0 * 1 + 1 * t0 + t0 * t0;
                    const int regs = (int)ceil_div(reg_paper * 100, MC::kRegRelaxPct);
                    // shared memory: double-buffered A and B tiles, rows padded by 4 floats
                    const int smem = 2 * bk * ((bm + 4) + (bn + 4)) * 4;
                    if (smem > L.smem_per_block_optin) continue;
                    const int blk = blocks_per_core(L, regs, threads, smem, 0);
                    if (blk < 1) continue;
                    const int64_t tiles = p.batch * ceil_div(M, bm) * ceil_div(N, bn);
                    for (int split : splits) {
                        if (split > 1 && (tiles * (split / 2) >= L.sm_count || K < 2LL * split * bk))
                            continue;
                        nnjit_candidate c = blank();
                        c.family = NNJIT_FAMILY_FFMA;
                        c.bm = bm; c.bn = bn; c.bk = bk;
                        c.tm = t0; c.tn = t0;
                        c.stages = 2;
                        c.split_k = split;
                        c.threads = threads;
                        c.smem_bytes = smem;
                        c.regs_per_thread = regs;
                        c.blocks_per_sm = blk;
                        const int64_t grid = tiles * split;
                        const int64_t slots = (int64_t)L.sm_count * blk;
                        const int64_t waves = ceil_div(grid, slots);
                        c.grid = (int32_t)grid;
                        c.wave_eff_ppm = (int32_t)(grid * 1000000 / (waves * slots));
                        const int64_t per_sm = ceil_div(grid, L.sm_count);
                        const int64_t resident = std::min<int64_t>(per_sm, blk);
                        const int64_t warps = resident * threads / 32;
                        const int64_t util_pct = std::min<int64_t>(100, std::max<int64_t>(1, warps * 100 / 16));
                        int64_t cost = per_sm * ceil_div((int64_t)bm * bn * ceil_div(K, split), 128) *
                                       100 / util_pct;
                        if (split > 1)
                            cost += MC::kLaunchClk +
                                    ceil_div(2LL * split * p.batch * M * N * 4, MC::kHbmBytesPerClk);
                        c.predicted_cost = cost;
                        c.instance = ffma_instance(t0, bm, bn, bk, p.b_layout);
                        v.push_back(c);
                    }
                }
            }
        }
    }
}

// ---------------------------------------------------------------------------------
// Split-K GEMV family (M <= 8, bf16 weights): bandwidth-bound, so the axes are those
// that set the bytes in flight per SM: threads per CTA, rows per warp, 16-byte loads in
// flight per lane and row (unroll), and split-K.
// ---------------------------------------------------------------------------------
// 4-bit weights (NNJIT_W4_BF16): the TMA-fed tensor-core kernel only.  A ring stage
// holds `rows` weight rows x 1024 codes (512 bytes a row, four 128-byte-swizzled boxes),
// the 1024-element slice of every row of x and the rows' 8 group scales, padded to 1 KB;
// axes rows per stage (16-row MMA tiles), ring stages, split-K.
void gemv_w4_space(const Problem& p, const nnjit_device_limits& L, std::vector<nnjit_candidate>& v,
                   int64_t* naive) {
    using MC = ModelConstants;
    const int64_t M = std::max<int64_t>(p.M, 1), N = std::max<int64_t>(p.N, 1);
    const int64_t K = std::max<int64_t>(p.K, 1);
    const int64_t wbytes = N * K / 2 + ceil_div(K, 128) * N * 2;
    const int64_t chunks = ceil_div(K, MC::kGemvW4Kc);
    *naive = 2 * 2 * 4;
    for (int rows : {16, 32}) {
        const int64_t groups = ceil_div(N, rows);
        for (int stages : {4, 8}) {
            for (int split : {1, 2, 4, 8}) {
                const int64_t cps = ceil_div(chunks, split);
                if (split > 1 && (cps < 2 || (split - 1) * cps >= chunks ||
                                  groups * (split / 2) >= 2LL * L.sm_count))
                    continue;
                const int64_t stage_bytes =
                    ceil_div(rows * (MC::kGemvW4Kc / 2 + 16) + M * MC::kGemvW4Kc * 2, 1024) * 1024;
                // dynamic (1 KB alignment slack + ring) and static (barriers, partial sums)
                const int64_t smem = 1024 + stages * stage_bytes + 256 + rows * 128;
                if (smem > L.smem_per_block_optin) continue;
                const int regs = rows == 16 ? 88 : 112;  // ptxas: 82 / 108
                const int blk = blocks_per_core(L, regs, MC::kGemvTmaThreads, (int)smem, 0);
                if (blk < 1) continue;
                const int64_t items = groups * split;
                const int64_t slots = (int64_t)L.sm_count * blk;
                const int64_t grid = std::min<int64_t>(items, slots);
                nnjit_candidate c = blank();
                c.family = NNJIT_FAMILY_GEMV;
                c.bm = (int)M; c.bn = rows; c.bk = MC::kGemvW4Kc;
                c.tm = rows / 16; c.tn = 1;
                c.stages = stages;
                c.split_k = split;
                c.threads = MC::kGemvTmaThreads;
                c.smem_bytes = (int)smem;
                c.regs_per_thread = regs;
                c.blocks_per_sm = blk;
                c.grid = (int32_t)grid;
                c.wave_eff_ppm = (int32_t)(grid * 1000000 / slots);
                const int64_t resident = std::min<int64_t>(ceil_div(grid, L.sm_count), blk);
                const int64_t inflight = resident * stages * rows * MC::kGemvW4Kc / 2;
                const int64_t eff_pct = std::min<int64_t>(100, std::max<int64_t>(1, inflight * 100 / 32768));
                int64_t cost = ceil_div(wbytes, MC::kHbmBytesPerClk) * 100 / eff_pct;
                cost = cost * ceil_div(items, L.sm_count) * L.sm_count / items;
                if (split > 1)
                    cost += MC::kLaunchClk + ceil_div(2LL * split * M * N * 4, MC::kHbmBytesPerClk);
                c.predicted_cost = cost;
                c.instance = gemv_w4_instance(rows);
                v.push_back(c);
            }
        }
    }
}

void gemv_space(const Problem& p, const nnjit_device_limits& L, std::vector<nnjit_candidate>& v,
                int64_t* naive) {
    using MC = ModelConstants;
    if (p.dtype == NNJIT_W4_BF16) {
        gemv_w4_space(p, L, v, naive);
        return;
    }
    const int64_t M = std::max<int64_t>(p.M, 1), N = std::max<int64_t>(p.N, 1);
    const int64_t K = std::max<int64_t>(p.K, 1);
    const int64_t wbytes = N * K * 2;
    if (p.b_layout == NNJIT_B_NK) {
        *naive = 2 * 3 * 2 * 4;
        for (int threads : {128, 256}) {
            for (int rows : {1, 2, 4}) {
                for (int unroll : {2, 4}) {
                    const int warps = threads / 32;
                    const int64_t ctas_n = ceil_div(N, (int64_t)warps * rows);
                    for (int split : {1, 2, 4, 8}) {
                        const int64_t kper = ceil_div(ceil_div(K, split), 8) * 8;
                        if (split > 1 && (kper < 256LL * unroll ||
                                          ctas_n * (split / 2) >= 2LL * L.sm_count))
                            continue;
                        const int64_t smem = ceil_div(M * kper * 2, 16) * 16;
                        if (smem > MC::kGemvMaxSmem || smem > L.smem_per_block_optin) continue;
                        const int regs = 40 + rows * (int)M + 4 * unroll * rows + 8;
                        const int blk = blocks_per_core(L, regs, threads, (int)smem, 0);
                        if (blk < 1) continue;
                        nnjit_candidate c = blank();
                        c.family = NNJIT_FAMILY_GEMV;
                        c.bm = (int)M; c.bn = warps * rows; c.bk = (int)std::min<int64_t>(kper, 1 << 30);
                        c.tm = rows; c.tn = 1;
                        c.stages = unroll;
                        c.split_k = split;
                        c.threads = threads;
                        c.smem_bytes = (int)smem;
                        c.regs_per_thread = regs;
                        c.blocks_per_sm = blk;
                        // at most as many CTAs as fit at once (bytes in flight are
                        // what a streaming kernel needs); beyond that the warps take
                        // row groups round-robin
                        const int64_t per_split = std::min<int64_t>(ctas_n, (int64_t)L.sm_count * blk);
                        const int64_t grid = per_split * split;
                        const int64_t slots = (int64_t)L.sm_count * blk;
                        const int64_t waves = ceil_div(grid, slots);
                        c.grid = (int32_t)grid;
                        c.wave_eff_ppm = (int32_t)(grid * 1000000 / (waves * slots));
                        const int64_t resident = std::min<int64_t>(ceil_div(grid, L.sm_count), blk);
                        const int64_t inflight = resident * threads * unroll * rows * 16;
                        const int64_t eff_pct = std::min<int64_t>(100, std::max<int64_t>(1, inflight * 100 / 32768));
                        int64_t cost = ceil_div(wbytes, MC::kHbmBytesPerClk) * 100 / eff_pct;
                        if (split > 1)
                            cost += MC::kLaunchClk +
                                    ceil_div(2LL * split * M * N * 4, MC::kHbmBytesPerClk);
                        c.predicted_cost = cost;
                        c.instance = gemv_instance(p.b_layout, rows, unroll);
                        v.push_back(c);
                    }
                }
            }
        }
        // TMA-fed instances: a producer warp keeps `stages` boxes of `rows` weight rows x
        // 256 K elements in flight; axes rows per stage, ring stages and split-K.
        const int maxm = M == 1 ? 1 : MC::kGemvMaxM;
        const int64_t chunks = ceil_div(K, MC::kGemvTmaKc);
        *naive += 3 * 2 * 4;
        for (int rows : {8, 16, 32}) {
            const int64_t groups = ceil_div(N, rows);
            for (int stages : {4, 8}) {
                for (int split : {1, 2, 4, 8}) {
                    const int64_t cps = ceil_div(chunks, split);
                    if (split > 1 && (cps < 2 || (split - 1) * cps >= chunks ||
                                      groups * (split / 2) >= 2LL * L.sm_count))
                        continue;
                    const int64_t smem = 128 + (int64_t)stages * (rows + M) * MC::kGemvTmaKc * 2;
                    if (smem > L.smem_per_block_optin) continue;
                    const int regs = maxm == 1 ? 40 : 96 + 3 * rows;
                    const int blk = blocks_per_core(L, regs, MC::kGemvTmaThreads, (int)smem, 0);
                    if (blk < 1) continue;
                    const int64_t items = groups * split;
                    const int64_t slots = (int64_t)L.sm_count * blk;
                    const int64_t grid = std::min<int64_t>(items, slots);
                    nnjit_candidate c = blank();
                    c.family = NNJIT_FAMILY_GEMV;
                    c.bm = (int)M; c.bn = rows; c.bk = MC::kGemvTmaKc;
                    c.tm = rows / 4; c.tn = 1;
                    c.stages = stages;
                    c.split_k = split;
                    c.threads = MC::kGemvTmaThreads;
                    c.smem_bytes = (int)smem;
                    c.regs_per_thread = regs;
                    c.blocks_per_sm = blk;
                    c.grid = (int32_t)grid;
                    c.wave_eff_ppm = (int32_t)(grid * 1000000 / slots);
                    const int64_t resident = std::min<int64_t>(ceil_div(grid, L.sm_count), blk);
                    const int64_t inflight = resident * stages * rows * MC::kGemvTmaKc * 2;
                    const int64_t eff_pct = std::min<int64_t>(100, std::max<int64_t>(1, inflight * 100 / 32768));
                    int64_t cost = ceil_div(wbytes, MC::kHbmBytesPerClk) * 100 / eff_pct;
                    // the SM with the most items finishes last
                    cost = cost * ceil_div(items, L.sm_count) * L.sm_count / items;
                    if (split > 1)
                        cost += MC::kLaunchClk + ceil_div(2LL * split * M * N * 4, MC::kHbmBytesPerClk);
                    c.predicted_cost = cost;
                    c.instance = gemv_tma_instance(rows, maxm);
                    v.push_back(c);
                }
            }
        }
    } else {
        *naive = 2 * 2 * 6;
        for (int threads : {128, 256}) {
            for (int unroll : {2, 4}) {
                const int warps = threads / 32;
                const int64_t ctas_n = ceil_div(N, 256);
                for (int split : {1, 2, 4, 8, 16, 32}) {
                    const int64_t kper = ceil_div(K, split);
                    if (split > 1 && (kper < (int64_t)warps * unroll ||
                                      ctas_n * (split / 2) >= 2LL * L.sm_count))
                        continue;
                    const int64_t smem = (int64_t)warps * M * 256 * 4;
                    if (smem > MC::kGemvMaxSmem || smem > L.smem_per_block_optin) continue;
                    const int regs = 40 + 8 * (int)M + 4 * unroll + 8;
                    const int blk = blocks_per_core(L, regs, threads, (int)smem, 0);
                    if (blk < 1) continue;
                    nnjit_candidate c = blank();
                    c.family = NNJIT_FAMILY_GEMV;
                    c.bm = (int)M; c.bn = 256; c.bk = (int)std::min<int64_t>(kper, 1 << 30);
                    c.tm = 1; c.tn = 8;
                    c.stages = unroll;
                    c.split_k = split;
                    c.threads = threads;
                    c.smem_bytes = (int)smem;
                    c.regs_per_thread = regs;
                    c.blocks_per_sm = blk;
                    const int64_t grid = ctas_n * split;
                    const int64_t slots = (int64_t)L.sm_count * blk;
                    const int64_t waves = ceil_div(grid, slots);
                    c.grid = (int32_t)grid;
                    c.wave_eff_ppm = (int32_t)(grid * 1000000 / (waves * slots));
                    const int64_t resident = std::min<int64_t>(ceil_div(grid, L.sm_count), blk);
                    const int64_t inflight = resident * threads * unroll * 16;
                    const int64_t eff_pct = std::min<int64_t>(100, std::max<int64_t>(1, inflight * 100 / 32768));
                    int64_t cost = ceil_div(wbytes, MC::kHbmBytesPerClk) * 100 / eff_pct;
                    if (split > 1)
                        cost += MC::kLaunchClk + ceil_div(2LL * split * M * N * 4, MC::kHbmBytesPerClk);
                    c.predicted_cost = cost;
                    c.instance = gemv_instance(p.b_layout, 1, unroll);
                    v.push_back(c);
                }
            }
        }
    }
}

}  // namespace

int tc_instance(int dtype, int b_layout, int bn, int cluster, int bm, int kg) {
    const int bi = bn == 64 ? 0 : bn == 128 ? 1 : bn == 256 ? 2 : -1;
    if (bi < 0 || (bm != 64 && bm != 128) || (bm == 64 && cluster)) return -1;
    const int di = dtype == NNJIT_BF16 ? 0 : 1;
    if (kg == 2) {
        if (bm != 128 || cluster || bn > 128) return -1;
        return 36 + (di * 2 + (b_layout == NNJIT_B_KN ? 1 : 0)) * 2 + bi;
    }
    if (kg != 1) return -1;
    const int variant = bm == 64 ? 2 : cluster ? 1 : 0;
    return variant * 12 + (di * 2 + (b_layout == NNJIT_B_KN ? 1 : 0)) * 3 + bi;
}

// The 12 (thread tile, block tile) pairs with 64..256 threads, in enumeration order.
static const int kFfmaTiles[12][3] = {
    {4, 32, 32}, {4, 32, 64}, {4, 32, 128}, {4, 64, 32}, {4, 64, 64}, {4, 128, 32},
    {8, 32, 128}, {8, 64, 64}, {8, 64, 128}, {8, 128, 32}, {8, 128, 64}, {8, 128, 128}};

int ffma_instance(int tm, int bm, int bn, int bk, int b_layout) {
    int ti = -1;
    for (int i = 0; i < 12; ++i)
        if (kFfmaTiles[i][0] == tm && kFfmaTiles[i][1] == bm && kFfmaTiles[i][2] == bn) ti = i;
    if (ti < 0 || bk != 16) return -1;
    return ti * 2 + (b_layout == NNJIT_B_NK ? 1 : 0);
}

int gemv_instance(int b_layout, int rows, int unroll) {
    const int ui = unroll == 2 ? 0 : unroll == 4 ? 1 : -1;
    if (ui < 0) return -1;
    if (b_layout == NNJIT_B_KN) return rows == 1 ? 6 + ui : -1;
    const int ri = rows == 1 ? 0 : rows == 2 ? 1 : rows == 4 ? 2 : -1;
    if (ri < 0) return -1;
    return ri * 2 + ui;
}

int gemv_w4_instance(int rows) {
    const int ri = rows == 16 ? 0 : rows == 32 ? 1 : -1;
    return ri < 0 ? -1 : kGemvW4FirstInstance + ri;
}

int gemv_tma_instance(int rows, int maxm) {
    const int ri = rows == 8 ? 0 : rows == 16 ? 1 : rows == 32 ? 2 : -1;
    const int mi = maxm == 1 ? 0 : maxm == ModelConstants::kGemvMaxM ? 1 : -1;
    if (ri < 0 || mi < 0) return -1;
    return kGemvTmaFirstInstance + ri * 2 + mi;
}

nnjit_status resolve_problem(const nnjit_matmul_desc* d, Problem* p, std::string* err) {
    if (!d || !p) { *err = "descriptor is NULL"; return NNJIT_ERR_INVALID_ARG; }
    if (d->M < 0 || d->N < 0 || d->K < 0) { *err = "M, N, K must be >= 0"; return NNJIT_ERR_INVALID_ARG; }
    if (d->batch < 1) { *err = "batch must be >= 1"; return NNJIT_ERR_INVALID_ARG; }
    if (d->dtype < NNJIT_F32_FFMA || d->dtype > NNJIT_W4_BF16) { *err = "unknown dtype"; return NNJIT_ERR_INVALID_ARG; }
    if (d->b_layout != NNJIT_B_KN && d->b_layout != NNJIT_B_NK) { *err = "unknown b_layout"; return NNJIT_ERR_INVALID_ARG; }
    if (d->has_bias != 0 && d->has_bias != 1) { *err = "has_bias must be 0 or 1"; return NNJIT_ERR_INVALID_ARG; }
    if ((d->epilogue & ~(NNJIT_EPI_RESIDUAL | 15)) != 0 || (d->epilogue & 15) > NNJIT_EPI_SILU) {
        *err = "unknown epilogue"; return NNJIT_ERR_INVALID_ARG;
    }
    const int64_t lim = (int64_t)1 << 31;
    if (d->M >= lim || d->N >= lim || d->K >= lim || d->batch >= lim) {
        *err = "dimensions must be < 2^31"; return NNJIT_ERR_INVALID_ARG;
    }
    if (d->lda < 0 || d->ldb < 0 || d->ldc < 0 || d->stride_a < 0 || d->stride_b < 0 || d->stride_c < 0) {
        *err = "leading dimensions and strides must be >= 0"; return NNJIT_ERR_INVALID_ARG;
    }
    Problem q;
    q.M = d->M; q.N = d->N; q.K = d->K; q.batch = d->batch;
    q.dtype = d->dtype; q.b_layout = d->b_layout; q.has_bias = d->has_bias; q.flags = d->flags;
    q.epilogue = d->epilogue;
    const int64_t b_rows = q.b_layout == NNJIT_B_KN ? q.K : q.N;
    const int64_t b_cols = q.b_layout == NNJIT_B_KN ? q.N : q.K;
    q.lda = d->lda ? d->lda : std::max<int64_t>(q.K, 1);
    q.ldb = d->ldb ? d->ldb : std::max<int64_t>(b_cols, 1);
    q.ldc = d->ldc ? d->ldc : std::max<int64_t>(q.N, 1);
    if (q.lda < q.K) { *err = "lda < K"; return NNJIT_ERR_INVALID_ARG; }
    if (q.ldb < b_cols) { *err = "ldb smaller than the row length of B"; return NNJIT_ERR_INVALID_ARG; }
    if (q.ldc < q.N) { *err = "ldc < N"; return NNJIT_ERR_INVALID_ARG; }
    q.stride_a = d->stride_a ? d->stride_a : q.M * q.lda;
    q.stride_b = d->stride_b ? d->stride_b : b_rows * q.ldb;
    q.stride_c = d->stride_c ? d->stride_c : q.M * q.ldc;
    if (q.batch > 1 && q.stride_c < q.M * q.ldc) {
        *err = "stride_c smaller than one C matrix: batch items would overlap";
        return NNJIT_ERR_INVALID_ARG;
    }
    const int64_t elim = (int64_t)1 << 40;
    if (q.batch * std::max<int64_t>(q.stride_a, q.M * q.lda) >= elim ||
        q.batch * std::max<int64_t>(q.stride_b, b_rows * q.ldb) >= elim ||
        q.batch * std::max<int64_t>(q.stride_c, q.M * q.ldc) >= elim) {
        *err = "operand extent too large"; return NNJIT_ERR_INVALID_ARG;
    }
    *p = q;
    return NNJIT_OK;
}

nnjit_status choose_family(const Problem& p, int* family, std::string* err) {
    if (p.dtype == NNJIT_F32_FFMA) { *family = NNJIT_FAMILY_FFMA; return NNJIT_OK; }
    if (p.dtype == NNJIT_W4_BF16) {
        if (p.M > ModelConstants::kGemvMaxM || p.batch != 1 || p.b_layout != NNJIT_B_NK) {
            *err = "4-bit weights are served for decode products: M <= 8, batch 1, B as [N][K]";
            return NNJIT_ERR_UNSUPPORTED;
        }
        if (!p.degenerate() && ((p.lda * 2) % 16 != 0 || p.ldb % 32 != 0 || p.N % 8 != 0)) {
            *err = "4-bit GEMV needs 16-byte rows of A (lda multiple of 8), of the codes (ldb "
                   "multiple of 32) and of the group-major scales (N multiple of 8)";
            return NNJIT_ERR_UNSUPPORTED;
        }
        *family = NNJIT_FAMILY_GEMV;
        return NNJIT_OK;
    }
    const int e = p.elem_bytes();
    if (p.dtype == NNJIT_BF16 && p.M <= ModelConstants::kGemvMaxM && p.batch == 1) {
        // B as [N][K]: x is staged and W streamed with 16-byte loads along K.  B as [K][N]
        // falls back to 2-byte loads when rows of W are not 16-byte aligned.
        if (!p.degenerate() && p.b_layout == NNJIT_B_NK &&
            ((p.lda * e) % 16 != 0 || (p.ldb * e) % 16 != 0)) {
            *err = "GEMV path with B as [N][K] needs 16-byte aligned rows of A and B "
                   "(lda, ldb multiples of 8)";
            return NNJIT_ERR_UNSUPPORTED;
        }
        *family = NNJIT_FAMILY_GEMV;
        return NNJIT_OK;
    }
    if (!p.degenerate()) {
        if ((p.lda * e) % 16 != 0 || (p.ldb * e) % 16 != 0) {
            *err = "tensor-core path needs 16-byte aligned row strides (TMA): lda*elem and "
                   "ldb*elem must be multiples of 16 bytes";
            return NNJIT_ERR_UNSUPPORTED;
        }
        if (p.batch > 1 && ((p.stride_a * e) % 16 != 0 || (p.stride_b * e) % 16 != 0)) {
            *err = "tensor-core path needs 16-byte aligned batch strides";
            return NNJIT_ERR_UNSUPPORTED;
        }
    }
    *family = NNJIT_FAMILY_TC;
    return NNJIT_OK;
}

nnjit_settings free_settings() {
    nnjit_settings s;
    s.raster = s.kgroup = s.reduce = NNJIT_SETTING_FREE;
    return s;
}

int setting_of(const nnjit_settings& s, int axis) {
    switch (axis) {
        case 0: return s.raster;
        case 1: return s.kgroup;
        case 2: return s.reduce;
        default: return NNJIT_SETTING_FREE;
    }
}

bool settings_valid(const nnjit_settings& s, std::string* err) {
    // reduce: 0 second kernel, 1 cluster (DSMEM), 2 CTA-pair stream-K
    const int lo[kSettingAxes] = {0, 1, 0}, hi[kSettingAxes] = {1, 2, 2};
    const char* names[kSettingAxes] = {"raster", "kgroup", "reduce"};
    for (int a = 0; a < kSettingAxes; ++a) {
        const int v = setting_of(s, a);
        if (v != NNJIT_SETTING_FREE && (v < lo[a] || v > hi[a])) {
            *err = std::string("setting ") + names[a] + " out of range";
            return false;
        }
    }
    return true;
}

int candidate_setting(const Problem& p, const nnjit_candidate& c, int axis) {
    if (c.family != NNJIT_FAMILY_TC) return -1;
    switch (axis) {
        case 0: return c.raster;
        case 1: return c.bk / (128 / p.elem_bytes());
        case 2: return c.reduce;
        default: return -1;
    }
}

bool setting_twins(const Problem& p, const nnjit_candidate& a, const nnjit_candidate& b, int axis) {
    if (a.family != NNJIT_FAMILY_TC || b.family != NNJIT_FAMILY_TC) return false;
    if (a.bm != b.bm || a.bn != b.bn || a.split_k != b.split_k) return false;
    for (int o = 0; o < kSettingAxes; ++o)
        if (o != axis && candidate_setting(p, a, o) != candidate_setting(p, b, o)) return false;
    return candidate_setting(p, a, axis) != candidate_setting(p, b, axis);
}

void apply_settings(const Problem& p, const nnjit_settings& s, std::vector<nnjit_candidate>* v) {
    for (int axis = 0; axis < kSettingAxes; ++axis) {
        const int fixed = setting_of(s, axis);
        if (fixed == NNJIT_SETTING_FREE) continue;
        std::vector<nnjit_candidate> kept;
        for (const auto& c : *v) {
            bool drop = false;
            if (c.family == NNJIT_FAMILY_TC && candidate_setting(p, c, axis) != fixed)
                for (const auto& t : *v)
                    if (candidate_setting(p, t, axis) == fixed && setting_twins(p, c, t, axis)) {
                        drop = true;
                        break;
                    }
            if (!drop) kept.push_back(c);
        }
        *v = std::move(kept);
    }
}

nnjit_status build_space(const Problem& p, const nnjit_device_limits& lim, const nnjit_settings& set,
                         std::vector<nnjit_candidate>* out, int64_t* naive, std::string* err) {
    if (!settings_valid(set, err)) return NNJIT_ERR_INVALID_ARG;
    if (lim.sm_count <= 0 || lim.smem_per_sm <= 0 || lim.smem_per_block_optin <= 0 ||
        lim.regs_per_sm <= 0 || lim.max_threads_per_sm <= 0 || lim.max_blocks_per_sm <= 0 ||
        lim.tmem_cols_per_sm < 0) {
        *err = "device limits must be positive";
        return NNJIT_ERR_INVALID_ARG;
    }
    int family = 0;
    nnjit_status st = choose_family(p, &family, err);
    if (st != NNJIT_OK) return st;
    std::vector<nnjit_candidate> v;
    int64_t nv = 0;
    if (family == NNJIT_FAMILY_TC) {
        if (lim.cc_major != 10 || lim.tmem_cols_per_sm < 128) {
            *err = "tensor-core family needs an sm_10x device with tensor memory";
            return NNJIT_ERR_UNSUPPORTED;
        }
        tc_space(p, lim, v, &nv);
    } else if (family == NNJIT_FAMILY_FFMA) {
        ffma_space(p, lim, v, &nv);
    } else {
        gemv_space(p, lim, v, &nv);
    }
    if (v.empty()) {
        *err = "no candidate fits the device limits";
        return NNJIT_ERR_UNSUPPORTED;
    }
    // Evaluation order (Sec. 5.2): most blocks per core first; then the predicted cost;
    // ties keep enumeration order.
    std::stable_sort(v.begin(), v.end(), [](const nnjit_candidate& a, const nnjit_candidate& b) {
        if (a.blocks_per_sm != b.blocks_per_sm) return a.blocks_per_sm > b.blocks_per_sm;
        return a.predicted_cost < b.predicted_cost;
    });
    apply_settings(p, set, &v);
    *out = std::move(v);
    if (naive) *naive = nv;
    return NNJIT_OK;
}

}  // namespace nnjit
