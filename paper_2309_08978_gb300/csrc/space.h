// Lite kernel-configuration space (host only).
//
// Sec. 5.2 and Table 1 of the paper: tile sizes decide how a kernel uses registers,
// L1/shared memory, threads and warps; formulas of those usages plus a few heuristics
// prune the space to a few dozen candidates, evaluated from the most to the fewest
// blocks per core.  This file restates that scheme for three sm_103a kernel families.
#pragma once

#include <cstdint>
#include <string>
#include <vector>

#include "../../include/nnjit.h"

namespace nnjit {

// Descriptor with every default resolved and validated.
struct Problem {
    int64_t M = 0, N = 0, K = 0, batch = 1;
    int dtype = NNJIT_BF16;
    int b_layout = NNJIT_B_NK;
    int64_t lda = 0, ldb = 0, ldc = 0;
    int64_t stride_a = 0, stride_b = 0, stride_c = 0;
    int has_bias = 0;
    uint32_t flags = 0;
    int epilogue = NNJIT_EPI_NONE;
    // bytes per element of A (and of B, except for 4-bit weights)
    int elem_bytes() const { return dtype == NNJIT_BF16 || dtype == NNJIT_W4_BF16 ? 2 : 4; }
    bool degenerate() const { return M == 0 || N == 0 || K == 0; }
    // 4-bit weight blob: scale block offset and total bytes (see nnjit.h)
    int64_t w4_scale_offset() const { return (N * (ldb / 2) + 255) / 256 * 256; }
    int64_t w4_groups() const { return (K + 127) / 128; }
    int64_t w4_blob_bytes() const { return w4_scale_offset() + w4_groups() * N * 2; }
    // extent of B in bytes over every batch item
    int64_t b_bytes() const {
        if (dtype == NNJIT_W4_BF16) return w4_blob_bytes();
        const int64_t rows = b_layout == NNJIT_B_KN ? K : N, cols = b_layout == NNJIT_B_KN ? N : K;
        return ((batch - 1) * stride_b + (rows - 1) * ldb + cols) * elem_bytes();
    }
};

// Model constants of the ordering cost (readings; see the design notes).
struct ModelConstants {
    static constexpr int kFeedBytesPerClk = 64;      // L2->SM operand feed per SM
    static constexpr int kHbmBytesPerClk = 3500;     // chip-wide HBM bytes per SM clock
    static constexpr int kLaunchClk = 4000;          // cost of one extra kernel launch (the
                                                     // split-K sum: about 2 us measured)
    static constexpr int kRegRelaxPct = 50;          // Table 1 register formula covers half
    static constexpr int kTcRegsPerThread = 176;     // tcgen05 kernel: ptxas reports 72-173
    static constexpr int kTcThreads = 192;           // 6 warps: TMA, MMA, 4 x epilogue
    static constexpr int kTcBM = 128;
    static constexpr int kTcFixedSmem = 1024 + 256 + 32768;  // alignment slack, barriers,
                                                              // epilogue staging buffers
    static constexpr int kTcMaxStages = 8;
    static constexpr int kTcPairAccCols = 512;        // TMEM columns of a CTA-pair tile kernel (2 x 256)
    static constexpr int kMmaN256Clk = 128;           // tensor pipe: one M = 128, N = 256 MMA
    static constexpr int kMmaIssueClk = 57;           // issuing thread: one tcgen05.mma
    static constexpr int kSlotSyncClk = 226;          // issuing thread: ring-slot wait + commit
    static constexpr int kIssueShowDiv = 8;           // 1/8 of the issue path is not hidden
                                                      // behind the operand feed
    static constexpr int kDsmemReduceBytesPerClk = 5; // cluster split-K: partial-tile exchange
                                                      // and sum through DSMEM, per SM
    static constexpr int kGemvMaxM = 8;
    static constexpr int kGemvMaxSmem = 64 * 1024;
    static constexpr int kGemvTmaKc = 256;           // K elements per TMA GEMV ring stage
    static constexpr int kGemvTmaThreads = 160;      // producer warp + 4 consumer warps
    static constexpr int kGemvW4Kc = 1024;           // K codes per 4-bit GEMV ring stage
};

// Resolve defaults and validate.  Returns NNJIT_OK or an error with `err` set.
nnjit_status resolve_problem(const nnjit_matmul_desc* d, Problem* p, std::string* err);

// Which family serves the problem (a1 of the hot path), or UNSUPPORTED with `err`.
nnjit_status choose_family(const Problem& p, int* family, std::string* err);

// Fixed settings (nnjit_settings, the primitive vector of Sec. 5.1).  Axis a of a
// tensor-core candidate: 0 raster, 1 k-blocks per ring slot, 2 split-K reduction; -1 for
// candidates of other families.
constexpr int kSettingAxes = 3;
nnjit_settings free_settings();
int setting_of(const nnjit_settings& s, int axis);
bool settings_valid(const nnjit_settings& s, std::string* err);
int candidate_setting(const Problem& p, const nnjit_candidate& c, int axis);
// True if a and b are the same candidate but for axis `axis` (every other searched field
// equal: bm, bn, split_k and the other settings).
bool setting_twins(const Problem& p, const nnjit_candidate& a, const nnjit_candidate& b, int axis);
// Drop, axis by axis in order, every candidate whose value differs from a fixed one while
// its twin with the fixed value is in the space.  Order is preserved.
void apply_settings(const Problem& p, const nnjit_settings& s, std::vector<nnjit_candidate>* v);

// Build the ordered lite space, then apply the fixed settings.  naive = size before
// pruning.
nnjit_status build_space(const Problem& p, const nnjit_device_limits& lim, const nnjit_settings& set,
                         std::vector<nnjit_candidate>* out, int64_t* naive, std::string* err);

// Precompiled-instance index helpers (kept in one place so the registry and the space
// agree).
// kg: k-blocks per ring slot (2 only for 128-row persistent tiles with BN <= 128)
int tc_instance(int dtype, int b_layout, int bn, int cluster, int bm, int kg = 1);  // 0..43
// 256 x 256 tiles on CTA pairs (tcgen05 cta_group::2), B as [N][K]: 44 (bf16), 45 (tf32).
constexpr int kTcPairFirstInstance = 44;
int ffma_instance(int tm, int bm, int bn, int bk, int b_layout);  // 0..23, -1 if none
int gemv_instance(int b_layout, int rows, int unroll);        // 0..7, -1 if none
// TMA-fed GEMV (B as [N][K]): rows per stage 8/16/32, M <= maxm (1 or 8).
constexpr int kGemvTmaFirstInstance = 8;
int gemv_tma_instance(int rows, int maxm);                     // 8..13, -1 if none
// TMA-fed GEMV over 4-bit weights (NNJIT_W4_BF16): rows per stage 16/32.
constexpr int kGemvW4FirstInstance = 14;
int gemv_w4_instance(int rows);                                // 14..15, -1 if none

}  // namespace nnjit
