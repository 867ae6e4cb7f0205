"""Oracle for the lite space (Sec. 5.2, Table 1, Table 2) -- TEST INFRASTRUCTURE ONLY.

Two parts, both plain Python over integers:

* ``table1_usage`` -- the tile-based hardware-usage formulas of Table 1 as the paper
  writes them (WebGPU variant): Reg_thread, L1_block, Thread_block, Warp_block and
  Block_core = min(RegLimit, L1Limit, WarpLimit).

* ``build_space`` -- the lite space the GPU library is specified to build for one
  problem on one device, restated rule by rule from its written description (Table 1
  usage formulas with the Blackwell resource limits, heuristic 2's power-of-two tiles,
  the split-K and pruning rules, the evaluation order of Sec. 5.2: most blocks per core
  first, then the predicted cost, then enumeration order).  Every quantity is an integer
  and every division a floor or ceiling of positive integers, so the library's
  enumeration must match element by element.

The library shares no code with this module.
"""
from __future__ import annotations

from dataclasses import dataclass

# enum values of the C ABI
F32_FFMA, TF32, BF16, W4_BF16 = 0, 1, 2, 3
B_KN, B_NK = 0, 1
FAMILY_FFMA, FAMILY_TC, FAMILY_GEMV = 0, 1, 2
INVALID_ARG, UNSUPPORTED = 1, 2

# model constants (readings of the paper's unstated relaxation ratio and cost model)
FEED_BYTES_PER_CLK = 64       # per-SM L2 -> SM operand feed
HBM_BYTES_PER_CLK = 3500      # chip-wide HBM bytes per SM clock
LAUNCH_CLK = 4000             # one extra kernel launch (the split-K sum after the GEMM)
REG_SHARE_PCT = 50            # Table 1's Reg_thread is this share of a thread's registers
TC_REGS = 176                 # registers per thread of the tensor-core kernel (ptxas: 72-173)
TC_THREADS = 192
TC_BM = 128
TC_FIXED_SMEM = 1024 + 256 + 32768   # alignment slack, barriers, epilogue staging
TC_MAX_STAGES = 8
TC_PAIR_ACC_COLS = 512        # TMEM columns of the CTA-pair tile kernel (2 x 256)
TC_PAIR_FIRST = 44            # instance ids of the CTA-pair tile kernel (bf16, tf32)
MMA_N256_CLK = 128            # tensor pipe: one M = 128, N = 256 MMA instruction
MMA_ISSUE_CLK = 57            # issuing thread: one tcgen05.mma
SLOT_SYNC_CLK = 226           # issuing thread: one ring-slot barrier wait + commit
ISSUE_SHOW = 8                # 1/8 of the issue path is not hidden behind the feed
DSMEM_REDUCE_BYTES_PER_CLK = 5   # cluster split-K partial exchange and sum, per SM
GEMV_MAX_M = 8
GEMV_MAX_SMEM = 64 * 1024
GEMV_TMA_KC = 256             # K elements per ring stage of the TMA-fed GEMV
GEMV_TMA_THREADS = 160        # producer warp + 4 consumer warps
GEMV_TMA_FIRST = 8            # first instance id of the TMA-fed GEMV kernels
GEMV_W4_FIRST = 14            # first instance id of the 4-bit-weight GEMV kernels
GEMV_W4_KC = 1024             # 4-bit codes per ring stage and row

CANDIDATE_FIELDS = ("family", "bm", "bn", "bk", "tm", "tn", "stages", "split_k", "raster",
                    "threads", "smem_bytes", "tmem_cols", "regs_per_thread", "blocks_per_sm",
                    "grid", "wave_eff_ppm", "instance", "predicted_cost", "reduce", "cluster_m")


def cdiv(a: int, b: int) -> int:
    return -(-a // b)


def pow2_at_least(x: int) -> int:
    p = 1
    while p < x:
        p *= 2
    return p


# ---------------------------------------------------------------------------- Table 1

def table1_usage(x0, r0, y0, x1, r1, y1, warp_width, total_regs_per_core, l1_size_per_core,
                 total_warps_per_core):
    """Table 1, hardware resource usage for WebGPU, in the paper's units (registers and
    elements; the caller scales L1 by the element size when comparing to bytes)."""
    reg_thread = x0 * r0 + r0 * y0 + x0 * y0
    l1_block = x1 * r1 + r1 * y1 + x1 * y1
    thread_block = (x1 // x0) * (y1 // y0)
    warp_block = thread_block // warp_width
    reg_limit = total_regs_per_core // (reg_thread * thread_block)
    l1_limit = l1_size_per_core // l1_block
    warp_limit = total_warps_per_core // warp_block
    return {"Reg_thread": reg_thread, "L1_block": l1_block, "Thread_block": thread_block,
            "Warp_block": warp_block, "RegLimit": reg_limit, "L1Limit": l1_limit,
            "WarpLimit": warp_limit, "Block_core": min(reg_limit, l1_limit, warp_limit)}


# ---------------------------------------------------------------------------- problems

@dataclass
class Problem:
    M: int
    N: int
    K: int
    batch: int
    dtype: int
    b_layout: int
    lda: int
    ldb: int
    ldc: int
    stride_a: int
    stride_b: int
    stride_c: int
    has_bias: int

    @property
    def elem(self) -> int:
        return 2 if self.dtype in (BF16, W4_BF16) else 4

    @property
    def degenerate(self) -> bool:
        return self.M == 0 or self.N == 0 or self.K == 0


class SpaceError(Exception):
    def __init__(self, status):
        super().__init__(status)
        self.status = status


def resolve(M, N, K, batch=1, dtype=BF16, b_layout=B_NK, lda=0, ldb=0, ldc=0, stride_a=0,
            stride_b=0, stride_c=0, has_bias=0) -> Problem:
    """Defaults and validation of the problem descriptor (packed when zero)."""
    if M < 0 or N < 0 or K < 0 or batch < 1:
        raise SpaceError(INVALID_ARG)
    if dtype not in (F32_FFMA, TF32, BF16, W4_BF16) or b_layout not in (B_KN, B_NK) or has_bias not in (0, 1):
        raise SpaceError(INVALID_ARG)
    if max(M, N, K, batch) >= 2 ** 31:
        raise SpaceError(INVALID_ARG)
    if min(lda, ldb, ldc, stride_a, stride_b, stride_c) < 0:
        raise SpaceError(INVALID_ARG)
    b_rows, b_cols = (K, N) if b_layout == B_KN else (N, K)
    lda = lda or max(K, 1)
    ldb = ldb or max(b_cols, 1)
    ldc = ldc or max(N, 1)
    if lda < K or ldb < b_cols or ldc < N:
        raise SpaceError(INVALID_ARG)
    stride_a = stride_a or M * lda
    stride_b = stride_b or b_rows * ldb
    stride_c = stride_c or M * ldc
    if batch > 1 and stride_c < M * ldc:
        raise SpaceError(INVALID_ARG)
    lim = 2 ** 40
    if (batch * max(stride_a, M * lda) >= lim or batch * max(stride_b, b_rows * ldb) >= lim or
            batch * max(stride_c, M * ldc) >= lim):
        raise SpaceError(INVALID_ARG)
    return Problem(M, N, K, batch, dtype, b_layout, lda, ldb, ldc, stride_a, stride_b, stride_c,
                   has_bias)


def family_of(p: Problem) -> int:
    """Exact FP32 -> SIMT; bf16 with M <= 8 (one matrix) -> GEMV; else tensor cores, which
    read operands with TMA and so need 16-byte row and batch strides."""
    if p.dtype == F32_FFMA:
        return FAMILY_FFMA
    e = p.elem
    if p.dtype == W4_BF16:
        # 4-bit weights: decode products only, 16-byte rows of x, codes and group scales
        if p.M > GEMV_MAX_M or p.batch != 1 or p.b_layout != B_NK:
            raise SpaceError(UNSUPPORTED)
        if not p.degenerate and ((p.lda * 2) % 16 or p.ldb % 32 or p.N % 8):
            raise SpaceError(UNSUPPORTED)
        return FAMILY_GEMV
    if p.dtype == BF16 and p.M <= GEMV_MAX_M and p.batch == 1:
        if not p.degenerate and p.b_layout == B_NK and ((p.lda * e) % 16 or (p.ldb * e) % 16):
            raise SpaceError(UNSUPPORTED)
        return FAMILY_GEMV
    if not p.degenerate:
        if (p.lda * e) % 16 or (p.ldb * e) % 16:
            raise SpaceError(UNSUPPORTED)
        if p.batch > 1 and ((p.stride_a * e) % 16 or (p.stride_b * e) % 16):
            raise SpaceError(UNSUPPORTED)
    return FAMILY_TC


# ---------------------------------------------------------------------------- helpers

def block_core(lim, regs, threads, smem, tmem):
    """Table 1's Block_core with the Blackwell resources: the fewest CTAs allowed by the
    register file, shared memory (the L1Limit), warps, tensor-memory columns, blocks."""
    reg_limit = lim["regs_per_sm"] // max(1, regs * threads)
    # each resident CTA also holds the SM's per-block shared-memory reservation
    reserved = max(0, lim["smem_per_sm"] - lim["smem_per_block_optin"])
    l1_limit = lim["smem_per_sm"] // (smem + reserved) if smem > 0 else lim["max_blocks_per_sm"]
    warp_limit = (lim["max_threads_per_sm"] // 32) // max(1, threads // 32)
    tmem_limit = lim["tmem_cols_per_sm"] // tmem if tmem > 0 else lim["max_blocks_per_sm"]
    return min(reg_limit, l1_limit, warp_limit, tmem_limit, lim["max_blocks_per_sm"])


def _blank():
    c = dict.fromkeys(CANDIDATE_FIELDS, 0)
    c["split_k"] = 1
    c["instance"] = -1
    c["cluster_m"] = 1
    return c


def tc_instance(dtype, b_layout, bn, cluster, bm, kg=1):
    if kg == 2:
        return 36 + ((0 if dtype == BF16 else 1) * 2 + (1 if b_layout == B_KN else 0)) * 2 + {64: 0, 128: 1}[bn]
    variant = 2 if bm == 64 else (1 if cluster else 0)
    return variant * 12 + ((0 if dtype == BF16 else 1) * 2 + (1 if b_layout == B_KN else 0)) * 3 + \
        {64: 0, 128: 1, 256: 2}[bn]


FFMA_TILES = [(4, 32, 32), (4, 32, 64), (4, 32, 128), (4, 64, 32), (4, 64, 64), (4, 128, 32),
              (8, 32, 128), (8, 64, 64), (8, 64, 128), (8, 128, 32), (8, 128, 64), (8, 128, 128)]


def ffma_instance(t0, bm, bn, layout):
    return FFMA_TILES.index((t0, bm, bn)) * 2 + (1 if layout == B_NK else 0)


def gemv_instance(layout, rows, unroll):
    u = {2: 0, 4: 1}[unroll]
    if layout == B_KN:
        return 6 + u
    return {1: 0, 2: 1, 4: 2}[rows] * 2 + u


def gemv_tma_instance(rows, maxm):
    return GEMV_TMA_FIRST + {8: 0, 16: 1, 32: 2}[rows] * 2 + {1: 0, GEMV_MAX_M: 1}[maxm]


# ---------------------------------------------------------------------------- families

def _tc(p, lim):
    e = p.elem
    bk = 128 // e
    M, N, K = max(p.M, 1), max(p.N, 1), max(p.K, 1)
    num_kb = cdiv(K, bk)
    out = []
    for bm, bn, kg in [(m, n, g) for m in (TC_BM, 64) for n in (64, 128, 256) for g in (1, 2)]:
        if bn > 64 and bn > pow2_at_least(N):
            continue
        # 64-row tiles only where 128-row tiles would leave SMs idle
        if bm == 64 and p.batch * cdiv(M, TC_BM) * cdiv(N, bn) >= lim["sm_count"]:
            continue
        # two k-blocks per ring slot where the MMA issue path, not the tensor pipe, sets
        # the pace: 128-row tiles with BN <= 128
        if kg == 2 and (bm != TC_BM or bn > 128):
            continue
        kb_bytes = (bm + bn) * 128
        stage = kg * kb_bytes
        stages = min(TC_MAX_STAGES, (lim["smem_per_block_optin"] - TC_FIXED_SMEM) // stage)
        if stages < 2:
            continue
        smem = stages * stage + TC_FIXED_SMEM
        tmem = pow2_at_least(max(32, 2 * bn))
        if tmem > lim["tmem_cols_per_sm"]:
            continue
        blk = block_core(lim, TC_REGS, TC_THREADS, smem, tmem)
        if blk < 1:
            continue
        tiles_m, tiles_n = cdiv(M, bm), cdiv(N, bn)
        tiles = p.batch * tiles_m * tiles_n
        for split in (1, 2, 4, 8):
            if split > 1 and (tiles * (split // 2) >= lim["sm_count"] or num_kb < 4 * split):
                continue
            for reduce in ((0, 1) if split > 1 and kg == 1 else (0,)):
                for raster in (0, 1):
                    if raster == 1 and (tiles_m == 1 or tiles_n == 1):
                        continue
                    if reduce == 1 and (bm != TC_BM or raster == 1 or stages * stage < TC_BM * (bn + 4) * 4):
                        continue
                    c = _blank()
                    work = tiles * split
                    slots = lim["sm_count"] * blk
                    live = min(work, slots)
                    waves = cdiv(work, live)
                    # per k-block: tensor pipe, issuing thread, operand feed
                    t_tensor = 4 * max(MMA_N256_CLK // 4, MMA_N256_CLK * bn // 256)
                    t_issue = 4 * MMA_ISSUE_CLK + SLOT_SYNC_CLK // kg
                    t_kb = max(t_tensor, t_issue, cdiv(kb_bytes, FEED_BYTES_PER_CLK)) + t_issue // ISSUE_SHOW
                    cost = waves * t_kb * cdiv(num_kb, split)
                    if split > 1 and reduce == 0:
                        cost += LAUNCH_CLK + cdiv(2 * split * p.batch * M * N * 4, HBM_BYTES_PER_CLK)
                    if split > 1 and reduce == 1:
                        cost += waves * (TC_BM * bn * 4 // DSMEM_REDUCE_BYTES_PER_CLK)
                    c.update(family=FAMILY_TC, bm=bm, bn=bn, bk=bk * kg, stages=stages, split_k=split,
                             raster=raster, threads=TC_THREADS, smem_bytes=smem, tmem_cols=tmem,
                             regs_per_thread=TC_REGS, blocks_per_sm=blk,
                             grid=work if reduce else live, wave_eff_ppm=work * 1000000 // (waves * live),
                             instance=tc_instance(p.dtype, p.b_layout, bn, reduce, bm, kg=kg),
                             predicted_cost=cost, reduce=reduce)
                    out.append(c)
    # 256 x 256 tiles on CTA pairs (tcgen05 cta_group::2), B as [N][K]: an SM receives its
    # 128 rows of A and half of the B tile per k-block; one thread issues for both SMs
    if p.b_layout == B_NK and M > TC_BM and lim["sm_count"] >= 2:
        kb_bytes = (TC_BM + 128) * 128
        stages = min(TC_MAX_STAGES, (lim["smem_per_block_optin"] - TC_FIXED_SMEM) // kb_bytes)
        smem = stages * kb_bytes + TC_FIXED_SMEM
        tmem = TC_PAIR_ACC_COLS
        blk = block_core(lim, TC_REGS, TC_THREADS, smem, tmem)
        tiles2_m, tiles_n = cdiv(M, 256), cdiv(N, 256)
        pairs = p.batch * tiles2_m * tiles_n
        if stages >= 2 and blk >= 1 and tmem <= lim["tmem_cols_per_sm"]:
            for raster in (0, 1):
                if raster == 1 and (tiles2_m == 1 or tiles_n == 1):
                    continue
                live = min(pairs, max(1, lim["sm_count"] * blk // 2))
                waves = cdiv(pairs, live)
                t_issue = 4 * MMA_ISSUE_CLK + SLOT_SYNC_CLK
                t_kb = max(4 * MMA_N256_CLK, t_issue, cdiv(kb_bytes, FEED_BYTES_PER_CLK)) + t_issue // ISSUE_SHOW
                c = _blank()
                c.update(family=FAMILY_TC, bm=256, bn=256, bk=bk, stages=stages, raster=raster,
                         threads=TC_THREADS, smem_bytes=smem, tmem_cols=tmem, regs_per_thread=TC_REGS,
                         blocks_per_sm=blk, cluster_m=2, grid=2 * live,
                         wave_eff_ppm=pairs * 1000000 // (waves * live),
                         predicted_cost=waves * t_kb * num_kb,
                         instance=TC_PAIR_FIRST + (0 if p.dtype == BF16 else 1))
                out.append(c)
                # stream-K over the last waves: whole waves but the last as whole tiles, the
                # k-blocks of the rest shared evenly by all pairs
                pair_slots = max(1, lim["sm_count"] * blk // 2)
                # only from two whole waves on (with all tiles in stream-K the hand-offs sit
                # on the critical path and the launch measured slower than whole tiles)
                if pairs % pair_slots and pairs // pair_slots >= 2:
                    waves_sk = pairs // pair_slots
                    dp = (waves_sk - 1) * pair_slots
                    iters = (pairs - dp) * num_kb
                    share = iters // pair_slots
                    if share >= 4:
                        per_pair = cdiv(iters, pair_slots)
                        t = dict(c)
                        t.update(reduce=2, grid=2 * pair_slots,
                                 wave_eff_ppm=pairs * num_kb * 1000000 // (dp * num_kb + pair_slots * per_pair),
                                 predicted_cost=(dp // pair_slots) * t_kb * num_kb + t_kb * per_pair +
                                 (1 + cdiv(num_kb, share)) * (128 * 256 * 4 // FEED_BYTES_PER_CLK))
                        out.append(t)
    return out, 2 * 3 * (TC_MAX_STAGES - 1) * 4 * 2 * 2 * 2 * 2


def _ffma(p, lim):
    M, N, K = max(p.M, 1), max(p.N, 1), max(p.K, 1)
    out = []
    for t0 in (4, 8):
        for bm in (32, 64, 128):
            for bn in (32, 64, 128):
                threads = (bm // t0) * (bn // t0)              # Thread_block
                if threads < 64 or threads > 256:              # heuristic 5 (and >= 2 warps)
                    continue
                if (bm > 32 and bm > pow2_at_least(M)) or (bn > 32 and bn > pow2_at_least(N)):
                    continue
                bk = 16
                reg_paper = t0 * 1 + 1 * t0 + t0 * t0          # Reg_thread, r0 = 1
                regs = cdiv(reg_paper * 100, REG_SHARE_PCT)
                smem = 2 * bk * ((bm + 4) + (bn + 4)) * 4      # double-buffered, padded rows
                if smem > lim["smem_per_block_optin"]:
                    continue
                blk = block_core(lim, regs, threads, smem, 0)
                if blk < 1:
                    continue
                tiles = p.batch * cdiv(M, bm) * cdiv(N, bn)
                for split in (1, 2, 4, 8):
                    if split > 1 and (tiles * (split // 2) >= lim["sm_count"] or K < 2 * split * bk):
                        continue
                    grid = tiles * split
                    slots = lim["sm_count"] * blk
                    waves = cdiv(grid, slots)
                    per_sm = cdiv(grid, lim["sm_count"])
                    warps = min(per_sm, blk) * threads // 32
                    util = min(100, max(1, warps * 100 // 16))
                    cost = per_sm * cdiv(bm * bn * cdiv(K, split), 128) * 100 // util
                    if split > 1:
                        cost += LAUNCH_CLK + cdiv(2 * split * p.batch * M * N * 4, HBM_BYTES_PER_CLK)
                    c = _blank()
                    c.update(family=FAMILY_FFMA, bm=bm, bn=bn, bk=bk, tm=t0, tn=t0, stages=2,
                             split_k=split, threads=threads, smem_bytes=smem, regs_per_thread=regs,
                             blocks_per_sm=blk, grid=grid, wave_eff_ppm=grid * 1000000 // (waves * slots),
                             instance=ffma_instance(t0, bm, bn, p.b_layout), predicted_cost=cost)
                    out.append(c)
    return out, 2 * 3 * 3 * 2 * 4


def gemv_w4_instance(rows):
    return GEMV_W4_FIRST + {16: 0, 32: 1}[rows]


def _gemv_w4(p, lim):
    """4-bit weights: a ring stage holds `rows` weight rows x 1024 codes (512 bytes a row),
    1024 elements of every row of x and the rows' 8 group scales, padded to 1 KB."""
    M, N, K = max(p.M, 1), max(p.N, 1), max(p.K, 1)
    wbytes = N * K // 2 + cdiv(K, 128) * N * 2
    chunks = cdiv(K, GEMV_W4_KC)
    out = []
    for rows in (16, 32):
        groups = cdiv(N, rows)
        for stages in (4, 8):
            for split in (1, 2, 4, 8):
                cps = cdiv(chunks, split)
                if split > 1 and (cps < 2 or (split - 1) * cps >= chunks or
                                  groups * (split // 2) >= 2 * lim["sm_count"]):
                    continue
                stage_bytes = cdiv(rows * (GEMV_W4_KC // 2 + 16) + M * GEMV_W4_KC * 2, 1024) * 1024
                smem = 1024 + stages * stage_bytes + 256 + rows * 128
                if smem > lim["smem_per_block_optin"]:
                    continue
                regs = 88 if rows == 16 else 112
                blk = block_core(lim, regs, GEMV_TMA_THREADS, smem, 0)
                if blk < 1:
                    continue
                items = groups * split
                slots = lim["sm_count"] * blk
                grid = min(items, slots)
                inflight = min(cdiv(grid, lim["sm_count"]), blk) * stages * rows * GEMV_W4_KC // 2
                eff = min(100, max(1, inflight * 100 // 32768))
                cost = cdiv(wbytes, HBM_BYTES_PER_CLK) * 100 // eff
                cost = cost * cdiv(items, lim["sm_count"]) * lim["sm_count"] // items
                if split > 1:
                    cost += LAUNCH_CLK + cdiv(2 * split * M * N * 4, HBM_BYTES_PER_CLK)
                c = _blank()
                c.update(family=FAMILY_GEMV, bm=M, bn=rows, bk=GEMV_W4_KC, tm=rows // 16, tn=1,
                         stages=stages, split_k=split, threads=GEMV_TMA_THREADS, smem_bytes=smem,
                         regs_per_thread=regs, blocks_per_sm=blk, grid=grid,
                         wave_eff_ppm=grid * 1000000 // slots,
                         instance=gemv_w4_instance(rows), predicted_cost=cost)
                out.append(c)
    return out, 2 * 2 * 4


def _gemv(p, lim):
    if p.dtype == W4_BF16:
        return _gemv_w4(p, lim)
    M, N, K = max(p.M, 1), max(p.N, 1), max(p.K, 1)
    wbytes = N * K * 2
    out = []
    if p.b_layout == B_NK:
        for threads in (128, 256):
            for rows in (1, 2, 4):
                for unroll in (2, 4):
                    warps = threads // 32
                    ctas_n = cdiv(N, warps * rows)
                    for split in (1, 2, 4, 8):
                        kper = cdiv(cdiv(K, split), 8) * 8
                        if split > 1 and (kper < 256 * unroll or ctas_n * (split // 2) >= 2 * lim["sm_count"]):
                            continue
                        smem = cdiv(M * kper * 2, 16) * 16
                        if smem > GEMV_MAX_SMEM or smem > lim["smem_per_block_optin"]:
                            continue
                        regs = 40 + rows * M + 4 * unroll * rows + 8
                        blk = block_core(lim, regs, threads, smem, 0)
                        if blk < 1:
                            continue
                        # at most as many CTAs as fit at once; beyond that warps take
                        # row groups round-robin
                        grid = min(ctas_n, lim["sm_count"] * blk) * split
                        slots = lim["sm_count"] * blk
                        waves = cdiv(grid, slots)
                        inflight = min(cdiv(grid, lim["sm_count"]), blk) * threads * unroll * rows * 16
                        eff = min(100, max(1, inflight * 100 // 32768))
                        cost = cdiv(wbytes, HBM_BYTES_PER_CLK) * 100 // eff
                        if split > 1:
                            cost += LAUNCH_CLK + cdiv(2 * split * M * N * 4, HBM_BYTES_PER_CLK)
                        c = _blank()
                        c.update(family=FAMILY_GEMV, bm=M, bn=warps * rows, bk=min(kper, 1 << 30), tm=rows,
                                 tn=1, stages=unroll, split_k=split, threads=threads, smem_bytes=smem,
                                 regs_per_thread=regs, blocks_per_sm=blk, grid=grid,
                                 wave_eff_ppm=grid * 1000000 // (waves * slots),
                                 instance=gemv_instance(B_NK, rows, unroll), predicted_cost=cost)
                        out.append(c)
        # TMA-fed kernels: `stages` boxes of `rows` weight rows x 256 K elements in flight
        maxm = 1 if M == 1 else GEMV_MAX_M
        chunks = cdiv(K, GEMV_TMA_KC)
        for rows in (8, 16, 32):
            groups = cdiv(N, rows)
            for stages in (4, 8):
                for split in (1, 2, 4, 8):
                    cps = cdiv(chunks, split)
                    if split > 1 and (cps < 2 or (split - 1) * cps >= chunks or
                                      groups * (split // 2) >= 2 * lim["sm_count"]):
                        continue
                    smem = 128 + stages * (rows + M) * GEMV_TMA_KC * 2
                    if smem > lim["smem_per_block_optin"]:
                        continue
                    regs = 40 if maxm == 1 else 96 + 3 * rows
                    blk = block_core(lim, regs, GEMV_TMA_THREADS, smem, 0)
                    if blk < 1:
                        continue
                    items = groups * split
                    slots = lim["sm_count"] * blk
                    grid = min(items, slots)
                    inflight = min(cdiv(grid, lim["sm_count"]), blk) * stages * rows * GEMV_TMA_KC * 2
                    eff = min(100, max(1, inflight * 100 // 32768))
                    cost = cdiv(wbytes, HBM_BYTES_PER_CLK) * 100 // eff
                    # the SM with the most items finishes last
                    cost = cost * cdiv(items, lim["sm_count"]) * lim["sm_count"] // items
                    if split > 1:
                        cost += LAUNCH_CLK + cdiv(2 * split * M * N * 4, HBM_BYTES_PER_CLK)
                    c = _blank()
                    c.update(family=FAMILY_GEMV, bm=M, bn=rows, bk=GEMV_TMA_KC, tm=rows // 4, tn=1,
                             stages=stages, split_k=split, threads=GEMV_TMA_THREADS, smem_bytes=smem,
                             regs_per_thread=regs, blocks_per_sm=blk, grid=grid,
                             wave_eff_ppm=grid * 1000000 // slots,
                             instance=gemv_tma_instance(rows, maxm), predicted_cost=cost)
                    out.append(c)
        return out, 2 * 3 * 2 * 4 + 3 * 2 * 4
    for threads in (128, 256):
        for unroll in (2, 4):
            warps = threads // 32
            ctas_n = cdiv(N, 256)
            for split in (1, 2, 4, 8, 16, 32):
                kper = cdiv(K, split)
                if split > 1 and (kper < warps * unroll or ctas_n * (split // 2) >= 2 * lim["sm_count"]):
                    continue
                smem = warps * M * 256 * 4
                if smem > GEMV_MAX_SMEM or smem > lim["smem_per_block_optin"]:
                    continue
                regs = 40 + 8 * M + 4 * unroll + 8
                blk = block_core(lim, regs, threads, smem, 0)
                if blk < 1:
                    continue
                grid = ctas_n * split
                slots = lim["sm_count"] * blk
                waves = cdiv(grid, slots)
                inflight = min(cdiv(grid, lim["sm_count"]), blk) * threads * unroll * 16
                eff = min(100, max(1, inflight * 100 // 32768))
                cost = cdiv(wbytes, HBM_BYTES_PER_CLK) * 100 // eff
                if split > 1:
                    cost += LAUNCH_CLK + cdiv(2 * split * M * N * 4, HBM_BYTES_PER_CLK)
                c = _blank()
                c.update(family=FAMILY_GEMV, bm=M, bn=256, bk=min(kper, 1 << 30), tm=1, tn=8,
                         stages=unroll, split_k=split, threads=threads, smem_bytes=smem,
                         regs_per_thread=regs, blocks_per_sm=blk, grid=grid,
                         wave_eff_ppm=grid * 1000000 // (waves * slots),
                         instance=gemv_instance(B_KN, 1, unroll), predicted_cost=cost)
                out.append(c)
    return out, 2 * 2 * 6


SETTING_AXES = ("raster", "kgroup", "reduce")
SETTING_RANGE = {"raster": (0, 1), "kgroup": (1, 2), "reduce": (0, 2)}


def setting_value(p: Problem, c: dict, axis: str):
    """The fixed-setting value of a tensor-core candidate (None for other families):
    tile order, k-blocks per ring slot (bk over one 128-byte k-block) and split-K
    reduction."""
    if c["family"] != FAMILY_TC:
        return None
    if axis == "raster":
        return c["raster"]
    if axis == "kgroup":
        return c["bk"] // (128 // p.elem)
    return c["reduce"]


def _twins(p: Problem, a: dict, b: dict, axis: str) -> bool:
    """a and b differ in `axis` and agree on every other searched field."""
    if a["family"] != FAMILY_TC or b["family"] != FAMILY_TC:
        return False
    if (a["bm"], a["bn"], a["split_k"]) != (b["bm"], b["bn"], b["split_k"]):
        return False
    for o in SETTING_AXES:
        if o != axis and setting_value(p, a, o) != setting_value(p, b, o):
            return False
    return setting_value(p, a, axis) != setting_value(p, b, axis)


def apply_settings(p: Problem, cands: list, settings: dict | None) -> list:
    """Sec. 5.1's fixed settings: for each fixed axis in SETTING_AXES order, drop a
    candidate whose value differs when its twin with the fixed value is present."""
    for axis in SETTING_AXES:
        fixed = (settings or {}).get(axis, -1)
        if fixed == -1:
            continue
        keep = []
        for c in cands:
            v = setting_value(p, c, axis)
            drop = v is not None and v != fixed and any(
                setting_value(p, t, axis) == fixed and _twins(p, c, t, axis) for t in cands)
            if not drop:
                keep.append(c)
        cands = keep
    return cands


def build_space(p: Problem, lim: dict, settings: dict | None = None):
    """Ordered candidates (list of dicts with CANDIDATE_FIELDS) and the unpruned count,
    after the fixed settings (a dict axis -> value; -1 or absent: searched)."""
    for axis, v in (settings or {}).items():
        lo, hi = SETTING_RANGE[axis]
        if v != -1 and not lo <= v <= hi:
            raise SpaceError(INVALID_ARG)
    if (lim["sm_count"] <= 0 or lim["smem_per_sm"] <= 0 or lim["smem_per_block_optin"] <= 0 or
            lim["regs_per_sm"] <= 0 or lim["max_threads_per_sm"] <= 0 or
            lim["max_blocks_per_sm"] <= 0 or lim["tmem_cols_per_sm"] < 0):
        raise SpaceError(INVALID_ARG)
    fam = family_of(p)
    if fam == FAMILY_TC:
        if lim["cc_major"] != 10 or lim["tmem_cols_per_sm"] < 128:
            raise SpaceError(UNSUPPORTED)
        cands, naive = _tc(p, lim)
    elif fam == FAMILY_FFMA:
        cands, naive = _ffma(p, lim)
    else:
        cands, naive = _gemv(p, lim)
    if not cands:
        raise SpaceError(UNSUPPORTED)
    # Sec. 5.2: from the most blocks per core to the fewest; then predicted cost; then
    # enumeration order (a stable sort)
    cands.sort(key=lambda c: (-c["blocks_per_sm"], c["predicted_cost"]))
    return apply_settings(p, cands, settings), naive
