"""The lite space: Table 1's formulas against hand-worked values, and the library's
enumeration (nnjit_space_enumerate, host only) against the oracle's restatement of the
space rules, element by element, with no GPU."""
import os

import pytest

from oracle import space as osp

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "table1_usage.txt")


def _golden_rows():
    for line in open(GOLDEN):
        if line.startswith("#") or not line.strip():
            continue
        lhs, rhs = line.split("|")
        yield [int(v) for v in lhs.split()], [int(v) for v in rhs.split()]


@pytest.mark.parametrize("args,want", list(_golden_rows()))
def test_table1_formulas_match_hand_worked_values(args, want):
    got = osp.table1_usage(*args)
    keys = ["Reg_thread", "L1_block", "Thread_block", "Warp_block", "RegLimit", "L1Limit",
            "WarpLimit", "Block_core"]
    assert [got[k] for k in keys] == want


GB300 = dict(sm_count=152, smem_per_sm=233472, smem_per_block_optin=232448, regs_per_sm=65536,
             max_threads_per_sm=2048, max_blocks_per_sm=32, tmem_cols_per_sm=512,
             l2_bytes=132120576, cc_major=10, cc_minor=3)
# a smaller hypothetical sm_10x part: fewer SMs, less shared memory, fewer blocks
SMALL = dict(sm_count=40, smem_per_sm=167936, smem_per_block_optin=166912, regs_per_sm=65536,
             max_threads_per_sm=1536, max_blocks_per_sm=24, tmem_cols_per_sm=512,
             l2_bytes=33554432, cc_major=10, cc_minor=0)


def _limits(d):
    import paper_2309_08978_gb300 as nj
    L = nj.nnjit_device_limits()
    for k, v in d.items():
        setattr(L, k, v)
    return L


def _problems():
    from synthetic import WORKLOADS
    code = {"f32_ffma": osp.F32_FFMA, "tf32": osp.TF32, "bf16": osp.BF16, "w4_bf16": osp.W4_BF16}
    out = []
    for w in WORKLOADS.values():
        for dt in w.dtypes:
            for s in w.shapes:
                out.append(dict(M=s.M, N=s.N, K=s.K, batch=s.batch, dtype=code[dt],
                                b_layout=osp.B_KN if s.b_layout == "KN" else osp.B_NK,
                                has_bias=int(s.has_bias)))
    extra = [
        (1, 1, 1, 1, osp.F32_FFMA, osp.B_KN), (7, 63, 65, 1, osp.F32_FFMA, osp.B_NK),
        (129, 130, 67, 3, osp.F32_FFMA, osp.B_KN), (9, 40, 24, 1, osp.BF16, osp.B_NK),
        (300, 264, 136, 1, osp.BF16, osp.B_KN), (5, 36, 12, 1, osp.TF32, osp.B_NK),
        (1, 1000, 4104, 1, osp.BF16, osp.B_NK), (8, 33, 24, 1, osp.BF16, osp.B_KN),
        (3, 5, 0, 1, osp.BF16, osp.B_KN), (0, 5, 8, 1, osp.TF32, osp.B_KN),
        (4096, 4096, 4096, 2, osp.BF16, osp.B_NK), (100, 90, 300, 1, osp.F32_FFMA, osp.B_NK),
        (2, 22016, 4096, 1, osp.BF16, osp.B_KN), (640, 3072, 768, 1, osp.TF32, osp.B_KN),
    ]
    for M, N, K, b, dt, lay in extra:
        out.append(dict(M=M, N=N, K=K, batch=b, dtype=dt, b_layout=lay, has_bias=0))
    # explicit strides, unaligned strides (UNSUPPORTED), invalid descriptors
    out.append(dict(M=2, N=77, K=100, dtype=osp.BF16, b_layout=osp.B_NK, lda=104, ldb=104))
    out.append(dict(M=64, N=64, K=30, dtype=osp.BF16, b_layout=osp.B_NK))
    # 4-bit weights: decode shapes, a padded row, a ragged N, and refusals
    for M, N, K, ldb in ((1, 4096, 4096, 0), (1, 4096, 11008, 0), (3, 1000, 2056, 2080),
                         (8, 520, 4096, 0), (1, 1000, 100, 0), (1, 1004, 4096, 0), (9, 64, 256, 0)):
        out.append(dict(M=M, N=N, K=K, dtype=osp.W4_BF16, b_layout=osp.B_NK, ldb=ldb))
    out.append(dict(M=1, N=64, K=256, dtype=osp.W4_BF16, b_layout=osp.B_KN))
    out.append(dict(M=64, N=30, K=64, dtype=osp.TF32, b_layout=osp.B_KN))
    out.append(dict(M=130, N=72, K=64, dtype=osp.BF16, b_layout=osp.B_NK, ldc=75))
    out.append(dict(M=4, N=4, K=8, dtype=osp.BF16, b_layout=osp.B_NK, lda=4))
    out.append(dict(M=-1, N=4, K=4, dtype=osp.BF16, b_layout=osp.B_NK))
    out.append(dict(M=3, N=4, K=8, batch=2, dtype=osp.BF16, b_layout=osp.B_NK, stride_c=5))
    return out


@pytest.mark.parametrize("dev", ["gb300", "small"])
def test_library_space_equals_oracle_space(dev):
    import paper_2309_08978_gb300 as nj
    from paper_2309_08978_gb300.build_lib import build
    build()
    lim = GB300 if dev == "gb300" else SMALL
    L = _limits(lim)
    checked = 0
    for prob in _problems():
        desc = nj.make_desc(prob["M"], prob["N"], prob["K"], prob["dtype"], prob["b_layout"],
                            batch=prob.get("batch", 1), has_bias=prob.get("has_bias", 0),
                            lda=prob.get("lda", 0), ldb=prob.get("ldb", 0), ldc=prob.get("ldc", 0),
                            stride_c=prob.get("stride_c", 0))
        try:
            p = osp.resolve(**prob)
            want, want_naive = osp.build_space(p, lim)
            want_status = 0
        except osp.SpaceError as e:
            want_status = e.status
        try:
            got, got_naive = nj.nnjit_space_enumerate(desc, L)
            got_status = 0
        except nj.NnjitError as e:
            got_status = e.status
        assert got_status == want_status, (prob, got_status, want_status)
        if want_status:
            continue
        assert got_naive == want_naive, prob
        assert len(got) == len(want), (prob, len(got), len(want))
        for i, (g, w) in enumerate(zip(got, want)):
            assert {k: g[k] for k in osp.CANDIDATE_FIELDS} == w, (prob, i, g, w)
        checked += 1
    assert checked >= 30


def test_space_invariants_on_gb300():
    for prob in _problems():
        try:
            p = osp.resolve(**prob)
            cands, naive = osp.build_space(p, GB300)
        except osp.SpaceError:
            continue
        assert 1 <= len(cands) <= naive
        assert all(b["blocks_per_sm"] <= a["blocks_per_sm"] for a, b in zip(cands, cands[1:]))
        for c in cands:
            for k in ("bm", "bn", "split_k"):              # heuristic 2: powers of two
                assert c[k] & (c[k] - 1) == 0 or c["family"] == osp.FAMILY_GEMV
            assert c["smem_bytes"] <= GB300["smem_per_block_optin"]
            assert c["tmem_cols"] <= GB300["tmem_cols_per_sm"]
            assert 32 <= c["threads"] <= 256 or c["threads"] == 192
            assert c["instance"] >= 0
        keys = [tuple(c[k] for k in osp.CANDIDATE_FIELDS) for c in cands]
        assert len(set(keys)) == len(keys)
