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


SETTINGS_CASES = [
    {"raster": 0}, {"raster": 1}, {"kgroup": 2}, {"kgroup": 1, "reduce": 1},
    {"reduce": 0}, {"reduce": 1, "raster": 1},
    {"raster": 0, "kgroup": 2, "reduce": 1},
]


@pytest.mark.parametrize("settings", SETTINGS_CASES, ids=lambda s: ",".join(f"{k}={v}" for k, v in s.items()))
def test_library_space_with_fixed_settings_equals_oracle(settings):
    """Sec. 5.1's fixed settings prune the same candidates in both implementations."""
    import paper_2309_08978_gb300 as nj
    from paper_2309_08978_gb300.build_lib import build
    build()
    L = _limits(GB300)
    nj.nnjit_settings_set(settings)
    try:
        checked = 0
        for prob in _problems():
            desc = nj.make_desc(prob["M"], prob["N"], prob["K"], prob["dtype"], prob["b_layout"],
                                batch=prob.get("batch", 1), has_bias=prob.get("has_bias", 0),
                                lda=prob.get("lda", 0), ldb=prob.get("ldb", 0), ldc=prob.get("ldc", 0),
                                stride_c=prob.get("stride_c", 0))
            try:
                want, _ = osp.build_space(osp.resolve(**prob), GB300, settings)
            except osp.SpaceError:
                continue
            got, _ = nj.nnjit_space_enumerate(desc, L)
            assert [{k: g[k] for k in osp.CANDIDATE_FIELDS} for g in got] == want, (prob, settings)
            checked += 1
        assert checked >= 30
    finally:
        nj.nnjit_settings_set(None)


def test_fixed_settings_prune_only_where_a_twin_exists():
    """A fixed setting keeps the space non-empty and ordered (a subsequence of the free
    space), removes every candidate with the other value whose twin is present, and
    keeps the only legal choice (kgroup = 2 keeps the 256-wide tiles, which exist only
    with one k-block per slot)."""
    seen_bn256 = False
    for prob in _problems():
        try:
            p = osp.resolve(**prob)
            free, _ = osp.build_space(p, GB300)
        except osp.SpaceError:
            continue
        for settings in SETTINGS_CASES:
            fixed, _ = osp.build_space(p, GB300, settings)
            assert fixed, (prob, settings)
            it = iter(free)
            assert all(any(c == f for f in it) for c in fixed)          # ordered subsequence
            for axis, v in settings.items():
                for c in fixed:
                    w = osp.setting_value(p, c, axis)
                    if w is not None and w != v:
                        assert not any(osp.setting_value(p, t, axis) == v and osp._twins(p, c, t, axis)
                                       for t in fixed), (prob, settings, c)
            if settings.get("kgroup") == 2:
                wide = [c for c in free if c["family"] == osp.FAMILY_TC and c["bn"] == 256]
                seen_bn256 |= bool(wide)
                assert all(c in fixed for c in wide if settings.keys() == {"kgroup"})
    assert seen_bn256


def test_setting_values_of_candidates():
    """The setting accessors read what the candidates encode: bk = 2 k-blocks of 128 bytes
    for kgroup 2 (64 bf16 elements per k-block); the only two-CTA clusters are the
    256-row CTA-pair tiles."""
    p = osp.resolve(M=4096, N=4096, K=4096, dtype=osp.BF16, b_layout=osp.B_NK)
    cands, _ = osp.build_space(p, GB300)
    kg = {osp.setting_value(p, c, "kgroup") for c in cands}
    assert kg == {1, 2}
    assert all(c["bk"] == 64 * osp.setting_value(p, c, "kgroup") for c in cands)
    pairs = [c for c in cands if c["cluster_m"] == 2]
    assert pairs and all(c["bm"] == 256 and c["bn"] == 256 for c in pairs)


BLACKWELL = os.path.join(os.path.dirname(__file__), "golden", "blackwell_usage.txt")
_DT = {"bf16": osp.BF16, "tf32": osp.TF32, "f32_ffma": osp.F32_FFMA, "w4_bf16": osp.W4_BF16}
_FAM = {"tc": osp.FAMILY_TC, "ffma": osp.FAMILY_FFMA, "gemv": osp.FAMILY_GEMV}


def _blackwell_rows(kind):
    for line in open(BLACKWELL):
        if line.startswith("#") or not line.strip():
            continue
        head, *rest = [part.strip() for part in line.split("|")]
        fam, dt, lay, M, N, K = head.split()
        if (fam == "order") != (kind == "order"):
            continue
        prob = dict(M=int(M), N=int(N), K=int(K), dtype=_DT[dt],
                    b_layout=osp.B_NK if lay == "NK" else osp.B_KN)
        if kind == "order":
            yield prob, [[int(v) for v in r.split()] for r in rest]
        else:
            pick = {k: int(v) for k, v in (t.split("=") for t in rest[0].split())}
            want = {k: int(v) for k, v in (t.split("=") for t in rest[1].split())}
            yield fam, prob, pick, want


def _both_spaces(prob):
    """The library's space (host only, GB300 limits) and the oracle restatement's."""
    import paper_2309_08978_gb300 as nj
    p = osp.resolve(**prob)
    ours, _ = osp.build_space(p, GB300)
    lay = "NK" if prob["b_layout"] == osp.B_NK else "KN"
    dt = {v: k for k, v in _DT.items()}[prob["dtype"]]
    lib, _ = nj.nnjit_space_enumerate(nj.make_desc(prob["M"], prob["N"], prob["K"], dt, lay),
                                      _limits(GB300))
    return {"oracle": ours, "library": lib}


@pytest.mark.parametrize("fam,prob,pick,want", list(_blackwell_rows("usage")),
                         ids=lambda v: str(v) if not isinstance(v, dict) else
                         ",".join(f"{k}={x}" for k, x in v.items() if k in ("M", "N", "K", "bm", "bn",
                                                                          "bk", "split_k", "reduce",
                                                                          "stages", "tm")))
def test_blackwell_usage_matches_hand_worked_values(fam, prob, pick, want):
    """Stages, shared memory, TMEM columns, registers, blocks per SM, grid, wave efficiency
    and the ordering cost of chosen candidates, worked by hand from the usage formulas
    (tests/golden/blackwell_usage.txt), for the library and the oracle restatement alike."""
    for who, space in _both_spaces(prob).items():
        hits = [c for c in space if c["family"] == _FAM[fam] and all(c[k] == v for k, v in pick.items())]
        assert len(hits) == 1, f"{who}: {len(hits)} candidates match {pick}"
        got = {k: hits[0][k] for k in want}
        assert got == want, f"{who}: {got} != {want}"


@pytest.mark.parametrize("prob,order", list(_blackwell_rows("order")))
def test_evaluation_order_matches_hand_ordering(prob, order):
    """The 4096^3 BF16 space, index by index, in the order worked out by hand (blocks per
    SM, then the cost, then enumeration order), stream-K CTA pairs included."""
    for who, space in _both_spaces(prob).items():
        assert len(space) == len(order), f"{who}: {len(space)} candidates"
        for idx, bm, bn, bk, split, reduce, raster, cluster in order:
            c = space[idx]
            assert (c["bm"], c["bn"], c["bk"], c["split_k"], c["reduce"], c["raster"], c["cluster_m"]) == \
                (bm, bn, bk, split, reduce, raster, cluster), f"{who}: index {idx} is {c}"
