"""GPU parity: the CUDA path through the C ABI against the oracle, element by element.

Integer-valued inputs in [-8, 8] are exact in bf16, tf32 and f32, and every partial sum
stays below 2^24, so every kernel must reproduce the oracle bit for bit in any
summation order (split-K included).  Random inputs with the workloads' distributions are
held to the relative-Frobenius tolerances 1e-5 (FP32-FFMA), 5e-3 (TF32), 1e-2 (BF16).
Shapes span several tiles and ragged tails in M, N and K.
"""
import numpy as np
import pytest

import oracle
from synthetic import Shape, make_operands
from gpu_util import compare, dev, layout_code, run_plan

pytestmark = pytest.mark.gpu

nj = pytest.importorskip("paper_2309_08978_gb300")


def _plan(shape, dtype, budget=0.0, flags=0, **kw):
    desc = nj.make_desc(shape.M, shape.N, shape.K, dtype, shape.b_layout, batch=shape.batch,
                        has_bias=shape.has_bias, flags=flags, **kw)
    return nj.nnjit_matmul_plan_ex(desc, budget)


FFMA_SHAPES = [(1, 1, 1, "KN"), (7, 63, 65, "NK"), (129, 130, 67, "KN"), (64, 768, 768, "KN"),
               (33, 257, 40, "NK")]
TC_BF16_SHAPES = [(9, 40, 24, "NK"), (129, 200, 72, "NK"), (300, 264, 136, "KN"),
                  (256, 512, 1024, "NK"), (130, 72, 200, "KN"), (512, 768, 64, "NK")]
TC_TF32_SHAPES = [(5, 36, 12, "NK"), (130, 96, 100, "KN"), (257, 300, 68, "NK"),
                  (64, 768, 768, "KN"), (512, 768, 256, "NK")]
GEMV_SHAPES = [(1, 1, 8, "NK"), (1, 7, 16, "NK"), (3, 300, 520, "NK"), (8, 4096, 256, "NK"),
               (1, 1000, 4104, "NK"), (2, 300, 520, "KN"), (1, 513, 4096, "KN"), (8, 33, 24, "KN")]

CASES = ([("f32_ffma",) + s for s in FFMA_SHAPES] + [("bf16",) + s for s in TC_BF16_SHAPES] +
         [("tf32",) + s for s in TC_TF32_SHAPES] + [("bf16",) + s for s in GEMV_SHAPES])


def _ids(c):
    return f"{c[0]}-{c[1]}x{c[2]}x{c[3]}-{c[4]}"


@pytest.mark.parametrize("case", CASES, ids=_ids)
@pytest.mark.parametrize("with_bias", [False, True])
def test_exact_integer_inputs(case, with_bias):
    dtype, M, N, K, layout = case
    shape = Shape("t", M, N, K, 1, layout, with_bias)
    A, B, bias = make_operands(shape, 7, dtype, ints=True)
    with _plan(shape, dtype) as plan:
        C = run_plan(plan, A, B, bias, M, N)
    compare(C, A, B, bias, layout, dtype, exact=True)


@pytest.mark.parametrize("case", CASES, ids=_ids)
def test_random_inputs_tolerance(case):
    dtype, M, N, K, layout = case
    shape = Shape("t", M, N, K, 1, layout, True)
    A, B, bias = make_operands(shape, 8, dtype)
    with _plan(shape, dtype) as plan:
        C = run_plan(plan, A, B, bias, M, N)
    compare(C, A, B, bias, layout, dtype)


EVERY_CANDIDATE = [("f32_ffma", 64, 768, 768, "KN"), ("f32_ffma", 100, 90, 300, "NK"),
                   ("tf32", 64, 768, 768, "KN"), ("tf32", 200, 300, 520, "NK"),
                   ("bf16", 300, 520, 1040, "NK"), ("bf16", 200, 600, 520, "KN"),
                   ("bf16", 1, 4096, 4096, "NK"), ("bf16", 4, 1000, 2048, "KN"),
                   ("bf16", 3, 1000, 2056, "NK"), ("bf16", 8, 520, 4096, "NK")]


@pytest.mark.parametrize("case", EVERY_CANDIDATE, ids=_ids)
def test_every_candidate_is_exact(case):
    """Legality invariant of the lite space: every enumerated candidate launches and
    reproduces the oracle exactly on integer inputs."""
    dtype, M, N, K, layout = case
    shape = Shape("t", M, N, K, 1, layout, True)
    A, B, bias = make_operands(shape, 9, dtype, ints=True)
    desc = nj.make_desc(M, N, K, dtype, layout, has_bias=True)
    lim = nj.nnjit_device_limits_query(0)
    cands, _ = nj.nnjit_space_enumerate(desc, lim)
    assert 1 <= len(cands) <= 96, len(cands)
    for i, c in enumerate(cands):
        with nj.nnjit_matmul_plan_candidate(desc, i) as plan:
            C = run_plan(plan, A, B, bias, M, N)
        try:
            compare(C, A, B, bias, layout, dtype, exact=True)
        except AssertionError as e:
            raise AssertionError(f"candidate {i} {c}: {e}") from None


BATCHED = [("bf16", 3, 130, 72, 64, "NK"), ("bf16", 4, 256, 64, 256, "KN"),
           ("tf32", 2, 129, 40, 36, "NK"), ("bf16", 5, 64, 128, 128, "NK"),
           ("f32_ffma", 3, 33, 20, 17, "KN")]


@pytest.mark.parametrize("case", BATCHED, ids=lambda c: f"{c[0]}-b{c[1]}-{c[2]}x{c[3]}x{c[4]}-{c[5]}")
@pytest.mark.parametrize("exact", [True, False])
def test_batched(case, exact):
    dtype, batch, M, N, K, layout = case
    shape = Shape("t", M, N, K, batch, layout, False)
    A, B, _ = make_operands(shape, 10, dtype, ints=exact)
    with _plan(shape, dtype) as plan:
        C = run_plan(plan, A, B, None, M, N, batch=batch)
    compare(C, A, B, None, layout, dtype, exact=exact)


@pytest.mark.parametrize("dtype", ["f32_ffma", "tf32", "bf16"])
def test_degenerate_shapes(dtype):
    import torch
    bias = np.arange(5, dtype=np.float32)
    # K = 0: C = bias
    with nj.nnjit_matmul_plan_ex(nj.make_desc(3, 5, 0, dtype, "KN", has_bias=True), 10.0) as plan:
        C = torch.full((3, 5), float("nan"), device="cuda")
        plan.run(None, None, torch.from_numpy(bias).cuda(), C)
        torch.cuda.synchronize()
        assert np.array_equal(C.cpu().numpy(), np.broadcast_to(bias, (3, 5)))
        C.fill_(float("nan"))
        plan.run(None, None, None, C)
        torch.cuda.synchronize()
        assert np.array_equal(C.cpu().numpy(), np.zeros((3, 5), np.float32))
    # M = 0 or N = 0: nothing to do, nothing written
    for M, N in [(0, 5), (3, 0)]:
        with nj.nnjit_matmul_plan_ex(nj.make_desc(M, N, 8, dtype, "KN"), 10.0) as plan:
            plan.run(None, None, None, None)


@pytest.mark.parametrize("M", [2, 1])
def test_gemv_ragged_k_with_padded_rows(M):
    """K = 100 is not a multiple of the 8-element vector: lda = ldb = 104 keeps rows
    16-byte aligned; the streaming kernels' scalar tail covers the last 4 elements and
    the TMA-fed kernels' zero fill past K does.  Every candidate of the space runs."""
    N, K, ld = 77, 100, 104
    shape = Shape("t", M, N, ld, 1, "NK", True)
    Ap, Bp, bias = make_operands(shape, 11, "bf16", ints=True)
    desc = nj.make_desc(M, N, K, "bf16", "NK", has_bias=True, lda=ld, ldb=ld)
    cands, _ = nj.nnjit_space_enumerate(desc, nj.nnjit_device_limits_query(0))
    assert any(c["instance"] >= 8 for c in cands)
    for i, c in enumerate(cands):
        with nj.nnjit_matmul_plan_candidate(desc, i) as plan:
            assert plan.describe()["family"] == nj.NNJIT_FAMILY_GEMV
            C = run_plan(plan, Ap, Bp, bias, M, N)
        try:
            compare(C, np.ascontiguousarray(Ap[:, :K]), np.ascontiguousarray(Bp[:, :K]), bias,
                    "NK", "bf16", exact=True)
        except AssertionError as e:
            raise AssertionError(f"candidate {i} {c}: {e}") from None


@pytest.mark.parametrize("ldc", [80, 75])
def test_tc_strided_c(ldc):
    """ldc > N: the epilogue honours the output row stride and leaves the gap alone.
    ldc = 80 keeps 16-byte rows (TMA-store epilogue); ldc = 75 does not (direct stores)."""
    import torch
    M, N, K = 130, 72, 64
    shape = Shape("t", M, N, K, 1, "NK", True)
    A, B, bias = make_operands(shape, 12, "bf16", ints=True)
    desc = nj.make_desc(M, N, K, "bf16", "NK", has_bias=True, ldc=ldc)
    with nj.nnjit_matmul_plan_ex(desc, 0.0) as plan:
        from gpu_util import dev
        Cbuf = torch.full((M, ldc), -7.0, device="cuda")
        plan.run(dev(A), dev(B), dev(bias), Cbuf)
        torch.cuda.synchronize()
    Cn = Cbuf.cpu().numpy()
    compare(np.ascontiguousarray(Cn[:, :N]), A, B, bias, "NK", "bf16", exact=True)
    assert np.all(Cn[:, N:] == -7.0)


CONST_B_CASES = [("bf16", 300, 520, 1040, "NK"), ("tf32", 130, 96, 100, "KN"),
                 ("bf16", 1, 4096, 4096, "NK"), ("bf16", 3, 300, 520, "NK"),
                 ("bf16", 512, 768, 3072, "NK")]


@pytest.mark.parametrize("case", CONST_B_CASES, ids=_ids)
def test_constant_b_flag_is_exact(case):
    """NNJIT_PLAN_B_CONSTANT lets the kernels start reading B before the dependency
    wait; results must not change."""
    dtype, M, N, K, layout = case
    shape = Shape("t", M, N, K, 1, layout, True)
    A, B, bias = make_operands(shape, 13, dtype, ints=True)
    desc = nj.make_desc(M, N, K, dtype, layout, has_bias=True,
                        flags=nj.NNJIT_PLAN_B_CONSTANT | nj.NNJIT_PLAN_NO_CACHE)
    lim = nj.nnjit_device_limits_query(0)
    cands, _ = nj.nnjit_space_enumerate(desc, lim)
    # the first few candidates, plus every tensor-core one with two k-blocks per ring slot
    # (whose preloaded B tiles are grouped two to a barrier)
    picks = sorted(set(range(min(len(cands), 6))) |
                   {i for i, c in enumerate(cands) if c["family"] == nj.NNJIT_FAMILY_TC and
                    (c["bk"] * (2 if dtype == "bf16" else 4) == 256 or c["cluster_m"] == 2)})
    for i in picks:
        with nj.nnjit_matmul_plan_candidate(desc, i) as plan:
            C = run_plan(plan, A, B, bias, M, N)
        compare(C, A, B, bias, layout, dtype, exact=True)


def test_chain_waits_for_the_producer_of_a():
    """Two TF32 products on one stream, the second reading the first's output as A while
    its (constant) B is fetched early: the second must still see the finished A.
    Integer operands keep every value exact (C1 <= 64 is exact in TF32)."""
    import torch
    from synthetic import small_ints
    M, K1, N1, N2 = 256, 16, 64, 128
    A0 = (small_ints(40, M * K1, -2, 2).reshape(M, K1)).astype(np.float32)
    B1 = (small_ints(41, N1 * K1, -2, 2).reshape(N1, K1)).astype(np.float32)
    B2 = (small_ints(42, N2 * N1).reshape(N2, N1)).astype(np.float32)
    flags = nj.NNJIT_PLAN_B_CONSTANT | nj.NNJIT_PLAN_NO_CACHE
    p1 = nj.nnjit_matmul_plan_ex(nj.make_desc(M, N1, K1, "tf32", "NK", flags=flags), 0.0)
    p2 = nj.nnjit_matmul_plan_ex(nj.make_desc(M, N2, N1, "tf32", "NK", flags=flags), 0.0)
    dA0, dB1, dB2 = (torch.from_numpy(x).cuda() for x in (A0, B1, B2))
    want1 = A0.astype(np.int64) @ B1.T.astype(np.int64)
    want2 = want1 @ B2.T.astype(np.int64)
    s = torch.cuda.Stream()
    for rep in range(20):
        C1 = torch.full((M, N1), float("nan"), device="cuda")
        C2 = torch.full((M, N2), float("nan"), device="cuda")
        torch.cuda.synchronize()
        with torch.cuda.stream(s):
            p1.run(dA0, dB1, None, C1, s)
            p2.run(C1, dB2, None, C2, s)
        s.synchronize()
        assert np.array_equal(C2.cpu().numpy(), want2.astype(np.float32)), f"repetition {rep}"
    p1.destroy()
    p2.destroy()


@pytest.mark.parametrize("M", [1, 3])
def test_gemv_tma_constant_b_every_candidate(M):
    """TMA-fed GEMV candidates with NNJIT_PLAN_B_CONSTANT: the weight boxes of the first
    ring are requested before the dependency wait, x boxes after it.  N and K are not
    multiples of the box (rows past N and K past 2056 are zero-filled)."""
    N, K = 1000, 2056
    shape = Shape("t", M, N, K, 1, "NK", True)
    A, B, bias = make_operands(shape, 15, "bf16", ints=True)
    desc = nj.make_desc(M, N, K, "bf16", "NK", has_bias=True,
                        flags=nj.NNJIT_PLAN_B_CONSTANT | nj.NNJIT_PLAN_NO_CACHE)
    cands, _ = nj.nnjit_space_enumerate(desc, nj.nnjit_device_limits_query(0))
    tma = [i for i, c in enumerate(cands) if c["instance"] >= 8]
    assert tma
    for i in tma:
        with nj.nnjit_matmul_plan_candidate(desc, i) as plan:
            C = run_plan(plan, A, B, bias, M, N)
        compare(C, A, B, bias, "NK", "bf16", exact=True)


def test_gemv_tma_writes_after_the_previous_kernel():
    """A slow product writes C, then a TMA-fed GEMV with constant weights writes the same
    C on the same stream: the second one's results must be the ones left in C."""
    import torch
    M, N, K1, K2 = 1, 4096, 8192, 512
    s1 = Shape("t", M, N, K1, 1, "NK", False)
    s2 = Shape("t", M, N, K2, 1, "NK", False)
    A1, B1, _ = make_operands(s1, 16, "bf16", ints=True)
    A2, B2, _ = make_operands(s2, 17, "bf16", ints=True)
    flags = nj.NNJIT_PLAN_B_CONSTANT | nj.NNJIT_PLAN_NO_CACHE
    d1 = nj.make_desc(M, N, K1, "bf16", "NK", flags=flags)
    d2 = nj.make_desc(M, N, K2, "bf16", "NK", flags=flags)
    c2, _ = nj.nnjit_space_enumerate(d2, nj.nnjit_device_limits_query(0))
    tma = [i for i, c in enumerate(c2) if c["instance"] >= 8]
    _, ref32 = oracle.matmul(A2, B2, None, layout_code("NK"))
    dA1, dB1, dA2, dB2 = dev(A1), dev(B1), dev(A2), dev(B2)
    p1 = nj.nnjit_matmul_plan_candidate(d1, 0)
    st = torch.cuda.Stream()
    try:
        for i in tma:
            with nj.nnjit_matmul_plan_candidate(d2, i) as p2:
                for rep in range(5):
                    C = torch.full((M, N), float("nan"), device="cuda")
                    torch.cuda.synchronize()
                    with torch.cuda.stream(st):
                        p1.run(dA1, dB1, None, C, st)
                        p2.run(dA2, dB2, None, C, st)
                    st.synchronize()
                    p2.check()
                    assert np.array_equal(C.cpu().numpy(), ref32), f"candidate {i} repetition {rep}"
    finally:
        p1.destroy()


FULL_WAVE_CASES = [("bf16", 2048, 2560, 192, "NK"), ("bf16", 2176, 2560, 136, "KN"),
                   ("tf32", 2048, 2560, 64, "NK"), ("tf32", 2200, 2560, 40, "KN")]


@pytest.mark.parametrize("case", FULL_WAVE_CASES, ids=_ids)
def test_full_wave_shapes_every_candidate_exact(case):
    """Shapes with more tiles than SMs, so persistent CTAs take several tiles and the
    accumulator barriers cycle: every candidate (CTA-pair tiles included where B is
    [N][K]), with and without a constant B.  Includes an odd number of 256-row tile
    rows, where the last pair tile lies partly past M."""
    dtype, M, N, K, layout = case
    shape = Shape("t", M, N, K, 1, layout, True)
    A, B, bias = make_operands(shape, 14, dtype, ints=True)
    for flags in (0, nj.NNJIT_PLAN_B_CONSTANT):
        desc = nj.make_desc(M, N, K, dtype, layout, has_bias=True, flags=flags)
        cands, _ = nj.nnjit_space_enumerate(desc, nj.nnjit_device_limits_query(0))
        assert all(c["cluster_m"] == 1 or c["bm"] == 256 for c in cands)
        if layout == "NK":
            assert any(c["cluster_m"] == 2 for c in cands), "expected CTA-pair candidates"
        for i in range(len(cands)):
            with nj.nnjit_matmul_plan_candidate(desc, i) as plan:
                C = run_plan(plan, A, B, bias, M, N)
            compare(C, A, B, bias, layout, dtype, exact=True)


EPI_CASES = [("f32_ffma", 64, 768, 768, "KN"), ("tf32", 200, 300, 520, "NK"),
             ("bf16", 300, 520, 1040, "NK"), ("bf16", 200, 600, 520, "KN"),
             ("bf16", 1, 4096, 4096, "NK"), ("bf16", 3, 1000, 2056, "NK"), ("bf16", 4, 1000, 2048, "KN")]


@pytest.mark.parametrize("case", EPI_CASES, ids=_ids)
def test_fused_activation_every_candidate(case):
    """C = act(A.B + bias) written by the kernel that writes C (split-K plans: by the
    reduction).  Every candidate of the space runs -- split-K reduces, cluster reduces,
    CTA pairs, TMA-fed GEMVs.  ReLU on integer inputs must be exact; GELU on random
    inputs stays within the dtype's tolerance; SiLU runs on the top-ranked plan."""
    dtype, M, N, K, layout = case
    shape = Shape("t", M, N, K, 1, layout, True)
    Ai, Bi, biasi = make_operands(shape, 30, dtype, ints=True)
    Ar, Br, biasr = make_operands(shape, 31, dtype)
    lim = nj.nnjit_device_limits_query(0)
    for act in ("relu", "gelu"):
        desc = nj.make_desc(M, N, K, dtype, layout, has_bias=True, epilogue=act,
                            flags=nj.NNJIT_PLAN_NO_CACHE)
        cands, _ = nj.nnjit_space_enumerate(desc, lim)
        for i, c in enumerate(cands):
            with nj.nnjit_matmul_plan_candidate(desc, i) as plan:
                if act == "relu":
                    C = run_plan(plan, Ai, Bi, biasi, M, N)
                else:
                    C = run_plan(plan, Ar, Br, biasr, M, N)
            try:
                if act == "relu":
                    compare(C, Ai, Bi, biasi, layout, dtype, exact=True, act=act)
                else:
                    compare(C, Ar, Br, biasr, layout, dtype, act=act)
            except AssertionError as e:
                raise AssertionError(f"{act} candidate {i} {c}: {e}") from None
    desc = nj.make_desc(M, N, K, dtype, layout, has_bias=True, epilogue="silu",
                        flags=nj.NNJIT_PLAN_NO_CACHE)
    with nj.nnjit_matmul_plan_ex(desc, 0.0) as plan:
        C = run_plan(plan, Ar, Br, biasr, M, N)
    compare(C, Ar, Br, biasr, layout, dtype, act="silu")


@pytest.mark.parametrize("act", ["relu", "gelu", "silu"])
def test_fused_activation_k0_applies_to_bias(act):
    """K = 0: C = act(bias) on every row.  The kernels evaluate GELU with the erf of
    Abramowitz & Stegun 7.1.26 (|error| <= 1.5e-7) and SiLU with the hardware exp2 and
    reciprocal approximations; against the FP64 definitions the error stays within
    2e-7 + 1e-6 |x| over [-10, 10]."""
    import torch
    from oracle.epilogue import apply
    bias = np.linspace(-10.0, 10.0, 801).astype(np.float32)
    N = bias.size
    with nj.nnjit_matmul_plan_ex(nj.make_desc(4, N, 0, "bf16", "NK", has_bias=True, epilogue=act), 0.0) as plan:
        C = torch.full((4, N), float("nan"), device="cuda")
        plan.run(None, None, torch.from_numpy(bias).cuda(), C)
        torch.cuda.synchronize()
    got = C.cpu().numpy().astype(np.float64)
    x = bias.astype(np.float64)
    err = np.abs(got - apply(x, act)[None, :])
    bound = 2e-7 + 1e-6 * np.abs(x)
    assert np.all(err <= bound[None, :]), f"max excess {np.max(err - bound):.3e} at x = {x[np.argmax(np.max(err, 0) - bound)]}"


W4_CASES = [(1, 4096, 4096, 0), (1, 4096, 11008, 0), (3, 1000, 2056, 2080), (8, 520, 4096, 0),
            (2, 264, 640, 0), (5, 4008, 4096, 0)]


def _w4_ids(c):
    return f"w4-{c[0]}x{c[1]}x{c[2]}" + (f"-ldb{c[3]}" if c[3] else "")


def _w4_compare(C, x, blob, N, K, ldb, bias, exact, act="none"):
    from oracle.quant import matmul as w4_matmul
    ref64, ref32 = w4_matmul(x, blob, N, K, ldb, bias, act)
    assert np.all(np.isfinite(C)), "non-finite output (unwritten element?)"
    if exact:
        bad = np.argwhere(C != ref32)
        assert bad.size == 0, f"{len(bad)} elements differ, first at {bad[:5].tolist()}"
    else:
        err = oracle.rel_fro(C, ref64)
        assert err <= 1e-2, f"rel_fro {err:.3e}"


@pytest.mark.parametrize("case", W4_CASES, ids=_w4_ids)
def test_w4_gemv_every_candidate(case):
    """4-bit weights: every candidate of the space, exact on integer x with unit scales
    (products (q - 8) x and all sums are integers below 2^24), within the BF16 tolerance
    on the workload's distributions, with and without constant-weight preloading.  K =
    2056 and 11008 end in a partial stage; K = 2056 also pads rows to ldb = 2080 codes."""
    from synthetic import make_w4_operands
    M, N, K, ldb = case
    shape = Shape("t", M, N, K, 1, "NK", True)
    xi, blob_i, bias_i = make_w4_operands(shape, 40, ints=True, ldb=ldb)
    xr, blob_r, bias_r = make_w4_operands(shape, 41, ldb=ldb)
    for flags in (nj.NNJIT_PLAN_NO_CACHE, nj.NNJIT_PLAN_NO_CACHE | nj.NNJIT_PLAN_B_CONSTANT):
        desc = nj.make_desc(M, N, K, "w4_bf16", "NK", has_bias=True, ldb=ldb, flags=flags)
        cands, _ = nj.nnjit_space_enumerate(desc, nj.nnjit_device_limits_query(0))
        assert cands and all(c["instance"] >= 14 for c in cands)
        for i, c in enumerate(cands):
            with nj.nnjit_matmul_plan_candidate(desc, i) as plan:
                Ce = run_plan(plan, xi, blob_i, bias_i, M, N)
                Cr = run_plan(plan, xr, blob_r, bias_r, M, N)
            try:
                _w4_compare(Ce, xi, blob_i, N, K, ldb, bias_i, exact=True)
                _w4_compare(Cr, xr, blob_r, N, K, ldb, bias_r, exact=False)
            except AssertionError as e:
                raise AssertionError(f"candidate {i} {c}: {e}") from None


def test_w4_gemv_tuned_plan_with_activation():
    from synthetic import make_w4_operands
    M, N, K = 1, 4096, 4096
    shape = Shape("t", M, N, K, 1, "NK", True)
    x, blob, bias = make_w4_operands(shape, 42)
    desc = nj.make_desc(M, N, K, "w4_bf16", "NK", has_bias=True, epilogue="silu",
                        flags=nj.NNJIT_PLAN_NO_CACHE)
    with nj.nnjit_matmul_plan_ex(desc, 50.0) as plan:
        C = run_plan(plan, x, blob, bias, M, N)
    _w4_compare(C, x, blob, N, K, 0, bias, exact=False, act="silu")


def test_w4_refusals():
    """Prefill-sized M, B as [K][N], unaligned code rows and a ragged N are refused."""
    L = nj.nnjit_device_limits_query(0)
    for d in (nj.make_desc(16, 64, 256, "w4_bf16", "NK"), nj.make_desc(1, 64, 256, "w4_bf16", "KN"),
              nj.make_desc(1, 64, 100, "w4_bf16", "NK"), nj.make_desc(1, 60, 256, "w4_bf16", "NK")):
        with pytest.raises(nj.NnjitError) as ei:
            nj.nnjit_space_enumerate(d, L)
        assert ei.value.status == nj.NNJIT_ERR_UNSUPPORTED


@pytest.mark.parametrize("case", EPI_CASES, ids=_ids)
def test_residual_epilogue_every_candidate(case):
    """C = act(A.B + bias) + C: the kernel that writes C adds the value C held before (split-K
    plans: the reduction, once).  Every candidate, ReLU + an integer residual on integer
    inputs (exact); the top-ranked plan with GELU + a random residual (tolerance)."""
    torch = pytest.importorskip("torch")
    dtype, M, N, K, layout = case
    shape = Shape("t", M, N, K, 1, layout, True)
    Ai, Bi, biasi = make_operands(shape, 32, dtype, ints=True)
    Ar, Br, biasr = make_operands(shape, 33, dtype)
    Ri = np.random.default_rng(7).integers(-8, 9, (M, N)).astype(np.float32)
    Rr = np.random.default_rng(8).normal(0.0, 1.0, (M, N)).astype(np.float32)
    lim = nj.nnjit_device_limits_query(0)
    desc = nj.make_desc(M, N, K, dtype, layout, has_bias=True, epilogue="relu", residual=True,
                        flags=nj.NNJIT_PLAN_NO_CACHE)
    cands, _ = nj.nnjit_space_enumerate(desc, lim)
    for i, c in enumerate(cands):
        with nj.nnjit_matmul_plan_candidate(desc, i) as plan:
            C = run_plan(plan, Ai, Bi, biasi, M, N, C=torch.from_numpy(Ri.copy()).cuda())
        try:
            compare(C, Ai, Bi, biasi, layout, dtype, exact=True, act="relu", residual=Ri)
        except AssertionError as e:
            raise AssertionError(f"candidate {i} {c}: {e}") from None
    desc = nj.make_desc(M, N, K, dtype, layout, has_bias=True, epilogue="gelu", residual=True,
                        flags=nj.NNJIT_PLAN_NO_CACHE)
    with nj.nnjit_matmul_plan_ex(desc, 0.0) as plan:
        C = run_plan(plan, Ar, Br, biasr, M, N, C=torch.from_numpy(Rr.copy()).cuda())
    compare(C, Ar, Br, biasr, layout, dtype, act="gelu", residual=Rr)


def test_residual_edge_cases():
    """Residual with direct stores (ldc = N + 1 rules the TMA store out), batched outputs
    (stride_c), K = 0 (C = bias + C), no activation, and a 4-bit weight GEMV."""
    torch = pytest.importorskip("torch")
    lim = nj.nnjit_device_limits_query(0)
    rng = np.random.default_rng(9)
    # direct stores, bf16 and tf32 tensor-core tiles
    for dtype in ("bf16", "tf32"):
        M, N, K = 130, 72, 64
        shape = Shape("t", M, N, K, 1, "NK", True)
        A, B, bias = make_operands(shape, 34, dtype, ints=True)
        R = rng.integers(-8, 9, (M, N + 1)).astype(np.float32)
        desc = nj.make_desc(M, N, K, dtype, "NK", has_bias=True, ldc=N + 1, residual=True,
                            flags=nj.NNJIT_PLAN_NO_CACHE)
        cands, _ = nj.nnjit_space_enumerate(desc, lim)
        for i in range(len(cands)):
            Cd = torch.from_numpy(R.copy()).cuda()
            with nj.nnjit_matmul_plan_candidate(desc, i) as plan:
                plan.run(dev(A), dev(B), dev(bias), Cd)
                torch.cuda.synchronize()
                plan.check()
            Cn = Cd.cpu().numpy()
            assert np.array_equal(Cn[:, N], R[:, N])                    # the gap is untouched
            compare(np.ascontiguousarray(Cn[:, :N]), A, B, bias, "NK", dtype, exact=True,
                    residual=R[:, :N])
    # batched (no bias), every candidate
    shape = Shape("t", 100, 96, 64, 3, "NK", False)
    A, B, _ = make_operands(shape, 35, "bf16", ints=True)
    R = rng.integers(-8, 9, (3, 100, 96)).astype(np.float32)
    desc = nj.make_desc(100, 96, 64, "bf16", "NK", batch=3, residual=True, flags=nj.NNJIT_PLAN_NO_CACHE)
    cands, _ = nj.nnjit_space_enumerate(desc, lim)
    for i in range(len(cands)):
        with nj.nnjit_matmul_plan_candidate(desc, i) as plan:
            C = run_plan(plan, A, B, None, 100, 96, batch=3, C=torch.from_numpy(R.copy()).cuda())
        compare(C, A, B, None, "NK", "bf16", exact=True, residual=R)
    # K = 0: C = bias + C
    bias = rng.integers(-8, 9, 40).astype(np.float32)
    R = rng.integers(-8, 9, (5, 40)).astype(np.float32)
    desc = nj.make_desc(5, 40, 0, "bf16", "NK", has_bias=True, residual=True, flags=nj.NNJIT_PLAN_NO_CACHE)
    with nj.nnjit_matmul_plan_ex(desc, 0.0) as plan:
        Cd = torch.from_numpy(R.copy()).cuda()
        plan.run(dev(np.zeros((5, 1), np.uint16)), dev(np.zeros((40, 1), np.uint16)), dev(bias), Cd)
        torch.cuda.synchronize()
        plan.check()
    assert np.array_equal(Cd.cpu().numpy(), R + bias)
    # 4-bit weights, every candidate
    from synthetic import make_w4_operands
    from oracle.quant import matmul as w4_matmul
    M, N, K = 2, 520, 4096
    shape = Shape("t", M, N, K, 1, "NK", True)
    x, blob, bias = make_w4_operands(shape, 36, ints=True)
    R = rng.integers(-8, 9, (M, N)).astype(np.float32)
    desc = nj.make_desc(M, N, K, "w4_bf16", "NK", has_bias=True, epilogue="relu", residual=True,
                        flags=nj.NNJIT_PLAN_NO_CACHE)
    cands, _ = nj.nnjit_space_enumerate(desc, lim)
    _, want = w4_matmul(x, blob, N, K, 0, bias, "relu", residual=R)
    for i in range(len(cands)):
        with nj.nnjit_matmul_plan_candidate(desc, i) as plan:
            C = run_plan(plan, x, blob, bias, M, N, C=torch.from_numpy(R.copy()).cuda())
        assert np.array_equal(C, want), i


STREAM_K_CASES = [("bf16", 4096, 2560, 1024, "NK"), ("tf32", 4096, 2560, 512, "NK"),
                  ("bf16", 4200, 2300, 1040, "NK"), ("bf16", 6144, 2560, 512, "NK"),
                  ("bf16", 4096, 4864, 1024, "NK"), ("bf16", 2048, 1024, 4096, "NK")]


@pytest.mark.parametrize("case", STREAM_K_CASES, ids=_ids)
def test_pair_stream_k_exact_repeated_and_in_graphs(case):
    """CTA-pair tiles with stream-K over the last waves (reduce 2): the k-blocks of the
    tiles past the whole waves but the last are shared evenly by the pairs; a tile cut
    between pairs is finished by the pair holding its first k-blocks, which adds the
    other pairs' partial sums after a flag hand-off and lowers the flags for the next
    launch.  Every stream-K candidate must be bit exact on integer inputs (with bias, and
    with ReLU), on three launches in a row and on two replays of a CUDA graph of two
    launches.  Cases: ragged M and N (4200 x 2300); 240 pair tiles of 8 k-blocks, so that
    each pair's range (9.3 k-blocks) ends inside a tile that another pair finishes
    (6144 x 2560 x 512); 304 tiles, a whole number of waves, where the space offers no
    stream-K and the test expects none (4096 x 4864); fewer tiles than two waves, where
    the space offers none either (2048 x 1024 x 4096)."""
    import torch
    dtype, M, N, K, layout = case
    shape = Shape("t", M, N, K, 1, layout, True)
    A, B, bias = make_operands(shape, 51, dtype, ints=True)
    dA, dB, dbias = (torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).view(torch.bfloat16).cuda()
                     if x.dtype == np.uint16 else torch.from_numpy(x).cuda() for x in (A, B, bias))
    lim = nj.nnjit_device_limits_query(0)
    for act in ("none", "relu"):
        desc = nj.make_desc(M, N, K, dtype, layout, has_bias=True, epilogue=act, flags=nj.NNJIT_PLAN_NO_CACHE)
        cands, _ = nj.nnjit_space_enumerate(desc, lim)
        tails = [i for i, c in enumerate(cands) if c["reduce"] == 2]
        pairs = (M + 255) // 256 * ((N + 255) // 256)
        if pairs % 76 == 0 or pairs // 76 < 2:
            assert not tails, "no stream-K where the tiles fill whole waves or fewer than two"
            return
        assert tails, "expected stream-K candidates"
        _, ref32 = oracle.matmul(A, B, bias, layout_code(layout), act=act)
        for i in tails:
            with nj.nnjit_matmul_plan_candidate(desc, i) as plan:
                for rep in range(3):
                    C = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
                    plan.run(dA, dB, dbias, C)
                    torch.cuda.synchronize()
                    plan.check()
                    got = C.cpu().numpy()
                    bad = np.argwhere(got != ref32)
                    assert bad.size == 0, f"candidate {i} {cands[i]} launch {rep}: {len(bad)} mismatches"
                st = torch.cuda.Stream()
                C1 = torch.empty((M, N), dtype=torch.float32, device="cuda")
                C2 = torch.empty((M, N), dtype=torch.float32, device="cuda")
                plan.run(dA, dB, dbias, C1, st)   # tensor maps cached outside the capture
                plan.run(dA, dB, dbias, C2, st)
                st.synchronize()
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=st):
                    plan.run(dA, dB, dbias, C1, st)
                    plan.run(dA, dB, dbias, C2, st)
                for rep in range(2):
                    C1.fill_(float("nan"))
                    C2.fill_(float("nan"))
                    g.replay()
                    torch.cuda.synchronize()
                    plan.check()
                    for Cx in (C1, C2):
                        assert np.array_equal(Cx.cpu().numpy(), ref32), f"candidate {i} graph replay {rep}"
