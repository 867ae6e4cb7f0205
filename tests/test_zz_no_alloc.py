"""The allocation-free decode GEMV (nnjit_gemv_bf16_noalloc) against the oracle and the
planned path.

Callers that cannot allocate device memory when they run a product (a process whose
memory a framework's caching allocator has reserved, a decode loop that must not pay for
cudaMalloc/cudaFree synchronisation) use this entry point: its split-K partial sums live
in a fixed array inside the library instead of a plan's workspace.  Each result is held
to the oracle (the MatMul definition in FP64) and to the planned entry point on the same
inputs.  This file is collected last so that a run stopping at the first failure has run
everything else.
"""
import numpy as np
import pytest

from synthetic import Shape, make_operands
from gpu_util import dev, run_plan, TOL
import oracle

pytestmark = pytest.mark.gpu

nj = pytest.importorskip("paper_2309_08978_gb300")


def _planned(A, B, bias, M, N, K):
    desc = nj.make_desc(M, N, K, "bf16", "NK", has_bias=bias is not None)
    with nj.nnjit_matmul_plan_ex(desc, 0.0) as plan:
        return run_plan(plan, A, B, bias, M, N)


def _noalloc(A, B, bias, M, N, K, split):
    import torch
    C = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    nj.nnjit_gemv_bf16_noalloc(M, N, K, dev(A), dev(B), dev(bias), C, split)
    torch.cuda.synchronize()
    return C.cpu().numpy()


@pytest.mark.parametrize("M,N,K,split,with_bias", [
    (1, 4096, 4096, 4, False),     # Llama-2-7B o-proj decode shape
    (3, 1000, 520, 2, True),       # ragged N, K not a multiple of the slice
    (8, 4096, 11008, 8, False),    # down-proj shape at M = 8
    (1, 513, 256, 1, True),        # no split: no scratch use
])
def test_noalloc_matches_oracle_and_planned_path_twice(M, N, K, split, with_bias):
    shape = Shape("t", M, N, K, 1, "NK", with_bias)
    for call, seed in enumerate((21, 22)):       # two calls in a row, new data each time
        A, B, bias = make_operands(shape, seed, "bf16")
        got = _noalloc(A, B, bias, M, N, K, split)
        assert np.all(np.isfinite(got)), f"call {call}: unwritten outputs"
        ref64, _ = oracle.matmul(A, B, bias, oracle.B_NK)
        assert oracle.rel_fro(got, ref64) <= TOL["bf16"], f"call {call}: vs oracle"
        want = _planned(A, B, bias, M, N, K)
        assert oracle.rel_fro(got, want.astype(np.float64)) <= TOL["bf16"], f"call {call}: vs plan"


def test_noalloc_exact_on_integer_inputs():
    # |sum| <= 64 K < 2^24: every order of f32 additions is exact, so the result must
    # equal the oracle's bit for bit (and so the planned path's)
    M, N, K, split = 2, 777, 1024, 4
    A, B, bias = make_operands(Shape("t", M, N, K, 1, "NK", True), 23, "bf16", ints=True)
    got = _noalloc(A, B, bias, M, N, K, split)
    _, ref32 = oracle.matmul(A, B, bias, oracle.B_NK)
    assert np.array_equal(got, ref32)
    assert np.array_equal(got, _planned(A, B, bias, M, N, K))


def test_noalloc_empty_trailing_slices_write_zero_partials():
    # K = 16 in 8 slices of 8 (rounded up): slices 2..7 are empty and must contribute
    # zero partials, whatever an earlier call left in the shared scratch array
    M, N = 8, 4096
    A, B, _ = make_operands(Shape("t", M, N, 4096, 1, "NK", False), 24, "bf16", ints=True)
    _noalloc(A, B, None, M, N, 4096, 8)          # fills 8 x M x N partials, non-zero
    M, N, K, split = 2, 300, 16, 8
    A, B, bias = make_operands(Shape("t", M, N, K, 1, "NK", True), 25, "bf16", ints=True)
    got = _noalloc(A, B, bias, M, N, K, split)
    _, ref32 = oracle.matmul(A, B, bias, oracle.B_NK)
    assert np.array_equal(got, ref32)
    assert np.array_equal(got, _planned(A, B, bias, M, N, K))


def test_noalloc_rejects_requests_beyond_the_scratch():
    import torch
    M, N, K = 8, 4096, 4096
    split = 64                     # 64 * 8 * 4096 = 2 Mi floats > 1 Mi
    x = torch.zeros((M, K), dtype=torch.bfloat16, device="cuda")
    W = torch.zeros((N, K), dtype=torch.bfloat16, device="cuda")
    C = torch.zeros((M, N), dtype=torch.float32, device="cuda")
    with pytest.raises(nj.NnjitError) as ei:
        nj.nnjit_gemv_bf16_noalloc(M, N, K, x, W, None, C, split)
    assert ei.value.status == nj.NNJIT_ERR_UNSUPPORTED
    assert "scratch" in str(ei.value)
    with pytest.raises(nj.NnjitError) as ei:
        nj.nnjit_gemv_bf16_noalloc(9, N, K, x, W, None, C, 1)
    assert ei.value.status == nj.NNJIT_ERR_INVALID_ARG


def test_noalloc_rejects_unaligned_operands():
    import torch
    M, N, K = 1, 256, 64
    x = torch.zeros((M, K + 8), dtype=torch.bfloat16, device="cuda")
    W = torch.zeros((N, K), dtype=torch.bfloat16, device="cuda")
    C = torch.zeros((M, N + 1), dtype=torch.float32, device="cuda")
    cases = [
        (M, N, 12, x, W, C[:, :N]),            # K not a multiple of 8
        (M, N, K, x[:, 1:], W, C[:, :N]),      # x 2 bytes past a 16-byte boundary
    ]
    for m, n, k, xx, ww, cc in cases:
        with pytest.raises(nj.NnjitError) as ei:
            nj.nnjit_gemv_bf16_noalloc(m, n, k, xx, ww, None, cc, 1)
        assert ei.value.status == nj.NNJIT_ERR_UNSUPPORTED
        assert "aligned" in str(ei.value)
