"""Pins for the oracle: facts fixed by mathematics, independent of the oracle's code.

Each test is chosen so that a plausible slip in the oracle (a dropped k term, a wrong
index or sign, a transposed operand, bias added per k, a lost batch stride) fails at
least one of them.
"""
import numpy as np
import pytest

import oracle
from oracle import B_KN, B_NK
from synthetic import small_ints, uniform, normal, to_f32, f32_to_bf16_bits

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def _int_operands(seed, batch, M, N, K, layout):
    A = small_ints(seed, batch * M * K).reshape(batch, M, K).astype(np.float32)
    bs = (K, N) if layout == B_KN else (N, K)
    B = small_ints(seed + 1, batch * K * N).reshape((batch,) + bs).astype(np.float32)
    bias = small_ints(seed + 2, N).astype(np.float32)
    return A, B, bias


def _exact_python(A, B, bias, layout):
    """Brute force with Python integers: independent of the C code and of floating point."""
    batch, M, K = A.shape
    N = B.shape[2] if layout == B_KN else B.shape[1]
    out = np.zeros((batch, M, N), dtype=object)
    for b in range(batch):
        for i in range(M):
            for j in range(N):
                s = 0
                for k in range(K):
                    bkj = B[b, k, j] if layout == B_KN else B[b, j, k]
                    s += int(A[b, i, k]) * int(bkj)
                out[b, i, j] = s + (int(bias[j]) if bias is not None else 0)
    return out


@pytest.mark.parametrize("layout", [B_KN, B_NK])
@pytest.mark.parametrize("dims", [(1, 1, 1, 1), (1, 3, 5, 7), (2, 4, 3, 9), (3, 7, 6, 1),
                                  (1, 5, 1, 11), (2, 1, 8, 4)])
@pytest.mark.parametrize("with_bias", [False, True])
def test_bruteforce_exact_integers(layout, dims, with_bias):
    batch, M, N, K = dims
    A, B, bias = _int_operands(100 + sum(dims), batch, M, N, K, layout)
    bias = bias if with_bias else None
    C64, C32 = oracle.matmul(A, B, bias, layout)
    ref = _exact_python(A, B, bias, layout)
    assert C64.shape == (batch, M, N)
    assert np.array_equal(C64, ref.astype(np.float64))
    assert np.array_equal(C32, ref.astype(np.float32))


@pytest.mark.parametrize("layout", [B_KN, B_NK])
def test_identity_bit_exact(layout):
    K = 37
    A = to_f32(uniform(7, 19 * K)).reshape(19, K)
    eye = np.eye(K, dtype=np.float32)
    C64, C32 = oracle.matmul(A, eye, None, layout)
    assert np.array_equal(C32, A)
    assert np.array_equal(C64, A.astype(np.float64))
    # identity on the left: I . B = B (B given in either storage)
    Bm = to_f32(normal(8, K * 23)).reshape(K, 23)
    Bs = Bm if layout == B_KN else np.ascontiguousarray(Bm.T)
    C64, _ = oracle.matmul(eye, Bs, None, layout)
    assert np.array_equal(C64, Bm.astype(np.float64))


def test_permutation_columns_exact():
    K = N = 29
    rng_perm = np.argsort(uniform(9, N))          # a permutation drawn from the generator
    P = np.zeros((K, N), dtype=np.float32)
    P[rng_perm, np.arange(N)] = 1.0               # column j of A.P is column perm[j] of A
    A = to_f32(normal(10, 11 * K)).reshape(11, K)
    C64, _ = oracle.matmul(A, P, None, B_KN)
    assert np.array_equal(C64, A[:, rng_perm].astype(np.float64))
    C64nk, _ = oracle.matmul(A, np.ascontiguousarray(P.T), None, B_NK)
    assert np.array_equal(C64nk, C64)


def test_all_ones_closed_form():
    M, N, K = 5, 6, 1000
    A = np.ones((M, K), dtype=np.float32)
    B = np.ones((K, N), dtype=np.float32)
    bias = to_f32(uniform(11, N))
    C64, _ = oracle.matmul(A, B, bias, B_KN)
    assert np.array_equal(C64, np.broadcast_to(K + bias.astype(np.float64), (M, N)))


def test_k1_outer_product():
    M, N = 13, 17
    a = to_f32(uniform(12, M)).reshape(M, 1)
    b = to_f32(uniform(13, N)).reshape(1, N)
    C64, _ = oracle.matmul(a, b, None, B_KN)
    # the product of two f32 values is exact in f64
    assert np.array_equal(C64, a.astype(np.float64) * b.astype(np.float64))


def test_zero_a_gives_bias_and_k0():
    bias = to_f32(normal(14, 9))
    C64, C32 = oracle.matmul(np.zeros((4, 5), np.float32), np.ones((5, 9), np.float32),
                             bias, B_KN)
    assert np.array_equal(C32, np.broadcast_to(bias, (4, 9)))
    C64, _ = oracle.matmul(np.zeros((4, 0), np.float32), np.zeros((0, 9), np.float32),
                           bias, B_KN)
    assert np.array_equal(C64, np.broadcast_to(bias.astype(np.float64), (4, 9)))


def test_empty_shapes():
    C64, C32 = oracle.matmul(np.zeros((0, 5), np.float32), np.zeros((5, 3), np.float32))
    assert C64.shape == (0, 3) and C32.shape == (0, 3)
    C64, _ = oracle.matmul(np.zeros((2, 5), np.float32), np.zeros((5, 0), np.float32))
    assert C64.shape == (2, 0)


@pytest.mark.parametrize("layout", [B_KN, B_NK])
def test_numpy_float64_matmul_agreement(layout):
    M, N, K = 67, 129, 300
    A = to_f32(normal(15, M * K)).reshape(M, K)
    Bm = to_f32(normal(16, K * N, 0.02)).reshape(K, N)
    Bs = Bm if layout == B_KN else np.ascontiguousarray(Bm.T)
    bias = to_f32(normal(17, N, 0.02))
    C64, _ = oracle.matmul(A, Bs, bias, layout)
    ref = A.astype(np.float64) @ Bm.astype(np.float64) + bias.astype(np.float64)
    assert oracle.rel_fro(C64, ref) <= 1e-12


def test_layouts_agree_bit_exact():
    M, N, K = 9, 21, 50
    A = to_f32(normal(18, M * K)).reshape(M, K)
    Bm = to_f32(normal(19, K * N)).reshape(K, N)
    c_kn, _ = oracle.matmul(A, Bm, None, B_KN)
    c_nk, _ = oracle.matmul(A, np.ascontiguousarray(Bm.T), None, B_NK)
    assert np.array_equal(c_kn, c_nk)


def test_batched_equals_per_matrix_and_broadcast_b():
    batch, M, N, K = 4, 6, 10, 12
    A = to_f32(normal(20, batch * M * K)).reshape(batch, M, K)
    B = to_f32(normal(21, batch * N * K)).reshape(batch, N, K)
    C64, _ = oracle.matmul(A, B, None, B_NK)
    for b in range(batch):
        cb, _ = oracle.matmul(A[b], B[b], None, B_NK)
        assert np.array_equal(C64[b], cb)
    Cbc, _ = oracle.matmul(A, B[1], None, B_NK)
    for b in range(batch):
        cb, _ = oracle.matmul(A[b], B[1], None, B_NK)
        assert np.array_equal(Cbc[b], cb)


def test_thread_count_invariance():
    A = to_f32(normal(22, 33 * 70)).reshape(33, 70)
    B = to_f32(normal(23, 70 * 45)).reshape(70, 45)
    c1, _ = oracle.matmul(A, B, None, B_KN, nthreads=1)
    c8, _ = oracle.matmul(A, B, None, B_KN, nthreads=8)
    assert np.array_equal(c1, c8)


def test_rows_subset_equals_full():
    A = to_f32(normal(24, 40 * 30)).reshape(40, 30)
    B = to_f32(normal(25, 30 * 20)).reshape(20, 30)
    full, _ = oracle.matmul(A, B, None, B_NK)
    rows = [0, 7, 39]
    sub, _ = oracle.matmul_rows(A, B, None, B_NK, rows)
    assert np.array_equal(sub, full[rows])


def test_bf16_widening_known_patterns():
    bits = np.array([0x0000, 0x8000, 0x3F80, 0xBF80, 0x4000, 0xC000, 0x3F81, 0x4049,
                     0x0001, 0x7F7F], dtype=np.uint16)
    want = np.array([0.0, -0.0, 1.0, -1.0, 2.0, -2.0, 1.0 + 2.0 ** -7,
                     2.0 * (1.0 + 73.0 / 128.0), 2.0 ** -133,
                     (2.0 - 2.0 ** -7) * 2.0 ** 127])
    got = oracle.bf16_bits_to_f64(bits)
    assert np.array_equal(got, want)
    assert np.signbit(got[1])


def test_bf16_operands_match_f32_operands():
    """An operand given as bf16 bits equals the same values given as f32."""
    A = to_f32(normal(26, 8 * 16)).reshape(8, 16)
    B = to_f32(normal(27, 16 * 4)).reshape(16, 4)
    Ab, Bb = f32_to_bf16_bits(A), f32_to_bf16_bits(B)
    from synthetic import bf16_bits_to_f32
    c_bits, _ = oracle.matmul(Ab, Bb, None, B_KN)
    c_f32, _ = oracle.matmul(bf16_bits_to_f32(Ab), bf16_bits_to_f32(Bb), None, B_KN)
    assert np.array_equal(c_bits, c_f32)


def test_rel_fro_closed_form():
    ref = np.array([[3.0, 4.0]])
    assert oracle.rel_fro(ref, ref) == 0.0
    assert oracle.rel_fro(np.array([[3.0, 0.0]]), ref) == pytest.approx(4.0 / 5.0)
    assert oracle.rel_fro(np.zeros((1, 1)), np.zeros((1, 1))) == 0.0


# ---------------------------------------------------------------- fused activations

def test_relu_exact():
    from oracle.epilogue import apply
    x = np.array([-3.5, -0.0, 0.0, 1e-300, 2.25, -1e300])
    assert np.array_equal(apply(x, "relu"), np.array([0.0, 0.0, 0.0, 1e-300, 2.25, 0.0]))


def test_gelu_known_values_and_odd_part():
    """gelu(x) = x Phi(x): Phi(1) = 0.8413447460685429 and Phi(2) = 0.9772498680518208
    (standard normal table); gelu(x) - gelu(-x) = x because Phi(x) + Phi(-x) = 1;
    gelu(0) = 0; for large x, gelu(x) -> x and gelu(-x) -> 0."""
    from oracle.epilogue import apply
    g = apply(np.array([1.0, -1.0, 2.0, 0.0, 12.0, -12.0]), "gelu")
    assert abs(g[0] - 0.8413447460685429) < 1e-15
    assert abs(g[1] + (1.0 - 0.8413447460685429)) < 1e-15
    assert abs(g[2] - 2.0 * 0.9772498680518208) < 1e-15
    assert g[3] == 0.0 and abs(g[4] - 12.0) < 1e-14 and abs(g[5]) < 1e-14
    x = np.random.default_rng(3).normal(0.0, 3.0, 1000)
    assert np.max(np.abs(apply(x, "gelu") - apply(-x, "gelu") - x)) < 1e-13


def test_silu_known_values_and_odd_part():
    """silu(x) = x sigma(x): sigma(ln 3) = 3/4 exactly; silu(x) - silu(-x) = x because
    sigma(x) + sigma(-x) = 1; silu(0) = 0; silu(-800) is -0 without overflow."""
    from oracle.epilogue import apply
    s = apply(np.array([np.log(3.0), 0.0, -800.0, 40.0]), "silu")
    assert abs(s[0] - 0.75 * np.log(3.0)) < 1e-15
    assert s[1] == 0.0 and s[2] == 0.0 and abs(s[3] - 40.0) < 1e-12
    x = np.random.default_rng(4).normal(0.0, 3.0, 1000)
    assert np.max(np.abs(apply(x, "silu") - apply(-x, "silu") - x)) < 1e-13


def test_matmul_applies_activation_after_bias():
    """The fused epilogue acts on the biased sum: with A = 0 the result is act(bias)."""
    from oracle.epilogue import apply
    bias = np.array([-2.0, -0.5, 0.0, 0.5, 2.0], dtype=np.float32)
    A = np.zeros((3, 4), np.float32)
    B = np.ones((4, 5), np.float32)
    for act in ("relu", "gelu", "silu"):
        C64, _ = oracle.matmul(A, B, bias, oracle.B_KN, act=act)
        assert np.array_equal(C64, np.broadcast_to(apply(bias.astype(np.float64), act), (3, 5)))
    # integer sums through relu: negative sums clamp to 0 exactly
    A = np.array([[1, -2], [3, 1]], np.float32)
    B = np.array([[1, 1], [2, -1]], np.float32)
    C64, _ = oracle.matmul(A, B, None, oracle.B_KN, act="relu")
    assert np.array_equal(C64, np.array([[0.0, 3.0], [5.0, 2.0]]))


# ---------------------------------------------------------------- 4-bit weights

def test_w4_dequant_hand_packed_blob():
    """A blob written byte by byte: row 1 holds codes 1, 2 (byte 0x21: the even k in the
    low nibble), code 15 at k = 127 and code 0 at k = 128; scales 0.5 (group 0) and 2.0
    (group 1) of row 1 sit at element N + 1 and 2N + 1 of the group-major scale block,
    which starts at the code block (8 rows x 128 bytes = 1024) rounded up to 256."""
    from oracle.quant import dequant
    N, K = 8, 256
    blob = np.full(1024 + 2 * N * 2, 0x88, dtype=np.uint8)      # every code 8 -> weight 0
    blob[1 * 128 + 0] = 0x21
    blob[1 * 128 + 63] = 0xF8                                     # k = 126 -> 8, k = 127 -> 15
    blob[1 * 128 + 64] = 0x80                                     # k = 128 -> 0, k = 129 -> 8
    scales = np.zeros((2, N), dtype=np.uint16)
    scales[0, 1] = 0x3F00                                         # 0.5
    scales[1, 1] = 0x4000                                         # 2.0
    blob[1024:] = scales.view(np.uint8).ravel()
    W = dequant(blob, N, K)
    assert W.shape == (N, K)
    assert W[1, 0] == (1 - 8) * 0.5 and W[1, 1] == (2 - 8) * 0.5
    assert W[1, 127] == 7 * 0.5 and W[1, 128] == -8 * 2.0
    nz = np.argwhere(W != 0).tolist()
    assert nz == [[1, 0], [1, 1], [1, 127], [1, 128]], nz


def test_w4_dequant_padded_rows_and_ragged_groups():
    """K = 200 (two groups, the second partial) with rows padded to ldb = 224 codes: the
    padding codes are ignored and k = 128..199 take the second group's scale."""
    from oracle.quant import dequant
    from synthetic import w4_blob
    N, K, ldb = 16, 200, 224
    rng = np.random.default_rng(5)
    codes = rng.integers(0, 16, (N, K)).astype(np.uint8)
    sb = np.array([[0x3F80] * N, [0x3E80] * N], dtype=np.uint16)   # 1.0, 0.25
    blob = w4_blob(codes, sb, ldb)
    assert blob.size == (N * ldb // 2 + 255) // 256 * 256 + 2 * N * 2
    W = dequant(blob, N, K, ldb)
    want = (codes.astype(np.float64) - 8) * np.where(np.arange(K) < 128, 1.0, 0.25)
    assert np.array_equal(W, want)


def test_w4_matmul_small_integers_bruteforce():
    """x . W^T with integer x and scale 1: the exact integer sums of (q - 8) x."""
    from oracle.quant import matmul as w4_matmul
    from synthetic import w4_blob
    rng = np.random.default_rng(6)
    M, N, K = 3, 8, 130
    codes = rng.integers(0, 16, (N, K)).astype(np.uint8)
    xi = rng.integers(-8, 9, (M, K))
    blob = w4_blob(codes, np.full((2, N), 0x3F80, np.uint16))
    x_bits = f32_to_bf16_bits(xi.astype(np.float32))
    C64, _ = w4_matmul(x_bits, blob, N, K)
    want = [[sum(int(xi[m, k]) * (int(codes[n, k]) - 8) for k in range(K)) for n in range(N)] for m in range(M)]
    assert np.array_equal(C64, np.array(want, dtype=np.float64))


def test_residual_is_added_after_the_activation():
    """C = act(A.Bt + bias) + R: with A = 0 the result is act(bias) + R; relu on integer
    sums then an integer residual stays exact; a residual of the wrong shape is refused."""
    from oracle.epilogue import apply
    bias = np.array([-2.0, 0.5, 3.0], dtype=np.float32)
    R = np.arange(6, dtype=np.float32).reshape(2, 3) - 2.5
    C64, C32 = oracle.matmul(np.zeros((2, 4), np.float32), np.ones((4, 3), np.float32), bias,
                             oracle.B_KN, act="gelu", residual=R)
    assert np.array_equal(C64, apply(np.broadcast_to(bias.astype(np.float64), (2, 3)), "gelu") + R)
    A = np.array([[1, -2], [3, 1]], np.float32)
    B = np.array([[1, 1], [2, -1]], np.float32)
    R = np.array([[10, -10], [0, 7]], np.float32)
    C64, _ = oracle.matmul(A, B, None, oracle.B_KN, act="relu", residual=R)
    assert np.array_equal(C64, np.array([[10.0, -7.0], [5.0, 9.0]]))
    with pytest.raises(ValueError):
        oracle.matmul(A, B, None, oracle.B_KN, residual=np.zeros((2, 3), np.float32))


# ---------------------------------------------------------------- attention

def _bf(x):
    return f32_to_bf16_bits(np.asarray(x, dtype=np.float32))


def test_attention_bruteforce_tiny():
    """Pure-Python loops with math.exp on a tiny causal and non-causal case."""
    import math
    from oracle.attention import attention
    rng = np.random.default_rng(10)
    Q = rng.integers(-3, 4, (1, 3, 4)).astype(np.float32)
    K = rng.integers(-3, 4, (1, 5, 4)).astype(np.float32)
    V = rng.integers(-3, 4, (1, 5, 4)).astype(np.float32)
    for causal in (False, True):
        O = attention(_bf(Q), _bf(K), _bf(V), 0.5, causal)
        for i in range(3):
            last = i + 2 if causal else 4
            s = [0.5 * sum(float(Q[0, i, c]) * float(K[0, j, c]) for c in range(4)) for j in range(last + 1)]
            mx = max(s)
            w = [math.exp(x - mx) for x in s]
            tot = sum(w)
            for c in range(4):
                want = sum(w[j] / tot * float(V[0, j, c]) for j in range(last + 1))
                assert abs(O[0, i, c] - want) < 1e-12


def test_attention_closed_forms():
    """One key: O = that value row.  Q = 0: uniform weights, O = the mean of the visible
    value rows (prefix means when causal).  A dominant key takes all the weight.  Causal
    with Lq > Lk: queries that see no key get 0, and query Lq - Lk sees key 0 only."""
    from oracle.attention import attention
    rng = np.random.default_rng(11)
    V = rng.integers(-4, 5, (2, 6, 8)).astype(np.float32)
    K = rng.integers(-4, 5, (2, 6, 8)).astype(np.float32)
    Q = rng.integers(-4, 5, (2, 3, 8)).astype(np.float32)
    O = attention(_bf(Q), _bf(K[:, :1]), _bf(V[:, :1]), 0.125)
    assert np.array_equal(O, np.broadcast_to(V[:, :1].astype(np.float64), O.shape))
    O = attention(_bf(np.zeros((2, 6, 8))), _bf(K), _bf(V), 1.0, causal=True)
    want = np.cumsum(V.astype(np.float64), axis=1) / np.arange(1, 7)[None, :, None]
    assert np.max(np.abs(O - want)) < 1e-12
    Kd = np.zeros((1, 4, 8), np.float32)
    Kd[0, 2] = 64.0
    Qd = np.full((1, 2, 8), 64.0, np.float32)
    O = attention(_bf(Qd), _bf(Kd), _bf(V[:1, :4]), 1.0)
    assert np.max(np.abs(O - V[0, 2].astype(np.float64))) < 1e-12
    O = attention(_bf(Q[:1, :3]), _bf(K[:1, :2]), _bf(V[:1, :2]), 0.5, causal=True)
    assert np.array_equal(O[0, 0], np.zeros(8))
    assert np.array_equal(O[0, 1], V[0, 0].astype(np.float64))


def test_attention_invariances():
    """Permuting keys and values together leaves O unchanged; adding one vector u to every
    key shifts each row's scores by a constant (softmax is shift-invariant); with every
    value row equal to ones, O is one (the weights sum to one)."""
    from oracle.attention import attention
    rng = np.random.default_rng(12)
    Q = rng.integers(-2, 3, (3, 5, 16)).astype(np.float32)
    K = rng.integers(-2, 3, (3, 7, 16)).astype(np.float32)
    V = rng.normal(0.0, 1.0, (3, 7, 16)).astype(np.float32)
    O = attention(_bf(Q), _bf(K), _bf(V), 0.25)
    perm = rng.permutation(7)
    assert np.max(np.abs(attention(_bf(Q), _bf(K[:, perm]), _bf(V[:, perm]), 0.25) - O)) < 1e-12
    u = rng.integers(-2, 3, 16).astype(np.float32)
    assert np.max(np.abs(attention(_bf(Q), _bf(K + u), _bf(V), 0.25) - O)) < 1e-12
    ones = attention(_bf(Q), _bf(K), _bf(np.ones_like(V)), 0.25, causal=True)
    assert np.max(np.abs(ones - 1.0)) < 1e-12
