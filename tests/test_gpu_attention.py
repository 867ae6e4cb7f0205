"""Fused attention (nnjit_attention) against the FP64 oracle, through the C ABI: ragged
lengths (partial key and query blocks), both head dimensions, the causal mask with
Lk > Lq and Lk < Lq (queries with no key), single queries, empty inputs, exact special
cases, and the T5-large and Llama-2 prefill attention shapes on sampled heads."""
import numpy as np
import pytest

import oracle
from oracle.attention import attention as attention_ref
from synthetic import f32_to_bf16_bits, normal

pytestmark = pytest.mark.gpu

nj = pytest.importorskip("paper_2309_08978_gb300")
torch = pytest.importorskip("torch")

TOL = 1e-2  # P is rounded to bf16 for the P V product


def _bf16(shape, seed):
    return f32_to_bf16_bits(normal(seed, int(np.prod(shape)), 1.0).astype(np.float32).reshape(shape))


def _dev(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()


KERNELS = {"tcgen05": 1, "mma": 2, "tcgen05_2t": 3}


def _run(Q, K, V, causal, scale, kernel=1):
    B, Lq, d = Q.shape
    O = torch.full((B, Lq, d), float("nan"), dtype=torch.float32, device="cuda")
    nj.nnjit_attention(_dev(Q), _dev(K), _dev(V), O, causal=causal, scale=scale, kernel=kernel)
    nj.nnjit_attention_check()
    return O.cpu().numpy()


CASES = [(2, 64, 64, 64, False), (3, 100, 130, 64, False), (2, 128, 128, 128, True),
         (1, 70, 200, 64, True), (1, 200, 70, 128, True), (4, 256, 256, 64, False),
         (2, 1, 300, 128, True), (2, 333, 333, 128, False), (1, 65, 1, 64, False),
         # more query blocks than SMs: persistent CTAs take several items each
         (160, 130, 200, 64, True), (90, 256, 130, 128, False)]


@pytest.mark.parametrize("kernel", list(KERNELS))
@pytest.mark.parametrize("case", CASES, ids=lambda c: "b{}-q{}-k{}-d{}{}".format(*c[:4], "-causal" if c[4] else ""))
def test_attention_matches_oracle(case, kernel):
    B, Lq, Lk, d, causal = case
    Q, K, V = _bf16((B, Lq, d), 1), _bf16((B, Lk, d), 2), _bf16((B, Lk, d), 3)
    scale = 1.0 / np.sqrt(d)
    O = _run(Q, K, V, causal, scale, KERNELS[kernel])
    ref = attention_ref(Q, K, V, scale, causal)
    assert np.all(np.isfinite(O))
    if causal and Lq > Lk:
        assert np.array_equal(O[:, :Lq - Lk], np.zeros_like(O[:, :Lq - Lk]))   # no visible key
    assert oracle.rel_fro(O, ref) <= TOL


@pytest.mark.parametrize("kernel", list(KERNELS))
def test_attention_exact_special_cases(kernel):
    """One key: every weight is exactly 1, so O is the value row bit for bit.  Lk = 0:
    O = 0.  Lq = 0: nothing is written."""
    V = _bf16((3, 1, 128), 4)
    O = _run(_bf16((3, 77, 128), 5), _bf16((3, 1, 128), 6), V, False, 0.3, KERNELS[kernel])
    want = oracle.bf16_bits_to_f64(V).astype(np.float32)
    assert np.array_equal(O, np.broadcast_to(want, O.shape))
    Q = _bf16((2, 10, 64), 7)
    O = torch.full((2, 10, 64), float("nan"), device="cuda")
    nj.nnjit_attention(_dev(Q), _dev(np.zeros((2, 1, 64), np.uint16)), _dev(np.zeros((2, 1, 64), np.uint16)),
                       O, scale=1.0, kernel=KERNELS[kernel])   # Lk = 1 with zero values
    torch.cuda.synchronize()
    assert np.array_equal(O.cpu().numpy(), np.zeros((2, 10, 64), np.float32))
    desc = nj.nnjit_attention_desc(2, 10, 0, 64, 0, 1.0, KERNELS[kernel])
    O.fill_(float("nan"))
    lib = nj.load_library()
    assert lib.nnjit_attention(desc, _dev(Q).data_ptr(), None, None, O.data_ptr(), None) == 0
    torch.cuda.synchronize()
    assert np.array_equal(O.cpu().numpy(), np.zeros((2, 10, 64), np.float32))


def test_attention_refusals():
    lib = nj.load_library()
    x = torch.zeros(64, dtype=torch.float32, device="cuda")
    p = x.data_ptr()
    for d, st in (((1, 4, 4, 96, 0, 1.0), nj.NNJIT_ERR_UNSUPPORTED), ((0, 4, 4, 64, 0, 1.0), nj.NNJIT_ERR_INVALID_ARG),
                  ((1, 4, 4, 64, 2, 1.0), nj.NNJIT_ERR_INVALID_ARG), ((1, -1, 4, 64, 0, 1.0), nj.NNJIT_ERR_INVALID_ARG),
                  ((1, 4, 4, 64, 0, float("inf")), nj.NNJIT_ERR_INVALID_ARG),
                  ((1, 4, 4, 64, 0, 1.0, 4), nj.NNJIT_ERR_INVALID_ARG)):
        assert lib.nnjit_attention(nj.nnjit_attention_desc(*d), p, p, p, p, None) == st
    assert lib.nnjit_attention(nj.nnjit_attention_desc(1, 4, 4, 64, 0, 1.0), p + 4, p, p, p, None) == \
        nj.NNJIT_ERR_UNSUPPORTED


@pytest.mark.parametrize("kernel", list(KERNELS))
@pytest.mark.parametrize("shape", [(128, 256, 256, 64, False), (128, 1024, 1024, 128, True)],
                         ids=["t5_large_heads", "llama2_prefill_heads"])
def test_attention_full_size_sampled_heads(shape, kernel):
    """The attention of the T5-large layer (8 x 16 heads, 256 tokens, d = 64) and of the
    Llama-2 prefill (4 x 32 heads, 1024 tokens, d = 128, causal), run in full; five heads
    compared with the oracle."""
    B, Lq, Lk, d, causal = shape
    Q, K, V = _bf16((B, Lq, d), 8), _bf16((B, Lk, d), 9), _bf16((B, Lk, d), 10)
    O = _run(Q, K, V, causal, 1.0 / np.sqrt(d), KERNELS[kernel])
    heads = [0, 1, B // 2, B - 2, B - 1]
    ref = attention_ref(Q[heads], K[heads], V[heads], 1.0 / np.sqrt(d), causal)
    assert oracle.rel_fro(O[heads], ref) <= TOL


def test_attention_tune_records_the_faster_kernel():
    """nnjit_attention_tune times the three kernels on the caller's buffers and records the
    fastest for the shape; AUTO calls then use it and stay within the oracle's tolerance."""
    B, Lq, Lk, d = 4, 200, 260, 64
    Q, K, V = _bf16((B, Lq, d), 11), _bf16((B, Lk, d), 12), _bf16((B, Lk, d), 13)
    dQ, dK, dV = _dev(Q), _dev(K), _dev(V)
    O = torch.empty((B, Lq, d), dtype=torch.float32, device="cuda")
    times, chosen = nj.nnjit_attention_tune(dQ, dK, dV, O, causal=True, reps=5)
    assert len(times) == 3 and all(t > 0 for t in times)
    kernels = (nj.NNJIT_ATTN_TCGEN05, nj.NNJIT_ATTN_MMA, nj.NNJIT_ATTN_TCGEN05_2T)
    assert chosen == kernels[min(range(3), key=lambda k: (times[k], k))]
    O.fill_(float("nan"))
    nj.nnjit_attention(dQ, dK, dV, O, causal=True)          # AUTO: the recorded kernel
    nj.nnjit_attention_check()
    assert oracle.rel_fro(O.cpu().numpy(), attention_ref(Q, K, V, 1.0 / np.sqrt(d), True)) <= TOL


def test_two_tile_work_counter_resets():
    """The two-tile kernel hands its items out from a per-launch work counter that the last
    CTA to finish taking items zeroes.  More launches than counter slots, and replays of one
    captured launch (the same slot every time), all give the first launch's output bit for
    bit; the first output matches the oracle on sampled heads."""
    B, Lq, Lk, d = 160, 600, 650, 64           # 160 x 3 items of 256 queries > the SM count
    Q, K, V = _bf16((B, Lq, d), 14), _bf16((B, Lk, d), 15), _bf16((B, Lk, d), 16)
    dQ, dK, dV = _dev(Q), _dev(K), _dev(V)
    kern = KERNELS["tcgen05_2t"]
    O0 = torch.full((B, Lq, d), float("nan"), dtype=torch.float32, device="cuda")
    nj.nnjit_attention(dQ, dK, dV, O0, causal=True, kernel=kern)
    nj.nnjit_attention_check()
    first = O0.cpu().numpy()
    heads = [0, 77, B - 1]
    assert oracle.rel_fro(first[heads], attention_ref(Q[heads], K[heads], V[heads], 1.0 / np.sqrt(d), True)) <= TOL
    O = torch.empty_like(O0)
    for _ in range(70):                        # the launcher cycles through 64 slots
        O.fill_(float("nan"))
        nj.nnjit_attention(dQ, dK, dV, O, causal=True, kernel=kern)
    nj.nnjit_attention_check()
    assert np.array_equal(O.cpu().numpy(), first)
    st = torch.cuda.Stream()
    st.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(st):
        Og = torch.full_like(O0, float("nan"))
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=st):
            nj.nnjit_attention(dQ, dK, dV, Og, causal=True, kernel=kern)
        for _ in range(3):
            Og.fill_(float("nan"))
            g.replay()
    torch.cuda.current_stream().wait_stream(st)
    torch.cuda.synchronize()
    nj.nnjit_attention_check()
    assert np.array_equal(Og.cpu().numpy(), first)


def test_attention_auto_without_a_record():
    """Without a tuning record, AUTO runs the two-tile kernel when its 256-query items fill
    at least half of the SMs and the one-tile tensor-memory kernel otherwise: bit for bit
    the chosen kernel's output."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    for B, kern in ((sms, KERNELS["tcgen05_2t"]), (2, KERNELS["tcgen05"])):
        Lq, Lk, d = 200, 300, 64
        Q, K, V = _bf16((B, Lq, d), 17), _bf16((B, Lk, d), 18), _bf16((B, Lk, d), 19)
        dQ, dK, dV = _dev(Q), _dev(K), _dev(V)
        want = torch.full((B, Lq, d), float("nan"), dtype=torch.float32, device="cuda")
        got = torch.full_like(want, float("nan"))
        nj.nnjit_attention(dQ, dK, dV, want, kernel=kern)
        nj.nnjit_attention(dQ, dK, dV, got)                  # AUTO, no record for this shape
        nj.nnjit_attention_check()
        assert torch.equal(got, want)
