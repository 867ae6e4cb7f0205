"""The bench's bookkeeping on the CPU: the flop count of fused attention (visible query-key
pairs against a brute-force count of the causal mask), whole-job throughput, the
algorithmic bytes of a product (each operand once, C in f32, the bias; written out for one
shape), the traffic table lookup and the kernel keys it is indexed by."""
import os

import numpy as np
import pytest

import bench
from synthetic import Shape, WORKLOADS


def _visible_pairs(Lq, Lk, causal):
    """Brute force: query i sees key j when j <= i + (Lk - Lq) under the causal mask."""
    i = np.arange(Lq)[:, None]
    j = np.arange(Lk)[None, :]
    mask = (j <= i + (Lk - Lq)) if causal else np.ones((Lq, Lk), bool)
    return int(mask.sum())


@pytest.mark.parametrize("Lq,Lk", [(1, 1), (5, 3), (3, 5), (128, 128), (200, 70), (70, 200), (1, 300)])
@pytest.mark.parametrize("causal", [False, True])
def test_attention_flops_count_visible_pairs(Lq, Lk, causal):
    B, d = 3, 64
    assert bench.attention_flops(B, Lq, Lk, d, causal) == 4 * d * B * _visible_pairs(Lq, Lk, causal)


def test_attention_flops_closed_forms():
    # square causal: n (n + 1) / 2 pairs; the Llama-2 prefill heads and the T5-large heads
    n = 1024
    assert bench.attention_flops(128, n, n, 128, True) == 4 * 128 * 128 * n * (n + 1) // 2
    assert bench.attention_flops(128, 256, 256, 64, False) == 4 * 64 * 128 * 256 * 256
    B, Lq, Lk, d, causal = bench.ATTENTION_WORKLOADS["llama2_7b_prefill_attention"]
    assert bench.attention_flops(B, Lq, Lk, d, causal) == 34393292800


def test_job_throughput():
    # 2 replicas x 1e12 flop x 10 steps in 5 ms = 4000 TFLOP/s
    assert bench.job_throughput(2, 10**12, 10, 5.0) == pytest.approx(4000.0)
    assert bench.max_over_ranks(3.5, 1) == 3.5


def test_shape_bytes_bart_qkv():
    s = WORKLOADS["bart_base_encoder_m512"].shapes[0]
    assert (s.M, s.N, s.K, s.has_bias) == (512, 2304, 768, True)
    want = 512 * 768 * 4 + 768 * 2304 * 4 + 512 * 2304 * 4 + 2304 * 4   # A, B, C (f32), bias
    assert bench.shape_bytes(s, "tf32") == want
    bf = Shape("x", M=4, N=8, K=16, has_bias=False)
    assert bench.shape_bytes(bf, "bf16") == 4 * 16 * 2 + 16 * 8 * 2 + 4 * 8 * 4


def test_kernel_key_format():
    s = Shape("ffn_down", M=512, N=768, K=3072, has_bias=True)
    cand = {"family": 1, "bm": 128, "bn": 256, "bk": 32, "stages": 4, "split_k": 8, "reduce": 0, "raster": 1}
    assert bench.kernel_key(s, "tf32", cand) == "tc tf32 1x512x768x3072 NK bm128 bn256 bk32 st4 split8 red0 rast1"


def test_traffic_table_lookup():
    assert bench.lookup_traffic("tc tf32 1x512x768x3072 NK bm128 bn256 bk32 st4 split8 red0 rast1") > 0
    assert bench.lookup_traffic("attention tcgen05 d128 B128 Lq1024 Lk1024 causal") > 0
    assert bench.lookup_traffic("no such kernel") is None
    # every entry is "key | integer bytes"
    path = os.path.join(bench.ROOT, "profiles", "dram_traffic.txt")
    with open(path) as f:
        rows = [ln.strip() for ln in f if ln.strip() and not ln.startswith("#")]
    assert rows and all("|" in r and int(r.rsplit("|", 1)[1]) > 0 for r in rows)
