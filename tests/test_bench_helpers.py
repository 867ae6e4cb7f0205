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
    # 1e12 flop x 10 steps in 5 ms = 2000 TFLOP/s
    assert bench.job_throughput(10**12, 10, 5.0) == pytest.approx(2000.0)


def test_prefix_curve():
    # candidate 3 of 8 is the fastest: prefixes shorter than 4 see 12 us at best
    times = {0: 20.0, 1: 12.0, 2: 15.0, 3: 10.0, 4: 11.0, 5: 30.0, 6: 10.5, 7: 40.0}
    c = bench.prefix_curve(times, 8)
    assert c["first_1"] == 2.0 and c["first_2"] == 1.2 and c["first_3"] == 1.2
    assert c["first_5"] == 1.0 and c["first_10"] == 1.0
    assert c["first_10pct"] == 2.0       # ceil(0.8) = 1 candidate
    assert c["first_25pct"] == 1.2       # 2 candidates
    assert c["first_50pct"] == 1.0       # 4 candidates
    # untimed (failed) candidates are skipped
    assert bench.prefix_curve({1: 5.0, 2: 4.0}, 3)["first_1"] is None


def test_more_than_one_gpu_is_refused_without_touching_a_gpu(capsys, monkeypatch):
    import json
    monkeypatch.delenv("WORLD_SIZE", raising=False)
    assert bench.main(["--gpus", "2"]) == 0
    line = json.loads(capsys.readouterr().out.strip())
    assert line["n_gpus"] == 2 and "unavailable" in line
    monkeypatch.setenv("WORLD_SIZE", "4")
    monkeypatch.setenv("RANK", "1")
    assert bench.main([]) == 0
    assert capsys.readouterr().out == ""         # only rank 0 prints


def test_both_arms_share_the_config():
    import argparse
    w = WORKLOADS[bench.DEFAULT_WORKLOAD]
    args = argparse.Namespace(epilogue="none")
    cfg = bench.workload_config(w, args)
    assert cfg["workload"] == "llama2_7b_prefill_m4096"
    assert cfg["shapes"][2] == [1, 4096, 22016, 4096, "NK"]
    assert cfg == bench.workload_config(w, args)


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
    assert bench.lookup_traffic("tc bf16 1x4096x22016x4096 NK bm256 bn256 bk64 st6 split1 red2 rast0") > 0
    assert bench.lookup_traffic("no such kernel") is None
    # every entry is "key | integer bytes"
    path = os.path.join(bench.ROOT, "profiles", "dram_traffic.txt")
    with open(path) as f:
        rows = [ln.strip() for ln in f if ln.strip() and not ln.startswith("#")]
    assert rows and all("|" in r and int(r.rsplit("|", 1)[1]) > 0 for r in rows)
