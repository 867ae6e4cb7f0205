"""The seeded input generators: published SplitMix64 values, rounding rules, workload
shapes (these inputs feed both the oracle and the GPU path)."""
import numpy as np
import pytest

from synthetic import (splitmix64, uniform, normal, small_ints, f32_to_bf16_bits,
                       bf16_bits_to_f32, WORKLOADS, make_operands)


def test_splitmix64_published_values():
    # seed 0: first output of the reference splitmix64.c
    assert int(splitmix64(0, 1)[0]) == 0xE220A8397B1DCDAF
    # seed 1234567: the first five outputs quoted with the reference implementation
    want = [6457827717110365317, 3203168211198807973, 9817491932198370423,
            4593380528125082431, 16408922859458223821]
    assert [int(v) for v in splitmix64(1234567, 5)] == want


def test_counter_based_offsets():
    full = splitmix64(42, 100)
    assert np.array_equal(splitmix64(42, 30, offset=70), full[70:])


def test_uniform_range_and_moments():
    u = uniform(3, 200000)
    assert u.min() >= -1.0 and u.max() < 1.0
    assert abs(u.mean()) < 0.01 and abs(u.var() - 1.0 / 3.0) < 0.01


def test_normal_moments():
    x = normal(4, 200001, 0.02)
    assert abs(x.mean()) < 0.001
    assert abs(x.std() - 0.02) < 0.0005


def test_small_ints_range():
    v = small_ints(5, 100000)
    assert v.min() == -8 and v.max() == 8
    assert np.all(v == np.round(v))


def test_bf16_round_to_nearest_even():
    one = 1.0
    vals = np.array([one, one + 2.0 ** -8, one + 3 * 2.0 ** -8, one + 2.0 ** -8 + 2.0 ** -20,
                     -2.5, 0.0], dtype=np.float32)
    bits = f32_to_bf16_bits(vals)
    assert [int(b) for b in bits] == [0x3F80, 0x3F80, 0x3F82, 0x3F81, 0xC020, 0x0000]
    assert np.array_equal(bf16_bits_to_f32(bits)[[0, 4]], np.array([1.0, -2.5], np.float32))


def test_workload_shapes():
    w = WORKLOADS["bart_base_encoder_m512"]
    assert [(s.M, s.N, s.K) for s in w.shapes] == [(512, 2304, 768), (512, 768, 768),
                                                   (512, 3072, 768), (512, 768, 3072)]
    p = WORKLOADS["llama2_7b_prefill_m4096"]
    assert p.shapes[-2].batch == 128 and (p.shapes[-2].M, p.shapes[-2].N, p.shapes[-2].K) == (1024, 1024, 128)
    ids = [i for s in p.shapes for i in s.ids[:2]]
    assert len(set(ids)) == len(ids)


def test_make_operands_row_prefix_and_types():
    s = WORKLOADS["bart_base_encoder_m512"].shapes[1]
    A, B, bias = make_operands(s, 1, "tf32")
    A8, B8, bias8 = make_operands(s, 1, "tf32", M=8)
    assert A.shape == (512, 768) and B.shape == (768, 768) and bias.shape == (768,)
    assert np.array_equal(A[:8], A8) and np.array_equal(B, B8)
    s3 = WORKLOADS["t5_large_layer_m2048"].shapes[4]
    Q, K, nb = make_operands(s3, 2, "bf16")
    assert Q.dtype == np.uint16 and Q.shape == (128, 256, 64) and K.shape == (128, 256, 64)
    assert nb is None


def test_int_mode_is_exact_in_bf16():
    s = WORKLOADS["llama2_7b_decode_m1"].shapes[1]
    A, B, _ = make_operands(s, 3, "bf16", ints=True)
    assert np.array_equal(bf16_bits_to_f32(A), np.round(bf16_bits_to_f32(A)))
    assert np.abs(bf16_bits_to_f32(B)).max() <= 8
