"""Counter-based seeded generators and the transformer-Linear workloads.

Generator: SplitMix64 (Steele, Lea and Flood, "Fast splittable pseudorandom number
generators", OOPSLA 2014).  Output i (i = 0, 1, ...) of the stream with seed s is
mix(s + (i + 1) * 0x9E3779B97F4A7C15) with the published 64-bit finaliser, so any
element can be drawn independently of the others (vectorised here with numpy uint64
arithmetic, which wraps modulo 2**64).

  * uniform[-1, 1): u = (z >> 11) * 2**-53 in [0, 1), then 2u - 1.
  * normal N(0, 1): Box-Muller on consecutive pairs (u1, u2):
        r = sqrt(-2 ln(1 - u1)),  out[2p] = r cos(2 pi u2),  out[2p+1] = r sin(2 pi u2).
  * small integers in [-8, 8]: floor(17 u) - 8 (exact in bf16, tf32 and f32).

Per-tensor seed: base_seed * 16 + tensor_id (base_seed = the workload's index 0..4).
Values are drawn in float64, scaled, rounded once to float32 (round-to-nearest-even,
numpy's conversion) and, for bf16 operands, from float32 to bf16 with
round-to-nearest-even on the bit pattern.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

_GAMMA = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
_CHUNK = 1 << 22


def _mix(z: np.ndarray) -> np.ndarray:
    z = (z ^ (z >> np.uint64(30))) * _M1
    z = (z ^ (z >> np.uint64(27))) * _M2
    return z ^ (z >> np.uint64(31))


def splitmix64(seed: int, n: int, offset: int = 0) -> np.ndarray:
    """Outputs offset .. offset+n-1 of the SplitMix64 stream seeded with `seed`."""
    with np.errstate(over="ignore"):
        idx = np.arange(offset + 1, offset + n + 1, dtype=np.uint64)
        return _mix(np.uint64(seed & 0xFFFFFFFFFFFFFFFF) + idx * _GAMMA)


def _unit(seed: int, n: int, offset: int = 0) -> np.ndarray:
    z = splitmix64(seed, n, offset)
    return (z >> np.uint64(11)).astype(np.float64) * (2.0 ** -53)


def uniform(seed: int, n: int, lo: float = -1.0, hi: float = 1.0) -> np.ndarray:
    out = np.empty(n, dtype=np.float64)
    for s in range(0, n, _CHUNK):
        e = min(n, s + _CHUNK)
        out[s:e] = lo + (hi - lo) * _unit(seed, e - s, s)
    return out


def normal(seed: int, n: int, std: float = 1.0) -> np.ndarray:
    out = np.empty(n, dtype=np.float64)
    pairs = (n + 1) // 2
    for s in range(0, pairs, _CHUNK):
        e = min(pairs, s + _CHUNK)
        u = _unit(seed, 2 * (e - s), 2 * s)
        r = np.sqrt(-2.0 * np.log1p(-u[0::2]))
        th = 2.0 * np.pi * u[1::2]
        blk = np.empty(2 * (e - s), dtype=np.float64)
        blk[0::2] = r * np.cos(th)
        blk[1::2] = r * np.sin(th)
        lo, hi = 2 * s, min(n, 2 * e)
        out[lo:hi] = std * blk[: hi - lo]
    return out


def small_ints(seed: int, n: int, lo: int = -8, hi: int = 8) -> np.ndarray:
    out = np.empty(n, dtype=np.float64)
    span = hi - lo + 1
    for s in range(0, n, _CHUNK):
        e = min(n, s + _CHUNK)
        out[s:e] = np.floor(span * _unit(seed, e - s, s)) + lo
    return out


def to_f32(x: np.ndarray) -> np.ndarray:
    return np.asarray(x, dtype=np.float64).astype(np.float32)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit patterns (uint16), round-to-nearest-even.  Inputs are finite."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    rounded = (u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))) >> np.uint64(16)
    return rounded.astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Inverse view used by the GPU-side tests (exact)."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


# ----------------------------------------------------------------------------------------
# Workloads: the transformer Linears / attention BatchMatMuls the operator is run on.
# ----------------------------------------------------------------------------------------

TENSOR_IDS = {"A": 0, "B": 1, "bias": 2, "Q": 12, "K": 13, "P": 14, "V": 15}


def tensor_seed(base_seed: int, tensor_id: int) -> int:
    return base_seed * 16 + tensor_id


@dataclass(frozen=True)
class Shape:
    name: str
    M: int
    N: int
    K: int
    batch: int = 1
    b_layout: str = "NK"          # "KN": B stored [K,N]; "NK": B stored [N,K]
    has_bias: bool = False
    a_dist: tuple = ("normal", 1.0)
    b_dist: tuple = ("normal", 0.02)
    bias_dist: tuple = ("normal", 0.02)
    ids: tuple = (0, 1, 2)        # tensor ids of A, B, bias
    b_is_weight: bool = True      # B is a model weight (constant across calls)

    @property
    def flops(self) -> int:
        return 2 * self.batch * self.M * self.N * self.K


@dataclass(frozen=True)
class Workload:
    key: str
    index: int                    # base seed
    title: str
    dtypes: tuple                 # operand dtype paths: "f32_ffma", "tf32", "bf16"
    shapes: tuple = field(default_factory=tuple)


def _linears(Ms, NKs, names, layout="NK", has_bias=False, a=("normal", 1.0),
             b=("normal", 0.02), bias=("normal", 0.02)):
    out = []
    for s, ((N, K), nm) in enumerate(zip(NKs, names)):
        out.append(Shape(nm, Ms, N, K, 1, layout, has_bias, a, b, bias,
                         (3 * s, 3 * s + 1, 3 * s + 2)))
    return tuple(out)


WORKLOADS = {
    "bart_linear_m64": Workload(
        "bart_linear_m64", 0,
        "Single FP32 MatMul C=A.B+bias, M=64 K=768 N=768, uniform[-1,1], seed 0, row-major",
        ("f32_ffma", "tf32"),
        (Shape("linear", 64, 768, 768, 1, "KN", True, ("uniform", 1.0), ("uniform", 1.0),
               ("uniform", 1.0), (0, 1, 2)),)),
    "bart_base_encoder_m512": Workload(
        "bart_base_encoder_m512", 1,
        "BART-base encoder layer Linears, batch 4 x seq 128 (M=512), TF32",
        ("tf32",),
        _linears(512, [(2304, 768), (768, 768), (3072, 768), (768, 3072)],
                 ["qkv", "out_proj", "ffn_up", "ffn_down"], has_bias=True)),
    "t5_large_layer_m2048": Workload(
        "t5_large_layer_m2048", 2,
        "T5-large layer, batch 8 x seq 256 (M=2048): Linears + attention QK^T / PV, BF16",
        ("bf16",),
        _linears(2048, [(1024, 1024), (4096, 1024), (1024, 4096), (4096, 4096)],
                 ["q_k_v_o", "wi", "wo", "n4096_k4096"]) + (
            Shape("qk_t", 256, 256, 64, 128, "NK", False, ("normal", 1.0), ("normal", 1.0),
                  ("normal", 0.0), (12, 13, 2), False),
            Shape("pv", 256, 64, 256, 128, "KN", False, ("normal", 1.0), ("normal", 1.0),
                  ("normal", 0.0), (14, 15, 2), False))),
    "llama2_7b_decode_m1": Workload(
        "llama2_7b_decode_m1", 3,
        "Llama-2-7B decoder block decode GEMVs, batch 1 (M=1), BF16",
        ("bf16",),
        _linears(1, [(12288, 4096), (4096, 4096), (22016, 4096), (4096, 11008)],
                 ["qkv", "o_proj", "gate_up", "down"])),
    "llama2_7b_prefill_m4096": Workload(
        "llama2_7b_prefill_m4096", 4,
        "Llama-2-7B decoder block prefill, batch 4 x seq 1024 (M=4096), BF16",
        ("bf16",),
        _linears(4096, [(12288, 4096), (4096, 4096), (22016, 4096), (4096, 11008)],
                 ["qkv", "o_proj", "gate_up", "down"]) + (
            Shape("qk_t", 1024, 1024, 128, 128, "NK", False, ("normal", 1.0), ("normal", 1.0),
                  ("normal", 0.0), (12, 13, 2), False),
            Shape("pv", 1024, 128, 1024, 128, "KN", False, ("normal", 1.0), ("normal", 1.0),
                  ("normal", 0.0), (14, 15, 2), False))),
    "llama2_7b_decode_w4_m1": Workload(
        "llama2_7b_decode_w4_m1", 6,
        "Llama-2-7B decoder block decode GEMVs, batch 1 (M=1), 4-bit weights with bf16 group "
        "scales (group 128), bf16 activations",
        ("w4_bf16",),
        _linears(1, [(12288, 4096), (4096, 4096), (22016, 4096), (4096, 11008)],
                 ["qkv", "o_proj", "gate_up", "down"])),
}


def _draw(dist: tuple, seed: int, n: int, ints: bool) -> np.ndarray:
    if ints:
        return small_ints(seed, n)
    kind, scale = dist
    if kind == "uniform":
        return uniform(seed, n, -scale, scale)
    if kind == "normal":
        return normal(seed, n, scale)
    raise ValueError(kind)


def w4_blob(codes: np.ndarray, scale_bits: np.ndarray, ldb: int = 0) -> np.ndarray:
    """The storage of 4-bit weights (nnjit_w4_layout): codes [N][K] in 0..15, two per byte
    (row n at byte n * ldb / 2, code k in byte k / 2, the low nibble holding the even k),
    then, from the code block rounded up to 256 bytes, the bf16 scale bit patterns
    [ceil(K / 128)][N] (group-major)."""
    N, K = codes.shape
    ldb = ldb or K
    row = ldb // 2
    off = (N * row + 255) // 256 * 256
    blob = np.zeros(off + scale_bits.size * 2, dtype=np.uint8)
    c = np.zeros((N, 2 * row), dtype=np.uint8)
    c[:, :K] = codes
    blob[:N * row] = (c[:, 0::2] | (c[:, 1::2] << 4)).ravel()
    blob[off:] = np.ascontiguousarray(scale_bits, dtype=np.uint16).view(np.uint8).ravel()
    return blob


def make_w4_operands(shape: Shape, base_seed: int, ints: bool = False, ldb: int = 0):
    """Operands of one product over 4-bit weights: x as bf16 bit patterns [M][K] (the
    shape's A distribution), the weight blob (codes drawn uniformly from 0..15, scales
    uniform in [0.002, 0.01) rounded to bf16 -- about the magnitude of a symmetric 4-bit
    quantisation of N(0, 0.02^2) weights), and the bias.  `ints`: x in [-8, 8] and every
    scale 1, so every product and sum is an exact integer."""
    ida, idb, idbias = shape.ids
    N, K = shape.N, shape.K
    x = _draw(shape.a_dist, tensor_seed(base_seed, ida), shape.M * K, ints)
    x_bits = f32_to_bf16_bits(to_f32(x).reshape(shape.M, K))
    seed_b = tensor_seed(base_seed, idb)
    codes = np.floor(16.0 * _unit(seed_b, N * K)).astype(np.uint8).reshape(N, K)
    groups = (K + 127) // 128
    if ints:
        scales = np.ones((groups, N), dtype=np.float32)
    else:
        scales = to_f32(uniform(seed_b ^ 0x5CA1E, groups * N, 0.002, 0.01)).reshape(groups, N)
    blob = w4_blob(codes, f32_to_bf16_bits(scales), ldb)
    bias = None
    if shape.has_bias:
        bias = to_f32(_draw(shape.bias_dist, tensor_seed(base_seed, idbias), N, ints))
    return x_bits, blob, bias


def make_operands(shape: Shape, base_seed: int, dtype: str, ints: bool = False,
                  M: int | None = None):
    """Operands of one product in their storage form.

    dtype "bf16": A, B as uint16 bf16 bit patterns; "f32_ffma"/"tf32": float32.
    bias (when the shape has one) is float32.  A is [batch,]M,K; B is [batch,]K,N (KN)
    or [batch,]N,K (NK).  `ints` draws integers in [-8, 8] instead (exact-mode tests).
    `M` overrides the row count (the first M rows of the full-size A are drawn, so a
    sample of rows equals the corresponding rows of the full operand).
    """
    if dtype == "w4_bf16":
        if M is not None:
            raise ValueError("row override not supported for 4-bit weights")
        return make_w4_operands(shape, base_seed, ints)
    Mr = shape.M if M is None else M
    ida, idb, idbias = shape.ids
    bshape = (shape.K, shape.N) if shape.b_layout == "KN" else (shape.N, shape.K)
    lead = (shape.batch,) if shape.batch > 1 else ()
    if shape.batch > 1 and M is not None:
        raise ValueError("row override only for non-batched shapes")
    a = _draw(shape.a_dist, tensor_seed(base_seed, ida), shape.batch * Mr * shape.K, ints)
    b = _draw(shape.b_dist, tensor_seed(base_seed, idb),
              shape.batch * shape.K * shape.N, ints)
    A = to_f32(a).reshape(lead + (Mr, shape.K))
    B = to_f32(b).reshape(lead + bshape)
    bias = None
    if shape.has_bias:
        bias = to_f32(_draw(shape.bias_dist, tensor_seed(base_seed, idbias), shape.N, ints))
    if dtype == "bf16":
        A, B = f32_to_bf16_bits(A), f32_to_bf16_bits(B)
    elif dtype not in ("f32_ffma", "tf32"):
        raise ValueError(dtype)
    return A, B, bias
