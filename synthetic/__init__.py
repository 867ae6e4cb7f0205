"""Seeded synthetic inputs shared by the oracle side and the GPU side of the tests and
the bench.  This package holds no arithmetic of the operator itself: it only draws
numbers and rounds them to the storage types (f32, bf16, packed 4-bit codes) the operator
consumes."""
from .gen import (  # noqa: F401
    splitmix64, uniform, normal, to_f32, f32_to_bf16_bits, bf16_bits_to_f32,
    small_ints, tensor_seed, TENSOR_IDS, WORKLOADS, Workload, Shape, make_operands,
    make_w4_operands, w4_blob,
)
