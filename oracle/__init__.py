"""Oracle for the nnJIT MatMul hot path -- TEST INFRASTRUCTURE ONLY.

A plain, slow, obviously correct CPU implementation of what the GPU path computes,
written from the paper:

  * ``matmul``  -- the MatMul / BatchMatMul operator (Sec. 2.2, Table 3) as its
    definition: an FP64 triple loop in plain C (matmul_f64.c), k ascending.
  * ``space``   -- the tile-based hardware-usage formulas and lite-space heuristics
    (Sec. 5.2, Table 1, Table 2) and the candidate evaluation order, restated in
    plain Python, plus the Blackwell readings of those rules used by the library.
  * ``epilogue`` -- the activations a kernel may apply after the bias (textbook
    definitions of ReLU, GELU and SiLU in FP64).
  * ``quant``   -- 4-bit weights with bf16 group scales, dequantised in FP64.
  * ``attention`` -- softmax attention between the two attention BatchMatMuls (Table 3,
    K2 and K3), its definition in FP64.

Only tests/, ``__graft_entry__.smoke()`` and bench.py's CPU-baseline / reference legs
may import this package.  The GPU library shares no code with it.
"""
from .matmul import (  # noqa: F401
    B_KN, B_NK, build, matmul, matmul_rows, rel_fro, bf16_bits_to_f64, to_f64, hw_threads,
)
