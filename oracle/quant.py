"""4-bit weights -- TEST INFRASTRUCTURE ONLY.

The paper runs Llama 2 7B "under 4-bit quantization" (Sec. 7) without stating the scheme.
The reading used here (and by the library's NNJIT_W4_BF16 path): symmetric 4-bit codes
with one bfloat16 scale per output row and group of 128 consecutive k,

    W[n][k] = (q[n][k] - 8) * s[k // 128][n],    q in 0..15,

stored as a blob: codes two per byte (row n at byte n * ldb / 2, code k in byte k // 2, the
low nibble holding the even k), then, from the code block rounded up to 256 bytes, the
scales group-major.  ``dequant`` rebuilds W in float64 from that blob; ``matmul`` is the
MatMul of oracle.matmul on it.
"""
from __future__ import annotations

import numpy as np

from .matmul import B_NK, bf16_bits_to_f64, matmul as _matmul


def dequant(blob: np.ndarray, N: int, K: int, ldb: int = 0) -> np.ndarray:
    """W [N][K] as float64 from a 4-bit weight blob."""
    ldb = ldb or K
    row = ldb // 2
    blob = np.asarray(blob, dtype=np.uint8)
    codes = blob[:N * row].reshape(N, row)
    q = np.empty((N, 2 * row), dtype=np.int64)
    q[:, 0::2] = codes & 0x0F
    q[:, 1::2] = codes >> 4
    q = q[:, :K]
    off = (N * row + 255) // 256 * 256
    groups = (K + 127) // 128
    s = bf16_bits_to_f64(blob[off:off + groups * N * 2].view(np.uint16).reshape(groups, N))
    return (q - 8).astype(np.float64) * s[np.arange(K) // 128, :].T


def matmul(x_bits: np.ndarray, blob: np.ndarray, N: int, K: int, ldb: int = 0, bias=None,
           act: str = "none", nthreads: int = 0, residual=None):
    """(C64, C32) of x (bf16 bit patterns [M][K]) times the dequantised W^T (+ bias, act,
    + residual)."""
    return _matmul(x_bits, dequant(blob, N, K, ldb), bias, B_NK, nthreads, act, residual)
