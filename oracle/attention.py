"""Attention -- TEST INFRASTRUCTURE ONLY.

The attention BatchMatMuls of the paper's workloads (Table 3, K2 = Q K^T and K3 = P V;
the transformer layers of BART, T5 and Llama 2, Sec. 7.1) with the softmax between them,
written as their definition in FP64:

    S[i][j] = scale * sum_c Q[i][c] K[j][c]
    P[i][j] = exp(S[i][j] - max_j' S[i][j']) / sum_j'' exp(S[i][j''] - max_j' S[i][j'])
    O[i][c] = sum_j P[i][j] V[j][c]

over the keys j a query may see (all of them, or with `causal`, j <= i + (Lk - Lq)); a
query that sees no key has O = 0.  Inputs are bf16 bit patterns, widened exactly.
"""
from __future__ import annotations

import numpy as np

from .matmul import bf16_bits_to_f64


def attention(Q_bits: np.ndarray, K_bits: np.ndarray, V_bits: np.ndarray, scale: float,
              causal: bool = False) -> np.ndarray:
    """O [batch][Lq][d] in float64 from Q [batch][Lq][d], K, V [batch][Lk][d]."""
    Q = bf16_bits_to_f64(np.asarray(Q_bits, dtype=np.uint16))
    K = bf16_bits_to_f64(np.asarray(K_bits, dtype=np.uint16))
    V = bf16_bits_to_f64(np.asarray(V_bits, dtype=np.uint16))
    batch, Lq, d = Q.shape
    Lk = K.shape[1]
    O = np.zeros((batch, Lq, d), dtype=np.float64)
    for b in range(batch):
        S = scale * (Q[b] @ K[b].T)                              # [Lq][Lk]
        for i in range(Lq):
            last = i + (Lk - Lq) if causal else Lk - 1           # last key query i sees
            if last < 0:
                continue
            row = S[i, :last + 1]
            e = np.exp(row - row.max())
            O[b, i] = (e / e.sum()) @ V[b, :last + 1]
    return O
