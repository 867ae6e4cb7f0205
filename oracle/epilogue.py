"""Elementwise activations fused after the bias -- TEST INFRASTRUCTURE ONLY.

The paper tunes the MatMul of transformer Linears (Sec. 2.2, Table 3); in the models it
evaluates (BART, T5, Llama 2, Sec. 7.1) an FFN Linear is followed by an activation, and
the library can apply it in the kernel that writes C (nnjit_epilogue).  The paper does
not define the activations; these are their textbook definitions, evaluated in FP64:

    relu(x) = max(x, 0)
    gelu(x) = x * Phi(x) = 0.5 * x * (1 + erf(x / sqrt(2)))      (exact GELU, erf form)
    silu(x) = x * sigmoid(x) = x / (1 + exp(-x))

``erf`` comes from the standard library (math.erf), applied element by element.
"""
from __future__ import annotations

import math

import numpy as np

EPILOGUES = ("none", "relu", "gelu", "silu")

_erf = np.vectorize(math.erf, otypes=[np.float64])


def apply(x: np.ndarray, act: str) -> np.ndarray:
    """act(x) in float64 for act in EPILOGUES."""
    x = np.asarray(x, dtype=np.float64)
    if act == "none":
        return x.copy()
    if act == "relu":
        return np.maximum(x, 0.0)
    if act == "gelu":
        return 0.5 * x * (1.0 + _erf(x / math.sqrt(2.0)))
    if act == "silu":
        with np.errstate(over="ignore"):
            return x / (1.0 + np.exp(-x))
    raise ValueError(f"unknown activation {act!r}")
