"""Python face of the C oracle (matmul_f64.c) -- TEST INFRASTRUCTURE ONLY.

Only tests/, ``__graft_entry__.smoke()`` and bench.py's CPU-baseline / reference legs
may import this module.  The GPU library never imports it, and it imports nothing
from the GPU library.

The operator (MatMul / BatchMatMul, Sec. 2.2 and Table 3 of the paper):

    C[b,i,j] = sum_k A[b,i,k] * Bt[b,k,j] + bias[j],   Bt = B (KN) or B^T (NK)

summed in FP64 with k ascending, bias added once at the end.  The result is returned
in FP64 and, rounded once, in FP32 (the output precision of every GPU path).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "matmul_f64.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "liboracle.so")

B_KN = 0  # B stored [K, N] row-major
B_NK = 1  # B stored [N, K] row-major (Linear weight layout, i.e. Bt = B^T)

_lib = None
_lock = threading.Lock()


def build(force: bool = False) -> str:
    """Compile matmul_f64.c with gcc into oracle/_build/liboracle.so (plain C, -O2)."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    # -ffp-contract=off: no fused multiply-add, so every product and sum is rounded
    # separately exactly as the definition reads, on x86 and on Arm alike.
    cmd = ["gcc", "-O2", "-ffp-contract=off", "-fPIC", "-shared", "-std=c11",
           "-o", tmp, _SRC, "-lpthread"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB_PATH)
            i64, dp = ctypes.c_int64, ctypes.c_void_p
            lib.oracle_matmul_f64.restype = ctypes.c_int
            lib.oracle_matmul_f64.argtypes = [
                i64, i64, i64, i64,
                dp, i64, i64,
                dp, ctypes.c_int, i64, i64,
                dp, dp, i64, i64, ctypes.c_int]
            lib.oracle_bf16_to_f64.restype = None
            lib.oracle_bf16_to_f64.argtypes = [dp, dp, i64]
            lib.oracle_hw_threads.restype = ctypes.c_int
            lib.oracle_hw_threads.argtypes = []
            _lib = lib
    return _lib


def hw_threads() -> int:
    return int(_load().oracle_hw_threads())


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns (uint16) to float64, via the C routine."""
    bits = np.ascontiguousarray(bits, dtype=np.uint16)
    out = np.empty(bits.shape, dtype=np.float64)
    _load().oracle_bf16_to_f64(bits.ctypes.data, out.ctypes.data, bits.size)
    return out


def to_f64(x: np.ndarray) -> np.ndarray:
    """Operand values as float64: uint16 arrays are bf16 bit patterns, floats widen."""
    if x.dtype == np.uint16:
        return bf16_bits_to_f64(x)
    if x.dtype in (np.float32, np.float64):
        return np.ascontiguousarray(x, dtype=np.float64)
    raise TypeError(f"unsupported operand dtype {x.dtype}")


def matmul(A: np.ndarray, B: np.ndarray, bias: np.ndarray | None = None,
           b_layout: int = B_KN, nthreads: int = 0, act: str = "none", residual=None):
    """Reference product.

    A: [M,K] or [batch,M,K]; B: [K,N] / [N,K] (KN / NK), optionally with a leading batch
    dimension.  uint16 arrays are bf16 bit patterns.  bias: [N] or None.  act: an
    activation of oracle.epilogue applied in FP64 after the bias (the fused epilogue).
    residual: None, or the prior content of C (shape of the result), added after the
    activation (the residual epilogue: C = act(A.Bt + bias) + C).
    Returns (C64, C32): float64 and float32 arrays of shape [M,N] or [batch,M,N].
    """
    A64, B64 = to_f64(A), to_f64(B)
    squeeze = A64.ndim == 2
    if squeeze:
        A64 = A64[None]
    if B64.ndim == 2:
        B64 = np.broadcast_to(B64, (A64.shape[0],) + B64.shape)
    batch, M, K = A64.shape
    if b_layout == B_KN:
        Kb, N = B64.shape[1:]
    elif b_layout == B_NK:
        N, Kb = B64.shape[1:]
    else:
        raise ValueError("b_layout must be B_KN or B_NK")
    if Kb != K or B64.shape[0] != batch:
        raise ValueError(f"shape mismatch A{A64.shape} B{B64.shape}")
    # a broadcast B has batch stride 0
    strideB = 0 if B64.strides[0] == 0 else B64.shape[1] * B64.shape[2]
    B64 = np.ascontiguousarray(B64[0]) if strideB == 0 else np.ascontiguousarray(B64)
    A64 = np.ascontiguousarray(A64)
    bias64 = None
    if bias is not None:
        bias64 = np.ascontiguousarray(to_f64(bias).reshape(-1))
        if bias64.size != N:
            raise ValueError("bias must have N elements")
    C = np.empty((batch, M, N), dtype=np.float64)
    ldb = N if b_layout == B_KN else K
    rc = _load().oracle_matmul_f64(
        batch, M, N, K,
        A64.ctypes.data, K, M * K,
        B64.ctypes.data, b_layout, ldb, strideB,
        bias64.ctypes.data if bias64 is not None else None,
        C.ctypes.data, N, M * N, nthreads)
    if rc != 0:
        raise RuntimeError(f"oracle_matmul_f64 failed with code {rc}")
    if squeeze:
        C = C[0]
    if act != "none":
        from .epilogue import apply
        C = apply(C, act)
    if residual is not None:
        R = np.asarray(residual, dtype=np.float64)
        if R.shape != C.shape:
            raise ValueError(f"residual shape {R.shape} != result shape {C.shape}")
        C = C + R
    return C, C.astype(np.float32)


def rel_fro(C_test: np.ndarray, C_ref64: np.ndarray) -> float:
    """Relative Frobenius error ||C_test - C_ref||_F / ||C_ref||_F, in float64."""
    d = np.asarray(C_test, dtype=np.float64) - C_ref64
    den = float(np.linalg.norm(C_ref64.ravel()))
    num = float(np.linalg.norm(d.ravel()))
    if den == 0.0:
        return 0.0 if num == 0.0 else float("inf")
    return num / den


def matmul_rows(A: np.ndarray, B: np.ndarray, bias, b_layout: int, rows,
                nthreads: int = 0, act: str = "none"):
    """Reference values for a subset of output rows (one full row each) of a single
    (non-batched) product: the oracle run on A[rows]."""
    rows = np.asarray(rows, dtype=np.int64)
    return matmul(np.ascontiguousarray(A[rows]), B, bias, b_layout, nthreads, act)
