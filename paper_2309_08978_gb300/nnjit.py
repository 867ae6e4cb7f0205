"""Python binding of the nnjit C ABI (include/nnjit.h): argument marshalling only.

Every function has the name of the C entry point it calls.  Device operands are torch
CUDA tensors (or raw integer device addresses); every step of the computation runs in
libnnjit.so.  There is no fallback: if the library is missing, loading it raises.
"""
from __future__ import annotations

import ctypes
import json
import os
import threading

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "_build", "libnnjit.so")

NNJIT_OK = 0
NNJIT_ERR_INVALID_ARG = 1
NNJIT_ERR_UNSUPPORTED = 2
NNJIT_ERR_CUDA = 3
NNJIT_ERR_OOM = 4
NNJIT_ERR_TIMEOUT = 5
NNJIT_ERR_BUDGET = 6

NNJIT_F32_FFMA = 0
NNJIT_TF32 = 1
NNJIT_BF16 = 2
NNJIT_W4_BF16 = 3

NNJIT_EPI_NONE = 0
NNJIT_EPI_RELU = 1
NNJIT_EPI_GELU = 2
NNJIT_EPI_SILU = 3
NNJIT_EPI_RESIDUAL = 0x10

NNJIT_B_KN = 0
NNJIT_B_NK = 1

NNJIT_FAMILY_FFMA = 0
NNJIT_FAMILY_TC = 1
NNJIT_FAMILY_GEMV = 2

NNJIT_PLAN_NO_CACHE = 0x1
NNJIT_PLAN_EXHAUSTIVE = 0x2
NNJIT_PLAN_REQUIRE_TIMED = 0x4
NNJIT_PLAN_B_CONSTANT = 0x8

DTYPES = {"f32_ffma": NNJIT_F32_FFMA, "tf32": NNJIT_TF32, "bf16": NNJIT_BF16, "w4_bf16": NNJIT_W4_BF16}
LAYOUTS = {"KN": NNJIT_B_KN, "NK": NNJIT_B_NK}


class nnjit_matmul_desc(ctypes.Structure):
    _fields_ = [("M", ctypes.c_int64), ("N", ctypes.c_int64), ("K", ctypes.c_int64),
                ("batch", ctypes.c_int64), ("dtype", ctypes.c_int32), ("b_layout", ctypes.c_int32),
                ("lda", ctypes.c_int64), ("ldb", ctypes.c_int64), ("ldc", ctypes.c_int64),
                ("stride_a", ctypes.c_int64), ("stride_b", ctypes.c_int64),
                ("stride_c", ctypes.c_int64), ("has_bias", ctypes.c_int32),
                ("flags", ctypes.c_uint32), ("epilogue", ctypes.c_int32)]


class nnjit_device_limits(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "sm_count", "smem_per_sm", "smem_per_block_optin", "regs_per_sm", "max_threads_per_sm",
        "max_blocks_per_sm", "tmem_cols_per_sm", "l2_bytes", "cc_major", "cc_minor")]


class nnjit_candidate(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "family", "bm", "bn", "bk", "tm", "tn", "stages", "split_k", "raster", "threads",
        "smem_bytes", "tmem_cols", "regs_per_thread", "blocks_per_sm", "grid", "wave_eff_ppm",
        "instance")] + [("predicted_cost", ctypes.c_int64), ("reduce", ctypes.c_int32),
                        ("cluster_m", ctypes.c_int32)]


class nnjit_attention_desc(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int64), ("Lq", ctypes.c_int64), ("Lk", ctypes.c_int64),
                ("d", ctypes.c_int64), ("causal", ctypes.c_int32), ("scale", ctypes.c_float),
                ("kernel", ctypes.c_int32)]


NNJIT_ATTN_AUTO, NNJIT_ATTN_TCGEN05, NNJIT_ATTN_MMA, NNJIT_ATTN_TCGEN05_2T = 0, 1, 2, 3


NNJIT_SETTING_FREE = -1
SETTING_AXES = ("raster", "kgroup", "reduce")


class nnjit_settings(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in SETTING_AXES]


def struct_to_dict(s) -> dict:
    return {name: getattr(s, name) for name, _ in s._fields_}


class NnjitError(RuntimeError):
    def __init__(self, status: int, func: str, detail: str):
        self.status = status
        super().__init__(f"{func}: {_status_name(status)}: {detail}")


_lib = None
_lock = threading.Lock()


def load_library(path: str = LIB_PATH):
    """Load libnnjit.so (raises if it has not been built)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(path):
            raise RuntimeError(f"libnnjit.so not found at {path}; build it first "
                               "(python -m paper_2309_08978_gb300.build_lib)")
        lib = ctypes.CDLL(path)
        P, vp, i32, i64, st = ctypes.POINTER, ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_int
        lib.nnjit_status_string.restype = ctypes.c_char_p
        lib.nnjit_status_string.argtypes = [st]
        lib.nnjit_last_error.restype = ctypes.c_char_p
        lib.nnjit_last_error.argtypes = []
        lib.nnjit_version.restype = i32
        lib.nnjit_version.argtypes = []
        sigs = {
            "nnjit_device_limits_query": [i32, P(nnjit_device_limits)],
            "nnjit_space_enumerate": [P(nnjit_matmul_desc), P(nnjit_device_limits),
                                      P(nnjit_candidate), i32, P(i32), P(i64)],
            "nnjit_matmul_plan": [i64, i64, i64, st, ctypes.c_double, P(vp)],
            "nnjit_matmul_plan_ex": [P(nnjit_matmul_desc), ctypes.c_double, P(vp)],
            "nnjit_matmul_plan_candidate": [P(nnjit_matmul_desc), i32, P(vp)],
            "nnjit_matmul_run": [vp, vp, vp, vp, vp, vp],
            "nnjit_matmul_run_batched": [vp, vp, vp, vp, vp],
            "nnjit_matmul_run_host": [vp, vp, vp, vp, vp, vp],
            "nnjit_matmul_run_host_seq": [i32, P(vp), P(vp), P(vp), P(vp), P(vp), vp],
            "nnjit_plan_check": [vp],
            "nnjit_plan_describe": [vp, ctypes.c_char_p, ctypes.c_size_t, P(ctypes.c_size_t)],
            "nnjit_plan_candidate": [vp, P(nnjit_candidate)],
            "nnjit_plan_destroy": [vp],
            "nnjit_cache_clear": [],
            "nnjit_gemv_bf16_noalloc": [i64, i64, i64, vp, vp, vp, vp, i32, vp],
            "nnjit_matmul_plan_online": [P(nnjit_matmul_desc), P(vp)],
            "nnjit_plan_online_progress": [vp, P(i32), P(i32), P(i32), P(i32)],
            "nnjit_cache_save": [ctypes.c_char_p],
            "nnjit_cache_load": [ctypes.c_char_p, P(i32)],
            "nnjit_w4_layout": [i64, i64, i64, P(i64), P(i64)],
            "nnjit_settings_set": [P(nnjit_settings)],
            "nnjit_attention": [P(nnjit_attention_desc), vp, vp, vp, vp, vp],
            "nnjit_attention_check": [],
            "nnjit_attention_tune": [P(nnjit_attention_desc), vp, vp, vp, vp, i32, P(ctypes.c_double), P(i32)],
            "nnjit_settings_get": [P(nnjit_settings)],
            "nnjit_settings_study": [P(nnjit_matmul_desc), i32, P(nnjit_settings), ctypes.c_char_p,
                                     ctypes.c_size_t, P(ctypes.c_size_t)],
        }
        for name, args in sigs.items():
            f = getattr(lib, name)
            f.restype = st
            f.argtypes = args
        lib.nnjit_cache_size.restype = i32
        lib.nnjit_cache_size.argtypes = []
        _lib = lib
        return lib


def _status_name(s: int) -> str:
    try:
        return load_library().nnjit_status_string(s).decode()
    except Exception:  # noqa: BLE001 - only used to format an error
        return str(s)


def _check(status: int, func: str):
    if status != NNJIT_OK:
        detail = load_library().nnjit_last_error().decode(errors="replace")
        raise NnjitError(status, func, detail)


def _ptr(x):
    """Device/host address of a tensor (data_ptr) or an integer address; None -> NULL."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


# ------------------------------------------------------------------------------ C ABI

def nnjit_status_string(s: int) -> str:
    return load_library().nnjit_status_string(s).decode()


def nnjit_last_error() -> str:
    return load_library().nnjit_last_error().decode(errors="replace")


def nnjit_version() -> int:
    return int(load_library().nnjit_version())


def nnjit_device_limits_query(device: int = 0) -> nnjit_device_limits:
    out = nnjit_device_limits()
    _check(load_library().nnjit_device_limits_query(device, ctypes.byref(out)),
           "nnjit_device_limits_query")
    return out


EPILOGUES = {"none": 0, "relu": 1, "gelu": 2, "silu": 3}


def make_desc(M, N, K, dtype, b_layout="KN", batch=1, has_bias=False, flags=0, lda=0, ldb=0,
              ldc=0, stride_a=0, stride_b=0, stride_c=0, epilogue="none",
              residual=False) -> nnjit_matmul_desc:
    """`epilogue`: an activation name or code; `residual`: C = act(A.Bt + bias) + C."""
    d = nnjit_matmul_desc()
    d.M, d.N, d.K, d.batch = M, N, K, batch
    d.dtype = DTYPES[dtype] if isinstance(dtype, str) else dtype
    d.b_layout = LAYOUTS[b_layout] if isinstance(b_layout, str) else b_layout
    d.lda, d.ldb, d.ldc = lda, ldb, ldc
    d.stride_a, d.stride_b, d.stride_c = stride_a, stride_b, stride_c
    d.has_bias = 1 if has_bias else 0
    d.flags = flags
    d.epilogue = (EPILOGUES[epilogue] if isinstance(epilogue, str) else epilogue) | \
        (NNJIT_EPI_RESIDUAL if residual else 0)
    return d


def nnjit_space_enumerate(desc: nnjit_matmul_desc, limits: nnjit_device_limits):
    """Returns (list of candidate dicts in evaluation order, naive space size)."""
    lib = load_library()
    count = ctypes.c_int32(0)
    naive = ctypes.c_int64(0)
    _check(lib.nnjit_space_enumerate(ctypes.byref(desc), ctypes.byref(limits), None, 0,
                                     ctypes.byref(count), ctypes.byref(naive)),
           "nnjit_space_enumerate")
    arr = (nnjit_candidate * max(1, count.value))()
    _check(lib.nnjit_space_enumerate(ctypes.byref(desc), ctypes.byref(limits), arr, count.value,
                                     ctypes.byref(count), ctypes.byref(naive)),
           "nnjit_space_enumerate")
    return [struct_to_dict(arr[i]) for i in range(count.value)], naive.value


class Plan:
    """Owning handle of an nnjit_plan."""

    def __init__(self, handle: int, desc: nnjit_matmul_desc | None = None):
        self.handle = handle
        self.desc = desc

    def run(self, A, B, bias, C, stream=None):
        nnjit_matmul_run(self, A, B, bias, C, stream)

    def describe(self) -> dict:
        return nnjit_plan_describe(self)

    def candidate(self) -> dict:
        return nnjit_plan_candidate(self)

    def check(self):
        nnjit_plan_check(self)

    def destroy(self):
        if self.handle:
            nnjit_plan_destroy(self)

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.destroy()


def nnjit_matmul_plan(M: int, N: int, K: int, dtype, tune_budget_ms: float) -> Plan:
    h = ctypes.c_void_p()
    dt = DTYPES[dtype] if isinstance(dtype, str) else dtype
    _check(load_library().nnjit_matmul_plan(M, N, K, dt, float(tune_budget_ms), ctypes.byref(h)),
           "nnjit_matmul_plan")
    return Plan(h.value, make_desc(M, N, K, dt, "KN", has_bias=True))


def nnjit_matmul_plan_ex(desc: nnjit_matmul_desc, tune_budget_ms: float) -> Plan:
    h = ctypes.c_void_p()
    _check(load_library().nnjit_matmul_plan_ex(ctypes.byref(desc), float(tune_budget_ms),
                                               ctypes.byref(h)), "nnjit_matmul_plan_ex")
    return Plan(h.value, desc)


def nnjit_matmul_plan_candidate(desc: nnjit_matmul_desc, index: int) -> Plan:
    h = ctypes.c_void_p()
    _check(load_library().nnjit_matmul_plan_candidate(ctypes.byref(desc), index, ctypes.byref(h)),
           "nnjit_matmul_plan_candidate")
    return Plan(h.value, desc)


def nnjit_matmul_plan_online(desc: nnjit_matmul_desc) -> Plan:
    h = ctypes.c_void_p()
    _check(load_library().nnjit_matmul_plan_online(ctypes.byref(desc), ctypes.byref(h)),
           "nnjit_matmul_plan_online")
    return Plan(h.value, desc)


def nnjit_plan_online_progress(plan: Plan) -> dict:
    v = [ctypes.c_int32(0) for _ in range(4)]
    _check(load_library().nnjit_plan_online_progress(plan.handle, *[ctypes.byref(x) for x in v]),
           "nnjit_plan_online_progress")
    return {"evaluated": v[0].value, "space_size": v[1].value, "current_index": v[2].value,
            "done": bool(v[3].value)}


def nnjit_matmul_run(plan: Plan, A, B, bias, C, stream=None):
    _check(load_library().nnjit_matmul_run(plan.handle, _ptr(A), _ptr(B), _ptr(bias), _ptr(C),
                                           _stream(stream)), "nnjit_matmul_run")


def nnjit_matmul_run_batched(plan: Plan, A, B, C, stream=None):
    _check(load_library().nnjit_matmul_run_batched(plan.handle, _ptr(A), _ptr(B), _ptr(C),
                                                   _stream(stream)), "nnjit_matmul_run_batched")


def nnjit_matmul_run_host(plan: Plan, hA, hB, hbias, hC, stream=None):
    _check(load_library().nnjit_matmul_run_host(plan.handle, _ptr(hA), _ptr(hB), _ptr(hbias),
                                                _ptr(hC), _stream(stream)),
           "nnjit_matmul_run_host")


def nnjit_matmul_run_host_seq(plans, hAs, hBs, hbiases, hCs, stream=None):
    """Sequence of products from host buffers with overlapped transfers (include/nnjit.h)."""
    n = len(plans)
    if not (len(hAs) == len(hBs) == len(hCs) == n) or (hbiases is not None and len(hbiases) != n):
        raise ValueError("plans and buffer lists must have the same length")
    vp = ctypes.c_void_p
    arr_p = (vp * max(1, n))(*[p.handle for p in plans])
    arr_a = (vp * max(1, n))(*[_ptr(x) for x in hAs])
    arr_b = (vp * max(1, n))(*[_ptr(x) for x in hBs])
    arr_c = (vp * max(1, n))(*[_ptr(x) for x in hCs])
    arr_bias = None if hbiases is None else (vp * max(1, n))(*[_ptr(x) for x in hbiases])
    _check(load_library().nnjit_matmul_run_host_seq(n, arr_p, arr_a, arr_b, arr_bias, arr_c, _stream(stream)),
           "nnjit_matmul_run_host_seq")


def nnjit_plan_check(plan: Plan):
    _check(load_library().nnjit_plan_check(plan.handle), "nnjit_plan_check")


def nnjit_plan_describe(plan: Plan) -> dict:
    lib = load_library()
    need = ctypes.c_size_t(0)
    _check(lib.nnjit_plan_describe(plan.handle, None, 0, ctypes.byref(need)), "nnjit_plan_describe")
    buf = ctypes.create_string_buffer(need.value)
    _check(lib.nnjit_plan_describe(plan.handle, buf, need.value, None), "nnjit_plan_describe")
    return json.loads(buf.value.decode())


def nnjit_plan_candidate(plan: Plan) -> dict:
    out = nnjit_candidate()
    _check(load_library().nnjit_plan_candidate(plan.handle, ctypes.byref(out)),
           "nnjit_plan_candidate")
    return struct_to_dict(out)


def nnjit_plan_destroy(plan: Plan):
    _check(load_library().nnjit_plan_destroy(plan.handle), "nnjit_plan_destroy")
    plan.handle = None


NNJIT_NOALLOC_SCRATCH_FLOATS = 1 << 20


def nnjit_gemv_bf16_noalloc(M: int, N: int, K: int, x, W, bias, C, split_k: int, stream=None):
    """Decode GEMV whose split-K partials live in a fixed array inside the library; it
    allocates nothing (see include/nnjit.h)."""
    _check(load_library().nnjit_gemv_bf16_noalloc(M, N, K, _ptr(x), _ptr(W), _ptr(bias), _ptr(C),
                                                  split_k, _stream(stream)),
           "nnjit_gemv_bf16_noalloc")


def nnjit_cache_clear():
    _check(load_library().nnjit_cache_clear(), "nnjit_cache_clear")


def nnjit_w4_layout(N: int, K: int, ldb: int = 0):
    """(scale_offset_bytes, total_bytes) of a 4-bit weight blob (ldb = 0: K)."""
    off, tot = ctypes.c_int64(0), ctypes.c_int64(0)
    _check(load_library().nnjit_w4_layout(N, K, ldb or K, ctypes.byref(off), ctypes.byref(tot)),
           "nnjit_w4_layout")
    return off.value, tot.value


def nnjit_cache_size() -> int:
    return int(load_library().nnjit_cache_size())


def nnjit_cache_save(path: str):
    _check(load_library().nnjit_cache_save(os.fsencode(path)), "nnjit_cache_save")


def nnjit_cache_load(path: str) -> int:
    n = ctypes.c_int32(0)
    _check(load_library().nnjit_cache_load(os.fsencode(path), ctypes.byref(n)), "nnjit_cache_load")
    return n.value


def nnjit_settings_set(settings: dict | None):
    """Fix settings process-wide ({axis: value}; missing axes stay searched); None clears."""
    lib = load_library()
    if settings is None:
        _check(lib.nnjit_settings_set(None), "nnjit_settings_set")
        return
    unknown = set(settings) - set(SETTING_AXES)
    if unknown:
        raise ValueError(f"unknown settings {sorted(unknown)}")
    s = nnjit_settings(*[int(settings.get(a, NNJIT_SETTING_FREE)) for a in SETTING_AXES])
    _check(lib.nnjit_settings_set(ctypes.byref(s)), "nnjit_settings_set")


def nnjit_settings_get() -> dict:
    s = nnjit_settings()
    _check(load_library().nnjit_settings_get(ctypes.byref(s)), "nnjit_settings_get")
    return struct_to_dict(s)


def nnjit_settings_study(descs) -> tuple[dict, dict]:
    """Run the one-variable-at-a-time settings study over `descs`; returns (settings it
    recommends, the JSON report as a dict).  Nothing is applied."""
    lib = load_library()
    arr = (nnjit_matmul_desc * len(descs))(*descs)
    out = nnjit_settings()
    need = ctypes.c_size_t(0)
    size = 4096 + 4096 * len(descs)      # the report takes well under 1 KB per product
    buf = ctypes.create_string_buffer(size)
    _check(lib.nnjit_settings_study(arr, len(descs), ctypes.byref(out), buf, size, ctypes.byref(need)),
           "nnjit_settings_study")
    if need.value > size:
        raise RuntimeError(f"settings report truncated ({need.value} > {size} bytes)")
    return struct_to_dict(out), json.loads(buf.value.decode())


def nnjit_attention(Q, K, V, O, causal=False, scale=None, stream=None, kernel=NNJIT_ATTN_AUTO):
    """O = softmax(scale Q K^T) V per leading index (batch x heads).  Q [B][Lq][d], K and V
    [B][Lk][d] bf16 tensors, O [B][Lq][d] float32 (device tensors); scale defaults to
    1 / sqrt(d); kernel: NNJIT_ATTN_AUTO / _TCGEN05 / _MMA / _TCGEN05_2T."""
    B, Lq, d = Q.shape
    Lk = K.shape[1]
    desc = nnjit_attention_desc(B, Lq, Lk, d, 1 if causal else 0,
                                float(scale) if scale is not None else 1.0 / float(d) ** 0.5, kernel)
    _check(load_library().nnjit_attention(ctypes.byref(desc), _ptr(Q), _ptr(K), _ptr(V), _ptr(O),
                                          _stream(stream)), "nnjit_attention")


def nnjit_attention_check():
    _check(load_library().nnjit_attention_check(), "nnjit_attention_check")


def nnjit_attention_tune(Q, K, V, O, causal=False, scale=None, reps=20):
    """Time the three attention kernels on these buffers (O is overwritten) and record the
    fastest for later kernel=AUTO calls; returns (times_us (tensor-memory, warp-MMA,
    two-tile tensor-memory), chosen)."""
    B, Lq, d = Q.shape
    desc = nnjit_attention_desc(B, Lq, K.shape[1], d, 1 if causal else 0,
                                float(scale) if scale is not None else 1.0 / float(d) ** 0.5, 0)
    times = (ctypes.c_double * 3)()
    chosen = ctypes.c_int32(0)
    _check(load_library().nnjit_attention_tune(ctypes.byref(desc), _ptr(Q), _ptr(K), _ptr(V), _ptr(O), reps,
                                               times, ctypes.byref(chosen)), "nnjit_attention_tune")
    return (times[0], times[1], times[2]), chosen.value
