"""Benchmark of the JIT-tuned MatMul hot path on one workload (one JSON line on stdout).

    python bench.py [--steps K] [--warmup W] [--impl ours|reference]
                    [--workload NAME] [--tune-budget-ms B] [--no-sweep]

A step is one pass of the workload's products over one batch of synthetic input.  The
default workload is the Llama-2-7B decoder block prefill at batch 4 x seq 1024 (M = 4096,
BF16): the four Linears (qkv, o-proj, gate/up, down) and the two attention BatchMatMuls
(QK^T and PV over 128 batch x heads).  Plans are tuned first under one total budget (the
JIT phase, timed separately and reported under "tune", with the exhaustive sweep of the
same spaces beside it); the timed region then runs K steps.  Each product's K launches
run as a block of CUDA-graph replays that rotate over enough operand copies to exceed the
L2, so operands come from HBM; CUDA events at the block boundaries give every kernel's
average launch duration.

The operator runs on one GPU: --gpus above 1 (or a torchrun world above 1) prints an
"unavailable" line and exits 0 without touching a GPU.

--impl reference times the oracle (the plain CPU definition) on the host cores on the
same workload and metric.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

DEFAULT_WORKLOAD = "llama2_7b_prefill_m4096"
METRIC = "GEMM TFLOP/s (GEMV GB/s) vs GB300 roofline per shape; JIT tune time to plan"
TF32_OVER_BF16 = 1.1 / 2.25     # nominal dense TF32 / BF16 tensor rates (fallback only)


def log(*a):
    print(*a, file=sys.stderr, flush=True)


# ------------------------------------------------------------------------- helpers

def ref_product(oracle, A, B, bias, s, dtype, nthreads=0, act="none"):
    """The oracle on one product's operands (4-bit weights: dequantised first)."""
    if dtype == "w4_bf16":
        from oracle.quant import matmul as w4_matmul
        return w4_matmul(A, B, s.N, s.K, 0, bias, act, nthreads)
    return oracle.matmul(A, B, bias, oracle.B_KN if s.b_layout == "KN" else oracle.B_NK,
                         nthreads=nthreads, act=act)


def shape_bytes(s, dtype):
    if dtype == "w4_bf16":  # x bf16, 4-bit codes, bf16 group scales, f32 C
        return s.M * s.K * 2 + s.N * s.K // 2 + (s.K + 127) // 128 * s.N * 2 + s.M * s.N * 4
    e = 2 if dtype in ("bf16",) else 4
    b = s.batch * (s.M * s.K * e + s.K * s.N * e + s.M * s.N * 4)
    return b + (4 * s.N if s.has_bias else 0)


def job_throughput(flops_per_step: int, steps: int, ms: float) -> float:
    """TFLOP/s of `steps` steps of `flops_per_step` in `ms` milliseconds."""
    return flops_per_step * steps / (ms / 1e3) / 1e12


def prefix_curve(times_us: dict, n: int) -> dict:
    """pick/best had the tuner timed only a prefix of the ordered space: for the first k
    candidates (k = 1, 2, 3, 5, 10) and the first 10 / 25 / 50 % of the space, the best
    time among them over the best time of the whole space."""
    best = min(times_us.values())
    out = {}

    def ratio(k):
        seen = [t for i, t in times_us.items() if i < k]
        return round(min(seen) / best, 4) if seen else None

    for k in (1, 2, 3, 5, 10):
        out[f"first_{k}"] = ratio(min(k, n))
    for pct in (10, 25, 50):
        out[f"first_{pct}pct"] = ratio(max(1, math.ceil(pct * n / 100)))
    return out


def workload_config(workload, args) -> dict:
    """The "config" object of the JSON line: the same for both arms."""
    return {"workload": workload.key, "title": workload.title, "epilogue": args.epilogue,
            "shapes": [[s.batch, s.M, s.N, s.K, s.b_layout] for s in workload.shapes],
            "parallelism": "single GPU",
            "l2": "each product rotates over operand copies totalling >= 3 x L2 (inputs larger "
                  "than L2), so every timed launch reads its operands from HBM",
            "schedule": "per product: K launches as CUDA-graph replays, products in sequence"}


def probe_peaks(dtype, dev):
    """Measured dense peaks for the non-BF16 paths, taken on this GPU at bench start:
    TF32 = torch.matmul on float32 8192^3 with TF32 allowed, FP32 FFMA = the same with
    TF32 off (cuBLAS SGEMM), each the best of several CUDA-event-timed launches."""
    import torch
    if dtype not in ("tf32", "f32_ffma"):
        return {}
    n = 8192
    a = torch.randn(n, n, device=dev)
    b = torch.randn(n, n, device=dev)
    out = {}
    old = torch.backends.cuda.matmul.allow_tf32
    try:
        for name, tf32, reps in (("tf32_tflops", True, 10), ("ffma_tflops", False, 4)):
            torch.backends.cuda.matmul.allow_tf32 = tf32
            for _ in range(2):
                torch.matmul(a, b)
            torch.cuda.synchronize()
            best = float("inf")
            for _ in range(reps):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                torch.matmul(a, b)
                e1.record()
                torch.cuda.synchronize()
                best = min(best, e0.elapsed_time(e1))
            out[name] = round(2 * n ** 3 / (best / 1e3) / 1e12, 2)
    finally:
        torch.backends.cuda.matmul.allow_tf32 = old
    del a, b
    torch.cuda.empty_cache()
    out["how"] = ("torch.matmul float32 8192^3 (cuBLAS), TF32 allowed / not allowed, best of "
                  "10 / 4 launches, CUDA events, on this GPU at bench start")
    return out


def kernel_key(s, dtype, cand):
    """Identifies one kernel configuration on one product (the traffic table's key)."""
    fam = {0: "ffma", 1: "tc", 2: "gemv"}[cand["family"]]
    return (f"{fam} {dtype} {s.batch}x{s.M}x{s.N}x{s.K} {s.b_layout} bm{cand['bm']} bn{cand['bn']} "
            f"bk{cand['bk']} st{cand['stages']} split{cand['split_k']} red{cand['reduce']} rast{cand['raster']}")


def lookup_traffic(key):
    """DRAM bytes per launch (ncu dram__bytes_read.sum + dram__bytes_write.sum) recorded in
    profiles/dram_traffic.txt for exactly this kernel configuration, else None."""
    path = os.path.join(ROOT, "profiles", "dram_traffic.txt")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#") or "|" not in line:
                continue
            k, v = line.rsplit("|", 1)
            if k.strip() == key:
                return int(float(v.strip()))
    return None


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
                "bf16_tflops_sustained": d.get("bf16_tflops_sustained"), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "source": "fallback"}


def sustained_run(clocks) -> bool:
    """A timed region long and hot enough to run under the power cap (the clock sampler
    saw sw_power_cap, or the median SM clock sat below 95 % of its maximum)."""
    if not clocks:
        return False
    return ("sw_power_cap" in clocks.get("reasons", []) or
            clocks["sm_mhz"] < 0.95 * clocks["sm_max_mhz"])


def peak_source(dtype, peaks, sustained, probes):
    """Where the tensor peak of the roofline comes from, in words."""
    if dtype == "tf32" and probes.get("tf32_tflops"):
        return "TF32 probe (cuBLAS float32 8192^3 with TF32, measured at bench start)"
    if dtype == "f32_ffma" and probes.get("ffma_tflops"):
        return "FP32 FFMA probe (cuBLAS SGEMM 8192^3, measured at bench start)"
    kind = ("sustained" if sustained else "burst") + " bf16"
    if dtype == "tf32":
        kind += " x nominal tf32/bf16 ratio"
    return f"{kind} ({peaks['source']})"


def dtype_peak_tflops(dtype, peaks, sm_mhz, sustained=False, probes=None, sm_count=152):
    """Dense peak for the dtype.  BF16: the measured figure (burst for a kernel timed in a
    short region, sustained under the power cap).  TF32 and FP32 FFMA: the probes taken at
    bench start (probe_peaks); without them, TF32 = BF16 x the nominal TF32/BF16 ratio and
    FFMA = SMs x 128 FMA/clk x 2 x the SM clock."""
    probes = probes or {}
    bf16 = peaks["bf16_tflops_sustained"] if sustained and peaks.get("bf16_tflops_sustained") \
        else peaks["bf16_tflops"]
    if dtype == "bf16":
        return bf16
    if dtype == "tf32":
        return probes.get("tf32_tflops") or bf16 * TF32_OVER_BF16
    return probes.get("ffma_tflops") or sm_count * 128 * 2 * sm_mhz * 1e6 / 1e12


class ClockSampler:
    """nvidia-smi sampling during the timed region."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index=0):
        self.index = index
        self.proc = None
        # the raw samples (the JSON line carries their summary); NNJIT_CLOCKS_DIR keeps them
        out_dir = os.environ.get("NNJIT_CLOCKS_DIR") or tempfile.gettempdir()
        self.path = os.path.join(out_dir, f"clocks_rank{index}.csv")

    def start(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"], stdout=self.f,
                stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.f.close()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 8:
                    continue
                try:
                    rows.append((float(parts[0]), float(parts[1]), parts[3:]))
                except ValueError:
                    continue
        if not rows:
            return None
        mx = max(r[1] for r in rows)
        load = sorted(r[0] for r in rows)
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = set()
        for r in rows:
            for n, v in zip(names, r[2][1:5]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": load[len(load) // 2], "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(rows)}


# ------------------------------------------------------------------------- reference arm

def run_reference(args, workload, rank):
    """The oracle as it stands, on the host cores, on the same workload and metric."""
    if rank != 0:
        return 0
    import numpy as np
    import oracle
    from synthetic import make_operands
    oracle.build()
    dtype = workload.dtypes[-1]
    cores = oracle.hw_threads()
    act = args.epilogue
    # one step = every product of the workload on a row sample of A (the oracle cost is
    # linear in the rows), sized to a few seconds of host work per step
    budget_s = float(os.environ.get("NNJIT_REF_STEP_S", "3.0"))
    ops = []
    for s in workload.shapes:
        A, B, bias = make_operands(s, workload.index, dtype)
        ops.append((s, A, B, bias))
    # calibrate the row fraction on one small probe
    t0 = time.perf_counter()
    s, A, B, bias = ops[0]
    probe_rows = max(1, min(s.M, 8))
    _ = ref_product(oracle, np.ascontiguousarray(A[..., :probe_rows, :] if s.batch > 1 else A[:probe_rows]),
                    B, bias, s, dtype)
    dt_probe = max(1e-4, time.perf_counter() - t0)
    probe_flops = 2 * s.batch * probe_rows * s.N * s.K
    rate = probe_flops / dt_probe
    full_flops = sum(x[0].flops for x in ops)
    frac = min(1.0, budget_s * rate / full_flops)
    sample_flops = 0
    timings = []
    for step in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        fl = 0
        for s, A, B, bias in ops:
            rows = max(1, int(round(s.M * frac)))
            Ar = A[:, :rows] if s.batch > 1 else A[:rows]
            ref_product(oracle, np.ascontiguousarray(Ar), B, bias, s, dtype, cores, act)
            fl += 2 * s.batch * rows * s.N * s.K
        dt = time.perf_counter() - t0
        if step >= args.warmup:
            timings.append(dt)
            sample_flops = fl
    total = sum(timings)
    value = sample_flops * len(timings) / total / 1e12
    sample = (f"each step: every product of the workload on the first {frac:.4f} of its rows "
              f"({sample_flops / 1e9:.3f} GFLOP of {full_flops / 1e9:.3f}), fp64 oracle")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "TFLOP/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1000 * total / len(timings), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": workload_config(workload, args),
        "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": cores, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def cpu_baseline(workload, dtype, seconds=12.0, act="none"):
    """Oracle throughput on the host cores on a bounded sample of the workload."""
    import numpy as np
    import oracle
    from synthetic import make_operands
    oracle.build()
    cores = oracle.hw_threads()
    ops = [(s,) + make_operands(s, workload.index, dtype) for s in workload.shapes]
    done_flops, t_used, reps = 0, 0.0, 0
    # rows of every product, grown until the sample takes ~`seconds`
    rows_frac = 1.0 / 64
    while t_used < seconds and reps < 64:
        t0 = time.perf_counter()
        fl = 0
        for s, A, B, bias in ops:
            rows = max(1, int(round(s.M * rows_frac)))
            Ar = A[:, :rows] if s.batch > 1 else A[:rows]
            ref_product(oracle, np.ascontiguousarray(Ar), B, bias, s, dtype, cores, act)
            fl += 2 * s.batch * rows * s.N * s.K
        dt = time.perf_counter() - t0
        done_flops += fl
        t_used += dt
        reps += 1
        if dt < seconds / 8 and rows_frac < 1.0:
            rows_frac = min(1.0, rows_frac * 2)
    return {"value": done_flops / t_used / 1e12, "unit": "TFLOP/s", "cores": cores,
            "kind": "oracle",
            "sample": f"{reps} passes over every product on up to {rows_frac:.4f} of its rows "
                      f"({done_flops / 1e9:.2f} GFLOP in {t_used:.1f} s, fp64, all host threads)"}


# ------------------------------------------------------------------------- attention

# Fused attention workloads: the attention BatchMatMuls of the T5-large layer and of the
# Llama-2 prefill (batch x heads, Lq, Lk, d, causal), with the softmax between them.
ATTENTION_WORKLOADS = {
    "t5_large_attention": (128, 256, 256, 64, False),
    "llama2_7b_prefill_attention": (128, 1024, 1024, 128, True),
}
ATTN_METRIC = "fused attention TFLOP/s (softmax(QK^T) V, visible query-key pairs)"


def attention_flops(B, Lq, Lk, d, causal):
    """4 d flops per visible (query, key) pair: 2 d for the score, 2 d for P V."""
    if not causal:
        pairs = Lq * Lk
    else:
        shift = Lk - Lq
        pairs = sum(max(0, min(Lk, i + shift + 1)) for i in range(Lq))
    return 4 * d * B * pairs


def run_attention(args, name):
    import numpy as np
    import torch
    import paper_2309_08978_gb300 as nj
    from synthetic import f32_to_bf16_bits, normal

    B, Lq, Lk, d, causal = ATTENTION_WORKLOADS[name]
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    peaks = load_peaks()
    lim = nj.nnjit_device_limits_query(0)
    scale = 1.0 / math.sqrt(d)

    def bf16(shape, seed):
        return f32_to_bf16_bits(normal(seed, int(np.prod(shape)), 1.0).astype(np.float32).reshape(shape))

    def to_dev(bits):
        return torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).to(dev)

    hQ, hK, hV = bf16((B, Lq, d), 20), bf16((B, Lk, d), 21), bf16((B, Lk, d), 22)
    set_bytes = (hQ.nbytes + hK.nbytes + hV.nbytes) + B * Lq * d * 4
    nsets = int(min(64, max(1, math.ceil(3 * lim.l2_bytes / set_bytes))))
    Q0, K0, V0 = to_dev(hQ), to_dev(hK), to_dev(hV)
    sets = [(Q0, K0, V0, torch.empty((B, Lq, d), dtype=torch.float32, device=dev))]
    for _ in range(nsets - 1):
        sets.append((Q0.clone(), K0.clone(), V0.clone(), torch.empty((B, Lq, d), dtype=torch.float32, device=dev)))
    stream = torch.cuda.Stream(device=dev)

    def launch(k):
        Q, K, V, O = sets[k % nsets]
        nj.nnjit_attention(Q, K, V, O, causal=causal, scale=scale, stream=stream)

    # the JIT phase: time the three kernels on these buffers, keep the fastest (kernel AUTO)
    t0 = time.perf_counter()
    (t_tc, t_mma, t_tc2), chosen = nj.nnjit_attention_tune(Q0, K0, V0, sets[0][3], causal=causal, scale=scale,
                                                           reps=10)
    tune = {"plan_ms": round(1000 * (time.perf_counter() - t0), 2), "tcgen05_us": round(t_tc, 3),
            "mma_us": round(t_mma, 3), "tcgen05_2t_us": round(t_tc2, 3),
            "chosen": {1: "tcgen05", 2: "mma", 3: "tcgen05_2t"}[chosen]}
    with torch.cuda.stream(stream):
        launch(0)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for k in range(nsets):
            launch(k)
    torch.cuda.synchronize()

    def block(n):
        for _ in range(n // nsets):
            g.replay()
        for k in range(n % nsets):
            launch(k)

    with torch.cuda.stream(stream):
        block(args.warmup)
    torch.cuda.synchronize()
    sampler = ClockSampler(0)
    sampler.start()
    time.sleep(0.3)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t_wall = time.perf_counter()
    torch.cuda.nvtx.range_push("timed_region")
    with torch.cuda.stream(stream):
        e0.record(stream)
        block(args.steps)
        e1.record(stream)
    stream.synchronize()
    torch.cuda.nvtx.range_pop()
    torch.cuda.synchronize()
    wall = time.perf_counter() - t_wall
    clocks = sampler.stop()
    ms = e0.elapsed_time(e1)
    flops = attention_flops(B, Lq, Lk, d, causal)
    value = job_throughput(flops, args.steps, ms)
    dur_s = ms / 1e3 / args.steps
    sustained = sustained_run(clocks)
    peak_t = peaks["bf16_tflops_sustained"] if sustained and peaks.get("bf16_tflops_sustained") else peaks["bf16_tflops"]
    ach = flops / dur_s / 1e12
    alg_bytes = set_bytes
    kernel_key = f"attention {tune['chosen']} d{d} B{B} Lq{Lq} Lk{Lk}" + (" causal" if causal else "")
    roof = {"bound": "tensor", "achieved": round(ach, 2), "peak": round(peak_t, 1), "unit": "TFLOP/s",
            "frac": round(ach / peak_t, 4), "traffic": lookup_traffic(kernel_key),
            "kernel": kernel_key,
            "peak_source": ("sustained" if sustained else "burst") + f" bf16 ({peaks['source']})",
            "units_per_launch": f"{flops} flop, {alg_bytes} algorithmic bytes"}

    # ---- context: the unfused path (this library's two BatchMatMuls with f32 scores, and a
    # torch softmax to bf16 between them); not part of the fused kernel's number
    unfused = None
    try:
        dq = nj.make_desc(Lq, Lk, d, "bf16", "NK", batch=B, flags=nj.NNJIT_PLAN_NO_CACHE)
        dv = nj.make_desc(Lq, d, Lk, "bf16", "KN", batch=B, flags=nj.NNJIT_PLAN_NO_CACHE)
        pq, pv = nj.nnjit_matmul_plan_ex(dq, 300.0), nj.nnjit_matmul_plan_ex(dv, 300.0)
        S = torch.empty((B, Lq, Lk), dtype=torch.float32, device=dev)
        Ou = torch.empty((B, Lq, d), dtype=torch.float32, device=dev)
        mask = None
        if causal:
            mask = torch.ones(Lq, Lk, dtype=torch.bool, device=dev).tril(Lk - Lq)

        def unfused_step():
            nj.nnjit_matmul_run_batched(pq, Q0, K0, S, stream)
            x = S * scale
            if mask is not None:
                x = x.masked_fill(~mask, float("-inf"))
            P = torch.softmax(x, dim=-1).to(torch.bfloat16)
            nj.nnjit_matmul_run_batched(pv, P, V0, Ou, stream)

        with torch.cuda.stream(stream):
            for _ in range(3):
                unfused_step()
            torch.cuda.synchronize()
            u0, u1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            reps = 20
            u0.record(stream)
            for _ in range(reps):
                unfused_step()
            u1.record(stream)
        stream.synchronize()
        unfused = {"us": round(1000 * u0.elapsed_time(u1) / reps, 3),
                   "how": "two nnjit BatchMatMul plans (f32 scores) and a torch softmax to bf16 "
                          "between them, operands L2-warm; context only"}
        pq.destroy()
        pv.destroy()
    except Exception as e:  # context only: report why it is missing
        unfused = {"unavailable": str(e)[:200]}

    # ---- end to end: host Q, K, V -> device, kernel, O -> host, per step
    e2e_steps = max(3, min(args.steps, args.e2e_steps))
    pQ, pK, pV = (torch.from_numpy(h.view(np.int16)).view(torch.bfloat16).pin_memory() for h in (hQ, hK, hV))
    pO = torch.empty((B, Lq, d), dtype=torch.float32).pin_memory()
    dQ, dK, dV, dO = sets[0]

    def e2e_step():
        dQ.copy_(pQ, non_blocking=True)
        dK.copy_(pK, non_blocking=True)
        dV.copy_(pV, non_blocking=True)
        nj.nnjit_attention(dQ, dK, dV, dO, causal=causal, scale=scale, stream=stream)
        pO.copy_(dO, non_blocking=True)

    with torch.cuda.stream(stream):
        e2e_step()
        stream.synchronize()
        f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        f0.record(stream)
        for _ in range(e2e_steps):
            e2e_step()
        f1.record(stream)
    stream.synchronize()
    e2e_ms = f0.elapsed_time(f1)
    e2e_value = job_throughput(flops, e2e_steps, e2e_ms)

    cpu = None
    if not args.no_cpu_baseline:
        from oracle.attention import attention as attention_ref
        t_used, heads = 0.0, 0
        while t_used < args.cpu_seconds and heads < B:
            t0 = time.perf_counter()
            attention_ref(hQ[heads:heads + 1], hK[heads:heads + 1], hV[heads:heads + 1], scale, causal)
            t_used += time.perf_counter() - t0
            heads += 1
        cpu = {"value": attention_flops(heads, Lq, Lk, d, causal) / t_used / 1e12, "unit": "TFLOP/s",
               "cores": 1, "kind": "oracle",
               "sample": f"{heads} of {B} heads ({t_used:.1f} s, fp64 numpy, one host thread for the "
                         "per-row softmax loop)"}

    line = {
        "metric": ATTN_METRIC, "value": round(value, 3), "unit": "TFLOP/s", "n_gpus": 1,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms / args.steps, 6),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded SplitMix64 N(0,1) Q, K, V; no trained weights)",
        "config": {"workload": name, "batch_heads": B, "Lq": Lq, "Lk": Lk, "d": d, "causal": causal,
                   "scale": scale, "parallelism": "single GPU",
                   "l2": f"rotates over {nsets} input/output copies (>= 3 x L2), so operands stream from HBM"},
        "roofline": roof,
        "tune": tune,
        "unfused": unfused,
        "e2e": {"value": round(e2e_value, 3), "unit": "TFLOP/s",
                "h2d_bytes_per_step": hQ.nbytes + hK.nbytes + hV.nbytes, "d2h_bytes_per_step": B * Lq * d * 4,
                "steps": e2e_steps,
                "how": "pinned host Q, K, V copied in, nnjit_attention, O copied out, all inside the timed region"},
        "gpu_launches": int(args.steps),
        "clocks": clocks,
        "wall_s": round(wall, 3),
    }
    if cpu is not None:
        line["cpu_baseline"] = cpu
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------------- our arm

def custom_workload(ap, spec):
    """A one-product workload from "MxNxK:dtype:layout" (weights-like B, no bias, the
    default distributions), seeded with index 5."""
    from synthetic import Shape, Workload
    try:
        dims, dtype, layout = spec.split(":")
        M, N, K = (int(x) for x in dims.lower().split("x"))
    except ValueError:
        ap.error(f"--shape: expected MxNxK:dtype:layout, got {spec!r}")
    if dtype not in ("f32_ffma", "tf32", "bf16", "w4_bf16") or layout not in ("NK", "KN") or min(M, N, K) < 1:
        ap.error(f"--shape: bad dtype, layout or size in {spec!r}")
    shape = Shape(f"{M}x{N}x{K}", M, N, K, 1, layout)
    return Workload(f"custom_{M}x{N}x{K}_{dtype}_{layout}", 5, f"custom product {spec}", (dtype,), (shape,))


def run_ours(args, workload):
    import numpy as np
    import torch
    import paper_2309_08978_gb300 as nj
    from synthetic import make_operands

    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    dtype = workload.dtypes[-1]
    peaks = load_peaks()
    lim = nj.nnjit_device_limits_query(0)
    l2 = lim.l2_bytes
    probes = probe_peaks(dtype, dev)

    def to_dev(x):
        if x is None:
            return None
        if x.dtype == np.uint16:
            return torch.from_numpy(x.view(np.int16)).view(torch.bfloat16).to(dev)
        return torch.from_numpy(x).to(dev)

    def to_pinned(x):
        if x is None:
            return None
        if x.dtype == np.uint16:
            t = torch.from_numpy(x.view(np.int16)).view(torch.bfloat16)
        else:
            t = torch.from_numpy(x)
        return t.pin_memory()

    # ---- operands, plans (the JIT phase), tuner vs exhaustive sweep
    if args.cache and os.path.exists(args.cache):
        nj.nnjit_cache_load(args.cache)
    items = []
    tune = {"budget_ms_total": args.tune_budget_ms, "shapes": []}
    budget_left = args.tune_budget_ms
    free_sizes = {}
    if args.study:
        # Sec. 5.1: fix the settings a one-variable-at-a-time microbenchmark finds
        # consistently better (a 4096^3 product per tensor-core dtype plus the workload's
        # own tensor-core products), then build every space with them
        tc_shapes = [s for s in workload.shapes if dtype in ("bf16", "tf32") and s.M > 8]
        descs = [nj.make_desc(4096, 4096, 4096, dt, "NK") for dt in ("bf16", "tf32")]
        descs += [nj.make_desc(s.M, s.N, s.K, dtype, s.b_layout, batch=s.batch, has_bias=s.has_bias)
                  for s in tc_shapes]
        for s in workload.shapes:
            d = nj.make_desc(s.M, s.N, s.K, dtype, s.b_layout, batch=s.batch, has_bias=s.has_bias)
            free_sizes[id(s)] = len(nj.nnjit_space_enumerate(d, lim)[0])
        t0 = time.perf_counter()
        fixed, report = nj.nnjit_settings_study(descs)
        study_ms = 1000 * (time.perf_counter() - t0)
        nj.nnjit_settings_set(fixed)
        tune["settings"] = {
            "fixed": fixed, "study_ms": round(study_ms, 1),
            "products": [{"shape": [p["batch"], p["M"], p["N"], p["K"]], "dtype": p["dtype"],
                          "space_size": p["space_size"], "best_us": round(p["best_us"], 3),
                          "verdicts": {a: [e["value"], e["twin_value"], round(e["twin_us"], 3), e["verdict"]]
                                       for a, e in p["settings"].items()}}
                         for p in report["products"]]}
    for si, s in enumerate(workload.shapes):
        A, B, bias = make_operands(s, workload.index, dtype)
        bflag = nj.NNJIT_PLAN_B_CONSTANT if s.b_is_weight else 0   # weights never change
        desc = nj.make_desc(s.M, s.N, s.K, dtype, s.b_layout, batch=s.batch,
                            has_bias=s.has_bias, flags=bflag, epilogue=args.epilogue)
        # the total budget is shared out evenly over the products still to plan
        budget = max(0.0, budget_left / (len(workload.shapes) - si))
        t0 = time.perf_counter()
        plan = nj.nnjit_matmul_plan_ex(desc, budget)
        plan_ms = 1000 * (time.perf_counter() - t0)
        budget_left -= plan_ms
        info = plan.describe()
        entry = {"shape": [s.batch, s.M, s.N, s.K], "budget_ms": round(budget, 1), "plan_ms": round(plan_ms, 2),
                 "timed": len(info["timings_us"]),
                 "space_size": info["space_size"], "naive_space": info["naive_space"],
                 **({"space_size_free": free_sizes[id(s)]} if id(s) in free_sizes else {}),
                 "chosen_index": info["chosen_index"], "family": info["family"],
                 "candidate": {k: info["candidate"][k] for k in ("bm", "bn", "bk", "stages", "split_k", "raster")}}
        if not args.no_sweep:
            sweep_desc = nj.make_desc(s.M, s.N, s.K, dtype, s.b_layout, batch=s.batch,
                                      has_bias=s.has_bias, epilogue=args.epilogue,
                                      flags=nj.NNJIT_PLAN_EXHAUSTIVE | nj.NNJIT_PLAN_NO_CACHE | bflag)
            t0 = time.perf_counter()
            sweep = nj.nnjit_matmul_plan_ex(sweep_desc, 0.0)
            sweep_ms = 1000 * (time.perf_counter() - t0)
            sinfo = sweep.describe()
            sweep.destroy()
            times = {int(i): t for i, t in sinfo["timings_us"]}
            best_i = min(times, key=lambda i: (times[i], i))
            pick = times.get(info["chosen_index"])
            entry.update({"sweep_ms": round(sweep_ms, 2), "best_index": best_i,
                          "best_us": round(times[best_i], 3),
                          "pick_us": round(pick, 3) if pick is not None else None,
                          "pick_over_best": round(pick / times[best_i], 4) if pick else None,
                          "prefix_curve": prefix_curve(times, info["space_size"])})
        tune["shapes"].append(entry)
        nsets = int(min(64, max(1, math.ceil(3 * l2 / shape_bytes(s, dtype)))))
        if s.batch > 1:
            out_shape = (s.batch, s.M, s.N)
        else:
            out_shape = (s.M, s.N)
        dA, dB, dbias = to_dev(A), to_dev(B), to_dev(bias)
        sets = [(dA, dB, dbias, torch.empty(out_shape, dtype=torch.float32, device=dev))]
        for _ in range(nsets - 1):
            sets.append((dA.clone(), dB.clone(), dbias.clone() if dbias is not None else None,
                         torch.empty(out_shape, dtype=torch.float32, device=dev)))
        cand = plan.candidate()
        launches = 1 + (1 if cand["split_k"] > 1 else 0)
        items.append({"shape": s, "plan": plan, "sets": sets, "host": (A, B, bias),
                      "launches": launches, "family": info["family"]})
    tune["total_plan_ms"] = round(sum(e["plan_ms"] for e in tune["shapes"]), 2)
    tune["within_budget"] = tune["total_plan_ms"] <= args.tune_budget_ms
    if args.cache:
        nj.nnjit_cache_save(args.cache)
    ratios = [e["pick_over_best"] for e in tune["shapes"] if e.get("pick_over_best")]
    if ratios:
        tune["max_pick_over_best"] = max(ratios)
    curves = [e["prefix_curve"] for e in tune["shapes"] if e.get("prefix_curve")]
    if curves:
        # the worst product at each prefix length
        tune["prefix_curve_max"] = {k: max(c[k] for c in curves) for k in curves[0]}
    torch.cuda.synchronize()

    stream = torch.cuda.Stream(device=dev)

    def run_item(it, k):
        A, B, bias, C = it["sets"][k % len(it["sets"])]
        it["plan"].run(A, B, bias, C, stream)

    # ---- graphs: per product, one replay = one launch on each operand copy
    graphs = []
    with torch.cuda.stream(stream):
        for it in items:
            run_item(it, 0)  # warm the tensor-map cache outside capture
        torch.cuda.synchronize()
        for it in items:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                for k in range(len(it["sets"])):
                    run_item(it, k)
            graphs.append(g)
    torch.cuda.synchronize()

    def block(i, n):
        """n launches of product i, as graph replays (+ a tail of single launches)."""
        it = items[i]
        G = len(it["sets"])
        for _ in range(n // G):
            graphs[i].replay()
        for k in range(n % G):
            run_item(it, k)

    # warm-up steps
    with torch.cuda.stream(stream):
        for i in range(len(items)):
            block(i, args.warmup)
    torch.cuda.synchronize()

    def barrier():
        torch.cuda.synchronize()

    sampler = ClockSampler(0)
    sampler.start()
    time.sleep(0.3)
    barrier()
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(len(items) + 1)]
    t_wall = time.perf_counter()
    torch.cuda.nvtx.range_push("timed_region")
    with torch.cuda.stream(stream):
        evs[0].record(stream)
        for i in range(len(items)):
            block(i, args.steps)
            evs[i + 1].record(stream)
    stream.synchronize()
    torch.cuda.nvtx.range_pop()
    barrier()
    wall = time.perf_counter() - t_wall
    clocks = sampler.stop()
    per_item_ms = [evs[i].elapsed_time(evs[i + 1]) for i in range(len(items))]
    total_ms = sum(per_item_ms)
    for it in items:
        it["plan"].check()

    flops_step = sum(it["shape"].flops for it in items)
    ms_per_step = total_ms / args.steps
    value = job_throughput(flops_step, args.steps, total_ms)

    # ---- roofline of the dominant kernel (largest share of the timed region)
    dom = max(range(len(items)), key=lambda i: per_item_ms[i])
    ds = items[dom]["shape"]
    dur_s = per_item_ms[dom] / 1e3 / args.steps
    alg_bytes = shape_bytes(ds, dtype)
    sm_mhz = clocks["sm_mhz"] if clocks else 1900.0
    sustained = sustained_run(clocks)
    peak_t = dtype_peak_tflops(dtype, peaks, sm_mhz, sustained, probes, lim.sm_count)
    ai = ds.flops / alg_bytes
    ridge = peak_t * 1e12 / (peaks["hbm_gbs"] * 1e9)
    if items[dom]["family"] == nj.NNJIT_FAMILY_GEMV or ai < ridge:
        ach = alg_bytes / dur_s / 1e9
        roof = {"bound": "hbm", "achieved": round(ach, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": round(ach / peaks["hbm_gbs"], 4)}
    else:
        ach = ds.flops / dur_s / 1e12
        roof = {"bound": "tensor", "achieved": round(ach, 2), "peak": round(peak_t, 1),
                "unit": "TFLOP/s", "frac": round(ach / peak_t, 4)}
    dom_key = kernel_key(ds, dtype, items[dom]["plan"].candidate())
    roof.update({"traffic": lookup_traffic(dom_key), "kernel": dom_key,
                 "peak_source": peak_source(dtype, peaks, sustained, probes) if roof["unit"] == "TFLOP/s"
                                else f"copy bandwidth ({peaks['source']})",
                 "units_per_launch": f"{ds.flops} flop, {alg_bytes} algorithmic bytes"})
    per_shape = []
    for i, it in enumerate(items):
        s = it["shape"]
        d = per_item_ms[i] / 1e3 / args.steps
        tf, gb = s.flops / d / 1e12, shape_bytes(s, dtype) / d / 1e9
        hbm_bound = it["family"] == nj.NNJIT_FAMILY_GEMV or s.flops / shape_bytes(s, dtype) < ridge
        per_shape.append({"shape": [s.batch, s.M, s.N, s.K], "us": round(d * 1e6, 3),
                          "tflops": round(tf, 2), "gbs": round(gb, 1),
                          "bound": "hbm" if hbm_bound else "tensor",
                          "frac": round(gb / peaks["hbm_gbs"] if hbm_bound else tf / peak_t, 4),
                          "share": round(per_item_ms[i] / sum(per_item_ms), 4)})

    # ---- end to end through the C ABI with host buffers (copies inside the region)
    e2e_steps = max(3, min(args.steps, args.e2e_steps))
    hosts = []
    for it in items:
        A, B, bias = it["host"]
        s = it["shape"]
        out = torch.empty(((s.batch, s.M, s.N) if s.batch > 1 else (s.M, s.N)),
                          dtype=torch.float32).pin_memory()
        hosts.append((to_pinned(A), to_pinned(B), to_pinned(bias), out))
    h2d = sum(h[0].numel() * h[0].element_size() + h[1].numel() * h[1].element_size() +
              (h[2].numel() * 4 if h[2] is not None else 0) for h in hosts)
    d2h = sum(h[3].numel() * 4 for h in hosts)
    plans = [it["plan"] for it in items]
    cols = list(zip(*hosts))          # hA, hB, hbias, hC lists
    has_bias = any(x is not None for x in cols[2])

    def e2e_step():
        nj.nnjit_matmul_run_host_seq(plans, cols[0], cols[1], cols[2] if has_bias else None, cols[3], stream)

    def e2e_serial_step():
        for it, h in zip(items, hosts):
            nj.nnjit_matmul_run_host(it["plan"], *h, stream)

    def time_e2e(step_fn):
        with torch.cuda.stream(stream):
            step_fn()
        stream.synchronize()
        barrier()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            e0.record(stream)
            for _ in range(e2e_steps):
                step_fn()
            e1.record(stream)
        stream.synchronize()
        barrier()
        return e0.elapsed_time(e1)

    e2e_ms = time_e2e(e2e_step)
    e2e_value = job_throughput(flops_step, e2e_steps, e2e_ms)
    serial_ms = time_e2e(e2e_serial_step)
    # every product's result must have come back intact: compare the host copy with the
    # device-side result of the same plan on the same operands
    for it, h in zip(items, hosts):
        A, B, bias, C = it["sets"][0]
        it["plan"].run(A, B, bias, C, stream)
    stream.synchronize()
    for it, h in zip(items, hosts):
        if not torch.equal(it["sets"][0][3].cpu(), h[3]):
            raise RuntimeError("end-to-end result differs from the device-side result")

    cpu = None
    if not args.no_cpu_baseline:
        cpu = cpu_baseline(workload, dtype, seconds=args.cpu_seconds, act=args.epilogue)

    line = {
        "metric": METRIC, "value": round(value, 3), "unit": "TFLOP/s", "n_gpus": 1,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_per_step, 6),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": dtype,
        "data": "synthetic (seeded SplitMix64, the workload's distributions; no trained weights)",
        "config": workload_config(workload, args),
        "operand_copies": {"per_product": [len(it["sets"]) for it in items],
                           "l2_bytes": l2, "rule": "copies x operand bytes >= 3 x L2 per product"},
        "roofline": roof,
        "per_shape": per_shape,
        "tune": tune,
        "e2e": {"value": round(e2e_value, 3), "unit": "TFLOP/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "steps": e2e_steps,
                "how": "nnjit_matmul_run_host_seq over the step's products: pinned host -> device "
                       "copies of every A, B (and bias) on a copy-in stream, the kernels, and every "
                       "C copied back on a copy-out stream, overlapped, all inside the timed region",
                "serial_value": round(job_throughput(flops_step, e2e_steps, serial_ms), 3),
                "serial_how": "nnjit_matmul_run_host per product (copies, kernel, copy back on one "
                              "stream, one product after another); context"},
        "gpu_launches": int(args.steps * sum(it["launches"] for it in items)),
        "clocks": clocks,
        "wall_s": round(wall, 3),
    }
    if cpu is not None:
        line["cpu_baseline"] = cpu
    if probes:
        line["peak_probes"] = probes
    for it in items:
        it["plan"].destroy()
    print(json.dumps(line), flush=True)
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--tune-budget-ms", type=float, default=30000.0,
                    help="total tuning budget of the workload, shared out over its products")
    ap.add_argument("--no-sweep", action="store_true", help="skip the exhaustive sweep")
    ap.add_argument("--study", action="store_true",
                    help="run the fixed-settings microbenchmark first and plan with its settings")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--e2e-steps", type=int, default=200)
    ap.add_argument("--cache", default=None,
                    help="plan-cache file: loaded before tuning if present, saved after")
    ap.add_argument("--only", default=None,
                    help="run a single product of the workload (by name), e.g. for profiling")
    ap.add_argument("--epilogue", default="none", choices=["none", "relu", "gelu", "silu"],
                    help="activation fused after the bias into every product (nnjit_epilogue)")
    ap.add_argument("--shape", default=None,
                    help="run one custom product instead of a workload: MxNxK:dtype:layout "
                         "(dtype f32_ffma, tf32, bf16 or w4_bf16; layout NK or KN), e.g. 4096x8192x4096:bf16:NK")
    args = ap.parse_args(argv)
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    from synthetic import WORKLOADS
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if args.impl == "ours" and (world > 1 or args.gpus > 1):
        # the operator runs on one GPU; several GPUs would only run independent replicas
        if rank == 0:
            print(json.dumps({"metric": METRIC, "n_gpus": max(world, args.gpus), "unavailable":
                              "single-GPU library: every product runs on one GPU, no multi-GPU "
                              "path is built"}), flush=True)
        return 0
    if args.workload in ATTENTION_WORKLOADS:
        if args.impl == "reference":
            print(json.dumps({"impl": "reference", "unavailable": "the reference arm covers the MatMul "
                              "workloads; the attention workloads have their oracle as cpu_baseline"}))
            return 0
        import __graft_entry__
        __graft_entry__.build()
        return run_attention(args, args.workload)
    workload = WORKLOADS[args.workload]
    if args.shape:
        workload = custom_workload(ap, args.shape)
    if args.only:
        import dataclasses
        shapes = tuple(s for s in workload.shapes if s.name == args.only)
        if not shapes:
            ap.error(f"--only: no product named {args.only} in {args.workload}")
        workload = dataclasses.replace(workload, shapes=shapes)
    if args.impl == "reference":
        return run_reference(args, workload, rank)
    import __graft_entry__
    __graft_entry__.build()
    return run_ours(args, workload)


if __name__ == "__main__":
    sys.exit(main())
