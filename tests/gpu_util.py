"""Helpers shared by the GPU tests: move seeded operands to the device, run a plan
through the C ABI, and compare with the oracle."""
from __future__ import annotations

import numpy as np

import oracle

TOL = {"f32_ffma": 1e-5, "tf32": 5e-3, "bf16": 1e-2, "w4_bf16": 1e-2}


def torch_mod():
    import torch
    return torch


def dev(x):
    """numpy operand -> CUDA tensor (uint16 arrays are bf16 bit patterns)."""
    torch = torch_mod()
    if x is None:
        return None
    if x.dtype == np.uint16:
        return torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).view(torch.bfloat16).cuda()
    return torch.from_numpy(np.ascontiguousarray(x)).cuda()


def layout_code(b_layout: str) -> int:
    return oracle.B_KN if b_layout == "KN" else oracle.B_NK


def run_plan(plan, A, B, bias, M, N, batch=1, C=None):
    """Run `plan` on numpy operands; returns C as numpy float32."""
    torch = torch_mod()
    dA, dB, dbias = dev(A), dev(B), dev(bias)
    shape = (batch, M, N) if batch > 1 else (M, N)
    if C is None:
        C = torch.full(shape, float("nan"), dtype=torch.float32, device="cuda")
    if batch > 1 and bias is None:
        plan_run_batched(plan, dA, dB, C)
    else:
        plan.run(dA, dB, dbias, C)
    torch.cuda.synchronize()
    plan.check()
    return C.cpu().numpy()


def plan_run_batched(plan, dA, dB, C):
    import paper_2309_08978_gb300 as nj
    nj.nnjit_matmul_run_batched(plan, dA, dB, C)


def compare(C_gpu, A, B, bias, b_layout, dtype, exact=False, act="none", residual=None):
    ref64, ref32 = oracle.matmul(A, B, bias, layout_code(b_layout), act=act, residual=residual)
    assert C_gpu.shape == ref64.shape
    assert np.all(np.isfinite(C_gpu)), "non-finite output (unwritten element?)"
    if exact:
        bad = np.argwhere(C_gpu != ref32)
        assert bad.size == 0, f"{len(bad)} elements differ, first at {bad[:5].tolist()}"
        return 0.0
    err = oracle.rel_fro(C_gpu, ref64)
    assert err <= TOL[dtype], f"rel_fro {err:.3e} > {TOL[dtype]}"
    return err
