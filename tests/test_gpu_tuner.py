"""The JIT tuner and plan cache on the GPU: budget semantics, cache hits, exhaustive
sweeps, the persisted kernel database, host-side fault injection, end-to-end host path."""
import os

import numpy as np
import pytest

from synthetic import Shape, make_operands
from gpu_util import run_plan, compare

pytestmark = pytest.mark.gpu

nj = pytest.importorskip("paper_2309_08978_gb300")


def _desc(flags=0):
    return nj.make_desc(512, 768, 768, "bf16", "NK", has_bias=True, flags=flags)


def test_budget_zero_takes_top_ranked_untimed():
    desc = _desc(nj.NNJIT_PLAN_NO_CACHE)
    lim = nj.nnjit_device_limits_query(0)
    cands, _ = nj.nnjit_space_enumerate(desc, lim)
    with nj.nnjit_matmul_plan_ex(desc, 0.0) as plan:
        info = plan.describe()
        assert info["chosen_index"] == 0 and info["timed"] is False
        assert plan.candidate() == cands[0]
    with pytest.raises(nj.NnjitError) as ei:
        nj.nnjit_matmul_plan_ex(_desc(nj.NNJIT_PLAN_NO_CACHE | nj.NNJIT_PLAN_REQUIRE_TIMED), 0.0)
    assert ei.value.status == nj.NNJIT_ERR_BUDGET


def test_exhaustive_times_every_candidate_and_picks_the_fastest():
    desc = _desc(nj.NNJIT_PLAN_EXHAUSTIVE)
    with nj.nnjit_matmul_plan_ex(desc, 0.0) as plan:
        info = plan.describe()
    assert len(info["timings_us"]) + len(info["failed"]) == info["space_size"]
    assert not info["failed"]
    # the pick is the fastest re-timed candidate (re-timing can reorder near-ties)
    times = dict((int(i), t) for i, t in info["timings_us"])
    assert times[info["chosen_index"]] <= min(times.values()) * 1.05


def test_cache_hit_and_persistence(tmp_path):
    nj.nnjit_cache_clear()
    desc = _desc()
    with nj.nnjit_matmul_plan_ex(desc, 200.0) as p1:
        i1 = p1.describe()
        assert i1["from_cache"] is False and i1["timed"] is True
    assert nj.nnjit_cache_size() == 1
    with nj.nnjit_matmul_plan_ex(desc, 200.0) as p2:
        i2 = p2.describe()
        assert i2["from_cache"] is True and i2["candidate"] == i1["candidate"]
    path = str(tmp_path / "plans.cache")
    nj.nnjit_cache_save(path)
    nj.nnjit_cache_clear()
    assert nj.nnjit_cache_load(path) == 1
    with nj.nnjit_matmul_plan_ex(desc, 200.0) as p3:
        i3 = p3.describe()
        assert i3["from_cache"] is True and i3["candidate"] == i1["candidate"]
        shape = Shape("t", 512, 768, 768, 1, "NK", True)
        A, B, bias = make_operands(shape, 30, "bf16", ints=True)
        compare(run_plan(p3, A, B, bias, 512, 768), A, B, bias, "NK", "bf16", exact=True)
    nj.nnjit_cache_clear()


def test_cached_candidate_outside_the_space_is_retuned(tmp_path):
    nj.nnjit_cache_clear()
    desc = _desc()
    with nj.nnjit_matmul_plan_ex(desc, 50.0):
        pass
    path = tmp_path / "plans.cache"
    nj.nnjit_cache_save(str(path))
    lines = path.read_text().splitlines()
    key, cand, rest, tim = lines[1].split("\t")
    fields = cand.split()
    fields[2] = "96"                      # BN = 96 is not a member of any space
    path.write_text(lines[0] + "\n" + "\t".join([key, " ".join(fields), rest, tim]) + "\n")
    nj.nnjit_cache_clear()
    assert nj.nnjit_cache_load(str(path)) == 1
    with nj.nnjit_matmul_plan_ex(desc, 50.0) as plan:
        info = plan.describe()
        assert info["from_cache"] is False and info["candidate"]["bn"] != 96
    nj.nnjit_cache_clear()


@pytest.mark.parametrize("kind", ["launch", "timeout"])
def test_fault_injection_skips_the_candidate(kind, monkeypatch):
    """Host-side injection: candidate 0 reports a launch error or an expired watchdog;
    the tuner must skip it and still deliver a correct plan."""
    monkeypatch.setenv("NNJIT_FAULT", f"{kind}:0")
    desc = _desc(nj.NNJIT_PLAN_NO_CACHE | nj.NNJIT_PLAN_EXHAUSTIVE)
    with nj.nnjit_matmul_plan_ex(desc, 0.0) as plan:
        info = plan.describe()
        assert 0 in info["failed"] and info["chosen_index"] != 0
        shape = Shape("t", 512, 768, 768, 1, "NK", True)
        A, B, bias = make_operands(shape, 31, "bf16", ints=True)
        compare(run_plan(plan, A, B, bias, 512, 768), A, B, bias, "NK", "bf16", exact=True)


def test_run_host_end_to_end():
    import torch
    shape = Shape("t", 300, 520, 264, 1, "KN", True)
    A, B, bias = make_operands(shape, 32, "tf32")
    desc = nj.make_desc(300, 520, 264, "tf32", "KN", has_bias=True)
    with nj.nnjit_matmul_plan_ex(desc, 20.0) as plan:
        hA = torch.from_numpy(A).pin_memory()
        hB = torch.from_numpy(B).pin_memory()
        hbias = torch.from_numpy(bias).pin_memory()
        hC = torch.empty((300, 520), dtype=torch.float32).pin_memory()
        nj.nnjit_matmul_run_host(plan, hA, hB, hbias, hC)
        torch.cuda.synchronize()
        plan.check()
        compare(hC.numpy(), A, B, bias, "KN", "tf32")


def test_run_host_seq_overlapped_sequence():
    """A sequence of products from host buffers with overlapped transfers: a tensor-core
    product with bias, a GEMV, a batched product and the first plan again with new
    inputs (its staging buffers are reused in order), all bit exact against the oracle on
    integer inputs; then twice in a row to check that a second call waits for the first."""
    import torch

    def pinned(x):
        if x is None:
            return None
        if x.dtype == np.uint16:
            return torch.from_numpy(x.view(np.int16)).view(torch.bfloat16).pin_memory()
        return torch.from_numpy(x).pin_memory()

    specs = [(Shape("a", 300, 520, 264, 1, "NK", True), 41),
             (Shape("b", 1, 1000, 512, 1, "NK", False), 42),
             (Shape("c", 130, 72, 64, 3, "KN", False), 43),
             (Shape("a", 300, 520, 264, 1, "NK", True), 44)]
    plans = {}
    items = []
    for shape, seed in specs:
        key = (shape.M, shape.N, shape.K, shape.batch, shape.b_layout)
        if key not in plans:
            desc = nj.make_desc(shape.M, shape.N, shape.K, "bf16", shape.b_layout, batch=shape.batch,
                                has_bias=shape.has_bias, flags=nj.NNJIT_PLAN_NO_CACHE)
            plans[key] = nj.nnjit_matmul_plan_ex(desc, 20.0)
        A, B, bias = make_operands(shape, seed, "bf16", ints=True)
        out = (shape.batch, shape.M, shape.N) if shape.batch > 1 else (shape.M, shape.N)
        hC = torch.full(out, float("nan"), dtype=torch.float32).pin_memory()
        items.append((plans[key], shape, A, B, bias, pinned(A), pinned(B), pinned(bias), hC))
    try:
        for _ in range(2):
            for it in items:
                it[8].fill_(float("nan"))
            nj.nnjit_matmul_run_host_seq([it[0] for it in items], [it[5] for it in items],
                                         [it[6] for it in items], [it[7] for it in items],
                                         [it[8] for it in items])
            torch.cuda.synchronize()
            for plan, shape, A, B, bias, *_, hC in items:
                plan.check()
                compare(hC.numpy(), A, B, bias, shape.b_layout, "bf16", exact=True)
    finally:
        for p in plans.values():
            p.destroy()


def test_invalid_run_arguments():
    import torch
    with nj.nnjit_matmul_plan_ex(nj.make_desc(256, 256, 256, "bf16", "NK"), 0.0) as plan:
        A = torch.zeros((256, 256), dtype=torch.bfloat16, device="cuda")
        C = torch.zeros((256, 256), dtype=torch.float32, device="cuda")
        with pytest.raises(nj.NnjitError) as ei:
            plan.run(A.data_ptr() + 2, A, None, C)          # misaligned A
        assert ei.value.status == nj.NNJIT_ERR_UNSUPPORTED
        with pytest.raises(nj.NnjitError) as ei:
            plan.run(A, None, None, C)
        assert ei.value.status == nj.NNJIT_ERR_INVALID_ARG


def test_online_plan_serves_exact_results_while_it_tunes():
    import torch
    from gpu_util import dev
    nj.nnjit_cache_clear()
    M, N, K = 512, 768, 768
    shape = Shape("t", M, N, K, 1, "NK", True)
    A, B, bias = make_operands(shape, 33, "bf16", ints=True)
    from oracle import matmul, B_NK
    _, ref32 = matmul(A, B, bias, B_NK)
    desc = nj.make_desc(M, N, K, "bf16", "NK", has_bias=True)
    plan = nj.nnjit_matmul_plan_online(desc)
    dA, dB, dbias = dev(A), dev(B), dev(bias)
    C = torch.empty((M, N), dtype=torch.float32, device="cuda")
    prog = nj.nnjit_plan_online_progress(plan)
    assert prog["done"] is False and prog["evaluated"] == 0
    calls = 0
    while not prog["done"] and calls < 1000:
        C.fill_(float("nan"))
        plan.run(dA, dB, dbias, C)
        torch.cuda.synchronize()
        assert np.array_equal(C.cpu().numpy(), ref32), f"call {calls}"
        calls += 1
        prog = nj.nnjit_plan_online_progress(plan)
    assert prog["done"], calls
    info = plan.describe()
    assert len(info["timings_us"]) + len(info["failed"]) == info["space_size"]
    times = dict((int(i), t) for i, t in info["timings_us"])
    # the incumbent is never beaten by more than the 2 % margin
    assert times[prog["current_index"]] <= min(times.values()) / 0.98 + 1e-9
    plan.run(dA, dB, dbias, C)
    torch.cuda.synchronize()
    assert np.array_equal(C.cpu().numpy(), ref32)
    plan.destroy()
    # the finished choice is in the kernel database
    with nj.nnjit_matmul_plan_ex(desc, 1000.0) as p2:
        i2 = p2.describe()
        assert i2["from_cache"] is True and i2["chosen_index"] == prog["current_index"]
    nj.nnjit_cache_clear()


def test_settings_study_and_fixed_settings():
    """The one-variable-at-a-time study (Sec. 5.1) times each product's full space, and
    each setting's verdict is consistent with the times it reports; the settings it
    recommends shrink the spaces (never to zero), are part of the plan-cache key and
    the plan description, and a plan from the shrunk space stays exact."""
    descs = [nj.make_desc(512, 2304, 768, "tf32", "NK", has_bias=True),
             nj.make_desc(1024, 1024, 1024, "bf16", "NK")]
    rec, report = nj.nnjit_settings_study(descs)
    assert set(rec) == set(nj.SETTING_AXES)
    assert len(report["products"]) == 2
    lim = nj.nnjit_device_limits_query(0)
    for prod, d in zip(report["products"], descs):
        cands, _ = nj.nnjit_space_enumerate(d, lim)
        assert prod["space_size"] == len(cands)
        for axis, ev in prod["settings"].items():
            assert ev["value"] == prod["best"][axis]
            if ev["verdict"] == "decisive":
                assert ev["twin_us"] > 1.02 * prod["best_us"]
                assert rec[axis] in (-1, ev["value"])
            elif ev["verdict"] == "tie":
                assert ev["twin_us"] <= 1.02 * prod["best_us"]
    for axis, v in rec.items():
        votes = {p["settings"][axis]["value"] for p in report["products"]
                 if p["settings"][axis]["verdict"] == "decisive"}
        assert (v == -1) == (len(votes) != 1) and (v == -1 or votes == {v})
    # apply a fixed setting set (the recommended one, or a hand-picked one when the study
    # found nothing decisive) and check the shrunk space and a plan from it
    fixed = {a: v for a, v in rec.items() if v != -1} or {"raster": 0, "kgroup": 2}
    full = [len(nj.nnjit_space_enumerate(d, lim)[0]) for d in descs]
    nj.nnjit_settings_set(fixed)
    try:
        shrunk = [len(nj.nnjit_space_enumerate(d, lim)[0]) for d in descs]
        assert all(1 <= s <= f for s, f in zip(shrunk, full))
        shape = Shape("t", 512, 2304, 768, 1, "NK", True)
        A, B, bias = make_operands(shape, 31, "tf32", ints=True)
        with nj.nnjit_matmul_plan_ex(descs[0], 200.0) as plan:
            info = plan.describe()
            assert info["settings"] == [fixed.get(a, -1) for a in nj.SETTING_AXES]
            C = run_plan(plan, A, B, bias, 512, 2304)
        compare(C, A, B, bias, "NK", "tf32", exact=True)
    finally:
        nj.nnjit_settings_set(None)
