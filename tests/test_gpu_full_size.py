"""Full-size parity: every product of the benchmark workloads -- the BART-base, T5-large and
Llama-2-7B Linears and attention BatchMatMuls (the MatMul / BatchMatMul kernels K0-K3 of
Table 3 at these models' sizes) -- planned the way the benchmark plans them, and every
candidate of each product's space, checked against the oracle at the full sizes.

The oracle computes sampled output rows: two rows of every 128-row tile plus every row of
the last tile (batched products: every row of a few batch items, the last included).
Exact mode draws integers in [-8, 8]: |sum| <= 64 K <= 704,512 < 2^24 for every K here,
so every summation order is exact in f32 and the GPU rows must equal the oracle's bit for
bit.  Random mode draws the workloads' own distributions and holds the tuned plan to the
dtype's relative-Frobenius tolerance on the same rows.
"""
import numpy as np
import pytest

import oracle
from gpu_util import TOL
from synthetic import WORKLOADS, make_operands

pytestmark = pytest.mark.gpu

nj = pytest.importorskip("paper_2309_08978_gb300")

# The benchmark's planning: weights are constant, and the workload's 30 s tuning budget
# is shared out over its products.
BENCH_TOTAL_BUDGET_MS = 30000.0

CASES = [(wk, i) for wk in ("bart_base_encoder_m512", "t5_large_layer_m2048",
                            "llama2_7b_decode_m1", "llama2_7b_prefill_m4096",
                            "llama2_7b_decode_w4_m1")
         for i in range(len(WORKLOADS[wk].shapes))]


def _ids(case):
    wk, i = case
    s = WORKLOADS[wk].shapes[i]
    return f"{wk}-{s.name}-{s.batch}x{s.M}x{s.N}x{s.K}"


def sample_rows(M, tile=128):
    """Two rows of every 128-row tile (a different pair per tile) and the whole last tile."""
    rows = set()
    for t in range((M + tile - 1) // tile):
        for r in ((7 * t + 3) % tile, tile - 1 - (13 * t) % tile):
            if t * tile + r < M:
                rows.add(t * tile + r)
    last = (M - 1) // tile * tile
    rows.update(range(last, M))
    return np.array(sorted(rows), dtype=np.int64)


def sample_items(batch):
    return np.array(sorted({0, batch // 3, (2 * batch) // 3, batch - 1}), dtype=np.int64)


def _dev(x):
    import torch
    if x is None:
        return None
    if x.dtype == np.uint16:
        return torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).view(torch.bfloat16).cuda()
    return torch.from_numpy(np.ascontiguousarray(x)).cuda()


class Product:
    """One workload product on the device, with the oracle's rows for it."""

    def __init__(self, wk, i, ints):
        w = WORKLOADS[wk]
        self.n_products = len(w.shapes)
        self.s = s = w.shapes[i]
        self.dtype = w.dtypes[-1]
        self.A, self.B, self.bias = make_operands(s, w.index, self.dtype, ints=ints)
        self.dA, self.dB, self.dbias = _dev(self.A), _dev(self.B), _dev(self.bias)
        self.flags = nj.NNJIT_PLAN_B_CONSTANT if s.b_is_weight else 0
        self.layout = oracle.B_KN if s.b_layout == "KN" else oracle.B_NK
        if s.batch > 1:
            self.items = sample_items(s.batch)
            self.rows = None
        else:
            self.items = None
            self.rows = sample_rows(s.M)
        self.ref64, self.ref32 = self._oracle()

    def _oracle(self):
        s = self.s
        if self.dtype == "w4_bf16":
            from oracle.quant import matmul as w4_matmul
            return w4_matmul(self.A[self.rows], self.B, s.N, s.K, 0, self.bias)
        if s.batch > 1:
            return oracle.matmul(self.A[self.items], self.B[self.items], None, self.layout)
        return oracle.matmul_rows(self.A, self.B, self.bias, self.layout, self.rows)

    def desc(self):
        s = self.s
        return nj.make_desc(s.M, s.N, s.K, self.dtype, s.b_layout, batch=s.batch,
                            has_bias=s.has_bias, flags=self.flags)

    def run(self, plan):
        """Run `plan` once; the sampled rows (or batch items) of C as numpy."""
        import torch
        s = self.s
        shape = (s.batch, s.M, s.N) if s.batch > 1 else (s.M, s.N)
        C = torch.full(shape, float("nan"), dtype=torch.float32, device="cuda")
        if s.batch > 1:
            nj.nnjit_matmul_run_batched(plan, self.dA, self.dB, C)
        else:
            plan.run(self.dA, self.dB, self.dbias, C)
        torch.cuda.synchronize()
        plan.check()
        idx = torch.from_numpy(self.items if s.batch > 1 else self.rows).cuda()
        out = C.index_select(0, idx).cpu().numpy()
        del C
        return out


def _bench_plan(prod):
    return nj.nnjit_matmul_plan_ex(prod.desc(), BENCH_TOTAL_BUDGET_MS / prod.n_products)


@pytest.mark.parametrize("case", CASES, ids=_ids)
def test_full_size_every_candidate_exact(case):
    """Integer inputs: the benchmark's tuned plan and then every candidate of the space
    must reproduce the oracle's rows bit for bit."""
    wk, i = case
    prod = Product(wk, i, ints=True)
    with _bench_plan(prod) as plan:
        got = prod.run(plan)
        chosen = plan.describe()["chosen_index"]
    bad = np.argwhere(got != prod.ref32)
    assert bad.size == 0, f"tuned plan (candidate {chosen}): {len(bad)} mismatches, first {bad[:3].tolist()}"
    cands, _ = nj.nnjit_space_enumerate(prod.desc(), nj.nnjit_device_limits_query(0))
    for j in range(len(cands)):
        with nj.nnjit_matmul_plan_candidate(prod.desc(), j) as plan:
            got = prod.run(plan)
        bad = np.argwhere(got != prod.ref32)
        assert bad.size == 0, f"candidate {j} {cands[j]}: {len(bad)} mismatches, first {bad[:3].tolist()}"


@pytest.mark.parametrize("case", CASES, ids=_ids)
def test_full_size_tuned_plan_within_tolerance(case):
    """The workload's own distributions: the tuned plan within the dtype's tolerance."""
    wk, i = case
    prod = Product(wk, i, ints=False)
    with _bench_plan(prod) as plan:
        got = prod.run(plan)
    assert np.all(np.isfinite(got))
    err = oracle.rel_fro(got, prod.ref64)
    assert err <= TOL[prod.dtype], f"rel_fro {err:.3e} > {TOL[prod.dtype]}"
