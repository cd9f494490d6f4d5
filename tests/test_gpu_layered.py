"""Per-layer budgets (PyramidKV schedule, ecokv_evict_layered, reading R18)
against the oracle's evict_layered: scores, lambda, each layer's selection
with its own budget, -1 in the slots past it, bit-exact rows."""
import numpy as np
import pytest
import torch

from oracle import ecokv_oracle as O
from paper_2609_06663_gb300 import ecokv as E
from paper_2609_06663_gb300.workloads import make_inputs, small_workload, workload
from tests.parity import TOL, check_rows, check_selection, oracle_params, score_error

DEV = "cuda"


def layers_of(w, n):
    return type(w)(**{**{f: getattr(w, f) for f in w.__dataclass_fields__}, "n_layers": n})


CASES = [
    # (workload, beta): bf16 tensor-core path, 4 layers
    (small_workload(3000, h_kv=2, group=2, window=8, budget=300, dtype="bf16", n_layers=4, clustered=True), 20.0),
    # fp32 CUDA-core path
    (small_workload(1500, h_kv=2, group=1, window=4, budget=150, pool_kernel=7, dtype="f32", n_layers=3), 5.0),
    # the first layer's budget exceeds N: kept whole
    (small_workload(300, h_kv=2, group=2, window=4, budget=200, dtype="bf16", n_layers=4), 20.0),
    # four layers of the 8k-token workload
    (layers_of(workload("c2"), 4), 20.0),
]
IDS = ["bf16_tc", "f32_simt", "first_layer_whole", "c2_four_layers"]


@pytest.mark.gpu
@pytest.mark.parametrize("case", CASES, ids=IDS)
def test_layered_budgets_match_oracle(case):
    w, beta = case
    budgets = E.pyramid_budgets(w.n_layers, w.budget, w.window, beta)
    stride = max(budgets)
    p = E.make_params(n_layers=w.n_layers, h_kv=w.h_kv, h_q=w.h_q, n=w.n, d=w.d, window=w.window, budget=stride,
                      pool_kernel=w.pool_kernel)
    K, V, Q = make_inputs(w)
    idx, Ko, Vo, S, lam = E.evict_layered(p, K.to(DEV), V.to(DEV), Q.to(DEV), budgets, want_scores=True)
    torch.cuda.synchronize()
    op = oracle_params(p)
    ref = O.evict_layered(K, V, Q, op, budgets)
    tol = TOL[w.dtype]
    S_np = S.cpu().double().numpy()
    idx_np = idx.cpu().numpy()
    for (l, h), r in ref.items():
        what = f"{w.name} unit ({l},{h}) budget {budgets[l]}"
        keep = min(budgets[l], w.n)
        assert score_error(S_np[l, h], r["S"]) <= tol, what
        assert abs(float(lam[l, h]) - r["lam"]) <= tol, what
        pl = O.Params(**{**op.__dict__, "budget": budgets[l]})
        check_selection(idx_np[l, h, :keep], r, pl, tol, what)
        assert (idx_np[l, h, keep:] == -1).all(), what
        check_rows(K[l, h].to(DEV), idx[l, h, :keep], Ko[l, h, :keep], what)
        check_rows(V[l, h].to(DEV), idx[l, h, :keep], Vo[l, h, :keep], what)
