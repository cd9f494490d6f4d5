"""ecokv_evict_noalloc (workspace held by the library, nothing allocated by the
call) against ecokv_evict with a caller workspace, bit for bit, on two calls in
a row, and its host-side size check.  The file name sorts last so that the entry point is
exercised both alone and after every other test in the same process."""
import numpy as np
import pytest
import torch

from paper_2609_06663_gb300 import ecokv as E
from paper_2609_06663_gb300.workloads import make_inputs, small_workload, workload
from tests.parity import check_rows

DEV = "cuda"


def params_of(w):
    return E.make_params(n_layers=w.n_layers, h_kv=w.h_kv, h_q=w.h_q, n=w.n, d=w.d, window=w.window,
                         budget=w.budget, pool_kernel=w.pool_kernel)


def one_layer(w, seed):
    return type(w)(**{**{f: getattr(w, f) for f in w.__dataclass_fields__}, "n_layers": 1, "seed": seed})


def test_oversize_request_rejected_on_host():
    """All 28 layers of the 32k-token workload need more than the fixed
    scratch: rejected with ECOKV_ERR_WORKSPACE before anything is launched
    (no GPU involved).  One layer of it fits."""
    E.lib()
    w = workload("c3_b10")
    p = params_of(w)
    assert E.ecokv_workspace_size(p) > E.ECOKV_NOALLOC_SCRATCH_BYTES
    code = E.ecokv_evict_noalloc(p, E.ECOKV_BF16, None, None, None, None, None, None, None, None, None)
    assert code == E.ECOKV_ERR_WORKSPACE
    assert E.ecokv_workspace_size(params_of(one_layer(w, w.seed))) <= E.ECOKV_NOALLOC_SCRATCH_BYTES


CASES = [
    # tensor-core path: bf16, several items per head, ragged tail
    (small_workload(5000, h_kv=2, group=4, window=8, budget=500, dtype="bf16", n_layers=2, clustered=True),
     small_workload(5000, h_kv=2, group=4, window=8, budget=500, dtype="bf16", n_layers=2, clustered=True,
                    seed=1)),
    # CUDA-core path: fp32
    (small_workload(3001, h_kv=2, group=1, window=8, budget=300, pool_kernel=7, dtype="f32"),
     small_workload(3001, h_kv=2, group=1, window=8, budget=300, pool_kernel=7, dtype="f32", seed=1)),
    # one layer of the 32k-token workload, at full length
    (one_layer(workload("c3_b10"), 11), one_layer(workload("c3_b10"), 12)),
]


@pytest.mark.gpu
@pytest.mark.parametrize("pair", CASES, ids=["bf16_tc", "f32_simt", "c3_one_layer"])
def test_noalloc_matches_workspace_entry_two_calls(pair):
    for w in pair:  # two calls in a row, on different inputs
        K, V, Q = make_inputs(w, device=DEV)
        p = params_of(w)
        assert E.ecokv_workspace_size(p) <= E.ECOKV_NOALLOC_SCRATCH_BYTES
        idx_r, Ko_r, Vo_r, S_r, lam_r = E.evict(p, K, V, Q, want_scores=True)
        idx, Ko, Vo, S, lam, code = E.evict_noalloc(p, K, V, Q, want_scores=True)
        torch.cuda.synchronize()
        assert code == 0, E.ecokv_status_string(code)
        # the same kernels on the same inputs with the same schedule: every
        # output is bit for bit the one the caller-workspace entry returns
        # (a stale or misplaced scratch region would show here)
        what = w.name
        assert torch.equal(S, S_r), f"{what}: scores differ from ecokv_evict"
        assert torch.equal(lam, lam_r), f"{what}: lambda differs from ecokv_evict"
        assert torch.equal(idx, idx_r), f"{what}: indices differ from ecokv_evict"
        assert torch.equal(Ko, Ko_r) and torch.equal(Vo, Vo_r), f"{what}: gathered rows differ"
        # and the pass itself is sound: rows are the ones idx names
        for h in range(w.h_kv):
            for l in range(w.n_layers):
                check_rows(K[l, h], idx[l, h], Ko[l, h], f"{what} unit ({l},{h})")
                check_rows(V[l, h], idx[l, h], Vo[l, h], f"{what} unit ({l},{h})")
        assert np.isfinite(S.cpu().numpy()).all()
