"""Layer-wide budget (AdaKV variant, ecokv_evict_adaptive) against the oracle:
the selection is the oracle's select_adaptive on the GPU's own scores, bit for
bit; the scores and lambda are those of ecokv_score (which the parity tests tie
to the oracle); the gathered rows are bit-exact copies.  Small cases also run
the oracle's whole adaptive pass and compare retained sets up to threshold ties."""
import numpy as np
import pytest
import torch

from oracle import ecokv_oracle as O
from paper_2609_06663_gb300 import ecokv as E
from paper_2609_06663_gb300.workloads import make_inputs, small_workload, workload
from tests.parity import TOL, oracle_params

DEV = "cuda"


def params_of(w):
    return E.make_params(n_layers=w.n_layers, h_kv=w.h_kv, h_q=w.h_q, n=w.n, d=w.d, window=w.window,
                         budget=w.budget, pool_kernel=w.pool_kernel)


def one_layer(w, seed):
    return type(w)(**{**{f: getattr(w, f) for f in w.__dataclass_fields__}, "n_layers": 1, "seed": seed})


CASES = [
    small_workload(5000, h_kv=4, group=2, window=8, budget=500, dtype="bf16", n_layers=2, clustered=True),
    small_workload(3001, h_kv=2, group=1, window=8, budget=300, pool_kernel=7, dtype="f32"),
    small_workload(700, h_kv=3, group=2, window=4, budget=900, dtype="bf16"),       # B >= N
    small_workload(600, h_kv=2, group=2, window=6, budget=6, dtype="bf16"),         # B = W: windows only
    one_layer(workload("c3_b10"), 7),
]
IDS = ["bf16_tc", "f32_simt", "keep_all", "windows_only", "c3_one_layer"]


@pytest.mark.gpu
@pytest.mark.parametrize("w", CASES, ids=IDS)
def test_adaptive_selection_and_rows(w):
    K, V, Q = make_inputs(w, device=DEV)
    p = params_of(w)
    S, lam_s, _ = E.score(p, K, Q)
    idx, off, Ko, Vo, lam = E.evict_adaptive(p, K, V, Q)
    torch.cuda.synchronize()
    assert torch.equal(lam, lam_s)
    op = oracle_params(p)
    S_np = S.cpu().double().numpy()
    idx_np, off_np = idx.cpu().numpy(), off.cpu().numpy()
    n_keep = min(p.budget, p.n)
    for l in range(w.n_layers):
        lists = O.select_adaptive([S_np[l, h] for h in range(w.h_kv)], op)
        ref_off = np.concatenate([[0], np.cumsum([len(x) for x in lists])])
        assert np.array_equal(off_np[l], ref_off), f"layer {l} offsets"
        assert np.array_equal(idx_np[l], np.concatenate(lists)), f"layer {l} indices"
        assert off_np[l, -1] == w.h_kv * n_keep
        for h in range(w.h_kv):
            seg = idx[l, off_np[l, h]:off_np[l, h + 1]].long()
            assert torch.equal(Ko[l, off_np[l, h]:off_np[l, h + 1]], K[l, h, seg])
            assert torch.equal(Vo[l, off_np[l, h]:off_np[l, h + 1]], V[l, h, seg])


@pytest.mark.gpu
@pytest.mark.parametrize("w", CASES[:2], ids=IDS[:2])
def test_adaptive_matches_whole_oracle_pass(w):
    K, V, Q = make_inputs(w)
    p = params_of(w)
    idx, off, _, _, lam = E.evict_adaptive(p, K.to(DEV), V.to(DEV), Q.to(DEV))
    S, _, _ = E.score(p, K.to(DEV), Q.to(DEV))
    torch.cuda.synchronize()
    op = oracle_params(p)
    ref = O.evict_adaptive(K, V, Q, op)
    tol = TOL[w.dtype]
    S_np = S.cpu().double().numpy()
    for l in range(w.n_layers):
        r = ref[l]
        for h in range(w.h_kv):
            assert abs(float(lam[l, h]) - r["heads"][h]["lam"]) <= tol
        # retained (head, position) pairs agree except at the layer threshold
        S_ref = np.concatenate([r["heads"][h]["S"] for h in range(w.h_kv)])
        scale = max(np.abs(S_ref).max(), np.abs(S_ref).mean())
        k_layer = w.h_kv * (p.budget - p.window)
        thr = np.sort(S_ref)[::-1][k_layer - 1]
        got = {(h, int(i)) for h in range(w.h_kv)
               for i in idx[l, off[l, h]:off[l, h + 1]].cpu().numpy() if i < op.t_v}
        want = {(h, int(i)) for h in range(w.h_kv)
                for i in r["idx"][r["head_off"][h]:r["head_off"][h + 1]] if i < op.t_v}
        for (h, i) in got ^ want:
            assert abs(S_ref[h * op.t_v + i] - thr) <= 4 * tol * scale, (l, h, i)
