"""Value-norm importance (ECOKV_FLAG_VNORM_IMP: S_imp = pooled vote * ||v||,
reading R17) against the oracle: scores within the tolerance, lambda, the
selection exact on the GPU's own scores and equal to the oracle's up to
threshold ties, bit-exact rows; the entry points without V refuse the flag."""
import numpy as np
import pytest
import torch

from oracle import ecokv_oracle as O
from paper_2609_06663_gb300 import ecokv as E
from paper_2609_06663_gb300.workloads import make_inputs, small_workload, sweep_workload, workload
from tests.parity import TOL, check_rows, check_selection, oracle_params, score_error

DEV = "cuda"


def params_of(w, flags=E.ECOKV_FLAG_VNORM_IMP):
    return E.make_params(n_layers=w.n_layers, h_kv=w.h_kv, h_q=w.h_q, n=w.n, d=w.d, window=w.window,
                         budget=w.budget, pool_kernel=w.pool_kernel, flags=flags)


def one_layer(w, seed):
    return type(w)(**{**{f: getattr(w, f) for f in w.__dataclass_fields__}, "n_layers": 1, "seed": seed})


CASES = [
    (small_workload(5000, h_kv=2, group=4, window=8, budget=500, dtype="bf16", n_layers=2, clustered=True), None),
    (small_workload(3001, h_kv=2, group=1, window=8, budget=300, pool_kernel=7, dtype="f32"), None),
    (small_workload(20000, h_kv=2, group=4, window=8, budget=2000, dtype="bf16", clustered=True), None),
    (one_layer(workload("c3_b10"), 9), [(0, 0), (0, 3)]),
]
IDS = ["bf16_tc", "f32_simt", "bf16_wide_cluster", "c3_one_layer"]


@pytest.mark.gpu
@pytest.mark.parametrize("case", CASES, ids=IDS)
def test_value_norm_importance(case):
    w, units = case
    K, V, Q = make_inputs(w)
    p = params_of(w)
    idx, Ko, Vo, S, lam = E.evict(p, K.to(DEV), V.to(DEV), Q.to(DEV), want_scores=True)
    torch.cuda.synchronize()
    op = oracle_params(p)
    assert op.flags & O.FLAG_VNORM_IMP
    units = units or [(l, h) for l in range(w.n_layers) for h in range(w.h_kv)]
    ref = O.evict(K, V, Q, op, heads=units)
    tol = TOL[w.dtype]
    S_np = S.cpu().double().numpy()
    for (l, h) in units:
        r = ref[(l, h)]
        what = f"{w.name} unit ({l},{h})"
        assert score_error(S_np[l, h], r["S"]) <= tol, what
        assert abs(float(lam[l, h]) - r["lam"]) <= tol, what
        check_selection(idx[l, h].cpu().numpy(), r, op, tol, what)
        check_rows(K[l, h].to(DEV), idx[l, h], Ko[l, h], what)
        check_rows(V[l, h].to(DEV), idx[l, h], Vo[l, h], what)


@pytest.mark.gpu
@pytest.mark.parametrize("flags", [
    E.ECOKV_FLAG_VNORM_IMP | E.ECOKV_FLAG_MAD,
    E.ECOKV_FLAG_VNORM_IMP | E.ECOKV_FLAG_WINSOR_1 | E.ECOKV_FLAG_CENTROID_NONWIN,
    E.ECOKV_FLAG_MAD | E.ECOKV_FLAG_CENTROID_NONWIN | E.ECOKV_FLAG_SC_MIXKV_SIGN,
], ids=["vnorm_mad", "vnorm_winsor1_nonwin", "mad_nonwin_mixsign"])
@pytest.mark.parametrize("case", CASES[:2], ids=IDS[:2])
def test_combined_variant_flags(case, flags):
    # the variants compose: each flag changes an independent term of the score
    w, units = case
    K, V, Q = make_inputs(w)
    p = params_of(w, flags)
    idx, Ko, Vo, S, lam = E.evict(p, K.to(DEV), V.to(DEV), Q.to(DEV), want_scores=True)
    torch.cuda.synchronize()
    op = oracle_params(p)
    assert op.flags == flags
    units = [(l, h) for l in range(w.n_layers) for h in range(w.h_kv)]
    ref = O.evict(K, V, Q, op, heads=units)
    tol = TOL[w.dtype]
    S_np = S.cpu().double().numpy()
    for (l, h) in units:
        r = ref[(l, h)]
        what = f"{w.name} unit ({l},{h}) flags {flags:#x}"
        assert score_error(S_np[l, h], r["S"]) <= tol, what
        assert abs(float(lam[l, h]) - r["lam"]) <= tol, what
        check_selection(idx[l, h].cpu().numpy(), r, op, tol, what)
        check_rows(V[l, h].to(DEV), idx[l, h], Vo[l, h], what)


@pytest.mark.gpu
def test_value_norm_flag_changes_the_scores_and_is_refused_without_values():
    w = CASES[0][0]
    K, V, Q = make_inputs(w, device=DEV)
    _, _, _, S0, _ = E.evict(params_of(w, 0), K, V, Q, want_scores=True)
    _, _, _, S1, _ = E.evict(params_of(w), K, V, Q, want_scores=True)
    assert not torch.equal(S0, S1)
    with pytest.raises(E.EcokvError) as e:
        E.score(params_of(w), K, Q)
    assert e.value.code == E.ECOKV_ERR_UNSUPPORTED


@pytest.mark.gpu
@pytest.mark.parametrize("n", [65536, 131072])
@pytest.mark.parametrize("flags", [E.ECOKV_FLAG_VNORM_IMP, E.ECOKV_FLAG_WINSOR_5, E.ECOKV_FLAG_MAD],
                         ids=["vnorm", "winsor5", "mad"])
def test_variants_on_long_heads(flags, n):
    # the sweep's long layers: clusters of 8 (65532 candidates) and 16 CTAs
    # (131068) finalize the heads, and the order statistics read the rows
    # from L2 instead of holding them in shared memory; two heads against the
    # oracle
    w = sweep_workload(n, 4)
    K, V, Q = make_inputs(w)
    p = params_of(w, flags)
    idx, Ko, Vo, S, lam = E.evict(p, K.to(DEV), V.to(DEV), Q.to(DEV), want_scores=True)
    torch.cuda.synchronize()
    op = oracle_params(p)
    units = [(0, 0), (0, 5)]
    ref = O.evict(K, V, Q, op, heads=units)
    tol = TOL[w.dtype]
    S_np = S.cpu().double().numpy()
    for (l, h) in units:
        r = ref[(l, h)]
        what = f"{w.name} unit ({l},{h}) flags {flags:#x}"
        assert score_error(S_np[l, h], r["S"]) <= tol, what
        assert abs(float(lam[l, h]) - r["lam"]) <= tol, what
        check_selection(idx[l, h].cpu().numpy(), r, op, tol, what)
        check_rows(V[l, h].to(DEV), idx[l, h], Vo[l, h], what)


@pytest.mark.gpu
def test_value_norm_refused_past_the_cluster_finalize():
    # past 16 x 8192 candidates no cluster shape takes the head
    w = small_workload(140000, h_kv=1, group=1, window=4, budget=400, dtype="bf16")
    K, V, Q = make_inputs(w, device=DEV)
    with pytest.raises(E.EcokvError) as e:
        E.evict(params_of(w), K, V, Q)
    assert e.value.code == E.ECOKV_ERR_UNSUPPORTED
