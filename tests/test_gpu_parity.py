"""CUDA path (through the C ABI) vs the fp64 oracle on the same seeded inputs.

Small shapes span several 128-key chunks and a ragged tail; the configs run
at their own shapes (layer subsets where the oracle would take long), and
every bf16 config also runs at full size in one call (the 32k-token one in
the same launch the benchmark times), checked on sampled (layer, head) units."""
import numpy as np
import pytest
import torch

from oracle import ecokv_oracle as O
from paper_2609_06663_gb300 import ecokv as E
from paper_2609_06663_gb300.workloads import CONFIGS, make_inputs, small_workload, sweep_workload, workload
from tests.parity import TOL, Guarded, check_rows, check_scores, check_selection, oracle_params, score_error

pytestmark = pytest.mark.gpu
DEV = "cuda"


def params_of(w, **kw):
    return E.make_params(n_layers=w.n_layers, h_kv=w.h_kv, h_q=w.h_q, n=w.n, d=w.d, window=w.window,
                         budget=w.budget, pool_kernel=w.pool_kernel, **kw)


def run_and_compare(w, layers=None, units=None, **kw):
    """Score + evict + split select on the GPU; compare with the oracle."""
    K, V, Q = make_inputs(w, layers=layers)
    nl = K.shape[0]
    wl = type(w)(**{**{f: getattr(w, f) for f in w.__dataclass_fields__}, "n_layers": nl})
    p = params_of(wl, **kw)
    Kd, Vd, Qd = K.to(DEV), V.to(DEV), Q.to(DEV)
    ws = E.alloc_workspace(p, DEV)
    # every output between guard regions (checked after the calls)
    n_keep, tv = min(p.budget, p.n), p.n - p.window
    dt = E.dtype_code(Kd)
    g = {k: Guarded(shape, t, DEV) for k, (shape, t) in {
        "S": ((nl, w.h_kv, tv), torch.float32), "lam": ((nl, w.h_kv), torch.float32),
        "dbg": ((nl, w.h_kv, 5, tv), torch.float32), "idx": ((nl, w.h_kv, n_keep), torch.int32),
        "Ko": ((nl, w.h_kv, n_keep, p.d), Kd.dtype), "Vo": ((nl, w.h_kv, n_keep, p.d), Kd.dtype),
        "S2": ((nl, w.h_kv, tv), torch.float32), "lam2": ((nl, w.h_kv), torch.float32),
        "idx_sel": ((nl, w.h_kv, n_keep), torch.int32)}.items()}
    S, lam, dbg = g["S"].view, g["lam"].view, g["dbg"].view
    idx, Ko, Vo, S2, lam2 = g["idx"].view, g["Ko"].view, g["Vo"].view, g["S2"].view, g["lam2"].view
    idx_sel = g["idx_sel"].view
    assert E.ecokv_score(p, dt, Kd, Qd, S, lam, dbg, ws, ws.numel()) == 0
    assert E.ecokv_evict(p, dt, Kd, Vd, Qd, idx, Ko, Vo, S2, lam2, ws, ws.numel()) == 0
    assert E.ecokv_select(p, S, idx_sel) == 0
    torch.cuda.synchronize()
    assert E.ecokv_device_status(ws) == 0
    for k, gk in g.items():
        gk.check(f"{w.name} {k}")
    # fused entry == split entries, bit for bit
    assert torch.equal(S, S2) and torch.equal(lam, lam2) and torch.equal(idx, idx_sel)
    op = oracle_params(p)
    units = units or [(l, h) for l in range(nl) for h in range(w.h_kv)]
    ref = O.evict(K, V, Q, op, heads=units)
    tol = TOL[w.dtype]
    S_np, D_np = S.cpu().double().numpy(), dbg.cpu().double().numpy()
    worst = 0.0
    for (l, h) in units:
        r = ref[(l, h)]
        what = f"{w.name} unit ({l},{h})"
        worst = max(worst, check_scores(S_np[l, h], r, tol, what))
        assert abs(float(lam[l, h]) - r["lam"]) <= tol, what
        if p.n > p.window:
            assert score_error(D_np[l, h, 1], r["s_imp"]) <= tol, what + " S_imp"
            assert score_error(D_np[l, h, 2], r["d_e"]) <= tol, what + " d_E"
            assert np.abs(D_np[l, h, 3] - r["c"]).max() <= tol, what + " cosine"
            assert score_error(D_np[l, h, 4], r["s_div"]) <= tol, what + " S_div"
        # select is exact given the same fp32 scores
        exact = O.select(S_np[l, h], op)
        assert (idx_sel[l, h].cpu().numpy() == exact).all(), what + " select"
        check_selection(idx[l, h].cpu().numpy(), r, op, tol, what)
        check_rows(Kd[l, h], idx[l, h], Ko[l, h], what)
        check_rows(Vd[l, h], idx[l, h], Vo[l, h], what)
    return worst


SMALL = [
    dict(n=1000, h_kv=2, group=1, window=8, budget=100, pool_kernel=7, dtype="f32"),
    dict(n=1000, h_kv=2, group=4, window=4, budget=100, pool_kernel=5, dtype="bf16", clustered=True),
    dict(n=129, h_kv=1, group=2, window=1, budget=17, pool_kernel=1, dtype="f32"),
    dict(n=127, h_kv=3, group=1, window=3, budget=30, pool_kernel=3, dtype="bf16"),
    dict(n=600, h_kv=1, group=8, window=32, budget=120, pool_kernel=5, dtype="bf16"),   # g*W = 256
    dict(n=600, h_kv=1, group=8, window=32, budget=120, pool_kernel=5, dtype="f32"),
    dict(n=300, h_kv=2, group=2, window=5, budget=5, pool_kernel=5, dtype="f32"),       # B == W
    dict(n=200, h_kv=2, group=1, window=4, budget=250, pool_kernel=5, dtype="bf16"),    # B >= N
    dict(n=8, h_kv=2, group=1, window=8, budget=8, pool_kernel=5, dtype="f32"),         # N == W
    dict(n=1, h_kv=1, group=1, window=1, budget=1, pool_kernel=1, dtype="f32"),         # N == 1
    dict(n=2, h_kv=1, group=3, window=1, budget=1, pool_kernel=3, dtype="bf16"),
    dict(n=5000, h_kv=2, group=7, window=8, budget=500, pool_kernel=5, dtype="bf16", n_layers=2,
         clustered=True),
    # more window rows than one launch of the tensor-core kernel holds (120):
    # g W = 224 in two row groups of 112, g W = 240 in two of 120
    dict(n=3000, h_kv=2, group=7, window=32, budget=300, pool_kernel=5, dtype="bf16", clustered=True),
    dict(n=1500, h_kv=1, group=8, window=30, budget=200, pool_kernel=5, dtype="bf16"),
]


@pytest.mark.parametrize("path", ["auto", "simt"])
@pytest.mark.parametrize("case", SMALL, ids=lambda c: f"n{c['n']}_g{c['group']}_w{c['window']}_b{c['budget']}_{c['dtype']}")
def test_small_shapes(case, path):
    # "auto" takes the tensor-core kernel for bf16 shapes it covers, "simt"
    # forces the CUDA-core passes; both must match the oracle.
    if path == "simt" and case["dtype"] == "f32":
        pytest.skip("fp32 always runs the CUDA-core passes")
    run_and_compare(small_workload(seed=11, **case), flags=E.ECOKV_FLAG_FORCE_SIMT if path == "simt" else 0)


# Streaming schedules of the tensor-core kernel: waves of one head to all of
# them, lags from one wave to all of pass 1 first.
SCHEDULES = [(1, 1), (1, 3), (2, 1), (5, 1), (3, 2), (6, 1)]


@pytest.mark.parametrize("wave,lag", SCHEDULES, ids=lambda v: str(v))
def test_streaming_schedules(wave, lag):
    w = small_workload(5000, h_kv=2, group=7, window=8, budget=500, pool_kernel=5, dtype="bf16", n_layers=3,
                       clustered=True)
    run_and_compare(w, sched_wave=wave, sched_lag=lag)


def test_streaming_schedule_row_groups():
    """Two window-row groups (g W = 128) with waves of one head: each group's
    pass 2 adds its vote to the earlier group's."""
    w = small_workload(3000, h_kv=2, group=8, window=16, budget=300, pool_kernel=5, dtype="bf16", n_layers=2,
                       clustered=True)
    run_and_compare(w, sched_wave=1, sched_lag=1)


def test_streaming_schedule_many_units():
    """Sixty heads of 1000 keys (8 tiles): slices that span several heads and
    heads split over several slices."""
    w = small_workload(1000, h_kv=4, group=2, window=4, budget=100, pool_kernel=5, dtype="bf16", n_layers=15)
    run_and_compare(w, units=[(0, 0), (3, 1), (7, 2), (14, 3)])


@pytest.mark.parametrize("flags,extra", [
    (O.FLAG_SC_MIXKV_SIGN, dict(alpha=0.0, beta=0.0)),          # MixKV special case
    (O.FLAG_LAMBDA_OVERRIDE, dict(lambda_override=0.0)),         # SnapKV importance only
    (0, dict(alpha=1.0, beta=1.0, tau=3.0)),
])
def test_variants(flags, extra):
    w = small_workload(n=777, h_kv=2, group=2, window=4, budget=64, dtype="f32", seed=5, clustered=True)
    run_and_compare(w, flags=flags, **extra)


def test_config_c0_full():
    run_and_compare(CONFIGS["c0"])


@pytest.mark.parametrize("key", ["c1_b10", "c1_b20"])
def test_config_c1_two_layers(key):
    run_and_compare(CONFIGS[key], layers=range(0, 2))


def test_config_c1_simt_path():
    run_and_compare(CONFIGS["c1_b10"], layers=range(0, 1), flags=E.ECOKV_FLAG_FORCE_SIMT)


def test_config_c2_two_layers():
    run_and_compare(CONFIGS["c2"], layers=range(5, 7))


@pytest.mark.parametrize("pool_kernel", [5, 7, 41])
def test_wide_cluster_ragged(pool_kernel):
    # 20000 candidates: three CTAs of 8192 in a cluster, the last one ragged;
    # kernel 41 pools from global memory instead of the shared halo
    w = small_workload(n=20000, h_kv=2, group=4, window=8, budget=2000, pool_kernel=pool_kernel, dtype="bf16",
                       clustered=True, seed=pool_kernel)
    run_and_compare(w)


# (32768, 8): the finalize takes clusters of four CTAs of 8192 candidates;
# (65536, 4): clusters of eight such CTAs
@pytest.mark.parametrize("n,window", [(1024, 1), (4096, 32), (16384, 4), (32768, 8), (65536, 4)])
def test_sweep_points(n, window):
    run_and_compare(sweep_workload(n, window))


def test_sweep_largest_point_sampled_heads():
    # the sweep's longest layer (131072 tokens, W = 16: g W = 64 rows on the
    # tensor cores; 131056 candidates, clusters of sixteen CTAs), every head
    # scored in one call, two heads against the oracle
    run_and_compare(sweep_workload(131072, 16), units=[(0, 0), (0, 5)])


def test_identical_keys_all_ties():
    # Every key equal: d_E = 0 and r_E = r_C = 1, so lambda = 1 and S_div is
    # constant; Sbar vanishes and S = 0 for every candidate in exact
    # arithmetic, so the relative score criterion has no scale here.  The
    # oracle (fp64) lands at |S| ~ 1e-18; the CUDA path must keep lambda and S
    # within the bf16 tolerance of that answer on the natural scale of the
    # scores (the pooled importance), and select exactly on its own scores.
    w = small_workload(n=400, h_kv=1, group=2, window=4, budget=40, dtype="bf16")
    K, V, Q = make_inputs(w)
    K[:] = K[:, :, :1]
    for flags in (0, E.ECOKV_FLAG_FORCE_SIMT):
        p = params_of(w, flags=flags)
        Kd, Vd, Qd = K.to(DEV), V.to(DEV), Q.to(DEV)
        S_g, lam_g, dbg = E.score(p, Kd, Qd, dbg=True)
        idx, Ko, Vo, S, lam = E.evict(p, Kd, Vd, Qd, want_scores=True)
        ref = O.evict(K, V, Q, oracle_params(p))[(0, 0)]
        imp_scale = ref["s_imp"].mean()
        tol = TOL["bf16"]
        assert abs(float(lam[0, 0]) - 1.0) <= tol and abs(ref["lam"] - 1.0) <= 1e-12
        assert np.abs(S[0, 0].cpu().double().numpy()).max() <= tol * imp_scale
        assert np.abs(ref["S"]).max() <= 1e-12 * imp_scale
        assert score_error(dbg[0, 0, 1].cpu().double().numpy(), ref["s_imp"]) <= tol
        assert np.abs(dbg[0, 0, 2].cpu().double().numpy()).max() <= tol * np.sqrt(128.0)  # d_E ~ 0
        S_np = S[0, 0].cpu().double().numpy()
        assert (idx[0, 0].cpu().numpy() == O.select(S_np, oracle_params(p))).all()
        if (S_np == 0).all():
            assert list(idx[0, 0].cpu().numpy()) == list(range(36)) + [396, 397, 398, 399]
        check_rows(Kd[0, 0], idx[0, 0], Ko[0, 0])


@pytest.mark.parametrize("n,window,budget", [(5000, 4, 300), (300, 1, 299), (20000, 8, 2000), (32768, 4, 30000),
                                             (70000, 8, 7000)])
def test_select_exact_on_crafted_scores(n, window, budget):
    # ties, negatives, +-0: radix select must equal (S desc, position asc)
    g = torch.Generator().manual_seed(n)
    tv = n - window
    S = (torch.randint(-6, 7, (2, 3, tv), generator=g).float() / 4)
    S[0, 0, ::7] = -0.0
    S[1, 2] = 1.5                                     # one head all ties
    p = E.make_params(n_layers=2, h_kv=3, h_q=3, n=n, window=window, budget=budget)
    idx = E.select(p, S.to(DEV)).cpu().numpy()
    op = oracle_params(p)
    for l in range(2):
        for h in range(3):
            assert (idx[l, h] == O.select(S[l, h].double().numpy(), op)).all()


def test_compact_reports_bad_index():
    w = small_workload(n=300, h_kv=2, group=1, window=4, budget=40, dtype="bf16")
    K, V, Q = make_inputs(w)
    p = params_of(w)
    Kd, Vd = K.to(DEV), V.to(DEV)
    idx = torch.arange(40, dtype=torch.int32, device=DEV).repeat(1, 2, 1).contiguous()
    idx[0, 1, 7] = 300                                   # out of range: zero row + status
    ws = E.alloc_workspace(p, DEV)
    Ko, Vo = E.compact(p, Kd, Vd, idx, ws=ws)
    assert E.ecokv_device_status(ws) == 6
    assert E.ecokv_device_status(ws) == 0              # cleared by the read
    assert torch.count_nonzero(Ko[0, 1, 7]) == 0 and torch.count_nonzero(Vo[0, 1, 7]) == 0
    good = idx[0, 0].long()
    assert torch.equal(Ko[0, 0], Kd[0, 0][good])


@pytest.mark.parametrize("key,units", [
    ("c3_b10", [(0, 0), (13, 2), (27, 3)]),      # as the benchmark launches it
    ("c3_b5", [(5, 1), (27, 0)]),
    ("c3_b20", [(0, 3), (20, 2)]),
    ("c2", [(0, 0), (17, 3), (27, 1)]),
    ("c1_b10", [(0, 0), (16, 31), (31, 7)]),
])
def test_full_size_sampled_units(key, units):
    # every layer and head of the configuration in one call, at full size;
    # sampled heads against the oracle
    w = workload(key)
    K, V, Q = make_inputs(w, device=DEV)
    p = params_of(w)
    ws = E.alloc_workspace(p, DEV)
    idx, Ko, Vo, S, lam = E.evict(p, K, V, Q, ws=ws, want_scores=True)
    torch.cuda.synchronize()
    assert E.ecokv_device_status(ws) == 0
    tol = TOL[w.dtype]
    for (l, h) in units:
        Kh = K[l:l + 1, h:h + 1].cpu()
        Qh = Q[l:l + 1, h * w.group:(h + 1) * w.group].cpu()
        r = O.evict(Kh, Kh, Qh, oracle_params(p, n_layers=1, h_kv=1, h_q=w.group))[(0, 0)]
        what = f"{key} unit ({l},{h})"
        check_scores(S[l, h].cpu().double().numpy(), r, tol, what)
        check_selection(idx[l, h].cpu().numpy(), r, oracle_params(p, n_layers=1, h_kv=1, h_q=w.group), tol, what)
        check_rows(K[l, h], idx[l, h], Ko[l, h], what)
        check_rows(V[l, h], idx[l, h], Vo[l, h], what)


# the non-window centroid (reading R19): both streaming paths against the oracle
@pytest.mark.parametrize("w,flags", [
    (small_workload(5000, h_kv=2, group=4, window=8, budget=500, dtype="bf16", n_layers=2, clustered=True), 0),
    (small_workload(5000, h_kv=2, group=4, window=8, budget=500, dtype="bf16", clustered=True),
     E.ECOKV_FLAG_FORCE_SIMT),
    (small_workload(3001, h_kv=2, group=1, window=8, budget=300, pool_kernel=7, dtype="f32"), 0),
], ids=["bf16_tc", "bf16_simt", "f32_simt"])
def test_non_window_centroid(w, flags):
    run_and_compare(w, flags=flags | E.ECOKV_FLAG_CENTROID_NONWIN)


def test_non_window_centroid_c2_two_layers():
    run_and_compare(CONFIGS["c2"], layers=range(3, 5), flags=E.ECOKV_FLAG_CENTROID_NONWIN)


# winsorised min-max of Eq. 2 (reading R20): both streaming paths and both
# clip levels against the oracle (scores, lambda, the per-token terms,
# selection, rows)
@pytest.mark.parametrize("w,flags", [
    (small_workload(5000, h_kv=2, group=4, window=8, budget=500, dtype="bf16", n_layers=2, clustered=True),
     E.ECOKV_FLAG_WINSOR_5),
    (small_workload(20000, h_kv=2, group=4, window=8, budget=2000, dtype="bf16", clustered=True),
     E.ECOKV_FLAG_WINSOR_1),
    (small_workload(3001, h_kv=2, group=1, window=8, budget=300, pool_kernel=7, dtype="f32"),
     E.ECOKV_FLAG_WINSOR_1),
], ids=["bf16_tc_5pct", "bf16_wide_1pct", "f32_simt_1pct"])
def test_winsorised_minmax(w, flags):
    run_and_compare(w, flags=flags)


def test_winsorised_minmax_c2_two_layers():
    run_and_compare(CONFIGS["c2"], layers=range(10, 12), flags=E.ECOKV_FLAG_WINSOR_5)


# MAD scaling of Eq. 2 (reading R21): both streaming paths, an odd and an even
# candidate count, against the oracle (scores, lambda, the per-token terms,
# selection, rows)
@pytest.mark.parametrize("w,flags", [
    (small_workload(5000, h_kv=2, group=4, window=8, budget=500, dtype="bf16", n_layers=2, clustered=True), 0),
    (small_workload(20001, h_kv=2, group=4, window=8, budget=2000, dtype="bf16", clustered=True), 0),
    (small_workload(5000, h_kv=2, group=4, window=8, budget=500, dtype="bf16", clustered=True),
     E.ECOKV_FLAG_FORCE_SIMT),
    (small_workload(3001, h_kv=2, group=1, window=8, budget=300, pool_kernel=7, dtype="f32"), 0),
], ids=["bf16_tc_even", "bf16_wide_odd", "bf16_simt", "f32_simt_odd"])
def test_mad_scaling(w, flags):
    run_and_compare(w, flags=flags | E.ECOKV_FLAG_MAD)


def test_mad_scaling_c2_two_layers():
    run_and_compare(CONFIGS["c2"], layers=range(6, 8), flags=E.ECOKV_FLAG_MAD)


# the order statistics behind the robust forms of Eq. 2 are exact: S_div
# recomputed in double from the GPU's own d_E and cosines, with numpy's order
# statistics of those single-precision distances (the median and MAD formed
# in single precision, as the kernels form them), agrees to rounding; a rank
# off by one moves s_E by ~1e-4
@pytest.mark.parametrize("flags", [E.ECOKV_FLAG_WINSOR_5, E.ECOKV_FLAG_WINSOR_1, E.ECOKV_FLAG_MAD],
                         ids=["winsor5", "winsor1", "mad"])
@pytest.mark.parametrize("n", [5000, 20001, 32768, 40000, 131072])
def test_robust_order_statistics_exact(flags, n):
    # past 32768 candidates the rows are read from L2 until the keys under the
    # ranks' prefixes fit the shared-memory slots
    w = small_workload(n, h_kv=2, group=4, window=8, budget=n // 10, dtype="bf16", clustered=True, seed=3)
    K, V, Q = make_inputs(w)
    p = params_of(w, flags=flags)
    ws = E.alloc_workspace(p, DEV)
    _, _, dbg = E.score(p, K.to(DEV), Q.to(DEV), ws=ws, dbg=True)
    torch.cuda.synchronize()
    assert E.ecokv_device_status(ws) == 0
    dbg = dbg.cpu().numpy()
    for h in range(w.h_kv):
        dE = dbg[0, h, 2].astype(np.float32)
        c = dbg[0, h, 3].astype(np.float64)
        T = dE.size
        srt = np.sort(dE)
        if flags & E.ECOKV_FLAG_MAD:
            half = np.float32(0.5)
            med = half * (srt[(T - 1) // 2] + srt[T // 2])
            dev = np.sort(np.abs(dE - med))
            mad = half * (dev[(T - 1) // 2] + dev[T // 2])
            sE = 1.0 / (1.0 + np.exp(-(dE.astype(np.float64) - float(med)) / (float(mad) + float(p.eps))))
        else:
            q = 0.01 if flags & E.ECOKV_FLAG_WINSOR_1 else 0.05
            lo, hi = float(srt[int(np.floor(q * (T - 1)))]), float(srt[int(np.ceil((1 - q) * (T - 1)))])
            sE = (np.clip(dE.astype(np.float64), lo, hi) - lo) / (hi - lo + float(p.eps))
        sdiv = float(p.alpha) * sE + (1.0 - float(p.alpha)) * (1.0 - c) / 2.0
        err = np.abs(dbg[0, h, 4].astype(np.float64) - sdiv).max()
        assert err <= 2e-6, f"n={n} head {h}: S_div differs by {err:.2e} from the exact order statistics"
