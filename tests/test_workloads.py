"""Seeded synthetic workloads: shapes, determinism, layouts, budgets."""
import torch

from paper_2609_06663_gb300.workloads import (CONFIGS, budget_fraction, make_inputs, small_workload,
                                              sweep_workload, _seg_len)


def test_budget_rounding_half_up():
    assert budget_fraction(2048, 0.10) == 205 and budget_fraction(2048, 0.20) == 410
    assert [budget_fraction(32768, f) for f in (0.05, 0.10, 0.20)] == [1638, 3277, 6554]


def test_layouts_cover_n():
    for w in CONFIGS.values():
        assert sum(_seg_len(s) for s in w.layout) == w.n
        assert w.h_q % w.h_kv == 0 and w.window <= w.budget
    for n in (1 << 10, 1 << 14, 1 << 17):
        w = sweep_workload(n, 4)
        assert sum(_seg_len(s) for s in w.layout) == n
        assert w.budget == budget_fraction(n, 0.1)


def test_shapes_dtypes_and_determinism():
    w = small_workload(n=300, h_kv=2, group=3, window=5, budget=40, dtype="bf16", clustered=True)
    K, V, Q = make_inputs(w)
    assert K.shape == (1, 2, 300, 128) and V.shape == K.shape and Q.shape == (1, 6, 5, 128)
    assert K.dtype == torch.bfloat16
    K2, V2, Q2 = make_inputs(w)
    assert torch.equal(K, K2) and torch.equal(V, V2) and torch.equal(Q, Q2)


def test_layer_subset_matches_full_draw():
    w = CONFIGS["c2"]
    w = type(w)(**{**{f: getattr(w, f) for f in w.__dataclass_fields__}, "n_layers": 3})
    K, V, Q = make_inputs(w)
    K1, V1, Q1 = make_inputs(w, layers=range(2, 3))
    assert torch.equal(K[2:3], K1) and torch.equal(Q[2:3], Q1)


def test_anisotropy_and_clusters():
    # text keys share a mean direction of norm 4 under N(0, I_128) noise: the
    # expected pairwise cosine is 16 / (16 + 128) = 0.111; cluster members are
    # near-duplicates (spread 0.1 per coordinate)
    w = small_workload(n=400, h_kv=1, window=4, budget=40, dtype="f32", clustered=True)
    K, _, _ = make_inputs(w)
    k = K[0, 0].double()
    kn = k / k.norm(dim=1, keepdim=True)
    mean_cos = (kn.sum(0).norm() ** 2 - 400) / (400 * 399)
    assert 0.08 < mean_cos < 0.15
    c0 = k[133:149]                      # first 16-token cluster after 133 text tokens
    assert (c0 - c0.mean(0)).norm(dim=1).max() < 0.1 * 128 ** 0.5 * 2
