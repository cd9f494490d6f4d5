"""Pins for the fp64 oracle: each check ties an oracle function to something
other than itself - a closed form, a special case that reduces to a library
routine, brute force on a tiny input, or an invariant the paper states - and
is chosen so that a plausible slip (dropped 1/sqrt(d), wrong causal mask,
centroid over the wrong set, flipped cosine sign, swapped alpha/beta, wrong
pooling divisor, wrong GQA mapping, wrong tie order) fails at least one.
"""
import math

import numpy as np
import pytest
import scipy.special

from oracle import ecokv_oracle as O


def rng(seed=0):
    return np.random.default_rng(seed)


def params(n, d, window, budget, h_kv=1, h_q=1, pool=1, **kw):
    return O.Params(n_layers=1, h_kv=h_kv, h_q=h_q, n=n, d=d, window=window, budget=budget,
                    pool_kernel=pool, **kw)


def aniso(r, n, d, scale=4.0):
    u = r.standard_normal(d)
    u /= np.linalg.norm(u)
    s = np.exp(0.5 * r.standard_normal(n))
    return s[:, None] * (scale * u[None, :] + r.standard_normal((n, d))), u


# ---------------------------------------------------------------- attention
def test_softmax_rows_sum_to_one_and_total_mass():
    r = rng(1)
    n, d, w, g = 40, 16, 5, 3
    K, u = aniso(r, n, d)
    Q = 4 * u + r.standard_normal((g, w, d))
    p = O.window_softmax(O.window_logits(K, Q))
    np.testing.assert_allclose(p.sum(-1), 1.0, rtol=0, atol=1e-14)
    # every window row puts mass 1 on visible keys: candidates + window = g*W
    raw = O.importance_raw(p, n - w)
    win_mass = p[:, :, n - w:].sum()
    assert abs(raw.sum() + win_mass - g * w) < 1e-12


def test_single_row_importance_is_textbook_softmax():
    # W = 1, g = 1, no pooling: S_imp is one softmax row restricted to T_v.
    r = rng(2)
    n, d = 33, 128
    K, u = aniso(r, n, d)
    q = 4 * u + r.standard_normal(d)
    pr = params(n, d, window=1, budget=8)
    out = O.score_head(K, q[None, None, :], pr)
    ref = scipy.special.softmax(K @ q / math.sqrt(d))[: n - 1]
    np.testing.assert_allclose(out["s_imp"], ref, rtol=1e-13, atol=0)
    np.testing.assert_allclose(out["s_imp_raw"], ref, rtol=1e-13, atol=0)


def test_causal_window_rows_by_slicing():
    # Window row j (position N-W+j) sees keys 0..N-W+j: recompute each row as a
    # library softmax over a slice, instead of a mask.
    r = rng(3)
    n, d, w, g = 29, 8, 3, 2
    K, u = aniso(r, n, d)
    Q = 4 * u + r.standard_normal((g, w, d))
    pr = params(n, d, window=w, budget=10, h_q=g)
    out = O.score_head(K, Q, pr)
    ref = np.zeros(n - w)
    for q in range(g):
        for j in range(w):
            vis = n - w + j + 1
            row = scipy.special.softmax(K[:vis] @ Q[q, j] / math.sqrt(d))
            ref += row[: n - w]
    np.testing.assert_allclose(out["s_imp_raw"], ref, rtol=1e-13)


def test_two_key_closed_form_scale():
    # d = 4 (sqrt(d) = 2), q = e1, k0 = 2 ln2 e1, k1 = k2 = 0, W = 1:
    # logits (ln 2, 0, 0) -> softmax (1/2, 1/4, 1/4).  Without the 1/sqrt(d)
    # scale the first probability would be 4/6.
    d = 4
    K = np.zeros((3, d))
    K[0, 0] = 2 * math.log(2.0)
    q = np.zeros((1, 1, d))
    q[0, 0, 0] = 1.0
    out = O.score_head(K, q, params(3, d, window=1, budget=2))
    np.testing.assert_allclose(out["s_imp_raw"], [0.5, 0.25], rtol=0, atol=1e-15)


def test_gqa_group_mapping():
    # KV head h gathers query heads h*g .. h*g+g-1 (consecutive grouping).
    r = rng(4)
    n, d, w, hkv, g = 24, 16, 2, 2, 3
    K = np.stack([aniso(r, n, d)[0] for _ in range(hkv)])[None]
    V = r.standard_normal(K.shape)
    Q = r.standard_normal((1, hkv * g, w, d))
    pr = params(n, d, window=w, budget=8, h_kv=hkv, h_q=hkv * g)
    res = O.evict(K, V, Q, pr)
    for h in range(hkv):
        acc = np.zeros(n - w)
        for q in range(h * g, h * g + g):
            one = params(n, d, window=w, budget=8)
            acc += O.score_head(K[0, h], Q[0, q:q + 1], one)["s_imp_raw"]
        np.testing.assert_allclose(res[(0, h)]["s_imp_raw"], acc, rtol=1e-13)


@pytest.mark.parametrize("t,k", [(1, 1), (3, 5), (4, 5), (10, 5), (17, 7), (6, 3), (9, 1)])
def test_avg_pool_matches_convolution(t, k):
    x = rng(t * 10 + k).random(t)
    full = np.convolve(x, np.ones(k) / k, mode="full")       # length t + k - 1
    ref = full[(k - 1) // 2:(k - 1) // 2 + t]                 # centred window
    np.testing.assert_allclose(O.avg_pool(x, k), ref, rtol=1e-14, atol=1e-16)


# ---------------------------------------------------------------- Euclidean
def test_centroid_includes_window_keys():
    # keys: N-1 copies of x, then one window key y.  kbar = ((N-1)x + y)/N, so
    # every candidate sits at distance ||y - x|| / N from it (0 if the centroid
    # were taken over the candidates only).
    r = rng(5)
    n, d = 16, 8
    x, y = r.standard_normal(d), r.standard_normal(d)
    K = np.vstack([np.tile(x, (n - 1, 1)), y])
    out = O.score_head(K, r.standard_normal((1, 1, d)), params(n, d, window=1, budget=4))
    gap = np.linalg.norm(y - x)
    np.testing.assert_allclose(out["d_e"], gap / n, rtol=1e-12)
    # Eq. 4 averages over all T keys: N-1 candidates at gap/N and the window
    # key at (N-1) gap/N give D_E = 2 (N-1) gap / N^2 (gap/N over T_v only).
    assert abs(out["D_E"] - 2 * (n - 1) * gap / n ** 2) < 1e-12 * gap


def test_distance_nonneg_zero_for_identical_and_expansion_identity():
    r = rng(6)
    n, d = 20, 128
    K, _ = aniso(r, n, d)
    kbar = O.key_centroid(K)
    dE = O.euclid_distance(K, kbar)
    assert (dE >= 0).all()
    # ECD(a,b)^2 = |a|^2 + |b|^2 - 2|a||b| CosSim(a,b)  (Sec. 4)
    na, nb = np.linalg.norm(K, axis=1), np.linalg.norm(kbar)
    cos = (K @ kbar) / (na * nb)
    np.testing.assert_allclose(dE ** 2, na ** 2 + nb ** 2 - 2 * na * nb * cos, rtol=1e-10)
    # identical keys with few significant bits (as bf16 keys have): the mean is
    # exact, so the distance is exactly 0
    same = np.tile(np.round(K[0] * 64) / 64, (7, 1))
    np.testing.assert_array_equal(O.euclid_distance(same, O.key_centroid(same)), 0.0)


def test_euclid_redundancy_closed_forms():
    d = 64
    # D_E = 0 -> sigma(0) = 1/2 -> r_E = 1
    K = np.tile(np.round(rng(7).standard_normal(d) * 64) / 64, (6, 1))
    out = O.score_head(K, np.ones((1, 1, d)), params(6, d, window=1, budget=3))
    assert out["D_E"] == 0.0 and out["r_E"] == 1.0
    # keys +-a e1 alternate: kbar = 0, every d_E = a.  With a = sqrt(d) ln 3:
    # sigma(ln 3) = 3/4 -> r_E = 1/2.
    a = math.sqrt(d) * math.log(3.0)
    K = np.zeros((8, d))
    K[0::2, 0], K[1::2, 0] = a, -a
    out = O.score_head(K, np.ones((1, 1, d)), params(8, d, window=2, budget=4))
    assert abs(out["D_E"] - a) < 1e-12
    assert abs(out["r_E"] - 0.5) < 1e-12
    # monotone decreasing in the spread, within (0, 1]
    vals = [O.euclid_redundancy(x, 8.0) for x in (0.0, 1.0, 5.0, 50.0)]
    assert vals[0] == 1.0 and all(a > b for a, b in zip(vals, vals[1:])) and vals[-1] > 0


def test_mean_distance_below_rms_distance():
    # Appendix C's standard-deviation alternative: D_std = sqrt(mean ||k_i -
    # kbar||^2), here by the variance identity sqrt(mean ||k||^2 - ||kbar||^2);
    # Jensen gives D_E <= D_std, with equality when every key is equally far
    # from the centroid
    r = rng(30)
    n, d = 40, 16
    K, _ = aniso(r, n, d)
    out = O.score_head(K, r.standard_normal((1, 2, d)), params(n, d, window=2, budget=10))
    kbar = K.mean(axis=0)
    d_std = math.sqrt((K * K).sum(axis=1).mean() - kbar @ kbar)
    assert out["D_E"] < d_std * (1 - 1e-3)                  # spread distances: strict
    # keys on a sphere about their centroid (pairs +-v_i): every distance equal
    V = r.standard_normal((n // 2, d))
    V *= 3.0 / np.linalg.norm(V, axis=1, keepdims=True)
    S2 = np.vstack([V, -V]) + 5.0
    out2 = O.score_head(S2, r.standard_normal((1, 2, d)), params(n, d, window=2, budget=10))
    c2 = S2.mean(axis=0)
    d_std2 = math.sqrt((S2 * S2).sum(axis=1).mean() - c2 @ c2)
    assert out2["D_E"] == pytest.approx(3.0, rel=1e-12) and d_std2 == pytest.approx(3.0, rel=1e-10)


def test_minmax_range_and_order():
    x = rng(8).random(50) * 7 - 3
    s = O.minmax(x, 1e-6)
    assert s.min() == 0.0 and s.max() < 1.0 and s.max() > 0.999
    assert (np.argsort(s, kind="stable") == np.argsort(x, kind="stable")).all()


# ---------------------------------------------------------------- cosine
def test_cosine_redundancy_is_mean_pairwise_cosine():
    # Closed form (T ||mu||^2 - 1)/(T - 1) == brute-force off-diagonal mean.
    r = rng(9)
    for n in (2, 3, 11):
        K, _ = aniso(r, n, 16, scale=1.5)
        KN = O.normalized_keys(K)
        mu = KN.mean(0)
        brute, cnt = 0.0, 0
        for i in range(n):
            for j in range(n):
                if i != j:
                    brute += float(KN[i] @ KN[j])
                    cnt += 1
        assert abs(O.cosine_redundancy(mu, n) - brute / cnt) < 1e-13


def test_cosine_sign_and_range():
    # keys (-e1, e1, e1, e1), W = 1: mu = e1/2, cosines (-1/2, 1/2, 1/2).
    # The anti-aligned key is the diverse one: s_C = (3/4, 1/4, 1/4).
    d = 8
    K = np.zeros((4, d))
    K[:, 0] = [-1, 1, 1, 1]
    K *= np.array([3.0, 1.0, 2.0, 5.0])[:, None]          # magnitudes do not matter
    pr = params(4, d, window=1, budget=2)
    out = O.score_head(K, np.ones((1, 1, d)), pr)
    np.testing.assert_allclose(out["c"], [-0.5, 0.5, 0.5], atol=1e-15)
    np.testing.assert_allclose(out["s_C"], [0.75, 0.25, 0.25], atol=1e-15)
    pr.flags = O.FLAG_SC_MIXKV_SIGN
    out = O.score_head(K, np.ones((1, 1, d)), pr)
    np.testing.assert_allclose(out["s_C"], [0.5, -0.5, -0.5], atol=1e-15)
    # general keys: |cos| <= 1 and r_C in [-1/(T-1), 1]
    r = rng(10)
    K, _ = aniso(r, 30, 16)
    out = O.score_head(K, np.ones((1, 1, 16)), params(30, 16, window=3, budget=8))
    assert np.abs(out["c"]).max() <= 1 + 1e-12
    assert -1 / 29 - 1e-12 <= out["r_C"] <= 1 + 1e-12


def test_zero_norm_key_has_zero_direction():
    d = 8
    K = np.zeros((5, d))
    K[1:, 1] = 2.0
    out = O.score_head(K, np.ones((1, 1, d)), params(5, d, window=1, budget=2))
    assert out["c"][0] == 0.0                      # khat of the zero key is 0
    np.testing.assert_allclose(out["mu"][1], 4 / 5)


# ---------------------------------------------------------------- combination
def test_alpha_weights_euclidean_term():
    # Positive per-key rescaling leaves directions (hence s_C) unchanged but
    # changes distances.  alpha = 0 -> S_div must not move; alpha = 1 -> it must.
    r = rng(11)
    n, d = 40, 32
    K, u = aniso(r, n, d)
    Q = (4 * u + r.standard_normal((1, 2, d)))
    K2 = K * np.exp(r.standard_normal(n))[:, None]
    for alpha, moves in ((0.0, False), (1.0, True)):
        pr = params(n, d, window=2, budget=10, alpha=alpha)
        a = O.score_head(K, Q, pr)["s_div"]
        b = O.score_head(K2, Q, pr)["s_div"]
        assert np.allclose(a, b, atol=1e-12) != moves


def test_beta_weights_euclidean_redundancy():
    # A global scale t changes D_E (so r_E) but not r_C.
    r = rng(12)
    n, d = 32, 16
    K, u = aniso(r, n, d)
    Q = 4 * u + r.standard_normal((1, 1, d))
    for beta, moves in ((0.0, False), (1.0, True)):
        pr = params(n, d, window=1, budget=6, beta=beta)
        la = O.score_head(K, Q, pr)["lam"]
        lb = O.score_head(3.0 * K, Q, pr)["lam"]
        assert (abs(la - lb) > 1e-6) == moves
    pr = params(n, d, window=1, budget=6)
    out = O.score_head(K, Q, pr)
    assert min(out["r_E"], out["r_C"]) - 1e-15 <= out["lam"] <= max(out["r_E"], out["r_C"]) + 1e-15


def test_rescale_matches_importance_mean_and_all_ties():
    r = rng(13)
    n, d = 64, 16
    K, u = aniso(r, n, d)
    Q = 4 * u + r.standard_normal((2, 4, d))
    out = O.score_head(K, Q, params(n, d, window=4, budget=16, h_q=2, pool=5))
    assert abs(out["s_tilde"].mean() - out["s_imp"].mean()) < 1e-15
    assert out["s_tilde"].min() == 0.0
    # identical keys: no diversity signal, S == (1 - lambda) S_imp and lambda = 1
    Ks = np.tile(np.round(K[0] * 64) / 64, (n, 1))
    out = O.score_head(Ks, Q, params(n, d, window=4, budget=16, h_q=2, pool=5))
    assert out["r_E"] == 1.0 and abs(out["r_C"] - 1.0) < 1e-12
    np.testing.assert_array_equal(out["s_tilde"], 0.0)


def test_collinear_keys_rank_by_distance():
    # Same direction, distinct norms: s_C is constant, so S_div follows d_E.
    r = rng(14)
    n, d = 25, 16
    u = r.standard_normal(d)
    K = np.outer(np.exp(r.standard_normal(n)), u)
    out = O.score_head(K, np.ones((1, 1, d)), params(n, d, window=1, budget=5))
    assert np.ptp(out["s_C"]) < 1e-12
    assert (np.argsort(out["s_div"], kind="stable") == np.argsort(out["d_e"], kind="stable")).all()


def test_lambda_zero_is_snapkv_selection():
    # lambda := 0 reduces the score to pooled window attention; the selection
    # must then equal SnapKV top-k built from library routines.
    r = rng(15)
    n, d, w, g, kp, B = 60, 16, 4, 2, 5, 20
    K, u = aniso(r, n, d)
    Q = 4 * u + r.standard_normal((g, w, d))
    pr = params(n, d, window=w, budget=B, h_q=g, pool=kp,
                flags=O.FLAG_LAMBDA_OVERRIDE, lambda_override=0.0)
    out = O.score_head(K, Q, pr)
    vote = np.zeros(n - w)
    for q in range(g):
        for j in range(w):
            vis = n - w + j + 1
            vote += scipy.special.softmax(K[:vis] @ Q[q, j] / math.sqrt(d))[: n - w]
    pooled = np.convolve(vote, np.ones(kp) / kp, mode="same")
    top = sorted(sorted(range(n - w), key=lambda i: (-pooled[i], i))[: B - w])
    assert list(O.select(out["S"], pr)) == top + list(range(n - w, n))


def test_mixkv_special_case():
    # alpha = beta = 0 gives MixKV's cosine-only diversity and lambda = r_C.
    r = rng(16)
    n, d = 50, 16
    K, u = aniso(r, n, d)
    Q = 4 * u + r.standard_normal((1, 2, d))
    pr = params(n, d, window=2, budget=12, alpha=0.0, beta=0.0, flags=O.FLAG_SC_MIXKV_SIGN)
    out = O.score_head(K, Q, pr)
    assert out["lam"] == out["r_C"]
    KN = K / np.linalg.norm(K, axis=1, keepdims=True)
    np.testing.assert_allclose(out["s_div"], -(KN[: n - 2] @ KN.mean(0)), rtol=1e-12)


# ---------------------------------------------------------------- selection
def test_select_brute_force_and_structure():
    r = rng(17)
    for trial in range(20):
        n = int(r.integers(3, 40))
        w = int(r.integers(1, n + 1))
        B = int(r.integers(w, n + 3))
        S = np.round(r.random(n - w) * 4) / 4          # many ties
        pr = params(n, 8, window=w, budget=B)
        idx = O.select(S, pr)
        assert len(idx) == min(B, n)
        if B >= n:
            assert list(idx) == list(range(n))
            continue
        k = B - w
        brute = sorted(sorted(range(n - w), key=lambda i: (-S[i], i))[:k])
        assert list(idx[:k]) == brute
        assert list(idx[k:]) == list(range(n - w, n))


def test_select_all_ties_takes_first_positions():
    pr = params(30, 8, window=3, budget=10)
    idx = O.select(np.full(27, 0.25), pr)
    assert list(idx) == list(range(7)) + [27, 28, 29]


def test_select_adaptive_one_head_is_per_head_select():
    # a layer of one head: the layer-wide budget is the head's budget
    r = rng(21)
    for trial in range(10):
        n = int(r.integers(5, 50))
        w = int(r.integers(1, n))
        B = int(r.integers(w, n + 2))
        S = np.round(r.random(n - w) * 8) / 8
        pr = params(n, 8, window=w, budget=B)
        got = O.select_adaptive([S], pr)
        assert len(got) == 1 and list(got[0]) == list(O.select(S, pr))


def test_select_adaptive_identical_heads_share_evenly():
    # heads with the same distinct scores: each keeps B - W of them, the same ones
    r = rng(22)
    n, w, B, h = 40, 4, 12, 3
    S = r.permutation(n - w).astype(float)
    pr = params(n, 8, window=w, budget=B, h_kv=h, h_q=h)
    got = O.select_adaptive([S, S.copy(), S.copy()], pr)
    for x in got:
        assert list(x) == list(O.select(S, pr))


def test_select_adaptive_threshold_invariant_and_structure():
    # brute force through the defining property, not through a sort: the
    # chosen set has H_kv (B - W) members, no unchosen score exceeds a chosen
    # one, and at equal scores the chosen ones come first in (head, position)
    r = rng(23)
    for trial in range(30):
        h = int(r.integers(1, 5))
        n = int(r.integers(4, 30))
        w = int(r.integers(1, n))
        B = int(r.integers(w, n + 2))
        S = [np.round(r.random(n - w) * 3) / 3 for _ in range(h)]   # many ties, across heads too
        pr = params(n, 8, window=w, budget=B, h_kv=h, h_q=h)
        got = O.select_adaptive(S, pr)
        assert len(got) == h
        if B >= n:
            assert all(list(x) == list(range(n)) for x in got)
            continue
        t_v = n - w
        for x in got:
            assert list(x[len(x) - w:]) == list(range(t_v, n))           # the window, last
            assert all(np.diff(x[:len(x) - w]) > 0)                      # ascending candidates
        chosen = {(hh, int(i)) for hh, x in enumerate(got) for i in x[:len(x) - w]}
        assert len(chosen) == h * (B - w)
        allc = [(hh, i) for hh in range(h) for i in range(t_v)]
        for (ha, ia) in chosen:
            for (hb, ib) in allc:
                if (hb, ib) in chosen:
                    continue
                sa, sb = S[ha][ia], S[hb][ib]
                assert sa > sb or (sa == sb and (ha, ia) < (hb, ib))


def test_evict_adaptive_layout():
    r = rng(24)
    n, d, w, B, h = 24, 8, 3, 8, 2
    K = r.standard_normal((1, h, n, d))
    V = r.standard_normal((1, h, n, d))
    Q = r.standard_normal((1, 2 * h, w, d))
    pr = O.Params(n_layers=1, h_kv=h, h_q=2 * h, n=n, d=d, window=w, budget=B, pool_kernel=3)
    res = O.evict_adaptive(K, V, Q, pr)[0]
    off = res["head_off"]
    assert off[0] == 0 and off[-1] == h * B and len(res["idx"]) == h * B
    for hh in range(h):
        seg = res["idx"][off[hh]:off[hh + 1]]
        assert np.array_equal(res["K_out"][off[hh]:off[hh + 1]], K[0, hh][seg])
        assert np.array_equal(res["V_out"][off[hh]:off[hh + 1]], V[0, hh][seg])
    lists = O.select_adaptive([res["heads"][hh]["S"] for hh in range(h)], pr)
    assert np.array_equal(np.concatenate(lists), res["idx"])


def test_value_norm_importance_scale_and_selection():
    # values of one common norm c: S_imp, the rescaled diversity and S all scale
    # by c (Eq. 7 is homogeneous in S_imp), so the selection is unchanged; a
    # value row of outsized norm lifts its candidate into the selection
    r = rng(25)
    n, d, w, B = 60, 16, 4, 14
    K, u = aniso(r, n, d)
    Qg = (4 * u + r.standard_normal((2, w, d)))[:, :, :]
    V = r.standard_normal((n, d))
    c = 2.5
    Vc = c * V / np.linalg.norm(V, axis=1, keepdims=True)
    base = params(n, d, window=w, budget=B, h_q=2, pool=3)
    vn = params(n, d, window=w, budget=B, h_q=2, pool=3, flags=O.FLAG_VNORM_IMP)
    r0 = O.score_head(K, Qg, base)
    r1 = O.score_head(K, Qg, vn, Vc)
    assert np.allclose(r1["s_imp"], c * r0["s_imp"], rtol=1e-12, atol=0)
    assert np.allclose(r1["S"], c * r0["S"], rtol=1e-11, atol=1e-15)
    assert np.array_equal(O.select(r1["S"], vn), O.select(r0["S"], base))
    assert np.allclose(O.value_norms(Vc), c)
    low = int(np.argmin(r0["S"]))
    Vb = Vc.copy()
    Vb[low] *= 1e6
    r2 = O.score_head(K, Qg, vn, Vb)
    assert low in set(O.select(r2["S"], vn))


@pytest.mark.parametrize("m,b_total,beta", [(28, 28 * 3277, 20.0), (32, 32 * 205, 20.0), (5, 500, 3.0),
                                             (2, 64, 1.5)])
def test_pyramid_schedule_closed_forms(m, b_total, beta):
    b = O.pyramid_budgets_real(m, b_total, beta)
    assert math.isclose(sum(b), b_total, rel_tol=1e-12)               # the total is kept
    assert math.isclose(b[-1], b_total / (beta * m), rel_tol=1e-12)   # the top layer
    assert math.isclose(b[0] + b[-1], 2 * b_total / m, rel_tol=1e-12)
    steps = np.diff(b)
    assert np.allclose(steps, steps[0], rtol=1e-9) and steps[0] <= 0  # linear, decreasing for beta >= 1


def test_pyramid_uniform_when_beta_is_one_and_integer_reading():
    assert O.pyramid_budgets_real(6, 600, 1.0) == pytest.approx([100.0] * 6)
    assert O.pyramid_budgets(6, 100, 1.0, 4) == [100] * 6
    got = O.pyramid_budgets(28, 3277, 20.0, 8)
    real = O.pyramid_budgets_real(28, 28 * 3277, 20.0)
    assert all(abs(g - r) <= 0.5 for g, r in zip(got, real))
    assert O.pyramid_budgets(4, 10, 100.0, 8)[-1] == 8                # raised to the window


def test_non_window_centroid_ignores_the_window_keys():
    # with the non-window centroid, moving the window keys leaves the
    # candidates' distances and s_E unchanged; with the default centroid they move
    r = rng(26)
    n, d, w = 50, 16, 6
    K, u = aniso(r, n, d)
    Qg = 4 * u + r.standard_normal((2, w, d))
    K2 = K.copy()
    K2[n - w:] += 7.0 * r.standard_normal((w, d))
    nonwin = params(n, d, window=w, budget=20, h_q=2, pool=3, flags=O.FLAG_CENTROID_NONWIN)
    a, b = O.score_head(K, Qg, nonwin), O.score_head(K2, Qg, nonwin)
    assert np.allclose(a["d_e"], b["d_e"], rtol=1e-12, atol=0) and np.allclose(a["s_E"], b["s_E"], rtol=1e-12)
    assert np.allclose(a["kbar"], K[:n - w].mean(axis=0), rtol=1e-12)
    base = params(n, d, window=w, budget=20, h_q=2, pool=3)
    c, e = O.score_head(K, Qg, base), O.score_head(K2, Qg, base)
    assert not np.allclose(c["d_e"], e["d_e"], rtol=1e-6)
    assert np.allclose(a["mu"], c["mu"]) and a["r_C"] == c["r_C"]        # the cosine terms keep all N


def test_winsorised_minmax_closed_forms_and_outlier_invariance():
    x = np.arange(100, dtype=float)                        # order statistics are the values
    assert np.allclose(O.winsor_minmax(x, 0.01, 1e-6), O.minmax(x, 1e-6))   # 1 %: ranks 0 and 99
    y = O.winsor_minmax(x, 0.05, 0.0)                      # 5 %: ranks floor(4.95) = 4, ceil(94.05) = 95
    assert (y[:5] == 0).all() and (y[95:] == 1).all()
    assert np.allclose(y[5:95], (x[5:95] - 4) / 91)
    r = rng(27)
    z = r.random(200)
    w = z.copy()
    w[17] = 1e9                                            # one extreme outlier
    a, b = O.winsor_minmax(z, 0.05, 1e-6), O.winsor_minmax(w, 0.05, 1e-6)
    keep = np.arange(200) != 17
    assert np.allclose(a[keep], b[keep], rtol=0, atol=0.02) and b[17] == pytest.approx(1.0, abs=1e-5)
    assert not np.allclose(O.minmax(z, 1e-6)[keep], O.minmax(w, 1e-6)[keep], atol=0.02)


def test_mad_scaling_closed_forms():
    # 0..100: median 50; the absolute deviations are 0 once and 1..50 twice,
    # so their median (the 51st smallest) is 25
    x = np.arange(101, dtype=float)
    s = O.mad_scale(x, 0.0)
    assert s[50] == 0.5
    assert s[75] == pytest.approx(0.7310585786300049, rel=1e-14)     # logistic(1)
    assert s[0] == pytest.approx(0.11920292202211755, rel=1e-14)     # logistic(-2)
    assert s[100] == pytest.approx(0.8807970779778823, rel=1e-14)    # logistic(2)
    # 0..99: median 49.5 (mean of the middle two); deviations 0.5 .. 49.5 twice
    # each, median (24.5 + 25.5) / 2 = 25
    y = np.arange(100, dtype=float)
    t = O.mad_scale(y, 0.0)
    assert t[62] == pytest.approx(0.6224593312018546, rel=1e-14)     # logistic(0.5)
    assert t[37] == pytest.approx(0.3775406687981454, rel=1e-14)     # logistic(-0.5)
    # eps enters the denominator
    assert O.mad_scale(x, 25.0)[100] == pytest.approx(0.7310585786300049, rel=1e-14)
    # the smallest heads: one candidate is its own median (s = 1/2); two have
    # their mean as median and half their gap as MAD (s = logistic(-1), logistic(1))
    assert O.mad_scale(np.array([7.25]), 1e-6).tolist() == [0.5]
    two = O.mad_scale(np.array([3.0, 11.0]), 0.0)
    assert two[0] == pytest.approx(0.2689414213699951, rel=1e-14) and two[1] == pytest.approx(0.7310585786300049, rel=1e-14)


def test_mad_scaling_invariances_and_outlier():
    r = rng(28)
    z = r.lognormal(0.0, 0.7, 301)
    s = O.mad_scale(z, 0.0)
    assert ((s > 0) & (s < 1)).all()
    assert (np.argsort(s, kind="stable") == np.argsort(z, kind="stable")).all()     # order kept
    assert np.allclose(O.mad_scale(3.5 * z + 11.0, 0.0), s, rtol=1e-12)          # affine invariant
    assert np.sum(s > 0.5) == np.sum(s < 0.5) == 150                              # median maps to 1/2
    assert O.mad_scale(np.full(9, 2.5), 1e-6).tolist() == [0.5] * 9               # MAD = 0
    w = z.copy()
    w[17] = 1e9
    b = O.mad_scale(w, 0.0)
    keep = np.arange(301) != 17
    assert np.allclose(b[keep], s[keep], atol=0.02) and b[17] == 1.0
    def std_scaled(v):                                     # a mean / std z-score is not robust to it
        return 1.0 / (1.0 + np.exp(-(v - v.mean()) / v.std()))
    assert not np.allclose(std_scaled(w)[keep], std_scaled(z)[keep], atol=0.02)


def test_mad_flag_replaces_the_minmax_of_eq2():
    # alpha = 1 and lambda = 1: S ranks the candidates by s_E; with the MAD
    # flag the candidate at the median distance has s_E = 1/2 exactly
    r = rng(29)
    n, d, w = 41, 16, 4                                    # 37 candidates
    K, u = aniso(r, n, d)
    Qg = 4 * u + r.standard_normal((1, w, d))
    pm = params(n, d, window=w, budget=12, pool=3, alpha=1.0, lambda_override=1.0,
                flags=O.FLAG_MAD | O.FLAG_LAMBDA_OVERRIDE)
    out = O.score_head(K, Qg, pm)
    mid = np.argsort(out["d_e"])[18]
    assert out["s_E"][mid] == 0.5
    assert (np.argsort(out["S"]) == np.argsort(out["d_e"])).all()
    plain = O.score_head(K, Qg, params(n, d, window=w, budget=12, pool=3, alpha=1.0, lambda_override=1.0,
                                       flags=O.FLAG_LAMBDA_OVERRIDE))
    assert plain["s_E"].min() == 0.0 and out["s_E"].min() > 0.0


def test_compact_rows():
    r = rng(18)
    X = r.standard_normal((12, 5))
    idx = np.array([0, 3, 4, 9, 11])
    out = O.compact(X, idx)
    for rr, i in enumerate(idx):
        for c in range(5):
            assert out[rr, c] == X[i, c]


def test_bf16_widening_is_exact():
    import torch
    x = torch.randn(1000).to(torch.bfloat16)
    bits = x.view(torch.int16).numpy().astype(np.uint16).astype(np.uint32) << 16
    ref = bits.view(np.float32).astype(np.float64)
    np.testing.assert_array_equal(O.to_f64(x), ref)


def test_degenerate_shapes():
    r = rng(19)
    d = 8
    # N == W: no candidates, the window is the whole retained set
    K = r.standard_normal((4, d))
    pr = params(4, d, window=4, budget=4)
    out = O.score_head(K, r.standard_normal((1, 4, d)), pr)
    assert out["S"].shape == (0,)
    assert list(O.select(out["S"], pr)) == [0, 1, 2, 3]
    # B == W: only the window survives
    K = r.standard_normal((10, d))
    pr = params(10, d, window=3, budget=3)
    out = O.score_head(K, r.standard_normal((1, 3, d)), pr)
    assert list(O.select(out["S"], pr)) == [7, 8, 9]
    # N == 1
    pr = params(1, d, window=1, budget=1)
    out = O.score_head(r.standard_normal((1, d)), r.standard_normal((1, 1, d)), pr)
    assert out["r_C"] == 1.0 and list(O.select(out["S"], pr)) == [0]


def test_oracle_regression_fixture():
    # Frozen oracle output (tests/golden/make_golden.py); guards against an
    # unannounced change of the oracle's arithmetic.
    import json
    import os
    import sys
    here = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
    sys.path.insert(0, here)
    import make_golden
    with open(os.path.join(here, "oracle_regression.json")) as f:
        gold = json.load(f)
    K, V, Q, p = make_golden.case()
    res = O.evict(K, V, Q, p)
    for key, g in gold["units"].items():
        l, h = map(int, key.split(","))
        r = res[(l, h)]
        assert list(r["idx"]) == g["idx"]
        for k in ("S", "lam", "r_E", "r_C", "D_E", "s_imp", "d_e", "c"):
            np.testing.assert_allclose(np.asarray(r[k]), np.asarray(g[k]), rtol=1e-12, atol=1e-15)
