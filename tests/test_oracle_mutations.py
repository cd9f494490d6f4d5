"""The oracle's pins are strong enough: each plausible slip below, planted in
the oracle (on the CPU, for the duration of one check), makes at least one pin
of tests/test_oracle_pins.py fail.  The regression fixture is left out: it was
written by the oracle itself, so it would catch every change and pin nothing.
"""
import inspect

import numpy as np
import pytest

from oracle import ecokv_oracle as O
from tests import test_oracle_pins as PINS

ORIG = {name: getattr(O, name) for name in dir(O) if callable(getattr(O, name))}


def _pins():
    out = []
    for name, fn in sorted(vars(PINS).items()):
        if not name.startswith("test_") or name == "test_oracle_regression_fixture":
            continue
        marks = getattr(fn, "pytestmark", [])
        args = [m.args for m in marks if m.name == "parametrize"]
        if args:
            names, values = args[0]
            for v in values:
                out.append((name, fn, dict(zip([s.strip() for s in names.split(",")], v))))
        else:
            assert not inspect.signature(fn).parameters, name
            out.append((name, fn, {}))
    return out


# ---- the planted slips -----------------------------------------------------
def no_scale(K, Qg):                      # 1/sqrt(d) dropped
    return ORIG["window_logits"](K, Qg) * np.sqrt(K.shape[1])


def no_causal_mask(K, Qg):                # every window row sees every key
    return np.einsum("qjd,id->qji", Qg, K) / np.sqrt(K.shape[1])


def average_not_sum(p, t_v):              # mean over rows and heads instead of the sum
    return p[:, :, :t_v].mean(axis=(0, 1))


def pool_counts_valid_only(x, kernel):    # zero padding not counted in the divisor
    t, half = x.shape[0], kernel // 2
    y, c = np.zeros(t), np.zeros(t)
    for o in range(-half, half + 1):
        lo, hi = max(0, -o), min(t, t - o)
        if lo < hi:
            y[lo:hi] += x[lo + o:hi + o]
            c[lo:hi] += 1
    return y / c


def pool_off_centre(x, kernel):           # window shifted by one
    return np.roll(ORIG["avg_pool"](x, kernel), 1)


def centroid_drops_last_key(K):           # centroid over the wrong set
    return K[:-1].mean(axis=0) if len(K) > 1 else K.mean(axis=0)


def distance_squared(K, kbar):            # ||.||^2 instead of ||.||
    diff = K - kbar[None, :]
    return (diff * diff).sum(axis=1)


def redundancy_sign(mean_dist, tau):      # sigma(.) instead of 2 - 2 sigma(.)
    return 1.0 / (1.0 + np.exp(-mean_dist / tau))


def cosine_similarity_not_diversity(c, flags):   # flipped sign
    return (1.0 + c) / 2.0


def r_c_drops_minus_one(mu, t):           # (T ||mu||^2) / (T - 1)
    return 1.0 if t == 1 else t * float(mu @ mu) / (t - 1.0)


def minmax_reversed(x, eps):              # distance read as similarity
    return 1.0 - ORIG["minmax"](x, eps)


def rescale_by_importance(s_div, s_imp, eps):    # divides by the wrong mean
    sbar = ORIG["minmax"](s_div, eps)
    return sbar * (sbar.mean() / max(s_imp.mean(), 1e-300))


def select_k_is_budget(S, p):             # the window not counted in B
    n, w = p.n, p.window
    if p.budget >= n:
        return np.arange(n, dtype=np.int64)
    k = min(p.budget, n - w)
    order = np.lexsort((np.arange(n - w), -S))
    return np.concatenate([np.sort(order[:k]), np.arange(n - w, n)]).astype(np.int64)


def select_ties_high_position(S, p):      # ties to the higher position
    n, w = p.n, p.window
    if p.budget >= n:
        return np.arange(n, dtype=np.int64)
    order = np.lexsort((-np.arange(n - w), -S))
    return np.concatenate([np.sort(order[:p.budget - w]), np.arange(n - w, n)]).astype(np.int64)


def adaptive_budget_counts_window(S_heads, p):   # layer budget H_kv B instead of H_kv (B - W)
    q = O.Params(**{**p.__dict__, "budget": min(p.budget + p.window, p.n)})
    return ORIG["select_adaptive"](S_heads, q) if p.budget < p.n else ORIG["select_adaptive"](S_heads, p)


def adaptive_ties_by_position(S_heads, p):       # ties across heads by position first
    n, w, t_v, h = p.n, p.window, p.t_v, len(S_heads)
    if p.budget >= n:
        return [np.arange(n, dtype=np.int64) for _ in range(h)]
    cat = np.concatenate(S_heads)
    pos = np.tile(np.arange(t_v), h)
    order = np.lexsort((np.repeat(np.arange(h), t_v), pos, -cat))
    chosen = np.zeros(cat.size, dtype=bool)
    chosen[order[:h * (p.budget - w)]] = True
    return [np.concatenate([np.nonzero(chosen[i * t_v:(i + 1) * t_v])[0], np.arange(t_v, n)]) for i in range(h)]


def adaptive_no_window(S_heads, p):       # the heads' windows left out
    return [x[x < p.t_v] if p.budget < p.n else x for x in ORIG["select_adaptive"](S_heads, p)]


def value_norm_squared(V):               # ||v||^2 instead of ||v||
    return (V * V).sum(axis=1)


def pyramid_top_without_m(m, b_total, beta):    # b^{m-1} = b_total / beta
    if m == 1:
        return [float(b_total)]
    b_last = b_total / beta
    b_first = 2.0 * b_total / m - b_last
    return [b_first - (b_first - b_last) / (m - 1) * l for l in range(m)]


def pyramid_step_over_m(m, b_total, beta):      # slope divided by m, not m - 1
    if m == 1:
        return [float(b_total)]
    b_last = b_total / (beta * m)
    b_first = 2.0 * b_total / m - b_last
    return [b_first - (b_first - b_last) / m * l for l in range(m)]


def winsor_interpolated(x, p, eps):        # percentiles interpolated instead of order statistics
    lo, hi = np.percentile(x, 100 * p), np.percentile(x, 100 * (1 - p))
    return (np.clip(x, lo, hi) - lo) / (hi - lo + eps)


def mad_lower_median(x, eps):              # the lower middle value as the median of an even count
    srt = np.sort(x)
    med = srt[(len(x) - 1) // 2]
    dev = np.sort(np.abs(x - med))
    mad = dev[(len(x) - 1) // 2]
    return 1.0 / (1.0 + np.exp(-(x - med) / (mad + eps)))


def mad_std_scale(x, eps):                 # mean and standard deviation instead of median and MAD
    return 1.0 / (1.0 + np.exp(-(x - x.mean()) / (x.std() + eps)))


def mad_signed_deviation(x, eps):          # median of x - med instead of |x - med|
    med = np.median(x)
    mad = np.median(x - med)
    return 1.0 / (1.0 + np.exp(-(x - med) / (mad + eps)))


def mad_flipped(x, eps):                   # logistic of -z
    return 1.0 - ORIG["mad_scale"](x, eps)


MUTANTS = {
    "no_scale": ("window_logits", no_scale),
    "no_causal_mask": ("window_logits", no_causal_mask),
    "average_not_sum": ("importance_raw", average_not_sum),
    "pool_counts_valid_only": ("avg_pool", pool_counts_valid_only),
    "pool_off_centre": ("avg_pool", pool_off_centre),
    "centroid_drops_last_key": ("key_centroid", centroid_drops_last_key),
    "distance_squared": ("euclid_distance", distance_squared),
    "redundancy_sign": ("euclid_redundancy", redundancy_sign),
    "cosine_similarity_not_diversity": ("cosine_diversity", cosine_similarity_not_diversity),
    "r_c_drops_minus_one": ("cosine_redundancy", r_c_drops_minus_one),
    "minmax_reversed": ("minmax", minmax_reversed),
    "rescale_by_importance": ("rescale_diversity", rescale_by_importance),
    "select_k_is_budget": ("select", select_k_is_budget),
    "select_ties_high_position": ("select", select_ties_high_position),
    "adaptive_budget_counts_window": ("select_adaptive", adaptive_budget_counts_window),
    "adaptive_ties_by_position": ("select_adaptive", adaptive_ties_by_position),
    "adaptive_no_window": ("select_adaptive", adaptive_no_window),
    "value_norm_squared": ("value_norms", value_norm_squared),
    "pyramid_top_without_m": ("pyramid_budgets_real", pyramid_top_without_m),
    "pyramid_step_over_m": ("pyramid_budgets_real", pyramid_step_over_m),
    "winsor_interpolated": ("winsor_minmax", winsor_interpolated),
    "mad_lower_median": ("mad_scale", mad_lower_median),
    "mad_std_scale": ("mad_scale", mad_std_scale),
    "mad_signed_deviation": ("mad_scale", mad_signed_deviation),
    "mad_flipped": ("mad_scale", mad_flipped),
}


@pytest.mark.parametrize("mutant", sorted(MUTANTS))
def test_planted_slip_fails_a_pin(mutant, monkeypatch):
    name, fn = MUTANTS[mutant]
    monkeypatch.setattr(O, name, fn)
    failed = []
    for pin, f, kw in _pins():
        try:
            with np.errstate(all="ignore"):
                f(**kw)
        except Exception:  # an assertion, or the slip breaking the pin outright
            failed.append(pin)
    assert failed, f"no pin catches {mutant}"


def test_pins_pass_on_the_oracle_as_it_stands():
    for pin, f, kw in _pins():
        f(**kw)
