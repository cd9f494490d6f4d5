"""ECOKV prefill eviction pass: plain, slow CPU oracle in fp64.

TEST INFRASTRUCTURE.  Only tests/, __graft_entry__.smoke() and bench.py's
cpu_baseline / reference leg may import this module.  The library
(paper_2609_06663_gb300) never imports it and shares no code with it.

What it computes, per layer l and KV head h (paper Sec. 3 problem statement,
Sec. 5.1-5.2 Eq. 1-7, Appendix A "SnapKV" and "MixKV", Algorithm 1):

  1. window attention: l[q,j,i] = Q[q,j] . K[i] / sqrt(d) for the g query
     heads of the group and the W window rows; softmax over the visible keys;
  2. importance: sum of the probabilities over window rows and group heads for
     the T_v = N - W non-window keys, then 1-D average pooling;
  3. Euclidean terms: centroid kbar, distances d_E (Eq. 1), min-max s_E (Eq. 2),
     mean distance D_E (Eq. 4), redundancy r_E (Eq. 5);
  4. cosine terms: mean normalised key mu, cosine to the mean, s_C, and the
     off-diagonal mean cosine r_C (Appendix A, MixKV);
  5. S_div = alpha s_E + (1 - alpha) s_C (Eq. 3), lambda = beta r_E +
     (1 - beta) r_C (Eq. 6), diversity rescale (Sec. 5.2), S (Eq. 7);
  6. top-(B - W) of S over the non-window keys plus the whole window
     (Sec. 3), and the gather of the retained K/V rows;
  7. (variant, AdaKV's layer-wide budget, Appendix A) one top-H_kv (B - W)
     over the concatenated scores of a layer's heads instead of one top-(B - W)
     per head;
  8. (variant, PyramidKV's per-layer budgets, Appendix A) budget b^l for the
     heads of layer l.

Readings of passages that are silent, ambiguous or garbled (each one is also
listed with its justification in the design notes):

  R1  s_C = (1 - khat_i . mu) / 2.  Algorithm 1 maps the cosine to [0, 1] with
      (x + 1)/2 but prints the similarity, while MixKV's definition (Appendix A)
      is the negated cosine, a diversity.  The reading keeps both: the sign of
      MixKV and the [0, 1] range of Algorithm 1.  FLAG_SC_MIXKV_SIGN gives
      MixKV's s_C = -khat_i . mu.
  R2  alpha and beta weight the Euclidean terms, as Eq. 3 and Eq. 6 print them.
  R3  The rescale divides by mean(Sbar_div) (the printed mean(sbar_C) is the
      MixKV formula carried over); mean(Stilde_div) then equals mean(S_imp).
      When Sbar_div is identically zero the rescaled diversity is zero.
  R4  kbar, mu and D_E are means over all N keys (Eq. 1, Eq. 4, Algorithm 1
      steps 2 and 5); d_E, s_C, the extrema of Eq. 2, the Sbar rescale and
      mean(S_imp) run over the T_v candidates.
  R5  eps = 1e-6 (a "small constant"), also added to the min-max of S_div.
  R6  S_imp is a sum (not an average) over window rows and group heads; a
      positive per-head scale of S_imp leaves the selection unchanged.
  R7  No value-norm factor in S_imp by default (its combination is
      unspecified); FLAG_VNORM_IMP adds one (R17).
  R8  Scale 1/sqrt(d); window row j sits at position N - W + j and sees keys
      0 .. N - W + j; only the T_v candidates are scored.
  R9  Average pooling, centred, stride 1, zero padding counted in the divisor,
      over the length-T_v candidate vector; pool_kernel is odd.
  R10 The budget B counts the window: k = B - W candidates are chosen.  B >= N
      keeps every row.
  R11 Ranking is by (S descending, position ascending); the retained list is
      the chosen candidates in ascending position followed by the window.
  R12 khat = k / max(||k||, 1e-12).
  R13 tau = sqrt(d) unless given; sigma is the logistic function.
  R14 Query head q belongs to KV head q // (h_q / h_kv).
  R15 r_C := 1 when N = 1 (a single key is fully redundant with itself).
  R16 Layer-wide budget (AdaKV): the layer's candidate budget is H_kv (B - W);
      ties across heads go to the lower head, then the lower position; every
      head keeps its whole window.
  R17 Value-norm importance (FLAG_VNORM_IMP; Sec. 5.2 says S_imp combines the
      l2 norm of the value vector with the window attention, without the
      form): S_imp(i) = pooled vote(i) * ||v_i||_2, the pooling first.
  R18 Per-layer budgets (PyramidKV, Appendix A): the total is the uniform
      budget's, m B; the real-valued schedule is rounded half up and raised to
      at least W; a layer budget >= N keeps the layer whole.
  R19 Non-window centroid (FLAG_CENTROID_NONWIN; Appendix B's alternative to
      Algorithm 1 step 5): kbar over the T_v candidates (all N keys when
      T_v = 0); d_E of every key to that centroid, D_E still over all N (Eq.
      4); mu and r_C unchanged.
  R20 Winsorised min-max of Eq. 2 (FLAG_WINSOR_1 / FLAG_WINSOR_5, the
      normalisation ablation of Appendix B): q_lo and q_hi are order
      statistics of d_E over the candidates, the floor(p (T_v - 1))-th and
      the ceil((1 - p) (T_v - 1))-th smallest (0-based; p = 0.01 or 0.05, no
      interpolation); s_E = (clip(d_E, q_lo, q_hi) - q_lo) / (q_hi - q_lo + eps).
      The min-max of S_div in the rescale stays plain.
  R21 MAD scaling of Eq. 2 (FLAG_MAD; the same ablation names per-head MAD
      scaling at temperature 1 without its formula): med = median of d_E over
      the candidates, MAD = median of |d_E - med| (a median of an even count
      is the mean of its two middle order statistics); s_E = sigma((d_E -
      med) / (MAD + eps)), the logistic function at temperature 1 mapping the
      robust z-score into (0, 1), the range Eq. 2's text gives the diversity
      scores.  The min-max of S_div stays plain; at most one of FLAG_MAD and
      the winsorising flags.

Parity pins: every function below is checked in tests/test_oracle_pins.py
against closed forms, invariants, special cases that reduce to a library
routine, and brute force on tiny inputs.  The composite score S on realistic
data has no printed example to compare with: beyond those pins its parity is
unpinned.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

FLAG_SC_MIXKV_SIGN = 0x1
FLAG_LAMBDA_OVERRIDE = 0x2
FLAG_VNORM_IMP = 0x4
FLAG_CENTROID_NONWIN = 0x8
FLAG_WINSOR_1 = 0x10   # 1 %-99 % winsorised min-max of Eq. 2
FLAG_WINSOR_5 = 0x20   # 5 %-95 %
FLAG_MAD = 0x40        # MAD scaling of Eq. 2

NORM_FLOOR = 1e-12


@dataclass
class Params:
    """Mirror of the library's parameter block (defaults: Appendix A.3 table)."""
    n_layers: int
    h_kv: int
    h_q: int
    n: int
    d: int
    window: int
    budget: int
    pool_kernel: int = 5
    alpha: float = 0.8
    beta: float = 0.6
    tau: float = 0.0          # <= 0 means sqrt(d)
    eps: float = 1e-6
    flags: int = 0
    lambda_override: float = 0.0

    @property
    def group(self) -> int:
        return self.h_q // self.h_kv

    @property
    def t_v(self) -> int:
        return self.n - self.window

    @property
    def n_keep(self) -> int:
        return min(self.budget, self.n)

    @property
    def tau_eff(self) -> float:
        return self.tau if self.tau > 0 else float(np.sqrt(self.d))


# --------------------------------------------------------------------------
# 1. observation-window attention (Sec. 3 softmax(QK^T / sqrt(d_k)); SnapKV
#    voting over the observation window, Appendix A)
# --------------------------------------------------------------------------
def window_logits(K: np.ndarray, Qg: np.ndarray) -> np.ndarray:
    """l[q, j, i] = Qg[q, j] . K[i] / sqrt(d), -inf where key i is not visible.

    K: [N, d]; Qg: [g, W, d].  Window row j is the query at position N - W + j
    and sees keys 0 .. N - W + j (causal prefill, reading R8).
    """
    n, d = K.shape
    g, w, _ = Qg.shape
    logits = np.einsum("qjd,id->qji", Qg, K) / np.sqrt(d)
    pos = np.arange(n)[None, :]
    last_visible = (n - w + np.arange(w))[:, None]
    visible = pos <= last_visible                      # [W, N]
    return np.where(visible[None, :, :], logits, -np.inf)


def window_softmax(logits: np.ndarray) -> np.ndarray:
    """Row-wise softmax over the visible keys (invisible entries are -inf)."""
    m = logits.max(axis=-1, keepdims=True)
    e = np.exp(logits - m)
    return e / e.sum(axis=-1, keepdims=True)


def importance_raw(p: np.ndarray, t_v: int) -> np.ndarray:
    """SnapKV vote: sum of the window probabilities over rows and group heads,
    for the non-window candidates 0 .. T_v - 1 (reading R6)."""
    return p[:, :, :t_v].sum(axis=(0, 1))


def avg_pool(x: np.ndarray, kernel: int) -> np.ndarray:
    """Centred average pooling, stride 1, zero padding counted (reading R9)."""
    t = x.shape[0]
    half = kernel // 2
    y = np.zeros(t)
    for o in range(-half, half + 1):
        lo, hi = max(0, -o), min(t, t - o)
        if lo < hi:
            y[lo:hi] += x[lo + o:hi + o]
    return y / kernel


# --------------------------------------------------------------------------
# 2. Euclidean diversity and redundancy (Eq. 1, 2, 4, 5)
# --------------------------------------------------------------------------
def key_centroid(K: np.ndarray) -> np.ndarray:
    """kbar = (1/T) sum_i k_i over all T = N keys (Eq. 1, reading R4)."""
    return K.mean(axis=0)


def euclid_distance(K: np.ndarray, kbar: np.ndarray) -> np.ndarray:
    """d_E(i) = ||k_i - kbar||_2 (Eq. 1)."""
    diff = K - kbar[None, :]
    return np.sqrt((diff * diff).sum(axis=1))


def minmax(x: np.ndarray, eps: float) -> np.ndarray:
    """(x - min x) / (max x - min x + eps) (Eq. 2)."""
    lo, hi = x.min(), x.max()
    return (x - lo) / (hi - lo + eps)


def winsor_minmax(x: np.ndarray, p: float, eps: float) -> np.ndarray:
    """Winsorised min-max (R20): clip to the p and 1 - p order statistics,
    then min-max between them."""
    t = x.shape[0]
    srt = np.sort(x)
    lo = srt[int(np.floor(p * (t - 1)))]
    hi = srt[int(np.ceil((1.0 - p) * (t - 1)))]
    return (np.clip(x, lo, hi) - lo) / (hi - lo + eps)


def mad_scale(x: np.ndarray, eps: float) -> np.ndarray:
    """Per-head MAD scaling (R21): the logistic function of (x - median x) /
    (MAD + eps), MAD the median absolute deviation from the median."""
    med = np.median(x)
    mad = np.median(np.abs(x - med))
    z = (x - med) / (mad + eps)
    with np.errstate(over="ignore"):
        return 1.0 / (1.0 + np.exp(-z))


def euclid_redundancy(mean_dist: float, tau: float) -> float:
    """r_E = 2 - 2 sigma(D_E / tau) (Eq. 5)."""
    return 2.0 - 2.0 / (1.0 + np.exp(-mean_dist / tau))


# --------------------------------------------------------------------------
# 3. cosine diversity and redundancy (MixKV, Appendix A; Algorithm 1)
# --------------------------------------------------------------------------
def normalized_keys(K: np.ndarray) -> np.ndarray:
    """K_N,i = k_i / ||k_i|| with the norm floored at 1e-12 (reading R12)."""
    nrm = np.sqrt((K * K).sum(axis=1))
    return K / np.maximum(nrm, NORM_FLOOR)[:, None]


def cosine_to_mean(KN: np.ndarray, mu: np.ndarray) -> np.ndarray:
    """khat_i . mu, the cosine-type similarity of each key to the mean direction."""
    return KN @ mu


def cosine_diversity(c: np.ndarray, flags: int) -> np.ndarray:
    """s_C (reading R1)."""
    if flags & FLAG_SC_MIXKV_SIGN:
        return -c
    return (1.0 - c) / 2.0


def cosine_redundancy(mu: np.ndarray, t: int) -> float:
    """r_C = (T^2 ||mu||^2 - T) / (T (T - 1)) = (T ||mu||^2 - 1) / (T - 1)."""
    if t == 1:
        return 1.0
    return (t * float(mu @ mu) - 1.0) / (t - 1.0)


# --------------------------------------------------------------------------
# 4. combination (Eq. 3, 6, 7 and the rescale of Sec. 5.2)
# --------------------------------------------------------------------------
def rescale_diversity(s_div: np.ndarray, s_imp: np.ndarray, eps: float) -> np.ndarray:
    """Sbar = minmax(S_div); Stilde = Sbar * mean(S_imp) / mean(Sbar) (R3, R5)."""
    sbar = minmax(s_div, eps)
    mb = sbar.mean()
    if mb == 0.0:
        return np.zeros_like(sbar)
    return sbar * (s_imp.mean() / mb)


# --------------------------------------------------------------------------
# 5. selection and compaction (Sec. 3)
# --------------------------------------------------------------------------
def select(S: np.ndarray, p: Params) -> np.ndarray:
    """Retained positions: top-(B - W) candidates by (S desc, position asc) in
    ascending position, then the window N - W .. N - 1 (R10, R11).
    B >= N keeps 0 .. N - 1."""
    n, w = p.n, p.window
    if p.budget >= n:
        return np.arange(n, dtype=np.int64)
    k = p.budget - w
    t_v = n - w
    assert S.shape == (t_v,)
    order = np.lexsort((np.arange(t_v), -S))        # primary -S, then position
    chosen = np.sort(order[:k])
    return np.concatenate([chosen, np.arange(t_v, n)]).astype(np.int64)


def select_adaptive(S_heads: list, p: Params) -> list:
    """Layer-wide budget (AdaKV, Appendix A: the heads' scores are concatenated,
    one top-K is taken over the concatenation, and each head keeps what it got
    there).  Readings: K = H_kv (B - W), the layer's candidate budget, so the
    layer keeps H_kv B rows in all; ties go to the lower (head, position); each
    head's list is its chosen candidates in ascending position, then its window.
    B >= N keeps every row of every head.  Returns one index array per head."""
    n, w, t_v = p.n, p.window, p.t_v
    h_kv = len(S_heads)
    if p.budget >= n:
        return [np.arange(n, dtype=np.int64) for _ in range(h_kv)]
    k_layer = h_kv * (p.budget - w)
    cat = np.concatenate([np.asarray(s, dtype=np.float64) for s in S_heads])
    assert cat.shape == (h_kv * t_v,)
    order = np.lexsort((np.arange(cat.size), -cat))       # primary -S, then (head, position)
    chosen = np.zeros(cat.size, dtype=bool)
    chosen[order[:k_layer]] = True
    out = []
    for h in range(h_kv):
        mine = np.nonzero(chosen[h * t_v:(h + 1) * t_v])[0]
        out.append(np.concatenate([mine, np.arange(t_v, n)]).astype(np.int64))
    return out


def compact(X: np.ndarray, idx: np.ndarray) -> np.ndarray:
    """Gather the retained rows: X_out[r] = X[idx[r]]."""
    return X[idx]


# --------------------------------------------------------------------------
# one KV head, then all layers and heads
# --------------------------------------------------------------------------
def value_norms(V: np.ndarray) -> np.ndarray:
    """||v_i||_2 of every value row (R17)."""
    return np.sqrt((V * V).sum(axis=1))


def score_head(K: np.ndarray, Qg: np.ndarray, p: Params, V: np.ndarray | None = None) -> dict:
    """Every intermediate of the score for one (layer, KV head).

    K: [N, d] float64, Qg: [g, W, d] float64 (the group's window queries);
    V: [N, d] float64, needed with FLAG_VNORM_IMP only.
    """
    n, d = K.shape
    t_v = n - p.window
    out: dict = {}

    logits = window_logits(K, Qg)
    prob = window_softmax(logits)
    out["m"] = logits.max(axis=-1)                                 # [g, W]
    out["lse"] = out["m"] + np.log(np.exp(logits - out["m"][..., None]).sum(-1))
    s_imp_raw = importance_raw(prob, t_v)
    s_imp = avg_pool(s_imp_raw, p.pool_kernel)
    if p.flags & FLAG_VNORM_IMP:
        assert V is not None, "FLAG_VNORM_IMP needs the values"
        s_imp = s_imp * value_norms(V[:t_v])                       # R17

    kbar = key_centroid(K[:t_v] if (p.flags & FLAG_CENTROID_NONWIN) and t_v > 0 else K)   # R4, R19
    d_e_all = euclid_distance(K, kbar)
    D_E = d_e_all.mean()                                          # Eq. 4, all T keys
    r_E = euclid_redundancy(D_E, p.tau_eff)

    KN = normalized_keys(K)
    mu = KN.mean(axis=0)
    r_C = cosine_redundancy(mu, n)

    if p.flags & FLAG_LAMBDA_OVERRIDE:
        lam = p.lambda_override
    else:
        lam = p.beta * r_E + (1.0 - p.beta) * r_C                 # Eq. 6

    out.update(kbar=kbar, mu=mu, D_E=D_E, r_E=r_E, r_C=r_C, lam=lam,
               s_imp_raw=s_imp_raw, s_imp=s_imp, d_e=d_e_all[:t_v])
    if t_v == 0:
        empty = np.zeros(0)
        out.update(c=empty, s_E=empty, s_C=empty, s_div=empty, s_tilde=empty, S=empty)
        return out

    c = cosine_to_mean(KN[:t_v], mu)
    s_C = cosine_diversity(c, p.flags)
    if p.flags & (FLAG_WINSOR_1 | FLAG_WINSOR_5):
        s_E = winsor_minmax(d_e_all[:t_v], 0.01 if p.flags & FLAG_WINSOR_1 else 0.05, p.eps)   # R20
    elif p.flags & FLAG_MAD:
        s_E = mad_scale(d_e_all[:t_v], p.eps)                      # R21
    else:
        s_E = minmax(d_e_all[:t_v], p.eps)                         # Eq. 2
    s_div = p.alpha * s_E + (1.0 - p.alpha) * s_C                 # Eq. 3
    s_tilde = rescale_diversity(s_div, s_imp, p.eps)
    S = lam * s_tilde + (1.0 - lam) * s_imp                        # Eq. 7
    out.update(c=c, s_E=s_E, s_C=s_C, s_div=s_div, s_tilde=s_tilde, S=S)
    return out


def to_f64(x) -> np.ndarray:
    """Widen an input (numpy array or torch tensor, fp32 or bf16) exactly to fp64."""
    if hasattr(x, "detach"):                      # torch tensor, without importing torch
        x = x.detach().cpu().double().numpy()
    return np.asarray(x, dtype=np.float64)


def pyramid_budgets_real(m: int, b_total: float, beta: float) -> list:
    """PyramidKV's per-layer budgets (Appendix A): b^{m-1} = b_total / (beta m),
    b^0 = 2 b_total / m - b^{m-1}, and b^l linear between them."""
    if m == 1:
        return [float(b_total)]
    b_last = b_total / (beta * m)
    b_first = 2.0 * b_total / m - b_last
    return [b_first - (b_first - b_last) / (m - 1) * l for l in range(m)]


def pyramid_budgets(m: int, budget: int, beta: float, window: int) -> list:
    """Integer per-layer budgets (reading R18): the uniform budget's total
    m B spread by pyramid_budgets_real, each rounded half up and raised to at
    least the window."""
    return [max(window, int(np.floor(x + 0.5))) for x in pyramid_budgets_real(m, m * budget, beta)]


def evict_layered(K, V, Q, p: Params, budgets: list, heads=None) -> dict:
    """The pass with budget budgets[l] for every head of layer l (PyramidKV
    schedule); otherwise as evict."""
    res = {}
    units = heads if heads is not None else [(l, h) for l in range(p.n_layers) for h in range(p.h_kv)]
    for l in sorted({l for l, _ in units}):
        pl = Params(**{**p.__dict__, "budget": int(budgets[l])})
        res.update(evict(K, V, Q, pl, heads=[(ll, h) for ll, h in units if ll == l]))
    return res


def evict_adaptive(K, V, Q, p: Params, layers=None) -> dict:
    """The pass with the layer-wide budget of select_adaptive.  Returns, per
    layer l, the per-head score intermediates ('heads'), 'idx' (the heads'
    lists concatenated in head order), 'head_off' (H_kv + 1 offsets into it)
    and the gathered 'K_out' / 'V_out' rows in the same order."""
    K, V, Q = to_f64(K), to_f64(V), to_f64(Q)
    g = p.group
    res = {}
    for l in (layers if layers is not None else range(p.n_layers)):
        heads = [score_head(K[l, h], Q[l, h * g:(h + 1) * g], p, V[l, h]) for h in range(p.h_kv)]
        lists = select_adaptive([r["S"] for r in heads], p)
        off = np.concatenate([[0], np.cumsum([len(x) for x in lists])]).astype(np.int64)
        res[l] = {"heads": heads, "idx": np.concatenate(lists), "head_off": off,
                  "K_out": np.concatenate([compact(K[l, h], lists[h]) for h in range(p.h_kv)]),
                  "V_out": np.concatenate([compact(V[l, h], lists[h]) for h in range(p.h_kv)])}
    return res


def evict(K, V, Q, p: Params, heads=None) -> dict:
    """The whole pass over all (layer, KV head) units.

    K, V: [L, H_kv, N, d]; Q: [L, H_q, W, d].  `heads` optionally restricts the
    run to a list of (layer, head) units (for sampled checks at large sizes).
    Returns per-unit results keyed by (layer, head): the score intermediates,
    'idx' and the compacted 'K_out' / 'V_out' rows.
    """
    K, V, Q = to_f64(K), to_f64(V), to_f64(Q)
    g = p.group
    units = heads if heads is not None else [(l, h) for l in range(p.n_layers) for h in range(p.h_kv)]
    res = {}
    for (l, h) in units:
        r = score_head(K[l, h], Q[l, h * g:(h + 1) * g], p, V[l, h])
        idx = select(r["S"], p)
        r["idx"] = idx
        r["K_out"] = compact(K[l, h], idx)
        r["V_out"] = compact(V[l, h], idx)
        res[(l, h)] = r
    return res
