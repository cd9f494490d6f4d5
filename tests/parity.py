"""Comparison helpers for CUDA-path vs oracle parity (used by the gpu tests
and smoke checks).  Tolerances: per-token scores within 1e-3 relative for
bf16 inputs and 1e-5 for fp32 inputs, measured as
|S_gpu - S_ref| <= tol * max(|S_ref|, mean_i |S_ref|); retained sets equal
except for candidates whose oracle score lies within that tolerance of the
oracle's k-th largest score; compacted rows bit-exact."""
import numpy as np
import torch

from oracle import ecokv_oracle as O

TOL = {"f32": 1e-5, "bf16": 1e-3}


def oracle_params(p, **over) -> O.Params:
    kw = {k: getattr(p, k) for k in ("n_layers", "h_kv", "h_q", "n", "d", "window", "budget", "pool_kernel",
                                      "alpha", "beta", "tau", "eps", "flags", "lambda_override")}
    kw["flags"] = kw["flags"] & (O.FLAG_SC_MIXKV_SIGN | O.FLAG_LAMBDA_OVERRIDE | O.FLAG_VNORM_IMP |
                                 O.FLAG_CENTROID_NONWIN | O.FLAG_WINSOR_1 | O.FLAG_WINSOR_5 |
                                 O.FLAG_MAD)  # path flags mean nothing here
    kw.update(over)
    return O.Params(**kw)


def score_error(S_gpu: np.ndarray, S_ref: np.ndarray) -> float:
    if S_ref.size == 0:
        return 0.0
    scale = np.maximum(np.abs(S_ref), np.abs(S_ref).mean())
    scale = np.where(scale > 0, scale, 1.0)
    return float((np.abs(S_gpu - S_ref) / scale).max())


def check_scores(S_gpu, ref, tol, what=""):
    err = score_error(np.asarray(S_gpu, dtype=np.float64), ref["S"])
    assert err <= tol, f"{what}: score error {err:.3e} > {tol:g}"
    return err


def check_selection(idx_gpu: np.ndarray, ref: dict, p: O.Params, tol: float, what=""):
    """Retained sets equal except for threshold ties within tolerance."""
    n, w = p.n, p.window
    idx_gpu = np.asarray(idx_gpu, dtype=np.int64)
    assert idx_gpu.shape == (min(p.budget, n),), what
    if p.budget >= n:
        assert (idx_gpu == np.arange(n)).all(), what
        return 0
    k = p.budget - w
    assert (idx_gpu[k:] == np.arange(n - w, n)).all(), f"{what}: window not retained at the end"
    cand = idx_gpu[:k]
    assert (np.diff(cand) > 0).all() if k > 1 else True, f"{what}: candidates not ascending"
    assert ((cand >= 0) & (cand < n - w)).all(), what
    if k == 0:
        return 0
    S = ref["S"]
    thr = np.sort(S)[::-1][k - 1]
    band = tol * max(abs(thr), np.abs(S).mean())
    diff = set(cand.tolist()) ^ set(ref["idx"][:k].tolist())
    bad = [i for i in diff if abs(S[i] - thr) > band]
    assert not bad, f"{what}: {len(bad)} retained-set differences outside the threshold band, e.g. {bad[:5]}"
    return len(diff)


def check_rows(K: torch.Tensor, idx: torch.Tensor, K_out: torch.Tensor, what=""):
    """K_out[r] must be a bit-exact copy of K[idx[r]]."""
    ref = K[idx.long().cpu()] if K.device.type == "cpu" else K[idx.long()]
    assert torch.equal(K_out.to(ref.device), ref), f"{what}: compacted rows differ"


# ---------------------------------------------------------------- canaries
GUARD_BYTES = 256  # keeps the guarded view 16-byte aligned
_CANARY = {torch.float32: float("nan"), torch.bfloat16: float("nan"), torch.int32: -0x5A5A5A5B}


class Guarded:
    """An output tensor with guard regions before and after it, filled with a
    sentinel that no call may overwrite (out-of-bounds writes of the kernels
    show up here, the sanitizer being unavailable)."""

    def __init__(self, shape, dtype, device):
        import math
        self.g = GUARD_BYTES // torch.tensor([], dtype=dtype).element_size()
        n = math.prod(shape)
        self.full = torch.empty(n + 2 * self.g, dtype=dtype, device=device)
        self.full.fill_(_CANARY[dtype])
        self.view = self.full[self.g:self.g + n].view(*shape)
        self.view.zero_()

    def check(self, what=""):
        for part in (self.full[:self.g], self.full[-self.g:]):
            bits = part.view(torch.int16 if part.element_size() == 2 else torch.int32)
            ref = torch.empty_like(part).fill_(_CANARY[part.dtype])
            ref_bits = ref.view(torch.int16 if ref.element_size() == 2 else torch.int32)
            assert torch.equal(bits, ref_bits), f"{what}: a guard region next to an output was overwritten"
