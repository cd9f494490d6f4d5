"""Seeded synthetic inputs for the ECOKV prefill eviction pass.

This module only draws inputs: keys K, values V and observation-window
queries Qwin.  It holds none of the eviction arithmetic, so that the CUDA
path's tests and the fp64 oracle's tests can take identical inputs from it
without sharing any of the method's code.

Shapes follow the paper's problem statement (Sec. 3: keys and values per
layer l and head h, an observation window of the most recent tokens) with
the layout used throughout this package:

    K, V : [n_layers, h_kv, n, d]      row-major, d contiguous
    Qwin : [n_layers, h_q, window, d]  the last `window` query rows

Value distributions.  The paper's workloads are MLLM prefills on document /
chart / scene-text benchmarks; those datasets and model weights are not
available, so every workload here is synthetic and seeded:

* text keys are anisotropic (the narrow-cone property discussed in Sec. 4):
  per (layer, KV head) a unit direction u ~ normalised N(0, I_d), then
  k_i = s_i * (4 u + z_i), z_i ~ N(0, I_d), s_i ~ LogNormal(0, 0.5);
* visual keys come in clusters of near-duplicates: cluster centres are drawn
  as anisotropic keys, members are centre + N(0, 0.1^2 I_d);
* video frames are temporally correlated: frame 0 is a clustered image,
  frame t = frame t-1 + N(0, 0.2^2 I_d);
* values are N(0, 1); window queries are 4 u + N(0, I_d) with the u of the
  KV head they attend to (query head q belongs to KV head q // (h_q/h_kv)).

bf16 workloads draw in fp32 and round once to bf16 (round-to-nearest-even).
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import torch

__all__ = ["Workload", "CONFIGS", "workload", "sweep_workload", "small_workload",
           "make_inputs", "budget_fraction"]


def budget_fraction(n: int, frac: float) -> int:
    """Percent budgets are rounded half up: 0.1 * 32768 = 3276.8 -> 3277."""
    return int(math.floor(frac * n + 0.5))


@dataclass(frozen=True)
class Workload:
    name: str
    n_layers: int
    h_kv: int
    h_q: int
    n: int
    d: int
    dtype: str            # "f32" or "bf16"
    window: int
    pool_kernel: int
    budget: int
    layout: tuple         # token segments, see _segments()
    seed: int = 0

    @property
    def group(self) -> int:
        return self.h_q // self.h_kv

    @property
    def units(self) -> int:
        return self.n_layers * self.h_kv

    @property
    def elem_bytes(self) -> int:
        return 4 if self.dtype == "f32" else 2

    def describe(self) -> dict:
        return {"workload": self.name, "n_layers": self.n_layers, "h_kv": self.h_kv,
                "h_q": self.h_q, "n": self.n, "d": self.d, "dtype": self.dtype,
                "window": self.window, "pool_kernel": self.pool_kernel,
                "budget": self.budget, "seed": self.seed}


def _img(n_clusters: int, size: int = 16) -> tuple:
    return ("img", n_clusters, size)


def _video(frames: int, n_clusters: int, size: int = 16) -> tuple:
    return ("video", frames, n_clusters, size)


def _text(n: int) -> tuple:
    return ("text", n)


# Workload shapes.  Model shapes: LLaVA-1.5-7B (MHA, 32 layers x 32 heads) and
# Qwen2-VL / Qwen2.5-VL-7B (GQA, 28 layers, 28 query / 4 KV heads, d = 128);
# the GQA shape is the one whose FullKV size the efficiency table prints
# (28 x 4 x 128 x 2 x 2 B x 8192 tokens = 0.4375 GiB).
_C0 = dict(name="c0_mha8_n1024_f32", n_layers=1, h_kv=8, h_q=8, n=1024, d=128, dtype="f32",
           window=8, pool_kernel=7, layout=(_text(1024),))
_C1 = dict(n_layers=32, h_kv=32, h_q=32, n=2048, d=128, dtype="bf16", window=8, pool_kernel=5,
           layout=(_text(32), _img(36), _text(1440)))
_C2 = dict(name="c2_qwen_gqa_n8192_bf16_b1024", n_layers=28, h_kv=4, h_q=28, n=8192, d=128,
           dtype="bf16", window=4, pool_kernel=5, budget=1024,
           layout=(_text(1024), _img(80), _text(512), _img(80), _text(512), _img(80),
                   _text(512), _img(80), _text(512)))
_C3 = dict(n_layers=28, h_kv=4, h_q=28, n=32768, d=128, dtype="bf16", window=8, pool_kernel=5,
           layout=(_text(1024), _video(24, 80), _text(1024)))

CONFIGS: dict[str, Workload] = {
    "c0": Workload(budget=128, **_C0),
    "c1_b10": Workload(name="c1_llava_mha_n2048_bf16_b10pct", budget=budget_fraction(2048, 0.10), **_C1),
    "c1_b20": Workload(name="c1_llava_mha_n2048_bf16_b20pct", budget=budget_fraction(2048, 0.20), **_C1),
    "c2": Workload(**_C2),
    "c3_b5": Workload(name="c3_qwen_video_n32768_bf16_b5pct", budget=budget_fraction(32768, 0.05), **_C3),
    "c3_b10": Workload(name="c3_qwen_video_n32768_bf16_b10pct", budget=budget_fraction(32768, 0.10), **_C3),
    "c3_b20": Workload(name="c3_qwen_video_n32768_bf16_b20pct", budget=budget_fraction(32768, 0.20), **_C3),
}


def workload(key: str, **override) -> Workload:
    w = CONFIGS[key]
    if override:
        d = {f: getattr(w, f) for f in w.__dataclass_fields__}
        d.update(override)
        w = Workload(**d)
    return w


def sweep_workload(n: int, window: int, seed: int = 0) -> Workload:
    """Bandwidth sweep: one layer, 8 KV / 32 query heads, bf16, budget 10 %.

    28.125 % of the tokens (the 576/2048 visual share of the LLaVA shape) are
    16-token clusters placed after a short text prefix of n/64 tokens.
    """
    n_vis = (int(round(0.28125 * n)) // 16) * 16
    pre = n // 64
    post = n - pre - n_vis
    layout = tuple(s for s in (_text(pre), _img(n_vis // 16), _text(post)) if _seg_len(s) > 0)
    return Workload(name=f"c4_sweep_n{n}_w{window}_bf16", n_layers=1, h_kv=8, h_q=32, n=n, d=128,
                    dtype="bf16", window=window, pool_kernel=5, budget=budget_fraction(n, 0.10),
                    layout=layout, seed=seed)


def small_workload(n: int, *, h_kv: int = 2, group: int = 1, window: int = 4, budget: int = 16,
                   pool_kernel: int = 5, dtype: str = "f32", n_layers: int = 1, d: int = 128,
                   seed: int = 0, clustered: bool = False, name: str | None = None) -> Workload:
    """A small shape for parity and edge-case tests (ragged n, tiny windows ...)."""
    if clustered and n >= 48:
        nc = (n // 3) // 16
        layout = (_text(n // 3), _img(nc), _text(n - n // 3 - 16 * nc))
        layout = tuple(s for s in layout if _seg_len(s) > 0)
    else:
        layout = (_text(n),)
    return Workload(name=name or f"small_n{n}_h{h_kv}x{group}_w{window}_b{budget}_{dtype}",
                    n_layers=n_layers, h_kv=h_kv, h_q=h_kv * group, n=n, d=d, dtype=dtype,
                    window=window, pool_kernel=pool_kernel, budget=budget, layout=layout, seed=seed)


def _seg_len(seg: tuple) -> int:
    kind = seg[0]
    if kind == "text":
        return seg[1]
    if kind == "img":
        return seg[1] * seg[2]
    if kind == "video":
        return seg[1] * seg[2] * seg[3]
    raise ValueError(kind)


def _aniso(u: torch.Tensor, m: int, g: torch.Generator) -> torch.Tensor:
    d = u.numel()
    s = torch.exp(0.5 * torch.randn(m, generator=g, device=u.device))
    z = torch.randn(m, d, generator=g, device=u.device)
    return s[:, None] * (4.0 * u[None, :] + z)


def _clustered(u: torch.Tensor, n_clusters: int, size: int, g: torch.Generator) -> torch.Tensor:
    d = u.numel()
    centres = _aniso(u, n_clusters, g)
    members = centres.repeat_interleave(size, dim=0)
    return members + 0.1 * torch.randn(n_clusters * size, d, generator=g, device=u.device)


def _keys_for_head(w: Workload, u: torch.Tensor, g: torch.Generator) -> torch.Tensor:
    parts = []
    for seg in w.layout:
        kind = seg[0]
        if kind == "text":
            parts.append(_aniso(u, seg[1], g))
        elif kind == "img":
            parts.append(_clustered(u, seg[1], seg[2], g))
        elif kind == "video":
            frames, nc, size = seg[1], seg[2], seg[3]
            f = _clustered(u, nc, size, g)
            parts.append(f)
            for _ in range(1, frames):
                f = f + 0.2 * torch.randn(f.shape, generator=g, device=u.device)
                parts.append(f)
        else:
            raise ValueError(kind)
    k = torch.cat(parts, 0)
    assert k.shape[0] == w.n, (k.shape, w.n)
    return k


def make_inputs(w: Workload, device: str | torch.device = "cpu", layers: range | None = None):
    """Draw K, V, Qwin for workload `w` on `device`.

    Every layer has its own generator seeded ``seed * 1000 + layer`` so that a
    subset of layers can be drawn alone and matches the full draw.
    Returns (K, V, Qwin) in the workload's dtype (torch.float32 / bfloat16).
    """
    device = torch.device(device)
    layers = range(w.n_layers) if layers is None else layers
    tdt = torch.float32 if w.dtype == "f32" else torch.bfloat16
    nl = len(layers)
    K = torch.empty(nl, w.h_kv, w.n, w.d, dtype=tdt, device=device)
    V = torch.empty_like(K)
    Q = torch.empty(nl, w.h_q, w.window, w.d, dtype=tdt, device=device)
    g_sz = w.group
    for li, layer in enumerate(layers):
        g = torch.Generator(device=device)
        g.manual_seed(w.seed * 1000 + layer)
        for h in range(w.h_kv):
            u = torch.randn(w.d, generator=g, device=device)
            u = u / torch.linalg.vector_norm(u)
            K[li, h] = _keys_for_head(w, u, g).to(tdt)
            V[li, h] = torch.randn(w.n, w.d, generator=g, device=device).to(tdt)
            q = 4.0 * u[None, None, :] + torch.randn(g_sz, w.window, w.d, generator=g, device=device)
            Q[li, h * g_sz:(h + 1) * g_sz] = q.to(tdt)
    return K, V, Q
