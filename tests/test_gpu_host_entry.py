"""ecokv_evict_host (KV cache in pinned host memory: K copied once, kept V rows
gathered over the host link, outputs written to host memory) against
ecokv_evict on device copies: identical indices, rows and lambda."""
import pytest
import torch

from paper_2609_06663_gb300 import ecokv as E
from paper_2609_06663_gb300.workloads import make_inputs, small_workload, workload

DEV = "cuda"


def params_of(w):
    return E.make_params(n_layers=w.n_layers, h_kv=w.h_kv, h_q=w.h_q, n=w.n, d=w.d, window=w.window,
                         budget=w.budget, pool_kernel=w.pool_kernel)


def one_layer(w, seed):
    return type(w)(**{**{f: getattr(w, f) for f in w.__dataclass_fields__}, "n_layers": 1, "seed": seed})


CASES = [
    small_workload(5000, h_kv=2, group=4, window=8, budget=500, dtype="bf16", n_layers=2, clustered=True),
    small_workload(3001, h_kv=2, group=1, window=8, budget=300, pool_kernel=7, dtype="f32"),
    small_workload(700, h_kv=2, group=2, window=4, budget=900, dtype="bf16"),  # B >= N keeps every row
    one_layer(workload("c3_b10"), 5),
]


@pytest.mark.gpu
@pytest.mark.parametrize("w", CASES, ids=["bf16_tc", "f32_simt", "keep_all", "c3_one_layer"])
def test_host_entry_matches_device_entry(w):
    K, V, Q = make_inputs(w)
    p = params_of(w)
    hK, hV, hQ = K.pin_memory(), V.pin_memory(), Q.pin_memory()
    idx, Ko, Vo, lam = E.evict_host(p, hK, hV, hQ)
    torch.cuda.synchronize()
    idx_r, Ko_r, Vo_r, _, lam_r = E.evict(p, K.to(DEV), V.to(DEV), Q.to(DEV))
    torch.cuda.synchronize()
    assert torch.equal(idx, idx_r.cpu())
    assert torch.equal(Ko, Ko_r.cpu()) and torch.equal(Vo, Vo_r.cpu())
    assert torch.equal(lam, lam_r.cpu())


@pytest.mark.gpu
def test_host_entry_rejects_pageable_memory():
    w = CASES[0]
    K, V, Q = make_inputs(w)                      # pageable host tensors
    p = params_of(w)
    dt = E.dtype_code(K)
    ws = E.alloc_workspace_host(p, dt)
    n_keep = min(p.budget, p.n)
    idx = torch.empty(p.n_layers, p.h_kv, n_keep, dtype=torch.int32).pin_memory()
    Ko = torch.empty(p.n_layers, p.h_kv, n_keep, p.d, dtype=K.dtype).pin_memory()
    Vo = torch.empty_like(Ko).pin_memory()
    code = E.ecokv_evict_host(p, dt, K, V.pin_memory(), Q.pin_memory(), idx, Ko, Vo, None, ws, ws.numel())
    assert code == E.ECOKV_ERR_INVALID_ARG
    # a workspace one byte short
    code = E.ecokv_evict_host(p, dt, K.pin_memory(), V.pin_memory(), Q.pin_memory(), idx, Ko, Vo, None, ws,
                              ws.numel() - 1)
    assert code == E.ECOKV_ERR_WORKSPACE
