"""Bounded device-side waits, made to run out on purpose without faulting the
GPU: with ECOKV_FLAG_TEST_STALL the statistics of the first unit never
complete (the streaming kernel expects one more pass-1 arrival than there are
pass-1 items), so the wait of its pass 2 gives up after timeout_us.  The call
must report ECOKV_ERR_TIMEOUT through ecokv_device_status, return well before
the default 2 s limit, and leave the context and the workspace usable: the
next call on the same workspace is bit for bit the call on a fresh one, and
matches the oracle."""
import time

import pytest
import torch

from oracle import ecokv_oracle as O
from paper_2609_06663_gb300 import ecokv as E
from paper_2609_06663_gb300.workloads import make_inputs, small_workload
from tests.parity import TOL, check_rows, check_scores, check_selection, oracle_params

pytestmark = pytest.mark.gpu
DEV = "cuda"


def params_of(w, **kw):
    return E.make_params(n_layers=w.n_layers, h_kv=w.h_kv, h_q=w.h_q, n=w.n, d=w.d, window=w.window,
                         budget=w.budget, pool_kernel=w.pool_kernel, **kw)


def test_stalled_statistics_time_out_and_the_workspace_recovers():
    w = small_workload(3000, h_kv=2, group=4, window=8, budget=300, dtype="bf16", n_layers=2, clustered=True)
    K, V, Q = make_inputs(w)
    Kd, Vd, Qd = K.to(DEV), V.to(DEV), Q.to(DEV)
    p_stall = params_of(w, flags=E.ECOKV_FLAG_TEST_STALL, timeout_us=20000)
    p = params_of(w)
    assert E.ecokv_workspace_size(p_stall) == E.ecokv_workspace_size(p)
    ws = E.alloc_workspace(p, DEV)
    torch.cuda.synchronize()

    t0 = time.perf_counter()
    E.evict(p_stall, Kd, Vd, Qd, ws=ws)  # enqueued; the failure shows on the device only
    status = E.ecokv_device_status(ws)   # synchronises
    elapsed = time.perf_counter() - t0
    assert status == E.ECOKV_ERR_TIMEOUT, E.STATUS.get(status, status)
    assert elapsed < 1.0, f"the 20 ms limit took {elapsed:.3f} s to fire"
    assert E.ecokv_device_status(ws) == 0  # reading the status cleared it

    # the same workspace right after the aborted call, and a fresh one
    idx, Ko, Vo, S, lam = E.evict(p, Kd, Vd, Qd, ws=ws, want_scores=True)
    idx2, Ko2, Vo2, S2, lam2 = E.evict(p, Kd, Vd, Qd, want_scores=True)
    torch.cuda.synchronize()
    assert E.ecokv_device_status(ws) == 0
    assert torch.equal(S, S2) and torch.equal(lam, lam2) and torch.equal(idx, idx2)
    assert torch.equal(Ko, Ko2) and torch.equal(Vo, Vo2)

    op = oracle_params(p)
    ref = O.evict(K, V, Q, op)
    S_np = S.cpu().double().numpy()
    for (l, h), r in ref.items():
        what = f"unit ({l},{h}) after a timed-out call"
        check_scores(S_np[l, h], r, TOL["bf16"], what)
        check_selection(idx[l, h].cpu().numpy(), r, op, TOL["bf16"], what)
        check_rows(Kd[l, h], idx[l, h], Ko[l, h], what)
        check_rows(Vd[l, h], idx[l, h], Vo[l, h], what)


def test_stall_flag_needs_the_tensor_core_path():
    """The injected stall exists only in the tensor-core kernel; elsewhere the
    flag is refused before anything is launched."""
    w = small_workload(1000, h_kv=2, group=1, window=8, budget=100, dtype="f32")
    K, V, Q = (t.to(DEV) for t in make_inputs(w))
    p = params_of(w, flags=E.ECOKV_FLAG_TEST_STALL, timeout_us=20000)
    with pytest.raises(E.EcokvError) as e:
        E.evict(p, K, V, Q)
    assert e.value.code == E.ECOKV_ERR_UNSUPPORTED
