"""ctypes binding of libecokv.so: the C ABI of include/ecokv.h under the same
names, plus small helpers that allocate outputs with torch.  Argument
marshalling only: every step of the eviction pass runs in the library's CUDA
kernels, and there is no fallback.  Importing this module does not load the
library; the first call does, and raises if it is missing.
"""
from __future__ import annotations

import ctypes
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libecokv.so")

ECOKV_F32, ECOKV_BF16 = 0, 1
ECOKV_FLAG_SC_MIXKV_SIGN = 0x1
ECOKV_FLAG_LAMBDA_OVERRIDE = 0x2
ECOKV_FLAG_VNORM_IMP = 0x4
ECOKV_FLAG_CENTROID_NONWIN = 0x8
ECOKV_FLAG_WINSOR_1 = 0x10
ECOKV_FLAG_WINSOR_5 = 0x20
ECOKV_FLAG_MAD = 0x40
ECOKV_FLAG_FORCE_SIMT = 0x100
ECOKV_FLAG_TEST_STALL = 0x80000000
ECOKV_NOALLOC_SCRATCH_BYTES = 16 << 20   # fixed scratch of ecokv_evict_noalloc, per device
ECOKV_OK, ECOKV_ERR_INVALID_ARG, ECOKV_ERR_UNSUPPORTED, ECOKV_ERR_WORKSPACE = 0, 1, 2, 3
ECOKV_ERR_CUDA, ECOKV_ERR_TIMEOUT, ECOKV_ERR_DEVICE_INDEX = 4, 5, 6

STATUS = {0: "ECOKV_OK", 1: "ECOKV_ERR_INVALID_ARG", 2: "ECOKV_ERR_UNSUPPORTED", 3: "ECOKV_ERR_WORKSPACE",
          4: "ECOKV_ERR_CUDA", 5: "ECOKV_ERR_TIMEOUT", 6: "ECOKV_ERR_DEVICE_INDEX"}

EXPORTS = ("ecokv_params_default", "ecokv_check_params", "ecokv_workspace_size", "ecokv_score",
           "ecokv_select", "ecokv_compact", "ecokv_evict", "ecokv_device_status", "ecokv_status_string",
           "ecokv_evict_noalloc", "ecokv_set_stage_events", "ecokv_workspace_size_host", "ecokv_evict_host",
           "ecokv_evict_adaptive", "ecokv_evict_layered", "ecokv_pyramid_budgets")


class EcokvError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        super().__init__(f"{where}: {STATUS.get(code, code)} ({ecokv_status_string(code)})")


class ecokv_params(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("h_kv", ctypes.c_int32), ("h_q", ctypes.c_int32),
                ("n", ctypes.c_int32), ("d", ctypes.c_int32), ("window", ctypes.c_int32),
                ("budget", ctypes.c_int32), ("pool_kernel", ctypes.c_int32),
                ("alpha", ctypes.c_float), ("beta", ctypes.c_float), ("tau", ctypes.c_float),
                ("eps", ctypes.c_float), ("flags", ctypes.c_uint32), ("lambda_override", ctypes.c_float),
                ("sched_wave", ctypes.c_int32), ("sched_lag", ctypes.c_int32), ("timeout_us", ctypes.c_uint32)]

    def as_dict(self) -> dict:
        return {f: getattr(self, f) for f, _ in self._fields_}


_lib = None
_P = ctypes.POINTER(ecokv_params)
_vp, _sz = ctypes.c_void_p, ctypes.c_size_t


def lib() -> ctypes.CDLL:
    """Load libecokv.so once (RuntimeError if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"libecokv.so not found at {LIB_PATH}; build it with "
                               "`python -m paper_2609_06663_gb300.build` (no CPU fallback exists)")
        L = ctypes.CDLL(LIB_PATH)
        L.ecokv_params_default.argtypes = [_P]
        L.ecokv_params_default.restype = None
        L.ecokv_check_params.argtypes = [_P]
        L.ecokv_check_params.restype = ctypes.c_int
        L.ecokv_workspace_size.argtypes = [_P]
        L.ecokv_workspace_size.restype = _sz
        L.ecokv_score.argtypes = [_P, ctypes.c_int, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]
        L.ecokv_score.restype = ctypes.c_int
        L.ecokv_select.argtypes = [_P, _vp, _vp, _vp, _sz, _vp]
        L.ecokv_select.restype = ctypes.c_int
        L.ecokv_compact.argtypes = [_P, ctypes.c_int, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]
        L.ecokv_compact.restype = ctypes.c_int
        L.ecokv_evict.argtypes = [_P, ctypes.c_int, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]
        L.ecokv_evict.restype = ctypes.c_int
        L.ecokv_evict_noalloc.argtypes = [_P, ctypes.c_int, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp]
        L.ecokv_evict_noalloc.restype = ctypes.c_int
        L.ecokv_workspace_size_host.argtypes = [_P, ctypes.c_int]
        L.ecokv_workspace_size_host.restype = _sz
        L.ecokv_evict_host.argtypes = [_P, ctypes.c_int, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]
        L.ecokv_evict_host.restype = ctypes.c_int
        L.ecokv_evict_adaptive.argtypes = [_P, ctypes.c_int, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]
        L.ecokv_evict_adaptive.restype = ctypes.c_int
        L.ecokv_evict_layered.argtypes = [_P, ctypes.c_int, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _sz,
                                          _vp]
        L.ecokv_evict_layered.restype = ctypes.c_int
        L.ecokv_pyramid_budgets.argtypes = [ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_float, _vp]
        L.ecokv_pyramid_budgets.restype = ctypes.c_int
        L.ecokv_set_stage_events.argtypes = [ctypes.POINTER(_vp), ctypes.c_int]
        L.ecokv_set_stage_events.restype = ctypes.c_int
        L.ecokv_device_status.argtypes = [_vp, _vp]
        L.ecokv_device_status.restype = ctypes.c_int
        L.ecokv_status_string.argtypes = [ctypes.c_int]
        L.ecokv_status_string.restype = ctypes.c_char_p
        _lib = L
    return _lib


def _ptr(x) -> int | None:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _stream(s) -> int | None:
    if s is None:
        return None
    if isinstance(s, int):
        return s
    return s.cuda_stream


def _check(code: int, where: str) -> None:
    if code != 0:
        raise EcokvError(code, where)


# ---------------------------------------------------------------- C ABI, same names
def ecokv_params_default() -> ecokv_params:
    p = ecokv_params()
    lib().ecokv_params_default(ctypes.byref(p))
    return p


def ecokv_check_params(p: ecokv_params) -> int:
    return lib().ecokv_check_params(ctypes.byref(p))


def ecokv_workspace_size(p: ecokv_params) -> int:
    return lib().ecokv_workspace_size(ctypes.byref(p))


def ecokv_status_string(code: int) -> str:
    return lib().ecokv_status_string(code).decode()


def ecokv_score(p, dtype, K, Qwin, S, lam, dbg, ws, ws_bytes, stream=None) -> int:
    return lib().ecokv_score(ctypes.byref(p), dtype, _ptr(K), _ptr(Qwin), _ptr(S), _ptr(lam), _ptr(dbg),
                             _ptr(ws), ws_bytes, _stream(stream))


def ecokv_select(p, S, idx, ws=None, ws_bytes=0, stream=None) -> int:
    return lib().ecokv_select(ctypes.byref(p), _ptr(S), _ptr(idx), _ptr(ws), ws_bytes, _stream(stream))


def ecokv_compact(p, dtype, K, V, idx, K_out, V_out, ws=None, ws_bytes=0, stream=None) -> int:
    return lib().ecokv_compact(ctypes.byref(p), dtype, _ptr(K), _ptr(V), _ptr(idx), _ptr(K_out), _ptr(V_out),
                               _ptr(ws), ws_bytes, _stream(stream))


def ecokv_evict(p, dtype, K, V, Qwin, idx, K_out, V_out, S, lam, ws, ws_bytes, stream=None) -> int:
    return lib().ecokv_evict(ctypes.byref(p), dtype, _ptr(K), _ptr(V), _ptr(Qwin), _ptr(idx), _ptr(K_out),
                             _ptr(V_out), _ptr(S), _ptr(lam), _ptr(ws), ws_bytes, _stream(stream))


def ecokv_evict_adaptive(p, dtype, K, V, Qwin, idx, head_off, K_out, V_out, lam, ws, ws_bytes, stream=None) -> int:
    return lib().ecokv_evict_adaptive(ctypes.byref(p), dtype, _ptr(K), _ptr(V), _ptr(Qwin), _ptr(idx),
                                      _ptr(head_off), _ptr(K_out), _ptr(V_out), _ptr(lam), _ptr(ws), ws_bytes,
                                      _stream(stream))


def ecokv_evict_layered(p, dtype, K, V, Qwin, layer_budget, idx, K_out, V_out, S, lam, ws, ws_bytes,
                        stream=None) -> int:
    return lib().ecokv_evict_layered(ctypes.byref(p), dtype, _ptr(K), _ptr(V), _ptr(Qwin), _ptr(layer_budget),
                                     _ptr(idx), _ptr(K_out), _ptr(V_out), _ptr(S), _ptr(lam), _ptr(ws), ws_bytes,
                                     _stream(stream))


def pyramid_budgets(n_layers: int, budget: int, window: int, beta: float) -> list:
    """PyramidKV's per-layer budgets from the library (host computation)."""
    out = (ctypes.c_int32 * n_layers)()
    _check(lib().ecokv_pyramid_budgets(n_layers, budget, window, beta, ctypes.addressof(out)), "ecokv_pyramid_budgets")
    return list(out)


def ecokv_workspace_size_host(p, dtype) -> int:
    return lib().ecokv_workspace_size_host(ctypes.byref(p), dtype)


def ecokv_evict_host(p, dtype, K, V, Qwin, idx, K_out, V_out, lam, ws, ws_bytes, stream=None) -> int:
    return lib().ecokv_evict_host(ctypes.byref(p), dtype, _ptr(K), _ptr(V), _ptr(Qwin), _ptr(idx), _ptr(K_out),
                                  _ptr(V_out), _ptr(lam), _ptr(ws), ws_bytes, _stream(stream))


def ecokv_evict_noalloc(p, dtype, K, V, Qwin, idx, K_out, V_out, S, lam, dev_status, stream=None) -> int:
    return lib().ecokv_evict_noalloc(ctypes.byref(p), dtype, _ptr(K), _ptr(V), _ptr(Qwin), _ptr(idx),
                                     _ptr(K_out), _ptr(V_out), _ptr(S), _ptr(lam), _ptr(dev_status),
                                     _stream(stream))


def ecokv_set_stage_events(events) -> int:
    """events: None (hook off) or 4 torch.cuda.Event objects (or raw handles)."""
    if events is None:
        return lib().ecokv_set_stage_events(None, 0)
    hs = [e.cuda_event if hasattr(e, "cuda_event") else int(e) for e in events]
    arr = (_vp * len(hs))(*hs)
    return lib().ecokv_set_stage_events(arr, len(hs))


def ecokv_device_status(ws, stream=None) -> int:
    return lib().ecokv_device_status(_ptr(ws), _stream(stream))


# ---------------------------------------------------------------- torch helpers
def make_params(*, n_layers, h_kv, h_q, n, d=128, window, budget, pool_kernel=5, alpha=0.8, beta=0.6,
                tau=0.0, eps=1e-6, flags=0, lambda_override=0.0, sched_wave=0, sched_lag=0,
                timeout_us=0) -> ecokv_params:
    p = ecokv_params()
    for k, v in dict(n_layers=n_layers, h_kv=h_kv, h_q=h_q, n=n, d=d, window=window, budget=budget,
                     pool_kernel=pool_kernel, alpha=alpha, beta=beta, tau=tau, eps=eps, flags=flags,
                     lambda_override=lambda_override, sched_wave=sched_wave, sched_lag=sched_lag,
                     timeout_us=timeout_us).items():
        setattr(p, k, v)
    return p


def dtype_code(t) -> int:
    import torch
    if t.dtype == torch.float32:
        return ECOKV_F32
    if t.dtype == torch.bfloat16:
        return ECOKV_BF16
    raise TypeError(f"unsupported dtype {t.dtype}")


def alloc_workspace(p: ecokv_params, device="cuda"):
    import torch
    nbytes = ecokv_workspace_size(p)
    if nbytes == 0:
        _check(ecokv_check_params(p) or 1, "ecokv_workspace_size")
    ws = torch.zeros(nbytes, dtype=torch.uint8, device=device)
    return ws


def score(p, K, Qwin, ws=None, dbg=False, stream=None):
    """Run ecokv_score; returns (S [L,H,N-W], lambda [L,H], dbg or None)."""
    import torch
    ws = alloc_workspace(p, K.device) if ws is None else ws
    S = torch.empty(p.n_layers, p.h_kv, p.n - p.window, dtype=torch.float32, device=K.device)
    lam = torch.empty(p.n_layers, p.h_kv, dtype=torch.float32, device=K.device)
    D = torch.empty(p.n_layers, p.h_kv, 5, p.n - p.window, dtype=torch.float32, device=K.device) if dbg else None
    _check(ecokv_score(p, dtype_code(K), K, Qwin, S, lam, D, ws, ws.numel(), stream), "ecokv_score")
    return S, lam, D


def select(p, S, stream=None):
    import torch
    idx = torch.empty(p.n_layers, p.h_kv, min(p.budget, p.n), dtype=torch.int32, device=S.device)
    _check(ecokv_select(p, S, idx, None, 0, stream), "ecokv_select")
    return idx


def compact(p, K, V, idx, ws=None, stream=None):
    import torch
    n_keep = min(p.budget, p.n)
    Ko = torch.empty(p.n_layers, p.h_kv, n_keep, p.d, dtype=K.dtype, device=K.device)
    Vo = torch.empty_like(Ko)
    _check(ecokv_compact(p, dtype_code(K), K, V, idx, Ko, Vo, ws, 0 if ws is None else ws.numel(), stream),
           "ecokv_compact")
    return Ko, Vo


def evict(p, K, V, Qwin, ws=None, want_scores=False, stream=None):
    """Run ecokv_evict; returns (idx, K_out, V_out, S or None, lambda)."""
    import torch
    ws = alloc_workspace(p, K.device) if ws is None else ws
    n_keep = min(p.budget, p.n)
    idx = torch.empty(p.n_layers, p.h_kv, n_keep, dtype=torch.int32, device=K.device)
    Ko = torch.empty(p.n_layers, p.h_kv, n_keep, p.d, dtype=K.dtype, device=K.device)
    Vo = torch.empty_like(Ko)
    S = torch.empty(p.n_layers, p.h_kv, p.n - p.window, dtype=torch.float32, device=K.device) \
        if want_scores else None
    lam = torch.empty(p.n_layers, p.h_kv, dtype=torch.float32, device=K.device)
    _check(ecokv_evict(p, dtype_code(K), K, V, Qwin, idx, Ko, Vo, S, lam, ws, ws.numel(), stream),
           "ecokv_evict")
    return idx, Ko, Vo, S, lam


def evict_adaptive(p, K, V, Qwin, ws=None, stream=None):
    """Run ecokv_evict_adaptive (layer-wide budget); returns (idx [L][h_kv*B],
    head_off [L][h_kv+1], K_out, V_out [L][h_kv*B][d], lambda)."""
    import torch
    ws = alloc_workspace(p, K.device) if ws is None else ws
    rows = p.h_kv * min(p.budget, p.n)
    idx = torch.empty(p.n_layers, rows, dtype=torch.int32, device=K.device)
    off = torch.empty(p.n_layers, p.h_kv + 1, dtype=torch.int32, device=K.device)
    Ko = torch.empty(p.n_layers, rows, p.d, dtype=K.dtype, device=K.device)
    Vo = torch.empty_like(Ko)
    lam = torch.empty(p.n_layers, p.h_kv, dtype=torch.float32, device=K.device)
    _check(ecokv_evict_adaptive(p, dtype_code(K), K, V, Qwin, idx, off, Ko, Vo, lam, ws, ws.numel(), stream),
           "ecokv_evict_adaptive")
    return idx, off, Ko, Vo, lam


def evict_layered(p, K, V, Qwin, budgets, ws=None, want_scores=False, stream=None):
    """Run ecokv_evict_layered with budgets[l] for layer l (p.budget is the
    per-head stride, at least max(budgets)); returns as evict()."""
    import torch
    ws = alloc_workspace(p, K.device) if ws is None else ws
    n_keep = min(p.budget, p.n)
    lb = torch.tensor(list(budgets), dtype=torch.int32)
    idx = torch.empty(p.n_layers, p.h_kv, n_keep, dtype=torch.int32, device=K.device)
    Ko = torch.zeros(p.n_layers, p.h_kv, n_keep, p.d, dtype=K.dtype, device=K.device)
    Vo = torch.zeros_like(Ko)
    S = torch.empty(p.n_layers, p.h_kv, p.n - p.window, dtype=torch.float32, device=K.device) \
        if want_scores else None
    lam = torch.empty(p.n_layers, p.h_kv, dtype=torch.float32, device=K.device)
    _check(ecokv_evict_layered(p, dtype_code(K), K, V, Qwin, lb.data_ptr(), idx, Ko, Vo, S, lam, ws, ws.numel(),
                               stream), "ecokv_evict_layered")
    return idx, Ko, Vo, S, lam


def alloc_workspace_host(p, dtype, device="cuda"):
    """Device workspace for ecokv_evict_host (uint8 tensor)."""
    import torch
    n = ecokv_workspace_size_host(p, dtype)
    if n == 0:
        raise EcokvError(ECOKV_ERR_INVALID_ARG, "ecokv_workspace_size_host")
    return torch.empty(n, dtype=torch.uint8, device=device)


def evict_host(p, K, V, Qwin, ws=None, stream=None):
    """Run ecokv_evict_host on pinned host tensors; returns pinned host
    (idx, K_out, V_out, lambda), valid once the stream has been synchronised."""
    import torch
    dt = dtype_code(K)
    ws = alloc_workspace_host(p, dt) if ws is None else ws
    n_keep = min(p.budget, p.n)
    idx = torch.empty(p.n_layers, p.h_kv, n_keep, dtype=torch.int32).pin_memory()
    Ko = torch.empty(p.n_layers, p.h_kv, n_keep, p.d, dtype=K.dtype).pin_memory()
    Vo = torch.empty(p.n_layers, p.h_kv, n_keep, p.d, dtype=K.dtype).pin_memory()
    lam = torch.empty(p.n_layers, p.h_kv, dtype=torch.float32).pin_memory()
    _check(ecokv_evict_host(p, dt, K, V, Qwin, idx, Ko, Vo, lam, ws, ws.numel(), stream), "ecokv_evict_host")
    return idx, Ko, Vo, lam


def evict_noalloc(p, K, V, Qwin, want_scores=False, stream=None):
    """Run ecokv_evict_noalloc (library-held scratch, no workspace argument);
    returns (idx, K_out, V_out, S or None, lambda, device status code)."""
    import torch
    n_keep = min(p.budget, p.n)
    idx = torch.empty(p.n_layers, p.h_kv, n_keep, dtype=torch.int32, device=K.device)
    Ko = torch.empty(p.n_layers, p.h_kv, n_keep, p.d, dtype=K.dtype, device=K.device)
    Vo = torch.empty_like(Ko)
    S = torch.empty(p.n_layers, p.h_kv, p.n - p.window, dtype=torch.float32, device=K.device) \
        if want_scores else None
    lam = torch.empty(p.n_layers, p.h_kv, dtype=torch.float32, device=K.device)
    code = torch.full((1,), -1, dtype=torch.int32, device=K.device)
    _check(ecokv_evict_noalloc(p, dtype_code(K), K, V, Qwin, idx, Ko, Vo, S, lam, code, stream),
           "ecokv_evict_noalloc")
    return idx, Ko, Vo, S, lam, int(code.item())
