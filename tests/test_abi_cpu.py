"""The C-ABI library builds, loads and exports every symbol include/ecokv.h
declares; host-side argument checks return the documented codes before
anything is launched (no compute calls here: no GPU is needed)."""
import ctypes
import os
import re

import pytest

from paper_2609_06663_gb300 import ecokv as E

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(E.LIB_PATH):
        from paper_2609_06663_gb300 import build
        build.build()
    return E.lib()


def declared_functions():
    names = []
    for h in os.listdir(os.path.join(ROOT, "include")):
        if h.endswith(".h"):
            txt = open(os.path.join(ROOT, "include", h)).read()
            txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
            names += re.findall(r"^\s*[A-Za-z_][\w\s\*]*?\b(ecokv_\w+)\s*\(", txt, flags=re.M)
    return sorted(set(names))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 9
    for n in names:
        assert hasattr(lib, n), n
    assert set(E.EXPORTS) <= set(names)


def good():
    return E.make_params(n_layers=2, h_kv=4, h_q=28, n=4096, window=4, budget=512, pool_kernel=5)


def test_defaults_follow_hyperparameter_table(lib):
    p = E.ecokv_params_default()
    assert abs(p.alpha - 0.8) < 1e-7 and abs(p.beta - 0.6) < 1e-7
    assert p.pool_kernel == 5 and p.window == 4 and p.tau == 0.0 and abs(p.eps - 1e-6) < 1e-12


@pytest.mark.parametrize("field,value,code", [
    ("h_q", 30, 1), ("window", 0, 1), ("window", 5000, 1), ("budget", 3, 1), ("pool_kernel", 4, 1),
    ("pool_kernel", 0, 1), ("alpha", 1.5, 1), ("beta", -0.1, 1), ("eps", 0.0, 1), ("flags", 0x80, 1),
    ("n", 0, 1), ("d", 64, 2), ("n", (1 << 24) + 1, 2), ("window", 64, 2),
])
def test_param_validation(lib, field, value, code):
    p = good()
    assert E.ecokv_check_params(p) == 0
    setattr(p, field, value)
    if field == "window" and value == 64:
        p.budget = 4096          # (h_q/h_kv) * W = 448 > 256
    if field == "n" and value > 4096:
        p.budget = 8
    assert E.ecokv_check_params(p) == code
    assert E.ecokv_workspace_size(p) == 0


def test_workspace_grows_with_problem(lib):
    p = good()
    a = E.ecokv_workspace_size(p)
    p.n_layers = 4
    assert E.ecokv_workspace_size(p) > a > 0


def test_entry_points_reject_bad_arguments_before_launch(lib):
    p = good()
    fake = 1 << 20                       # aligned, never dereferenced: checks fail first
    ws_need = E.ecokv_workspace_size(p)
    # misaligned input
    assert E.ecokv_score(p, 1, fake + 2, fake, fake, None, None, fake, ws_need) == 1
    # null output
    assert E.ecokv_evict(p, 1, fake, fake, fake, None, fake, fake, None, None, fake, ws_need) == 1
    # workspace too small / missing
    assert E.ecokv_score(p, 1, fake, fake, fake, None, None, fake, ws_need - 1) == 3
    assert E.ecokv_evict(p, 1, fake, fake, fake, fake, fake, fake, None, None, None, 0) == 3
    # bad dtype code
    assert E.ecokv_compact(p, 7, fake, fake, fake, fake, fake) == 1
    # host entry: pointers the device cannot address (no device here at all)
    ws_host = E.ecokv_workspace_size_host(p, 1)
    assert ws_host >= ws_need + 2 * 4 * 4096 * 128 * 2          # holds the device copy of K
    assert E.ecokv_workspace_size_host(p, 7) == 0
    assert E.ecokv_evict_host(p, 1, fake, fake, fake, fake, fake, fake, None, fake, ws_host) == 1
    # invalid params win over everything
    p.d = 64
    assert E.ecokv_evict(p, 1, fake, fake, fake, fake, fake, fake, None, None, fake, ws_need) == 2


@pytest.mark.parametrize("m,B,W,beta", [(28, 3277, 8, 20.0), (32, 205, 8, 20.0), (28, 1024, 4, 5.0), (1, 50, 4, 20.0),
                                       (4, 10, 8, 100.0), (6, 100, 4, 1.0)])
def test_pyramid_budgets_match_the_oracle(lib, m, B, W, beta):
    from oracle import ecokv_oracle as O
    import numpy as np
    beta32 = float(np.float32(beta))
    assert E.pyramid_budgets(m, B, W, beta) == O.pyramid_budgets(m, B, beta32, W)


def test_pyramid_budgets_and_layered_entry_reject_bad_arguments(lib):
    import ctypes
    out = (ctypes.c_int32 * 4)()
    assert lib.ecokv_pyramid_budgets(4, 3, 8, 20.0, ctypes.addressof(out)) == 1   # budget below the window
    assert lib.ecokv_pyramid_budgets(4, 100, 8, 0.0, ctypes.addressof(out)) == 1  # beta must be > 0
    p = good()
    fake = 1 << 20
    ws = E.ecokv_workspace_size(p)
    lb = (ctypes.c_int32 * 2)(600, 100)                                            # above p.budget = 512
    assert E.ecokv_evict_layered(p, 1, fake, fake, fake, ctypes.addressof(lb), fake, fake, fake, None, None, fake,
                                 ws) == 1
    lb = (ctypes.c_int32 * 2)(2, 100)                                              # below the window
    assert E.ecokv_evict_layered(p, 1, fake, fake, fake, ctypes.addressof(lb), fake, fake, fake, None, None, fake,
                                 ws) == 1


def test_adaptive_entry_rejects_bad_arguments(lib):
    p = good()
    fake = 1 << 20
    ws = E.ecokv_workspace_size(p)
    # head offsets missing, then misaligned
    assert E.ecokv_evict_adaptive(p, 1, fake, fake, fake, fake, None, fake, fake, None, fake, ws) == 1
    assert E.ecokv_evict_adaptive(p, 1, fake, fake, fake, fake, fake + 2, fake, fake, None, fake, ws) == 1
    assert E.ecokv_evict_adaptive(p, 1, fake, fake, fake, fake, fake, fake, fake, None, fake, ws - 1) == 3
    # both winsorising levels at once
    p.flags = E.ECOKV_FLAG_WINSOR_1 | E.ECOKV_FLAG_WINSOR_5
    assert E.ecokv_check_params(p) == 1
    # MAD scaling with a winsorising level
    for wf in (E.ECOKV_FLAG_WINSOR_1, E.ECOKV_FLAG_WINSOR_5):
        p.flags = E.ECOKV_FLAG_MAD | wf
        assert E.ecokv_check_params(p) == 1
    p.flags = E.ECOKV_FLAG_MAD
    assert E.ecokv_check_params(p) == 0


def test_status_strings(lib):
    for c in range(7):
        assert E.ecokv_status_string(c)
    assert "workspace" in E.ecokv_status_string(3)


def test_no_cpu_fallback_when_library_missing(monkeypatch, tmp_path):
    monkeypatch.setattr(E, "_lib", None)
    monkeypatch.setattr(E, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        E.lib()


def test_binding_constants_match_header():
    txt = open(os.path.join(ROOT, "include", "ecokv.h")).read()
    m = re.search(r"#define ECOKV_NOALLOC_SCRATCH_BYTES \((\d+)u << (\d+)\)", txt)
    assert m and int(m.group(1)) << int(m.group(2)) == E.ECOKV_NOALLOC_SCRATCH_BYTES


def test_stage_events_hook_arguments(lib):
    assert E.ecokv_set_stage_events(None) == 0
    assert lib.ecokv_set_stage_events((ctypes.c_void_p * 2)(None, None), 2) == 1
