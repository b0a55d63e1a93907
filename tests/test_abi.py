"""The C-ABI library builds, loads, exports every entry point the headers declare,
and rejects bad arguments on the host (no compute calls: no GPU needed)."""
import ctypes as C
import glob
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        src = open(h).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        for m in re.finditer(r"^[A-Za-z_][\w\s\*]*?\b(wm_\w+)\s*\(", src, flags=re.M):
            names.add(m.group(1))
    return names


@pytest.fixture(scope="module")
def lib():
    import paper_2205_01435_gb300 as pkg
    path = pkg._build.build()
    return C.CDLL(path)


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert {"wm_create", "wm_rollout", "wm_mdn_nll", "wm_sync", "wm_destroy",
            "wm_last_error", "wm_last_path"} <= names
    for n in sorted(names):
        assert hasattr(lib, n), f"{n} declared in include/ but not exported by libwm.so"


def test_binding_loads_and_mirrors_names():
    import paper_2205_01435_gb300 as pkg
    wm = pkg.load()
    for n in ("wm_create", "wm_rollout", "wm_mdn_nll", "wm_sync", "wm_destroy", "wm_last_path",
              "wm_last_launches", "wm_rollout_noalloc", "wm_set_timing", "wm_kernel_time",
              "wm_set_controllers", "wm_returns", "wm_mdn_nll_backward"):
        assert callable(getattr(wm, n))


def test_timing_entry_points_reject_null_handle(lib):
    lib.wm_set_timing.argtypes = [C.c_void_p, C.c_int]
    lib.wm_kernel_time.argtypes = [C.c_void_p, C.c_int, C.POINTER(C.c_double), C.POINTER(C.c_longlong)]
    assert lib.wm_set_timing(None, 1) == 1
    ms, n = C.c_double(-1.0), C.c_longlong(-1)
    assert lib.wm_kernel_time(None, 0, C.byref(ms), C.byref(n)) == 1
    assert ms.value == -1.0 and n.value == -1  # outputs untouched on error


def test_invalid_config_rejected_on_host():
    import numpy as np
    import paper_2205_01435_gb300 as pkg
    wm = pkg.load()
    import synth
    cfg = synth.model_config("tiny_fp32")
    w = synth.weights(cfg)
    for bad in (dict(z_dim=0), dict(k_mix=0), dict(k_mix=33), dict(mdn_tau=-1.0),
                dict(ctrl_tau=-0.5), dict(h_dim=-4), dict(precision_code=7), dict(reward_mode=5),
                dict(reward_mode=1, w_missing="w_rt"), dict(value_head=1, w_missing="w_val")):
        c = dict(cfg)
        if "precision_code" in bad:
            c["precision"] = "fp8"
            c2 = wm.wm_config(c["z_dim"], c["a_dim"], c["h_dim"], c["k_mix"], 7, 1.0, 0, 0, 1.0,
                              0, 0, 0, 0)
            h = C.c_void_p()
            keep = {k: np.ascontiguousarray(w[k], np.float32) for k in
                    ("W_lstm", "b_lstm", "W_mdn", "b_mdn", "w_rew", "w_done", "W_ctrl", "b_ctrl")}
            ws = wm.wm_weights(*[keep[k].ctypes.data if k in keep else 0.0 for k in
                                 ("W_lstm", "b_lstm", "W_mdn", "b_mdn", "w_rew")], 0.0,
                               keep["w_done"].ctypes.data, 0.0, keep["W_ctrl"].ctypes.data,
                               keep["b_ctrl"].ctypes.data)
            assert wm._lib.wm_create(C.byref(c2), C.byref(ws), C.byref(h)) == wm.WM_ERR_INVALID_ARG
            continue
        ww = dict(w)
        if "w_missing" in bad:
            ww[bad.pop("w_missing")] = None
        c.update(bad)
        with pytest.raises(wm.WMError) as ei:
            wm.wm_create(c, ww)
        assert ei.value.status == wm.WM_ERR_INVALID_ARG


def test_null_handle_calls_are_rejected():
    import paper_2205_01435_gb300 as pkg
    wm = pkg.load()
    assert wm._lib.wm_rollout(None, 1, 1, 0, 0, None, None) == wm.WM_ERR_INVALID_ARG
    assert wm._lib.wm_mdn_nll(None, 1, 1, *([None] * 8)) == wm.WM_ERR_INVALID_ARG
    assert wm._lib.wm_sync(None) == wm.WM_ERR_INVALID_ARG
    assert wm._lib.wm_set_controllers(None, 1, 1, None, None) == wm.WM_ERR_INVALID_ARG
    assert wm._lib.wm_returns(None, 1, 1, 0, 0.9, 1, *([None] * 6)) == wm.WM_ERR_INVALID_ARG
    assert wm._lib.wm_mdn_nll_backward(None, 1, 1, None, None, None, None, None, None) == wm.WM_ERR_INVALID_ARG
    assert wm._lib.wm_last_error(None) == b"null handle"
    wm._lib.wm_destroy(None)  # no-op
