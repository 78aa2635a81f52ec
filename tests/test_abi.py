"""The C-ABI library loads and behaves at its boundary without a GPU.

No compute call is made here: only symbol lookup, status strings and the
argument validation that hwr_create / hwr_route_batch perform before touching
the device.
"""
import ctypes as ct
import os
import re
import subprocess

import numpy as np
import pytest

import paper_2608_14575_gb300 as H
from paper_2608_14575_gb300 import _hwr

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    H.build()
    return H.load()


def header_functions():
    text = open(os.path.join(ROOT, "include", "hwr.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(hwr_[a-z_]+)\s*\(", text)))


def test_every_declared_function_is_exported(lib):
    names = header_functions()
    assert len(names) >= 9, names
    out = subprocess.run(["nm", "-D", "--defined-only", H.lib_path()],
                         capture_output=True, text=True, check=True).stdout
    exported = set(l.split()[-1] for l in out.splitlines() if l.strip())
    for n in names:
        assert n in exported, n
        assert hasattr(lib, n)
    assert set(_hwr.EXPORTS) == set(names)


def test_status_strings(lib):
    for s in range(8):
        assert H.hwr_status_string(s)
    assert "unknown" in H.hwr_status_string(99)


def _structs(p):
    keep = []

    def ptr(a, dt):
        a = np.ascontiguousarray(a, dtype=dt)
        keep.append(a)
        return a.ctypes.data
    wdt = np.uint16 if p["dtype"] == "bf16" else np.float32
    t = _hwr.hwr_deployment_table(p["M"], p["G"], p["D"], ptr(p["dep_model"], np.int32),
                                  ptr(p["dep_gpu"], np.int32), ptr(p["log10p"], np.float32))
    pr = _hwr.hwr_predictor(p["F"], p["H1"], p["H2"], 1 if p["dtype"] == "bf16" else 0,
                            ptr(p["W1"], wdt), ptr(p["W2"], wdt), ptr(p["W3"], wdt),
                            ptr(p["b1"], np.float32), ptr(p["b2"], np.float32),
                            ptr(p["b3"], np.float32), ptr(p["mu"], np.float32),
                            ptr(p["sd"], np.float32), ptr(p["xform"], np.uint8))
    memb = ptr(p["memb"], wdt)
    return t, pr, memb, keep


def _create(lib, t, pr, memb, E, dt):
    ctx = ct.c_void_p(123)
    st = lib.hwr_create(ct.byref(t) if t is not None else None,
                        ct.byref(pr) if pr is not None else None, memb, E, dt, None,
                        ct.byref(ctx))
    return st, ctx


def test_create_validation(lib):
    import workload as W
    p = W.make_config(0, Q=4)
    t, pr, memb, keep = _structs(p)
    st, ctx = _create(lib, None, pr, memb, p["E"], 0)
    assert st == _hwr.HWR_ERR_INVALID_ARG and ctx.value is None
    assert "NULL" in H.hwr_last_error(None)
    st, _ = _create(lib, t, pr, memb, p["E"], 1)          # dtype mismatch
    assert st == _hwr.HWR_ERR_DTYPE
    st, _ = _create(lib, t, pr, memb, 63, 0)              # E % 8
    assert st == _hwr.HWR_ERR_INVALID_ARG
    pr.F = 8                                              # F < M + G + 9
    st, _ = _create(lib, t, pr, memb, p["E"], 0)
    assert st == _hwr.HWR_ERR_INVALID_ARG
    pr.F = p["F"]
    pr.H2 = 512
    st, _ = _create(lib, t, pr, memb, p["E"], 0)
    assert st == _hwr.HWR_ERR_UNSUPPORTED
    pr.H2 = p["H2"]
    bad = np.array([0, 5, 0, 1], np.int32)                # model id out of range
    t.dep_model = bad.ctypes.data
    st, _ = _create(lib, t, pr, memb, p["E"], 0)
    assert st == _hwr.HWR_ERR_INVALID_ARG
    t.dep_model = keep[0].ctypes.data
    sd = np.array(p["sd"], np.float32)
    sd[3] = 0.0
    pr.feat_std = sd.ctypes.data
    st, _ = _create(lib, t, pr, memb, p["E"], 0)
    assert st == _hwr.HWR_ERR_INVALID_ARG and "std" in H.hwr_last_error(None)


def test_calls_on_null_context(lib):
    assert lib.hwr_update_snapshot(None, None) == _hwr.HWR_ERR_INVALID_ARG
    assert lib.hwr_get_snapshot(None, None) == _hwr.HWR_ERR_INVALID_ARG
    assert lib.hwr_route_batch(None, 1, None, None, None, 1.0, 0.5, 0,
                               None, None, None) == _hwr.HWR_ERR_INVALID_ARG
    assert lib.hwr_synchronize(None) == _hwr.HWR_ERR_INVALID_ARG
    assert lib.hwr_destroy(None) == _hwr.HWR_OK


def test_binding_fails_loudly_without_library(tmp_path):
    with pytest.raises(RuntimeError, match="not built"):
        _hwr.load(str(tmp_path / "missing.so"))


def test_binding_address_helper_matches_ndarray_ctypes():
    # the binding takes data addresses through the buffer protocol where it
    # can; it must give the same address as ndarray.ctypes in every case
    from paper_2608_14575_gb300._hwr import _addr
    a = np.arange(12, dtype=np.float32).reshape(3, 4)
    cases = [a, a[1:], a[2], np.zeros((2, 8), np.uint16)[1],
             np.frombuffer(b"abcdabcd", dtype=np.float32),      # read-only
             np.empty(0, np.float32)]                          # empty
    for x in cases:
        assert _addr(x) == x.ctypes.data
