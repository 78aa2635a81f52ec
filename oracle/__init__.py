"""CPU oracle for HW-Router route scoring -- TEST INFRASTRUCTURE ONLY.

Only tests/, ``__graft_entry__.smoke()`` and bench.py's CPU-baseline leg may
import this package.  The library (``paper_2608_14575_gb300``) never does, and
this package never imports the library: the two share no code.

The arithmetic lives in ``hwr_oracle.c`` (plain C loops, see its header for the
definition and the two numeric modes).  This module only compiles it with gcc,
loads it with ctypes and marshals numpy arrays in and out.

Parity status of each function (what pins it, in tests/test_oracle_pins.py and
tests/test_oracle_mutants.py):
  features / predict / route   closed-form hand weights, invariants, brute force
  quality                      numpy.matmul in fp64 and sigmoid special values
  select                       brute-force enumeration on tiny inputs
  sequential mode              reduces to batch mode (Q = 1, zero running weight)
No function is left unpinned.
"""
from __future__ import annotations

import ctypes as ct
import os
import platform
import subprocess
import threading

import numpy as np

F64, F32 = 0, 1
_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "hwr_oracle.c")
_lock = threading.Lock()
_lib = None


def _so_path(src=_SRC, tag="oracle"):
    return os.path.join(_HERE, "_build", f"lib{tag}_{platform.machine()}.so")


def build(src: str = _SRC, out: str | None = None, extra=()) -> str:
    """Compile the oracle with gcc (no fast-math, no FP contraction)."""
    out = out or _so_path(src)
    os.makedirs(os.path.dirname(out), exist_ok=True)
    flags = ["-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off",
             "-fno-fast-math", "-fopenmp"]
    if platform.machine() in ("x86_64", "AMD64"):
        flags.append("-mfma")  # fmaf as one instruction; results are identical
    cmd = ["gcc", *flags, *extra, src, "-o", out + ".tmp", "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(out + ".tmp", out)
    return out


def load(path: str | None = None, rebuild: bool = False):
    """Load (building if needed) the oracle shared library."""
    global _lib
    with _lock:
        if path is None and _lib is not None and not rebuild:
            return _lib
        p = path or _so_path()
        if rebuild or not os.path.exists(p) or (
                path is None and os.path.getmtime(p) < os.path.getmtime(_SRC)):
            build(out=p)
        lib = ct.CDLL(p)
        _declare(lib)
        if path is None:
            _lib = lib
        return lib


class _Model(ct.Structure):
    _fields_ = [(n, ct.c_int32) for n in ("M", "G", "D", "F", "H1", "H2", "E", "n_heads")] + [
        ("dep_model", ct.c_void_p), ("dep_gpu", ct.c_void_p),
        ("log10p", ct.c_void_p), ("W1", ct.c_void_p), ("b1", ct.c_void_p),
        ("W2", ct.c_void_p), ("b2", ct.c_void_p), ("W3", ct.c_void_p),
        ("b3", ct.c_void_p), ("mu", ct.c_void_p), ("sd", ct.c_void_p),
        ("xform", ct.c_void_p), ("memb", ct.c_void_p)]


class _Snap(ct.Structure):
    _fields_ = [(n, ct.c_void_p) for n in
                ("running", "waiting", "kv", "gpu_util", "ttft", "tpot")]


def _declare(lib):
    P, I, F, D_ = ct.c_void_p, ct.c_int, ct.c_float, ct.c_double
    lib.orc_route.argtypes = [P, P, ct.c_int32, P, P, P, I, F, F, I, I, I, P,
                              P, P, P, I]
    lib.orc_route.restype = I
    lib.orc_score_all.argtypes = [P, P, ct.c_int32, P, P, P, I, F, I, I, P, P, I]
    lib.orc_route_q.argtypes = [P, P, ct.c_int32, P, P, P, I, P, F, I, I, I, P, P, P, P, I]
    lib.orc_route_q.restype = I
    lib.orc_slo_budget.argtypes = [F, F, F, F, F, F, I]
    lib.orc_slo_budget.restype = D_
    lib.orc_score_all.restype = I
    lib.orc_features.argtypes = [P, P, I, F, F, I, P]
    lib.orc_predict.argtypes = [P, P, I, P, P, P]
    lib.orc_quality.argtypes = [P, P, I, ct.c_size_t, I, P]
    lib.orc_select.argtypes = [I, P, P, D_, I]
    lib.orc_select.restype = I
    for n in ("orc_softplus_f64", "orc_sigmoid_f64"):
        getattr(lib, n).argtypes = [D_]
        getattr(lib, n).restype = D_
    for n in ("orc_softplus_f32", "orc_sigmoid_f32"):
        getattr(lib, n).argtypes = [F]
        getattr(lib, n).restype = F


def _widen(a):
    """bf16 bit patterns (uint16) -> float32; float32 passes through."""
    a = np.asarray(a)
    if a.dtype == np.uint16:
        return (a.astype(np.uint32) << 16).view(np.float32)
    return np.ascontiguousarray(a, dtype=np.float32)


class Problem:
    """ctypes views of one problem dict (see workload.gen.make_problem)."""

    def __init__(self, p: dict, snap: dict | None = None, lib=None):
        self.lib = lib or load()
        self.p = p
        keep = []

        def arr(a, dt):
            a = np.ascontiguousarray(a, dtype=dt)
            keep.append(a)
            return a.ctypes.data

        m = _Model()
        for n in ("M", "G", "D", "F", "H1", "H2", "E"):
            setattr(m, n, int(p[n]))
        m.n_heads = int(p.get("n_heads", 2))
        m.dep_model = arr(p["dep_model"], np.int32)
        m.dep_gpu = arr(p["dep_gpu"], np.int32)
        m.log10p = arr(p["log10p"], np.float32)
        for n in ("W1", "W2", "W3", "memb"):
            setattr(m, n, arr(_widen(p[n]), np.float32))
        for n in ("b1", "b2", "b3", "mu", "sd"):
            setattr(m, n, arr(p[n], np.float32))
        m.xform = arr(p["xform"], np.uint8)
        self.model = m
        self._keep = keep
        self.set_snapshot(snap if snap is not None else p["snap"])

    def set_snapshot(self, snap: dict):
        s = _Snap()
        self._snap_arrays = []
        for n, dt in (("running", np.int32), ("waiting", np.int32),
                      ("kv", np.float32), ("gpu_util", np.float32),
                      ("ttft", np.float32), ("tpot", np.float32)):
            a = np.ascontiguousarray(snap[n], dtype=dt)
            self._snap_arrays.append(a)
            setattr(s, n, a.ctypes.data)
        self.snap = s

    # -- queries -------------------------------------------------------
    @staticmethod
    def _queries(in_len, out_len, emb):
        il = np.ascontiguousarray(in_len, dtype=np.float32)
        ol = np.ascontiguousarray(out_len, dtype=np.float32)
        emb = np.asarray(emb)
        if emb.dtype == np.uint16:
            e, bf = np.ascontiguousarray(emb), 1
        else:
            e, bf = np.ascontiguousarray(emb, dtype=np.float32), 0
        return il, ol, e, bf

    def route(self, in_len=None, out_len=None, emb=None, *, slo=None, lam=None,
              mode=F64, sequential=False, convex=False, running=None,
              nthreads=1):
        """Route a batch. Returns (chosen int32, latency f64, utility f64, running)."""
        p = self.p
        il, ol, e, bf = self._queries(p["in_len"] if in_len is None else in_len,
                                      p["out_len"] if out_len is None else out_len,
                                      p["emb"] if emb is None else emb)
        Q = il.size
        slo = p["slo"] if slo is None else slo
        lam = p["lam"] if lam is None else lam
        run = np.array(self._snap_arrays[0] if running is None else running,
                       dtype=np.int32, copy=True)
        chosen = np.empty(Q, np.int32)
        lat = np.empty(Q, np.float64)
        util = np.empty(Q, np.float64)
        rc = self.lib.orc_route(ct.byref(self.model), ct.byref(self.snap), Q,
                                il.ctypes.data, ol.ctypes.data, e.ctypes.data,
                                bf, float(slo), float(lam), int(convex),
                                int(mode), int(sequential), run.ctypes.data,
                                chosen.ctypes.data, lat.ctypes.data,
                                util.ctypes.data, int(nthreads))
        if rc != 0:
            raise MemoryError("oracle allocation failed")
        return chosen, lat, util, run

    def route_slo(self, slo_q, in_len=None, out_len=None, emb=None, *, lam=None,
                  mode=F64, sequential=False, convex=False, running=None):
        """Route with one SLO budget per query (float32 array of length Q)."""
        p = self.p
        il, ol, e, bf = self._queries(p["in_len"] if in_len is None else in_len,
                                      p["out_len"] if out_len is None else out_len,
                                      p["emb"] if emb is None else emb)
        Q = il.size
        sq = np.ascontiguousarray(slo_q, dtype=np.float32)
        assert sq.size == Q
        lam = p["lam"] if lam is None else lam
        run = np.array(self._snap_arrays[0] if running is None else running,
                       dtype=np.int32, copy=True)
        chosen = np.empty(Q, np.int32)
        lat = np.empty(Q, np.float64)
        util = np.empty(Q, np.float64)
        rc = self.lib.orc_route_q(ct.byref(self.model), ct.byref(self.snap), Q,
                                  il.ctypes.data, ol.ctypes.data, e.ctypes.data, bf,
                                  sq.ctypes.data, float(lam), int(convex), int(mode),
                                  int(sequential), run.ctypes.data, chosen.ctypes.data,
                                  lat.ctypes.data, util.ctypes.data, 1)
        if rc != 0:
            raise MemoryError("oracle allocation failed")
        return chosen, lat, util, run

    def score_all(self, in_len=None, out_len=None, emb=None, *, lam=None,
                  mode=F64, convex=False, nthreads=1):
        """Latency and utility of every (query, deployment) pair, [Q][D]."""
        p = self.p
        il, ol, e, bf = self._queries(p["in_len"] if in_len is None else in_len,
                                      p["out_len"] if out_len is None else out_len,
                                      p["emb"] if emb is None else emb)
        Q, D = il.size, p["D"]
        lam = p["lam"] if lam is None else lam
        C = np.empty((Q, D), np.float64)
        U = np.empty((Q, D), np.float64)
        rc = self.lib.orc_score_all(ct.byref(self.model), ct.byref(self.snap),
                                    Q, il.ctypes.data, ol.ctypes.data,
                                    e.ctypes.data, bf, float(lam), int(convex),
                                    int(mode), C.ctypes.data, U.ctypes.data,
                                    int(nthreads))
        if rc != 0:
            raise MemoryError("oracle allocation failed")
        return C, U

    def features(self, d, in_len, out_len, mode=F64):
        x = np.empty(self.p["F"], np.float64)
        self.lib.orc_features(ct.byref(self.model), ct.byref(self.snap), int(d),
                              float(in_len), float(out_len), int(mode),
                              x.ctypes.data)
        return x

    def predict(self, x, mode=F64, heads=False):
        """(TTFT, TPOT), or (TTFT, TPOT, N_out) with heads=True."""
        x = np.ascontiguousarray(x, dtype=np.float64)
        a, b, c = ct.c_double(), ct.c_double(), ct.c_double()
        self.lib.orc_predict(ct.byref(self.model), x.ctypes.data, int(mode),
                             ct.byref(a), ct.byref(b), ct.byref(c))
        return (a.value, b.value, c.value) if heads else (a.value, b.value)

    def quality(self, emb_row, mode=F64):
        e = np.asarray(emb_row)
        bf = 1 if e.dtype == np.uint16 else 0
        e = np.ascontiguousarray(e, dtype=np.uint16 if bf else np.float32)
        out = np.empty(self.p["M"], np.float64)
        self.lib.orc_quality(ct.byref(self.model), e.ctypes.data, bf, 0,
                             int(mode), out.ctypes.data)
        return out


def slo_budget(a, b, slack, tpot_slo, in_len, out_len, mode=F64, lib=None):
    """Per-query SLO budgets of Eq. 4-5 (one value per query)."""
    lib = lib or load()
    il = np.asarray(in_len, np.float32).ravel()
    ol = np.asarray(out_len, np.float32).ravel()
    return np.array([lib.orc_slo_budget(float(a), float(b), float(slack), float(tpot_slo),
                                        float(x), float(y), int(mode))
                     for x, y in zip(il, ol)])


def select(C, U, slo, mode=F64, lib=None):
    lib = lib or load()
    C = np.ascontiguousarray(C, dtype=np.float64)
    U = np.ascontiguousarray(U, dtype=np.float64)
    return lib.orc_select(int(C.size), C.ctypes.data, U.ctypes.data, float(slo),
                          int(mode))


def softplus(z, mode=F64, lib=None):
    lib = lib or load()
    return lib.orc_softplus_f64(z) if mode == F64 else lib.orc_softplus_f32(z)


def sigmoid(s, mode=F64, lib=None):
    lib = lib or load()
    return lib.orc_sigmoid_f64(s) if mode == F64 else lib.orc_sigmoid_f32(s)
