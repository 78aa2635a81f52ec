"""ctypes binding of libhwr (include/hwr.h).

Argument marshalling only: every step of route scoring runs in the library's
CUDA kernels.  There is no fallback -- if the library has not been built, or
cannot be loaded, ``load()`` raises.

Low-level functions keep the C names (``hwr_create``, ``hwr_update_snapshot``,
``hwr_get_snapshot``, ``hwr_route_batch``, ``hwr_synchronize``,
``hwr_destroy``, ``hwr_status_string``, ``hwr_last_error``, ``hwr_get_stats``)
and take the same arguments (pointers as Python ints).  ``Router`` wraps one
context for numpy host arrays or CUDA tensors.
"""
from __future__ import annotations

import ctypes as ct
import os
import threading

import numpy as np

from . import build as _build

HWR_OK, HWR_ERR_INVALID_ARG, HWR_ERR_DTYPE, HWR_ERR_OOM = 0, 1, 2, 3
HWR_ERR_CUDA, HWR_ERR_TIMEOUT, HWR_ERR_STATE, HWR_ERR_UNSUPPORTED = 4, 5, 6, 7
HWR_F32, HWR_BF16 = 0, 1
HWR_SEQUENTIAL = 1 << 0
HWR_DEVICE_PTRS = 1 << 1
HWR_ASYNC = 1 << 2
HWR_SCORE_CONVEX = 1 << 3
HWR_PATH_SIMT = 1 << 4
HWR_PATH_TENSOR = 1 << 5
HWR_PROFILE = 1 << 6
KERNELS = ("snapshot", "route_simt", "seq_table", "qual_tc", "mlp_tc")
HWR_K_COUNT = len(KERNELS)

EXPORTS = ("hwr_create", "hwr_update_snapshot", "hwr_get_snapshot",
           "hwr_route_batch", "hwr_route_batch_slo", "hwr_route_batch_multi",
           "hwr_score_batch", "hwr_route_batch_noalloc", "hwr_synchronize",
           "hwr_destroy", "hwr_status_string", "hwr_last_error", "hwr_get_stats")
HWR_NOALLOC_MAX_Q = 32768


class hwr_deployment_table(ct.Structure):
    _fields_ = [("n_models", ct.c_int32), ("n_gpu_types", ct.c_int32),
                ("n_deployments", ct.c_int32), ("dep_model", ct.c_void_p),
                ("dep_gpu", ct.c_void_p), ("model_log10_params", ct.c_void_p)]


class hwr_predictor(ct.Structure):
    _fields_ = [("F", ct.c_int32), ("H1", ct.c_int32), ("H2", ct.c_int32),
                ("dtype", ct.c_int), ("W1", ct.c_void_p), ("W2", ct.c_void_p),
                ("W3", ct.c_void_p), ("b1", ct.c_void_p), ("b2", ct.c_void_p),
                ("b3", ct.c_void_p), ("feat_mean", ct.c_void_p),
                ("feat_std", ct.c_void_p), ("feat_xform", ct.c_void_p),
                ("n_heads", ct.c_int32)]


class hwr_snapshot(ct.Structure):
    _fields_ = [(n, ct.c_void_p) for n in
                ("running", "waiting", "kv_util", "gpu_util", "ttft_avg", "tpot_avg")]


class hwr_slo_spec(ct.Structure):
    _fields_ = [("budget", ct.c_void_p), ("ttft_a", ct.c_float), ("ttft_b", ct.c_float),
                ("slack", ct.c_float), ("tpot", ct.c_float)]


class hwr_stats(ct.Structure):
    _fields_ = [("queries_routed", ct.c_int64), ("kernel_launches", ct.c_int64),
                ("launches", ct.c_int64 * HWR_K_COUNT),
                ("profiled_launches", ct.c_int64 * HWR_K_COUNT),
                ("profiled_ms", ct.c_double * HWR_K_COUNT)]


class HwrError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{message} [{status}]")
        self.status = status


_lib = None
_lock = threading.Lock()


def lib_path() -> str:
    return _build.lib_path()


def load(path: str | None = None):
    """Load libhwr.  Raises if it is not built: no fallback path exists."""
    global _lib
    with _lock:
        if _lib is not None and path is None:
            return _lib
        p = path or lib_path()
        if not os.path.exists(p):
            raise RuntimeError(f"libhwr is not built ({p} missing); run "
                               "__graft_entry__.build() or paper_2608_14575_gb300/build.py")
        lib = ct.CDLL(p)
        P, I = ct.c_void_p, ct.c_int
        lib.hwr_create.argtypes = [P, P, P, ct.c_int32, I, P, ct.POINTER(P)]
        lib.hwr_update_snapshot.argtypes = [P, P]
        lib.hwr_get_snapshot.argtypes = [P, P]
        lib.hwr_route_batch.argtypes = [P, ct.c_int32, P, P, P, ct.c_float,
                                        ct.c_float, ct.c_uint32, P, P, P]
        lib.hwr_route_batch_noalloc.argtypes = lib.hwr_route_batch.argtypes
        lib.hwr_route_batch_slo.argtypes = [P, ct.c_int32, P, P, P, P, ct.c_float,
                                            ct.c_uint32, P, P, P]
        lib.hwr_route_batch_multi.argtypes = [P, ct.c_int32, P, P, P, ct.c_float, P,
                                              ct.c_int32, ct.c_uint32, P, P, P]
        lib.hwr_score_batch.argtypes = [P, ct.c_int32, P, P, P, ct.c_uint32, P, P]
        lib.hwr_synchronize.argtypes = [P]
        lib.hwr_destroy.argtypes = [P]
        lib.hwr_status_string.argtypes = [I]
        lib.hwr_status_string.restype = ct.c_char_p
        lib.hwr_last_error.argtypes = [P]
        lib.hwr_last_error.restype = ct.c_char_p
        lib.hwr_get_stats.argtypes = [P, P, I]
        for n in ("hwr_create", "hwr_update_snapshot", "hwr_get_snapshot",
                  "hwr_route_batch", "hwr_route_batch_slo", "hwr_route_batch_multi",
                  "hwr_score_batch", "hwr_route_batch_noalloc", "hwr_synchronize",
                  "hwr_destroy", "hwr_get_stats"):
            getattr(lib, n).restype = I
        if path is None:
            _lib = lib
        return lib


# ---- C names ----------------------------------------------------------------

def hwr_create(table, pred, model_emb, E, emb_dtype, stream, out):
    return load().hwr_create(table, pred, model_emb, E, emb_dtype, stream, out)


def hwr_update_snapshot(ctx, snap):
    return load().hwr_update_snapshot(ctx, snap)


def hwr_get_snapshot(ctx, running_out):
    return load().hwr_get_snapshot(ctx, running_out)


def hwr_route_batch(ctx, Q, in_len, out_len, q_emb, slo, lam, flags, chosen,
                    pred_latency, utility):
    return load().hwr_route_batch(ctx, Q, in_len, out_len, q_emb, slo, lam, flags,
                                  chosen, pred_latency, utility)


def hwr_route_batch_slo(ctx, Q, in_len, out_len, q_emb, slo, lam, flags, chosen,
                        pred_latency, utility):
    return load().hwr_route_batch_slo(ctx, Q, in_len, out_len, q_emb, slo, lam, flags,
                                      chosen, pred_latency, utility)


def hwr_route_batch_multi(ctx, Q, in_len, out_len, q_emb, slo, lambdas, K, flags, chosen,
                          pred_latency, utility):
    return load().hwr_route_batch_multi(ctx, Q, in_len, out_len, q_emb, slo, lambdas, K, flags,
                                        chosen, pred_latency, utility)


def hwr_score_batch(ctx, Q, in_len, out_len, q_emb, flags, cost, quality):
    return load().hwr_score_batch(ctx, Q, in_len, out_len, q_emb, flags, cost, quality)


def hwr_route_batch_noalloc(ctx, Q, in_len, out_len, q_emb, slo, lam, flags, chosen,
                            pred_latency, utility):
    return load().hwr_route_batch_noalloc(ctx, Q, in_len, out_len, q_emb, slo, lam, flags,
                                          chosen, pred_latency, utility)


def hwr_synchronize(ctx):
    return load().hwr_synchronize(ctx)


def hwr_destroy(ctx):
    return load().hwr_destroy(ctx)


def hwr_status_string(status):
    return load().hwr_status_string(status).decode()


def hwr_last_error(ctx):
    return load().hwr_last_error(ctx).decode()


def hwr_get_stats(ctx, out, reset):
    return load().hwr_get_stats(ctx, out, reset)


# ---- convenience wrapper ------------------------------------------------------

def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def _addr(a):
    """Address of a contiguous array's data.  Through the buffer protocol for
    writable non-empty arrays (about a third of the cost of ndarray.ctypes,
    which a small call pays several times), else through ndarray.ctypes."""
    try:
        return ct.addressof(ct.c_char.from_buffer(a))
    except (TypeError, ValueError):
        return a.ctypes.data


class Router:
    """One routing context built from a problem dict (see workload.gen).

    Host routing takes numpy arrays; device routing takes CUDA tensors (the
    context must then be created on the tensors' stream)."""

    def __init__(self, p: dict, stream: int | None = None):
        self.lib = load()
        self.p = p
        self.D, self.E = int(p["D"]), int(p["E"])
        self.bf16 = p["dtype"] == "bf16"
        self.wdt = np.uint16 if self.bf16 else np.float32
        keep = []

        def ptr(a, dt):
            a = _c(a, dt)
            keep.append(a)
            return a.ctypes.data

        t = hwr_deployment_table(int(p["M"]), int(p["G"]), int(p["D"]),
                                 ptr(p["dep_model"], np.int32),
                                 ptr(p["dep_gpu"], np.int32),
                                 ptr(p["log10p"], np.float32))
        pr = hwr_predictor(int(p["F"]), int(p["H1"]), int(p["H2"]),
                           HWR_BF16 if self.bf16 else HWR_F32,
                           ptr(p["W1"], self.wdt), ptr(p["W2"], self.wdt),
                           ptr(p["W3"], self.wdt), ptr(p["b1"], np.float32),
                           ptr(p["b2"], np.float32), ptr(p["b3"], np.float32),
                           ptr(p["mu"], np.float32), ptr(p["sd"], np.float32),
                           ptr(p["xform"], np.uint8), int(p.get("n_heads", 2)))
        ctx = ct.c_void_p()
        st = self.lib.hwr_create(ct.byref(t), ct.byref(pr), ptr(p["memb"], self.wdt),
                                 self.E, HWR_BF16 if self.bf16 else HWR_F32,
                                 stream, ct.byref(ctx))
        if st != HWR_OK:
            raise HwrError(st, self.lib.hwr_last_error(None).decode())
        self.ctx = ctx
        # snapshot staging: one persistent buffer whose six slices the
        # prebuilt hwr_snapshot points at, so an update copies six small
        # arrays instead of taking six pointers
        D = self.D
        self._snap_buf = np.empty(6 * D, np.uint32)
        b = self._snap_buf
        self._snap_views = (b[0:D].view(np.int32), b[D:2 * D].view(np.int32),
                            b[2 * D:3 * D].view(np.float32), b[3 * D:4 * D].view(np.float32),
                            b[4 * D:5 * D].view(np.float32), b[5 * D:6 * D].view(np.float32))
        base = b.ctypes.data
        self._snap_struct = hwr_snapshot(*[base + 4 * D * k for k in range(6)])
        self._snap_ref = ct.byref(self._snap_struct)
        self.update_snapshot(p["snap"])

    def _check(self, st):
        if st != HWR_OK:
            raise HwrError(st, self.lib.hwr_last_error(self.ctx).decode())

    def update_snapshot(self, snap: dict):
        shape = (self.D,)
        for v, name in zip(self._snap_views, ("running", "waiting", "kv", "gpu_util", "ttft", "tpot")):
            a = snap[name]
            if a.__class__ is not np.ndarray:
                a = np.asarray(a)
            if a.shape != shape:
                raise ValueError(f"snapshot {name}: shape {a.shape}, want {shape}")
            v[...] = a
        self._check(self.lib.hwr_update_snapshot(self.ctx, self._snap_ref))

    def get_snapshot(self) -> np.ndarray:
        out = np.empty(self.D, np.int32)
        self._check(self.lib.hwr_get_snapshot(self.ctx, _addr(out)))
        return out

    def route(self, in_len=None, out_len=None, emb=None, *, slo=None, lam=None,
              flags=0):
        """Host arrays in, host arrays out (chosen, latency, utility)."""
        p = self.p
        il = _c(p["in_len"] if in_len is None else in_len, np.float32)
        ol = _c(p["out_len"] if out_len is None else out_len, np.float32)
        em = _c(p["emb"] if emb is None else emb, self.wdt)
        Q = il.size
        # the three outputs as views of one allocation (one pointer to take)
        out = np.empty(3 * Q, np.uint32)
        o = _addr(out)
        self._check(self.lib.hwr_route_batch(
            self.ctx, Q, _addr(il), _addr(ol), _addr(em),
            float(p["slo"] if slo is None else slo),
            float(p["lam"] if lam is None else lam), int(flags) & ~HWR_DEVICE_PTRS,
            o, o + 4 * Q, o + 8 * Q))
        return out[:Q].view(np.int32), out[Q:2 * Q].view(np.float32), out[2 * Q:].view(np.float32)

    def score(self, in_len=None, out_len=None, emb=None, *, flags=0, quality=True):
        """Cost [Q][D] and quality [Q][M] (None unless `quality`) of a host batch."""
        p = self.p
        il = _c(p["in_len"] if in_len is None else in_len, np.float32)
        ol = _c(p["out_len"] if out_len is None else out_len, np.float32)
        em = _c(p["emb"] if emb is None else emb, self.wdt)
        Q = il.size
        cost = np.empty((Q, p["D"]), np.float32)
        qual = np.empty((Q, p["M"]), np.float32) if quality else None
        self._check(self.lib.hwr_score_batch(
            self.ctx, Q, _addr(il), _addr(ol), _addr(em),
            int(flags) & ~HWR_DEVICE_PTRS, _addr(cost),
            _addr(qual) if quality else None))
        return cost, qual

    def score_device(self, in_len, out_len, emb, cost, quality=None, *, flags=0):
        """Device scoring into CUDA tensors cost [Q][D] and quality [Q][M]."""
        self._check(self.lib.hwr_score_batch(
            self.ctx, int(in_len.numel()), in_len.data_ptr(), out_len.data_ptr(),
            emb.data_ptr(), int(flags) | HWR_DEVICE_PTRS, cost.data_ptr(),
            None if quality is None else quality.data_ptr()))

    def route_multi(self, lambdas, in_len=None, out_len=None, emb=None, *, slo=None,
                    flags=0):
        """Host routing for several lambdas; outputs have shape [K][Q]."""
        p = self.p
        il = _c(p["in_len"] if in_len is None else in_len, np.float32)
        ol = _c(p["out_len"] if out_len is None else out_len, np.float32)
        em = _c(p["emb"] if emb is None else emb, self.wdt)
        lam = _c(lambdas, np.float32)
        Q, K = il.size, lam.size
        chosen = np.empty((K, Q), np.int32)
        lat = np.empty((K, Q), np.float32)
        util = np.empty((K, Q), np.float32)
        self._check(self.lib.hwr_route_batch_multi(
            self.ctx, Q, _addr(il), _addr(ol), _addr(em),
            float(p["slo"] if slo is None else slo), _addr(lam), K,
            int(flags) & ~HWR_DEVICE_PTRS, _addr(chosen), _addr(lat),
            _addr(util)))
        return chosen, lat, util

    def route_device_multi(self, lambdas, in_len, out_len, emb, chosen, lat, util, *, slo,
                           flags=0):
        """Device routing for several lambdas into [K][Q] CUDA tensors."""
        lam = _c(lambdas, np.float32)
        self._check(self.lib.hwr_route_batch_multi(
            self.ctx, int(in_len.numel()), in_len.data_ptr(), out_len.data_ptr(),
            emb.data_ptr(), float(slo), _addr(lam), int(lam.size),
            int(flags) | HWR_DEVICE_PTRS, chosen.data_ptr(), lat.data_ptr(), util.data_ptr()))

    def route_slo(self, in_len=None, out_len=None, emb=None, *, budgets=None,
                  model=None, lam=None, flags=0):
        """Host routing with per-query budgets (array) or the Eq. 4-5 model
        (a, b, slack, tpot)."""
        p = self.p
        il = _c(p["in_len"] if in_len is None else in_len, np.float32)
        ol = _c(p["out_len"] if out_len is None else out_len, np.float32)
        em = _c(p["emb"] if emb is None else emb, self.wdt)
        Q = il.size
        spec, keep = self._spec(budgets, model, Q)
        out = np.empty(3 * Q, np.uint32)
        o = _addr(out)
        self._check(self.lib.hwr_route_batch_slo(
            self.ctx, Q, _addr(il), _addr(ol), _addr(em), ct.byref(spec),
            float(p["lam"] if lam is None else lam), int(flags) & ~HWR_DEVICE_PTRS,
            o, o + 4 * Q, o + 8 * Q))
        return out[:Q].view(np.int32), out[Q:2 * Q].view(np.float32), out[2 * Q:].view(np.float32)

    def route_device_slo(self, in_len, out_len, emb, chosen, lat, util, *, budgets=None,
                         model=None, lam, flags=0):
        """Device routing with per-query budgets (CUDA tensor) or the model."""
        spec = hwr_slo_spec(budgets.data_ptr() if budgets is not None else None,
                            *(model if model is not None else (0.0, 0.0, 1.0, 0.0)))
        self._check(self.lib.hwr_route_batch_slo(
            self.ctx, int(in_len.numel()), in_len.data_ptr(), out_len.data_ptr(),
            emb.data_ptr(), ct.byref(spec), float(lam), int(flags) | HWR_DEVICE_PTRS,
            chosen.data_ptr(), lat.data_ptr(), util.data_ptr()))

    @staticmethod
    def _spec(budgets, model, Q):
        if budgets is not None:
            b = _c(budgets, np.float32)
            assert b.size == Q
            return hwr_slo_spec(b.ctypes.data, 0.0, 0.0, 1.0, 0.0), b
        a, bb, slack, tpot = model
        return hwr_slo_spec(None, float(a), float(bb), float(slack), float(tpot)), None

    def route_host_ptrs(self, Q, in_len_ptr, out_len_ptr, emb_ptr, chosen_ptr,
                        lat_ptr, util_ptr, *, slo, lam, flags=0):
        """Host pointers (e.g. pinned tensors' data_ptr()) in and out."""
        self._check(self.lib.hwr_route_batch(
            self.ctx, int(Q), in_len_ptr, out_len_ptr, emb_ptr, float(slo),
            float(lam), int(flags) & ~HWR_DEVICE_PTRS, chosen_ptr, lat_ptr, util_ptr))

    def route_device(self, in_len, out_len, emb, chosen, lat, util, *, slo, lam,
                     flags=0):
        """CUDA tensors in and out, ordered on the context's stream."""
        self._check(self.lib.hwr_route_batch(
            self.ctx, int(in_len.numel()), in_len.data_ptr(), out_len.data_ptr(),
            emb.data_ptr(), float(slo), float(lam), int(flags) | HWR_DEVICE_PTRS,
            chosen.data_ptr(), lat.data_ptr(), util.data_ptr()))

    def route_device_noalloc(self, in_len, out_len, emb, chosen, lat, util, *, slo, lam,
                             flags=0):
        """As route_device, through hwr_route_batch_noalloc (no allocation)."""
        self._check(self.lib.hwr_route_batch_noalloc(
            self.ctx, int(in_len.numel()), in_len.data_ptr(), out_len.data_ptr(),
            emb.data_ptr(), float(slo), float(lam), int(flags) | HWR_DEVICE_PTRS,
            chosen.data_ptr(), lat.data_ptr(), util.data_ptr()))

    def synchronize(self):
        self._check(self.lib.hwr_synchronize(self.ctx))

    def stats(self, reset=False) -> dict:
        s = hwr_stats()
        self._check(self.lib.hwr_get_stats(self.ctx, ct.byref(s), int(reset)))
        return dict(queries_routed=s.queries_routed,
                    kernel_launches=s.kernel_launches,
                    launches={k: s.launches[i] for i, k in enumerate(KERNELS)},
                    profiled_launches={k: s.profiled_launches[i]
                                       for i, k in enumerate(KERNELS)},
                    profiled_ms={k: s.profiled_ms[i] for i, k in enumerate(KERNELS)})

    def close(self):
        if getattr(self, "ctx", None):
            self.lib.hwr_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
