"""Error paths of the C ABI on a GPU: every failure is a status, never a crash.

* HWR_TEST_FAIL_ALLOC=n fails the n-th allocation of hwr_create on the host;
  every n must give HWR_ERR_OOM and leave the process able to create the next
  context.
* Argument errors leave the context usable.
* A snapshot value outside the domain of its feature's transform (negative
  queue, non-finite value, <= 0 under log, <= -1 under log1p) is rejected and
  the previous snapshot stays in force.
* HWR_TEST_STALL=1 makes the tensor-path producers never signal their tiles,
  so the predictor kernel's bounded waits (about a second) run out: the call
  returns HWR_ERR_TIMEOUT, the context refuses further work (HWR_ERR_STATE),
  and a new context on the same device routes correctly -- the GPU is not
  faulted and nothing hangs.
"""
import ctypes as ct

import numpy as np
import pytest

import workload as W
import paper_2608_14575_gb300 as H
from paper_2608_14575_gb300 import _hwr

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def built():
    H.build()


def test_every_allocation_failure_is_reported(monkeypatch):
    p = W.make_config(1, Q=8)
    n, seen = 1, 0
    while True:
        monkeypatch.setenv("HWR_TEST_FAIL_ALLOC", str(n))
        try:
            r = H.Router(p)
        except H.HwrError as e:
            assert e.status == _hwr.HWR_ERR_OOM, e
            assert "test hook" in str(e)
            seen += 1
            n += 1
            continue
        r.close()
        break
    assert seen >= 20                      # every allocation of create was exercised
    monkeypatch.delenv("HWR_TEST_FAIL_ALLOC")
    r = H.Router(p)
    assert r.route()[0].shape == (8,)
    r.close()


def test_route_before_snapshot_and_argument_errors():
    lib = H.load()
    p = W.make_config(0, Q=4)
    keep = []

    def ptr(a, dt):
        a = np.ascontiguousarray(a, dtype=dt)
        keep.append(a)
        return a.ctypes.data
    t = _hwr.hwr_deployment_table(p["M"], p["G"], p["D"], ptr(p["dep_model"], np.int32),
                                  ptr(p["dep_gpu"], np.int32), ptr(p["log10p"], np.float32))
    pr = _hwr.hwr_predictor(p["F"], p["H1"], p["H2"], 0, ptr(p["W1"], np.float32),
                            ptr(p["W2"], np.float32), ptr(p["W3"], np.float32),
                            ptr(p["b1"], np.float32), ptr(p["b2"], np.float32),
                            ptr(p["b3"], np.float32), ptr(p["mu"], np.float32),
                            ptr(p["sd"], np.float32), ptr(p["xform"], np.uint8))
    ctx = ct.c_void_p()
    assert lib.hwr_create(ct.byref(t), ct.byref(pr), ptr(p["memb"], np.float32), p["E"], 0,
                          None, ct.byref(ctx)) == 0
    il, ol, em = (ptr(p["in_len"], np.float32), ptr(p["out_len"], np.float32),
                  ptr(p["emb"], np.float32))
    ch, lat, ut = np.empty(4, np.int32), np.empty(4, np.float32), np.empty(4, np.float32)
    args = (il, ol, em, 5.0, 0.5)
    outs = (ch.ctypes.data, lat.ctypes.data, ut.ctypes.data)
    assert lib.hwr_route_batch(ctx, 4, *args, 0, *outs) == _hwr.HWR_ERR_INVALID_ARG
    assert "snapshot" in H.hwr_last_error(ctx)
    s = p["snap"]
    snap = _hwr.hwr_snapshot(*(ptr(s[k], dt) for k, dt in (
        ("running", np.int32), ("waiting", np.int32), ("kv", np.float32),
        ("gpu_util", np.float32), ("ttft", np.float32), ("tpot", np.float32))))
    assert lib.hwr_update_snapshot(ctx, ct.byref(snap)) == 0
    assert lib.hwr_route_batch(ctx, 0, None, None, None, 5.0, 0.5, 0, None, None, None) == 0
    assert lib.hwr_route_batch(ctx, -1, *args, 0, *outs) == _hwr.HWR_ERR_INVALID_ARG
    assert lib.hwr_route_batch(ctx, 4, *args, 1 << 12, *outs) == _hwr.HWR_ERR_INVALID_ARG
    assert lib.hwr_route_batch(ctx, 4, *args, H.HWR_PATH_SIMT | H.HWR_PATH_TENSOR,
                               *outs) == _hwr.HWR_ERR_INVALID_ARG
    assert lib.hwr_route_batch(ctx, 4, il, ol, em, float("nan"), 0.5, 0,
                               *outs) == _hwr.HWR_ERR_INVALID_ARG
    assert lib.hwr_route_batch(ctx, 4, il, ol, em, 5.0, float("inf"), 0,
                               *outs) == _hwr.HWR_ERR_INVALID_ARG
    assert lib.hwr_route_batch(ctx, 4, None, ol, em, 5.0, 0.5, 0, *outs) == _hwr.HWR_ERR_INVALID_ARG
    assert lib.hwr_route_batch_noalloc(ctx, 4, *args, 0, *outs) == _hwr.HWR_ERR_UNSUPPORTED
    assert lib.hwr_route_batch(ctx, 4, *args, 0, *outs) == 0      # still usable
    assert ch.min() >= 0
    assert lib.hwr_destroy(ctx) == 0


def test_sequential_tensor_needs_a_bf16_context():
    p = W.make_config(2, Q=100)            # fp32: no tensor-core path
    r = H.Router(p)
    with pytest.raises(H.HwrError) as e:
        r.route(flags=H.HWR_SEQUENTIAL | H.HWR_PATH_TENSOR)
    assert e.value.status == _hwr.HWR_ERR_UNSUPPORTED
    assert r.route(flags=H.HWR_SEQUENTIAL)[0].shape == (100,)     # still usable
    r.close()


def test_bounded_wait_expires_into_timeout_status(monkeypatch):
    p = W.make_config(1, Q=1024)
    monkeypatch.setenv("HWR_TEST_STALL", "1")
    r = H.Router(p)
    monkeypatch.delenv("HWR_TEST_STALL")
    with pytest.raises(H.HwrError) as e:
        r.route(flags=H.HWR_PATH_TENSOR)
    assert e.value.status == _hwr.HWR_ERR_TIMEOUT
    with pytest.raises(H.HwrError) as e:
        r.route()
    assert e.value.status == _hwr.HWR_ERR_STATE
    r.close()
    # the device is healthy: a new context routes and matches the SIMT path
    r = H.Router(p)
    tc = r.route(flags=H.HWR_PATH_TENSOR)
    simt = r.route(flags=H.HWR_PATH_SIMT)
    same = tc[0] == simt[0]
    assert same.mean() > 0.95
    r.close()


@pytest.mark.parametrize("key,value", [("running", -1), ("waiting", -2), ("kv", np.nan),
                                       ("gpu_util", np.inf), ("ttft", 0.0), ("tpot", -1e-3)])
def test_snapshot_values_outside_their_domain_are_rejected(key, value):
    p = W.make_config(0, Q=32)
    r = H.Router(p)
    want = r.route()
    bad = {k: np.array(v, copy=True) for k, v in p["snap"].items()}
    bad[key][1] = value
    with pytest.raises(H.HwrError) as e:
        r.update_snapshot(bad)
    assert e.value.status == _hwr.HWR_ERR_INVALID_ARG, e.value
    assert "[1]" in str(e.value)
    # the context keeps its previous snapshot and routes as before
    got = r.route()
    assert all(np.array_equal(a, b) for a, b in zip(got, want))
    r.close()


def test_log1p_slot_accepts_values_above_minus_one_only():
    p = W.make_config(0, Q=8)
    P = p["M"] + p["G"]
    p["xform"] = np.array(p["xform"], copy=True)
    p["xform"][P + 3] = 1                  # KV utilisation through log1p
    r = H.Router(p)
    snap = {k: np.array(v, copy=True) for k, v in p["snap"].items()}
    snap["kv"][0] = -0.5                   # log1p(-0.5) is defined
    r.update_snapshot(snap)
    snap["kv"][0] = -1.0
    with pytest.raises(H.HwrError) as e:
        r.update_snapshot(snap)
    assert e.value.status == _hwr.HWR_ERR_INVALID_ARG and "log1p" in str(e.value)
    assert r.route()[0].min() >= 0
    r.close()
