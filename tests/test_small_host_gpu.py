"""Small synchronous calls with host buffers (the small-batch kernel, and
sequential routes on the SIMT kernels).

Such a call stages its inputs in mapped host memory and, instead of
synchronising the stream, waits for the kernel to write each query's chosen
deployment (stored last, with release semantics at system scope).  Two
fallbacks must give the same results as that fast path:
* when the wait runs out (its limit, HWR_TEST_POLL_US, set to 0 here) the call
  synchronises the stream and reads the outputs;
* when earlier work is still queued on the stream (an HWR_ASYNC route), the
  call synchronises instead of spinning on outputs the kernel has not begun.
Results are compared bit for bit with the oracle's canonical fp32 order.
"""
import numpy as np
import pytest

import oracle as O
import workload as W
import paper_2608_14575_gb300 as H
from tc_check import check_against_oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    H.build()


def _exact(got, p):
    want = O.Problem(p).route(mode=O.F32)
    assert np.array_equal(got[0], want[0])
    assert np.array_equal(got[1], want[1].astype(np.float32))
    assert np.array_equal(got[2], want[2].astype(np.float32))


@pytest.mark.parametrize("Q", [1, 16])
def test_wait_limit_zero_takes_the_synchronising_path(monkeypatch, Q):
    monkeypatch.setenv("HWR_TEST_POLL_US", "0")
    p = W.make_config(4, Q=Q)              # D = 32: Q * D <= 768 pairs
    r = H.Router(p)
    monkeypatch.delenv("HWR_TEST_POLL_US")
    for _ in range(3):
        _exact(r.route(), p)
    r.close()


def test_small_call_queued_behind_an_async_route():
    p = W.make_config(4, Q=8192)           # a tensor-path batch, then one query
    r = H.Router(p)
    big = r.route(flags=H.HWR_ASYNC)
    one = r.route(p["in_len"][:1], p["out_len"][:1], p["emb"][:1])
    _exact(one, W.query_slice(p, 0, 1))
    r.synchronize()
    check_against_oracle(p, big, idx=np.arange(0, p["Q"], 17))
    # with the stream idle again, the next small call takes the fast path
    _exact(r.route(p["in_len"][:4], p["out_len"][:4], p["emb"][:4]), W.query_slice(p, 0, 4))
    r.close()


@pytest.mark.parametrize("no_ats", ["0", "1"])
def test_staged_and_direct_host_paths_agree(monkeypatch, no_ats):
    """Where the GPU reaches pageable host memory (address translation over the
    CPU-GPU link), small synchronous calls read the caller's arrays and write
    its outputs directly; HWR_TEST_NO_ATS=1 forces the pinned staging copies.
    Both give the oracle's canonical results, batch and sequential."""
    monkeypatch.setenv("HWR_TEST_NO_ATS", no_ats)
    p = W.make_config(4, Q=8)
    r = H.Router(p)
    _exact(r.route(), p)
    r.close()
    p = W.make_config(2, Q=64)
    r = H.Router(p)
    got = r.route(flags=H.HWR_SEQUENTIAL)
    want = O.Problem(p).route(mode=O.F32, sequential=True)
    assert np.array_equal(got[0], want[0])
    assert np.array_equal(got[1], want[1].astype(np.float32))
    assert np.array_equal(r.get_snapshot(), want[3])
    r.close()


def _exact_seq(got, r, p):
    want = O.Problem(p).route(mode=O.F32, sequential=True)
    assert np.array_equal(got[0], want[0])
    assert np.array_equal(got[1], want[1].astype(np.float32))
    assert np.array_equal(got[2], want[2].astype(np.float32))
    assert np.array_equal(r.get_snapshot(), want[3])


@pytest.mark.parametrize("poll_us", [None, "0"])
@pytest.mark.parametrize("cfg,Q", [(2, 64), (4, 64)])
def test_sequential_calls_wait_on_outputs_or_synchronise(monkeypatch, poll_us, cfg, Q):
    """A small sequential call returns once the chain has written every
    output (the default) or, with the wait limit at 0, after synchronising the
    stream; both give the canonical results and the persisted counts.  At
    D = 32 a 64-query call spans two chunks, whose chains write disjoint parts
    of the outputs."""
    if poll_us is not None:
        monkeypatch.setenv("HWR_TEST_POLL_US", poll_us)
    p = W.make_config(cfg, Q=Q)
    r = H.Router(p)
    for _ in range(2):
        r.update_snapshot(p["snap"])
        _exact_seq(r.route(flags=H.HWR_SEQUENTIAL), r, p)
    r.close()


def test_sequential_call_queued_behind_an_async_route():
    p = W.make_config(4, Q=8192)
    r = H.Router(p)
    big = r.route(flags=H.HWR_ASYNC)
    got = r.route(p["in_len"][:16], p["out_len"][:16], p["emb"][:16], flags=H.HWR_SEQUENTIAL)
    r.synchronize()
    check_against_oracle(p, big, idx=np.arange(0, p["Q"], 17))
    _exact_seq(got, r, W.query_slice(p, 0, 16))
    r.close()
