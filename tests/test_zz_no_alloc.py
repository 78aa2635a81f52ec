"""hwr_route_batch_noalloc: routing with no allocation at call time.

For callers that cannot allocate GPU memory while they route (a router inside
an LLM serving process whose engine reserved nearly all of HBM for its KV
cache, or a serving loop that must not take cudaMalloc's device-wide
synchronisation).  The call must give the same decisions as hwr_route_batch
on the same inputs -- on two calls in a row, with different batches, so that
what the first call leaves in the shared scratch cannot leak into the second
-- and agree with the fp64 oracle within the tensor path's tolerance; it must
not allocate, and must reject batches larger than its fixed scratch.

Collected last on purpose (file name), so a run that stops at the first
failure has run every other test before this one.
"""
import numpy as np
import pytest

import workload as W
import paper_2608_14575_gb300 as H
from tc_check import check_against_oracle

pytestmark = pytest.mark.gpu
TOL = 2e-2


def _dev(p, lo, hi, dev):
    import torch
    return (torch.from_numpy(p["in_len"][lo:hi]).to(dev),
            torch.from_numpy(p["out_len"][lo:hi]).to(dev),
            torch.from_numpy(p["emb"][lo:hi].view(np.int16)).to(dev))


def _outs(n, dev):
    import torch
    return (torch.empty(n, dtype=torch.int32, device=dev),
            torch.empty(n, dtype=torch.float32, device=dev),
            torch.empty(n, dtype=torch.float32, device=dev))


def _close(a, b):
    ch, lat, ut = (x.cpu().numpy() for x in a)
    wch, wlat, wut = (x.cpu().numpy() for x in b)
    assert np.array_equal(ch, wch)
    assert np.all(np.abs(lat - wlat) <= TOL * np.maximum(np.abs(wlat), 1e-3))
    assert np.all(np.abs(ut - wut) <= TOL * np.maximum(np.abs(wut), 1.0))


def test_noalloc_matches_route_batch_on_two_calls():
    import torch
    H.build()
    dev = torch.device("cuda:0")
    p = W.make_config(3, Q=30_000)
    r = H.Router(p, stream=torch.cuda.current_stream().cuda_stream)
    for lo, hi in ((0, 20_000), (20_000, 30_000)):       # two calls, different batches
        inp = _dev(p, lo, hi, dev)
        ref = _outs(hi - lo, dev)
        r.route_device(*inp, *ref, slo=p["slo"], lam=p["lam"], flags=H.HWR_PATH_TENSOR)
        got = _outs(hi - lo, dev)
        r.route_device_noalloc(*inp, *got, slo=p["slo"], lam=p["lam"])
        torch.cuda.synchronize()
        _close(got, ref)
        # and against the oracle, on every 13th query of the batch
        full = [np.zeros(p["Q"], dt) for dt in (np.int32, np.float32, np.float32)]
        for f, x in zip(full, got):
            f[lo:hi] = x.cpu().numpy()
        check_against_oracle(p, full, idx=np.arange(lo, hi, 13))
    r.close()


def test_route_reading_noalloc_outputs_waits_for_them():
    """A normal route queued right behind an allocation-free one, reading
    that call's latencies as its output lengths, must see them complete."""
    import torch
    H.build()
    dev = torch.device("cuda:0")
    p = W.make_config(4, Q=4096)
    r = H.Router(p, stream=torch.cuda.current_stream().cuda_stream)
    il, ol, em = _dev(p, 0, p["Q"], dev)
    o1, o2 = _outs(p["Q"], dev), _outs(p["Q"], dev)
    for _ in range(3):
        r.route_device_noalloc(il, ol, em, *o1, slo=p["slo"], lam=p["lam"], flags=H.HWR_ASYNC)
        r.route_device(il, o1[1], em, *o2, slo=p["slo"], lam=p["lam"],
                       flags=H.HWR_PATH_TENSOR | H.HWR_ASYNC)
    r.synchronize()
    lat1 = o1[1].clone()
    o3 = _outs(p["Q"], dev)
    r.route_device(il, lat1, em, *o3, slo=p["slo"], lam=p["lam"], flags=H.HWR_PATH_TENSOR)
    torch.cuda.synchronize()
    for a, b in zip(o2, o3):
        assert np.array_equal(a.cpu().numpy(), b.cpu().numpy(), equal_nan=True)
    r.close()


def test_noalloc_allocates_nothing_and_rejects_oversize():
    import torch
    H.build()
    dev = torch.device("cuda:0")
    p = W.make_config(1, Q=4096)
    r = H.Router(p, stream=torch.cuda.current_stream().cuda_stream)
    inp = _dev(p, 0, 4096, dev)
    out = _outs(4096, dev)
    r.route_device_noalloc(*inp, *out, slo=p["slo"], lam=p["lam"])   # first call: set-up
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for _ in range(3):
        r.route_device_noalloc(*inp, *out, slo=p["slo"], lam=p["lam"])
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] >= free0
    ref = _outs(4096, dev)
    r.route_device(*inp, *ref, slo=p["slo"], lam=p["lam"], flags=H.HWR_PATH_TENSOR)
    torch.cuda.synchronize()
    _close(out, ref)
    big = H.HWR_NOALLOC_MAX_Q + 1
    z = torch.zeros(big, dtype=torch.float32, device=dev)
    e = torch.zeros((big, p["E"]), dtype=torch.int16, device=dev)
    o = _outs(big, dev)
    with pytest.raises(H.HwrError) as exc:
        r.route_device_noalloc(z, z, e, *o, slo=p["slo"], lam=p["lam"])
    assert exc.value.status == 7 and "maximum" in str(exc.value)
    r.close()
