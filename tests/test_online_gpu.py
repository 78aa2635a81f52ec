"""Online routing on the GPU against the oracle (Sec. 4.4 evaluation metrics).

The serving world (workload/serve.py) is driven once by the library (routing
and hwr_score_batch through the C ABI) and once by the oracle in canonical
fp32, from the same seeds.  With the fp32 predictor every decision is
bit-exact, so the two traces, and every metric computed from them, must be
identical: chosen deployments, predicted and realised latencies, quality, and
the queue histories the world produced from those choices.
"""
import numpy as np
import pytest

import oracle as O
import workload as W
from workload import serve as S
import paper_2608_14575_gb300 as H
from paper_2608_14575_gb300 import metrics as MX
from paper_2608_14575_gb300.online import OnlineRouter, compare

pytestmark = pytest.mark.gpu
MODEL = (0.35, 2.0 ** -9, 1.2, 0.0119)          # a (s), b (s/token), slack, TPOT_SLO (s)


@pytest.fixture(scope="module", autouse=True)
def built():
    H.build()


def _oracle_callbacks(p, sequential, budgets=None):
    orc = O.Problem(p)

    def route(snap, lo, hi):
        orc.set_snapshot(snap)
        q = (p["in_len"][lo:hi], p["out_len"][lo:hi], p["emb"][lo:hi])
        if budgets is not None:
            ch, lat, util, _ = orc.route_slo(budgets[lo:hi], *q, mode=O.F32,
                                             sequential=sequential, running=snap["running"])
        else:
            ch, lat, util, _ = orc.route(*q, mode=O.F32, sequential=sequential,
                                         running=snap["running"], nthreads=8)
        return ch, lat.astype(np.float32), util.astype(np.float32)

    def score(snap, lo, hi):
        orc.set_snapshot(snap)
        C, _ = orc.score_all(p["in_len"][lo:hi], p["out_len"][lo:hi], p["emb"][lo:hi],
                             mode=O.F32, nthreads=8)
        qual = np.array([orc.quality(p["emb"][i], mode=O.F32) for i in range(lo, hi)])
        return C.astype(np.float32), qual.astype(np.float32).reshape(hi - lo, p["M"])

    return route, score


def _same(a, b):
    for k in ("chosen", "latency", "utility", "realised", "quality", "running", "waiting"):
        assert np.array_equal(a[k], b[k], equal_nan=True), k


SCENARIOS = {
    # the online sequential workload itself: Poisson at 200 req/s, batches of 64
    "online_sequential": dict(),
    "micro_burst_cap": dict(pattern="micro_burst", rate=150.0, window=0.05, cap=8,
                            drain="per_time", service_s=0.4, burst_factor=10.0),
    "overload_static": dict(pattern="sustained_overload", rate=120.0, window=0.1, cap=8,
                            drain="per_time", service_s=0.4, overload=1.5, static=True),
    "overload_batch_mode": dict(pattern="sustained_overload", rate=120.0, batch=100, cap=6,
                                drain="per_time", service_s=0.4, seq=False),
}


@pytest.mark.parametrize("name", list(SCENARIOS))
def test_online_trace_matches_oracle(name):
    kw = dict(SCENARIOS[name])
    seq = kw.pop("seq", True)
    p = W.make_config(2, Q=2500)
    with OnlineRouter(p, sequential=seq) as r:
        g = S.run_online(p, r.route, r.score, **kw)
    route, score = _oracle_callbacks(p, seq)
    c = S.run_online(p, route, score, **kw)
    _same(g, c)
    mg = MX.summarize(g, p["dep_gpu"], p["G"])
    assert mg == MX.summarize(c, p["dep_gpu"], p["G"])
    if not seq and not kw.get("static"):
        # batch routing on the live state: the realised latency is the prediction
        assert np.array_equal(g["realised"], g["latency"], equal_nan=True)


def test_online_per_query_budgets_match_oracle():
    p = W.make_config(2, Q=1500)
    b = O.slo_budget(*MODEL, p["in_len"], p["out_len"], mode=O.F32).astype(np.float32)
    kw = dict(pattern="micro_burst", rate=150.0, window=0.05, cap=8, drain="per_time",
              service_s=0.4, budgets=b)
    with OnlineRouter(p, budgets=b) as r:
        g = S.run_online(p, r.route, r.score, **kw)
    route, score = _oracle_callbacks(p, True, budgets=b)
    c = S.run_online(p, route, score, **kw)
    _same(g, c)
    assert np.array_equal(g["budget"], b)


def test_score_batch_matches_oracle_and_route():
    """hwr_score_batch on the small-batch, fused SIMT and tensor paths."""
    for cfg, Q, flags in ((0, 7, 0), (0, 300, 0), (1, 300, H.HWR_PATH_SIMT)):
        p = W.make_config(cfg, Q=Q)
        r = H.Router(p)
        C, qual = r.score(flags=flags)
        orc = O.Problem(p)
        Cw, _ = orc.score_all(mode=O.F32, nthreads=8)
        assert np.array_equal(C, Cw.astype(np.float32)), (cfg, Q)
        qw = np.array([orc.quality(p["emb"][i], mode=O.F32) for i in range(Q)])
        assert np.array_equal(qual, qw.astype(np.float32)), (cfg, Q)
        ch, lat, _ = r.route(flags=flags)
        assert np.array_equal(lat, C[np.arange(Q), ch])
        r.close()
    # tensor path: the route's latencies are the stored costs of its choices
    p = W.make_config(3, Q=3000)
    r = H.Router(p)
    C, qual = r.score(flags=H.HWR_PATH_TENSOR)
    ch, lat, _ = r.route(flags=H.HWR_PATH_TENSOR)
    assert np.array_equal(lat, C[np.arange(p["Q"]), ch])
    Cw, _ = O.Problem(p).score_all(nthreads=16)
    rel = np.abs(C - Cw) / np.maximum(np.abs(Cw), 1e-3)
    assert rel.max() <= 2e-2, rel.max()
    C2, none = r.score(flags=H.HWR_PATH_TENSOR, quality=False)
    assert none is None and np.array_equal(C, C2)
    with pytest.raises(H.HwrError) as e:
        r.score(flags=H.HWR_SEQUENTIAL)
    assert e.value.status == 7
    r.close()


def test_score_device_pipelined_equals_host():
    import torch
    p = W.make_config(3, Q=20_000)
    r = H.Router(p, stream=torch.cuda.current_stream().cuda_stream)
    C, qual = r.score()                              # chunked host copies
    dev = torch.device("cuda:0")
    il = torch.from_numpy(p["in_len"]).to(dev)
    ol = torch.from_numpy(p["out_len"]).to(dev)
    em = torch.from_numpy(p["emb"].view(np.int16)).to(dev)
    Cd = torch.empty((p["Q"], p["D"]), dtype=torch.float32, device=dev)
    Qd = torch.empty((p["Q"], p["M"]), dtype=torch.float32, device=dev)
    r.score_device(il, ol, em, Cd, Qd)
    torch.cuda.synchronize()
    assert np.array_equal(Cd.cpu().numpy(), C)
    assert np.array_equal(Qd.cpu().numpy(), qual)
    r.close()


def test_compare_reports_both_modes():
    p = W.make_config(2, Q=2000)
    out = compare(p, S.run_online, pattern="sustained_overload", rate=100.0, window=0.1,
                  cap=8, drain="per_time", service_s=0.4, overload=1.5)
    for name in ("hw_router", "static_cost"):
        m = out[name]
        assert m["requests"] == 2000
        assert 0.0 <= m["slo_attainment"] <= 1.0
        assert abs(m["running_fraction"] + m["waiting_fraction"] - 1.0) < 1e-12
        assert m["load_skew"] >= 0.0
