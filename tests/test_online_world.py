"""Online evaluation on the CPU: arrival patterns, micro-batching, the serving
world's dynamics and the paper's online metrics (Sec. 4.4, Eq. 6).

Metrics are pinned by hand-computed examples; arrival patterns by their
defining statistics and by reductions to one another; the world by
conservation laws and by reproducing the online sequential workload.  The
oracle drives the world as the router in the last tests.
"""
import numpy as np
import pytest

import oracle as O
import workload as W
from workload import serve as S
from paper_2608_14575_gb300 import metrics as MX


# ---------------------------------------------------------------------------
# metrics: hand-computed cases

def test_slo_attainment_counts_inclusive_and_nan_as_miss():
    assert MX.slo_attainment([1.0, 2.0, 3.0, np.nan], 2.0) == 0.5
    assert MX.slo_attainment([1.0, 2.0], [0.5, 2.0]) == 0.5
    assert np.isnan(MX.slo_attainment([], 1.0))


def test_queue_composition_by_hand():
    r = [[1, 2], [3, 0]]
    w = [[0, 2], [1, 1]]
    assert MX.queue_composition(r, w) == (0.6, 0.4)
    assert all(np.isnan(MX.queue_composition([[0]], [[0]])))


def test_skews_by_hand():
    # deployments 0 and 2 on GPU 0, deployment 1 on GPU 1
    dep_gpu = [0, 1, 0]
    r = [[1, 2, 3], [3, 0, 1]]     # GPU means: (4 + 4) / 2 = 4, (2 + 0) / 2 = 1
    w = [[0, 1, 0], [2, 2, 2]]     # (0 + 4) / 2 = 2, (1 + 2) / 2 = 1.5
    s = MX.skews(r, w, dep_gpu, 2)
    assert s == dict(load_skew=3.5, running_skew=3.0, waiting_skew=0.5)
    # Eq. 6 for two GPUs is |Qbar_0 - Qbar_1|: relabelling the GPUs changes nothing
    assert MX.skews(r, w, [1, 0, 1], 2) == s
    # three GPUs: the spread max - min
    assert MX.skew([[1, 5, 2]], [0, 1, 2], 3) == 4.0
    # a GPU with no deployment has an empty queue
    assert MX.skew([[3, 3]], [0, 0], 2) == 6.0


def test_summarize_by_hand():
    tr = dict(chosen=np.array([0, 1, 1, -1]), latency=np.array([1.0, 3.0, 1.0, 9.0]),
              realised=np.array([1.5, 1.0, 2.5, np.nan]), budget=np.full(4, 2.0),
              quality=np.array([0.5, 0.7, 0.9, np.nan]),
              running=np.array([[2, 0], [1, 1]]), waiting=np.array([[0, 0], [0, 2]]))
    s = MX.summarize(tr, dep_gpu=[0, 1], G=2)
    assert s["slo_attainment"] == 0.5 and s["predicted_attainment"] == 0.5
    assert s["running_fraction"] == 4 / 6
    assert s["allocation"] == [1 / 3, 2 / 3]
    assert s["load_skew"] == 0.0 and s["running_skew"] == 1.0 and s["waiting_skew"] == 1.0
    assert abs(s["mean_quality"] - 0.7) < 1e-12


# ---------------------------------------------------------------------------
# arrivals and micro-batches

def _rng(k=0):
    return np.random.default_rng(1234 + k)


def test_poisson_statistics():
    t = S.arrival_times("poisson", 200_000, 200.0, _rng())
    assert np.all(np.diff(t) > 0)
    assert abs(np.diff(t).mean() * 200.0 - 1.0) < 0.01
    counts = np.bincount(np.floor(t).astype(int))[:-1]      # per-second counts
    assert abs(counts.var() / counts.mean() - 1.0) < 0.15    # Poisson: var = mean


def test_sustained_overload_is_poisson_above_rate():
    t = S.arrival_times("sustained_overload", 100_000, 100.0, _rng(1), overload=1.5)
    assert abs(np.diff(t).mean() * 150.0 - 1.0) < 0.015
    with pytest.raises(ValueError):
        S.arrival_times("sustained_overload", 10, 100.0, _rng(), overload=1.0)


def test_micro_burst_rates():
    rate, bf, bl, per = 50.0, 8.0, 0.05, 1.0
    t = S.arrival_times("micro_burst", 200_000, rate, _rng(2), burst_factor=bf,
                        burst_len=bl, period=per)
    assert np.all(np.diff(t) >= 0)
    phase = np.mod(t, per)
    inside = phase < bl
    T = np.floor(t[-1] / per) * per                          # whole periods only
    keep = t < T
    rate_in = np.sum(inside & keep) / (T / per * bl)
    rate_out = np.sum(~inside & keep) / (T / per * (per - bl))
    assert abs(rate_in / (bf * rate) - 1.0) < 0.03
    assert abs(rate_out / rate - 1.0) < 0.02
    # burst factor 1 reduces to the homogeneous process of the same draws
    a = S.arrival_times("micro_burst", 1000, rate, _rng(3), burst_factor=1.0,
                        burst_len=bl, period=per)
    b = np.cumsum(_rng(3).exponential(1.0, 1000)) / rate
    assert np.allclose(a, b, rtol=1e-9, atol=1e-9)


def test_micro_batches_by_count_and_window():
    s, e, d = S.micro_batches(np.arange(1, 11, dtype=float), batch=4)
    assert s.tolist() == [0, 4, 8] and e.tolist() == [4, 8, 10] and d.tolist() == [4.0, 8.0, 10.0]
    t = np.array([0.1, 0.2, 1.5, 3.2])
    s, e, d = S.micro_batches(t, window=1.0)
    assert s.tolist() == [0, 2, 3, 3] and e.tolist() == [2, 3, 3, 4]   # (2, 3) is empty
    assert d.tolist() == [1.0, 2.0, 3.0, 4.0]
    for fn in (lambda: S.micro_batches(t), lambda: S.micro_batches(t, batch=2, window=1.0)):
        with pytest.raises(ValueError):
            fn()


# ---------------------------------------------------------------------------
# the world, driven by simple host routers

def _least_loaded(p, record=None, frozen=None):
    """Sequential least-running-queue router (ties to the lowest index)."""
    def route(snap, lo, hi):
        if frozen is not None:
            for k in frozen:
                assert np.array_equal(snap[k], frozen[k])
        run = snap["running"].astype(np.int64).copy()
        out = np.empty(hi - lo, np.int32)
        for i in range(hi - lo):
            out[i] = int(np.argmin(run))
            run[out[i]] += 1
        if record is not None:
            record.append(out)
        n = hi - lo
        return out, np.zeros(n, np.float32), np.zeros(n, np.float32)
    return route


def _fake_score(p):
    def score(snap, lo, hi):
        n = hi - lo
        cost = (np.arange(n)[:, None] * 0.01 + snap["running"][None, :]).astype(np.float32)
        qual = np.tile(np.linspace(0.1, 0.9, p["M"], dtype=np.float32), (n, 1))
        return cost, qual
    return score


def test_reproduces_online_sequential_workload():
    p = W.make_config(2, Q=1000)
    rec = []
    tr = S.run_online(p, _least_loaded(p, rec), _fake_score(p))
    want, hist = W.simulate_online(p, lambda snap, lo, hi: _least_loaded(p)(snap, lo, hi)[0])
    assert np.array_equal(tr["chosen"], want)
    assert np.array_equal(tr["running"], np.array([h["running"] for h in hist]))
    assert np.array_equal(tr["waiting"], np.array([h["waiting"] for h in hist]))


@pytest.mark.parametrize("pattern,kw", [
    ("poisson", dict(batch=64)),
    ("micro_burst", dict(window=0.05, burst_factor=10.0)),
    ("sustained_overload", dict(window=0.1, overload=2.0)),
])
def test_capacity_and_conservation(pattern, kw):
    p = W.make_config(2, Q=3000)
    cap = 6
    tr = S.run_online(p, _least_loaded(p), _fake_score(p), pattern=pattern, rate=80.0,
                      drain="per_time", service_s=0.5, cap=cap, **kw)
    r, w = tr["running"], tr["waiting"]
    assert (r >= 0).all() and (w >= 0).all() and (r <= cap).all()
    # a waiting request exists only where every slot is busy
    assert ((w == 0) | (r == cap)).all()
    # realised latency and quality are read at the chosen deployment
    assert np.all(tr["chosen"] >= 0)
    assert np.isfinite(tr["realised"]).all()
    assert tr["budget"].shape == (3000,)
    # requests in the system never exceed those that have arrived plus the start
    start = np.minimum(p["snap"]["running"], cap).sum() + p["snap"]["waiting"].sum() + \
        np.maximum(p["snap"]["running"] - cap, 0).sum()
    inside = (r + w).sum(axis=1)
    assert np.all(inside <= start + tr["batch_start"])


def test_zero_capacity_everything_waits():
    p = W.make_config(2, Q=300)
    tr = S.run_online(p, _least_loaded(p), _fake_score(p), cap=0)
    assert (tr["running"][1:] == 0).all()
    w_total = tr["waiting"].sum(axis=1)
    assert np.array_equal(np.diff(w_total), np.full(len(w_total) - 1, 64))


def test_static_mode_sees_the_frozen_snapshot():
    p = W.make_config(2, Q=640)
    rec_s = []
    tr = S.run_online(p, _least_loaded(p, rec_s, frozen=p["snap"]), _fake_score(p),
                      static=True, cap=10, drain="per_time")
    # with the state frozen every batch is routed identically
    assert all(np.array_equal(rec_s[0], x) for x in rec_s[:-1])
    # but the world moved on
    assert not np.array_equal(tr["running"][0], tr["running"][-1])


def test_oracle_router_in_the_world():
    """Dynamic batch routing: realised latency is the router's own prediction."""
    p = W.make_config(0, Q=256)
    orc = O.Problem(p)

    def route(snap, lo, hi, seq=False):
        orc.set_snapshot(snap)
        ch, lat, util, _ = orc.route(p["in_len"][lo:hi], p["out_len"][lo:hi], p["emb"][lo:hi],
                                     mode=O.F32, sequential=seq, running=snap["running"])
        return ch, lat.astype(np.float32), util.astype(np.float32)

    def score(snap, lo, hi):
        orc.set_snapshot(snap)
        C, _ = orc.score_all(p["in_len"][lo:hi], p["out_len"][lo:hi], p["emb"][lo:hi],
                             mode=O.F32)
        q = np.array([orc.quality(p["emb"][i], mode=O.F32) for i in range(lo, hi)])
        return C.astype(np.float32), q.astype(np.float32)

    tr = S.run_online(p, route, score, batch=32, cap=4, drain="per_time", service_s=0.2)
    assert np.array_equal(tr["realised"], tr["latency"])
    s = MX.summarize(tr, p["dep_gpu"], p["G"])
    assert s["slo_attainment"] == s["predicted_attainment"]
    assert 0.0 <= s["waiting_fraction"] <= 1.0
    # sequential routing: the first request of each batch sees the live state
    tr2 = S.run_online(p, lambda s_, lo, hi: route(s_, lo, hi, True), score, batch=32,
                       cap=4, drain="per_time", service_s=0.2)
    first = tr2["batch_start"]
    assert np.array_equal(tr2["realised"][first], tr2["latency"][first])
