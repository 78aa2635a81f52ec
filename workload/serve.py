"""Synthetic serving world for online routing experiments.

The paper evaluates routers on live vLLM servers (Sec. 4.4, Sec. 5); here the
servers are replaced by a seeded stand-in that evolves the per-deployment
hardware snapshot between micro-batches.  Nothing in this module computes any
part of the routing method: it draws arrivals, groups them into micro-batches,
hands each batch to caller-supplied routing and scoring functions and moves
the world on with their choices.

Arrival patterns (Sec. 4.5 load generator):
  * "poisson"            exponential gaps with mean 1/rate;
  * "micro_burst"        Poisson whose rate is burst_factor x higher during
                         the first burst_len seconds of every period;
  * "sustained_overload" Poisson at overload x rate, `rate` being the world's
                         nominal capacity (a load held above what it serves).

World dynamics, after each micro-batch has been routed:
  1. placement: each routed request joins its deployment's running queue if a
     slot is free (running < cap), else its waiting queue; with cap None
     every request runs (the online sequential workload: waiting is held);
  2. drain: every running request completes with probability p, either per
     micro-batch (p = drain_p, the online sequential workload) or per elapsed
     time (p = 1 - exp(-dt / service_s), dt = time since the last dispatch);
  3. admission: waiting requests take the freed slots, first come first served;
  4. KV utilisation random-walks with N(0, kv_walk), clipped to [0, 1].
Other signals (GPU utilisation, recent TTFT/TPOT) are held.

The "static cost" comparison mode hands the router the initial snapshot on
every batch (the hardware signals frozen, as routers with static cost models
see them) while the world, and the scoring of realised latency, use the live
state.
"""
from __future__ import annotations

import numpy as np

from .gen import BASE_SEED

PATTERNS = ("poisson", "micro_burst", "sustained_overload")


def arrival_times(pattern: str, n: int, rate: float, rng, *, burst_factor: float = 8.0,
                  burst_len: float = 0.05, period: float = 1.0,
                  overload: float = 1.25) -> np.ndarray:
    """Arrival times (s, ascending, float64) of n requests."""
    if n < 0 or not rate > 0:
        raise ValueError("need n >= 0 and rate > 0")
    if pattern == "poisson":
        return np.cumsum(rng.exponential(1.0 / rate, size=n))
    if pattern == "sustained_overload":
        if not overload > 1.0:
            raise ValueError("sustained overload needs overload > 1")
        return np.cumsum(rng.exponential(1.0 / (overload * rate), size=n))
    if pattern == "micro_burst":
        if not (burst_factor >= 1.0 and 0.0 < burst_len < period):
            raise ValueError("micro-burst needs burst_factor >= 1 and 0 < burst_len < period")
        # time-rescaling: unit-rate points s_i in integrated-intensity space,
        # mapped back through the inverse of the piecewise-linear Lambda(t)
        s = np.cumsum(rng.exponential(1.0, size=n))
        hi = rate * burst_factor
        per = hi * burst_len + rate * (period - burst_len)
        k = np.floor(s / per)
        r = s - k * per
        t = np.where(r < hi * burst_len, r / hi, burst_len + (r - hi * burst_len) / rate)
        return k * period + t
    raise ValueError(f"unknown arrival pattern {pattern!r}; one of {PATTERNS}")


def nominal_capacity(cap, D: int, service_s: float) -> float:
    """Requests/s the world completes with every slot busy: sum(cap) / service_s."""
    c = np.broadcast_to(np.asarray(cap, np.float64), (D,))
    return float(c.sum() / service_s)


def micro_batches(t: np.ndarray, *, batch: int | None = None, window: float | None = None):
    """Split arrival-ordered requests into micro-batches.

    By count (`batch` requests each, the last one ragged; dispatched when the
    last request arrives) or by time window (all arrivals in [kW, (k+1)W),
    dispatched at (k+1)W; empty windows are kept so the world still drains).
    Returns (starts, ends, dispatch_times) with batch k = requests [starts[k], ends[k]).
    """
    n = len(t)
    if (batch is None) == (window is None):
        raise ValueError("give exactly one of batch and window")
    if batch is not None:
        if batch < 1:
            raise ValueError("batch >= 1")
        starts = np.arange(0, n, batch)
        ends = np.minimum(starts + batch, n)
        disp = t[ends - 1] if n else np.zeros(0)
        return starts, ends, np.asarray(disp, np.float64)
    if not window > 0:
        raise ValueError("window > 0")
    nwin = int(np.floor(t[-1] / window)) + 1 if n else 0
    edges = np.arange(nwin + 1) * window
    idx = np.searchsorted(t, edges, side="left")
    idx[-1] = n
    return idx[:-1].copy(), idx[1:].copy(), edges[1:].astype(np.float64)


def run_online(p: dict, route_fn, score_fn, *, n_requests: int | None = None,
               pattern: str = "poisson", rate: float | None = None,
               batch: int | None = None, window: float | None = None,
               drain: str = "per_batch", drain_p: float | None = None,
               service_s: float = 1.0, cap=None, static: bool = False,
               budgets=None, seed_offset: int = 0, **pattern_args) -> dict:
    """Run the online micro-batch loop; returns the per-request and per-batch trace.

    route_fn(snapshot, lo, hi) -> (chosen, latency, utility) routes requests
    [lo, hi) of `p` against `snapshot`; score_fn(snapshot, lo, hi) -> (cost
    [n][D], quality [n][M]) scores them (both called with copies).  The
    realised latency of a request is the cost of its chosen deployment under
    the live snapshot at the start of its micro-batch, and its quality is the
    chosen model's quality score.  `budgets` (one per request) replaces the
    scalar SLO p["slo"] for the attainment record.
    """
    n = p["Q"] if n_requests is None else int(n_requests)
    D = p["D"]
    if n > p["Q"]:
        raise ValueError("more requests than queries in the problem")
    if drain not in ("per_batch", "per_time"):
        raise ValueError("drain is 'per_batch' or 'per_time'")
    if batch is None and window is None:
        batch = p.get("batch", 64)
    rate = p.get("rate", 200.0) if rate is None else rate
    dp = p.get("drain_p", 0.3) if drain_p is None else drain_p
    kv_walk = p.get("kv_walk", 0.02)
    capv = None if cap is None else np.broadcast_to(np.asarray(cap, np.int64), (D,)).copy()
    if capv is not None and (capv < 0).any():
        raise ValueError("cap >= 0")
    # the world's stream is the online sequential workload's drain stream
    # (so count batches, per-batch drain and no cap reproduce that workload)
    cfg = (p.get("cfg") or 0) + 7919 * seed_offset
    rng_world = np.random.Generator(np.random.PCG64(np.random.SeedSequence(BASE_SEED + 1000 + cfg)))
    rng_arr = np.random.Generator(np.random.PCG64(np.random.SeedSequence(BASE_SEED + 2000 + cfg)))
    t = arrival_times(pattern, n, rate, rng_arr, **pattern_args)
    starts, ends, disp = micro_batches(t, batch=batch, window=window)

    snap = {k: np.array(v, copy=True) for k, v in p["snap"].items()}
    if capv is not None:    # start from a consistent state: overflow waits
        over = np.maximum(snap["running"].astype(np.int64) - capv, 0)
        snap["running"] = (snap["running"] - over).astype(np.int32)
        snap["waiting"] = (snap["waiting"] + over).astype(np.int32)
    frozen = {k: np.array(v, copy=True) for k, v in p["snap"].items()}
    dep_model = np.asarray(p["dep_model"])
    slo = np.full(n, p["slo"], np.float32) if budgets is None else \
        np.asarray(budgets, np.float32)[:n]

    chosen = np.full(n, -1, np.int32)
    lat = np.full(n, np.nan, np.float32)
    util = np.full(n, np.nan, np.float32)
    real = np.full(n, np.nan, np.float32)
    qual = np.full(n, np.nan, np.float32)
    K = len(starts)
    run_hist = np.zeros((K, D), np.int32)
    wait_hist = np.zeros((K, D), np.int32)
    t_prev = 0.0
    for k in range(K):
        lo, hi = int(starts[k]), int(ends[k])
        run_hist[k] = snap["running"]
        wait_hist[k] = snap["waiting"]
        if hi > lo:
            live = {kk: v.copy() for kk, v in snap.items()}
            view = {kk: v.copy() for kk, v in (frozen if static else snap).items()}
            c, l, u = route_fn(view, lo, hi)
            cost, q = score_fn(live, lo, hi)
            c = np.asarray(c, np.int32)
            chosen[lo:hi], lat[lo:hi], util[lo:hi] = c, l, u
            ok = c >= 0
            rows = np.nonzero(ok)[0]
            real[lo + rows] = np.asarray(cost)[rows, c[ok]]
            qual[lo + rows] = np.asarray(q)[rows, dep_model[c[ok]]]
            placed = np.bincount(c[ok], minlength=D).astype(np.int64)
        else:
            placed = np.zeros(D, np.int64)
        # 1. placement
        r = snap["running"].astype(np.int64)
        w = snap["waiting"].astype(np.int64)
        if capv is None:
            r += placed
        else:
            take = np.minimum(placed, np.maximum(capv - r, 0))
            r += take
            w += placed - take
        # 2. drain
        if drain == "per_batch":
            pd = dp
        else:
            pd = 1.0 - np.exp(-max(disp[k] - t_prev, 0.0) / service_s)
        r -= rng_world.binomial(r, pd)
        # 3. admission
        if capv is not None:
            move = np.minimum(w, np.maximum(capv - r, 0))
            r += move
            w -= move
        snap["running"] = r.astype(np.int32)
        snap["waiting"] = w.astype(np.int32)
        # 4. KV walk
        kv = snap["kv"].astype(np.float64) + rng_world.normal(0.0, kv_walk, D)
        snap["kv"] = np.clip(kv, 0.0, 1.0).astype(np.float32)
        t_prev = float(disp[k])
    return dict(arrival=t, batch_start=starts, batch_end=ends, dispatch=disp,
                chosen=chosen, latency=lat, utility=util, realised=real, quality=qual,
                budget=slo, running=run_hist, waiting=wait_hist, static=static,
                pattern=pattern, rate=rate)
