"""Online routing metrics of HW-Router's evaluation (Sec. 4.4, Eq. 6).

Host-side reductions over a trace of routed requests and of queue snapshots
sampled at each micro-batch (the monitor's view when decisions are made):

  * SLO attainment: the fraction of requests whose latency is within their
    budget (latency <= budget, the same inclusive test as the SLO mask);
  * queue composition: running and waiting requests as fractions of the total
    queue, summed over deployments and samples;
  * load, running and waiting skew: with Qbar_g the mean over samples of the
    total (running + waiting), running or waiting queue on GPU g (summed over
    the deployments placed on g), the spread max_g Qbar_g - min_g Qbar_g.
    For the paper's two GPUs this is |Qbar_0 - Qbar_1| (Eq. 6).

The functions take plain arrays, so they serve traces from the synthetic
serving world as well as queue samples scraped from real servers.
"""
from __future__ import annotations

import numpy as np


def slo_attainment(latency, budget) -> float:
    """Fraction of requests with latency <= budget (NaN latency counts as a miss)."""
    lat = np.asarray(latency, np.float64)
    b = np.broadcast_to(np.asarray(budget, np.float64), lat.shape)
    if lat.size == 0:
        return float("nan")
    return float(np.mean(lat <= b))


def queue_composition(running, waiting) -> tuple[float, float]:
    """(running fraction, waiting fraction) of all queued requests over all samples."""
    r = float(np.sum(np.asarray(running, np.int64)))
    w = float(np.sum(np.asarray(waiting, np.int64)))
    if r + w == 0:
        return float("nan"), float("nan")
    return r / (r + w), w / (r + w)


def gpu_means(queue, dep_gpu, G: int) -> np.ndarray:
    """Mean over samples of each GPU's queue: queue [samples][D] -> [G]."""
    q = np.asarray(queue, np.float64)
    if q.ndim != 2 or q.shape[0] == 0:
        raise ValueError("queue must be [samples][deployments] with at least one sample")
    g = np.asarray(dep_gpu, np.int64)
    per = np.zeros((q.shape[0], G))
    for d in range(q.shape[1]):
        per[:, g[d]] += q[:, d]
    return per.mean(axis=0)


def skew(queue, dep_gpu, G: int) -> float:
    """max_g Qbar_g - min_g Qbar_g (|Qbar_0 - Qbar_1| for two GPUs)."""
    m = gpu_means(queue, dep_gpu, G)
    return float(m.max() - m.min())


def skews(running, waiting, dep_gpu, G: int) -> dict:
    """Load, running and waiting skew of Eq. 6."""
    r = np.asarray(running, np.int64)
    w = np.asarray(waiting, np.int64)
    return dict(load_skew=skew(r + w, dep_gpu, G), running_skew=skew(r, dep_gpu, G),
                waiting_skew=skew(w, dep_gpu, G))


def latency_stats(latency) -> dict:
    lat = np.asarray(latency, np.float64)
    lat = lat[np.isfinite(lat)]
    if lat.size == 0:
        return dict(mean=float("nan"), p50=float("nan"), p95=float("nan"), p99=float("nan"))
    return dict(mean=float(lat.mean()), p50=float(np.percentile(lat, 50)),
                p95=float(np.percentile(lat, 95)), p99=float(np.percentile(lat, 99)))


def summarize(trace: dict, dep_gpu, G: int, D: int | None = None) -> dict:
    """All metrics of one online run (a trace of workload.serve.run_online's form)."""
    ch = np.asarray(trace["chosen"])
    D = int(np.asarray(trace["running"]).shape[1]) if D is None else D
    routed = ch >= 0
    alloc = np.bincount(ch[routed], minlength=D) / max(int(routed.sum()), 1)
    rf, wf = queue_composition(trace["running"], trace["waiting"])
    lat = np.asarray(trace["latency"], np.float64)
    out = dict(requests=int(ch.size),
               slo_attainment=slo_attainment(trace["realised"], trace["budget"]),
               predicted_attainment=slo_attainment(lat, trace["budget"]),
               running_fraction=rf, waiting_fraction=wf,
               realised_latency=latency_stats(trace["realised"]),
               mean_quality=float(np.nanmean(trace["quality"])) if ch.size else float("nan"),
               allocation=[float(a) for a in alloc])
    out.update(skews(trace["running"], trace["waiting"], dep_gpu, G))
    return out
