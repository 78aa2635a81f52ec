"""Online routing through the library: callbacks for the micro-batch loop.

`callbacks(p)` gives the routing and scoring functions that the online loop
(`workload.serve.run_online`) calls for each micro-batch: the router context
takes the snapshot the router is shown (live, or frozen in the static-cost
mode), a second context holds the live snapshot and scores realised latency
and quality with `hwr_score_batch`.  Every step runs in the library's
kernels; this module only moves arrays.
"""
from __future__ import annotations

import numpy as np

from ._hwr import HWR_SEQUENTIAL, Router
from . import metrics


class OnlineRouter:
    def __init__(self, p: dict, *, sequential: bool = True, flags: int = 0, lam=None,
                 slo=None, budgets=None):
        self.p = p
        self.router = Router(p)
        self.world = Router(p)
        self.flags = int(flags) | (HWR_SEQUENTIAL if sequential else 0)
        self.lam = p["lam"] if lam is None else lam
        self.slo = p["slo"] if slo is None else slo
        self.budgets = None if budgets is None else np.asarray(budgets, np.float32)

    def route(self, snap, lo, hi):
        p = self.p
        self.router.update_snapshot(snap)
        il, ol, em = p["in_len"][lo:hi], p["out_len"][lo:hi], p["emb"][lo:hi]
        if self.budgets is not None:
            return self.router.route_slo(il, ol, em, budgets=self.budgets[lo:hi],
                                         lam=self.lam, flags=self.flags)
        return self.router.route(il, ol, em, slo=self.slo, lam=self.lam, flags=self.flags)

    def score(self, snap, lo, hi):
        p = self.p
        self.world.update_snapshot(snap)
        return self.world.score(p["in_len"][lo:hi], p["out_len"][lo:hi], p["emb"][lo:hi],
                                flags=self.flags & ~HWR_SEQUENTIAL)

    def close(self):
        self.router.close()
        self.world.close()

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()


def compare(p: dict, run_online, *, sequential: bool = True, **world) -> dict:
    """Metrics of the hardware-aware router and of the static-cost mode on one world.

    `run_online` is the loop (workload.serve.run_online); `world` its options
    (pattern, rate, batch or window, drain, cap, ...).
    """
    out = {}
    for name, static in (("hw_router", False), ("static_cost", True)):
        with OnlineRouter(p, sequential=sequential) as r:
            tr = run_online(p, r.route, r.score, static=static, **world)
        out[name] = metrics.summarize(tr, p["dep_gpu"], p["G"], p["D"])
    return out
