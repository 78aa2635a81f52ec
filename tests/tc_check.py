"""Tolerance check of the bf16 tensor-core path against the fp64 oracle.

Predicted latency and utility must sit within 2e-2 relative of the oracle's
scores of the deployment the GPU chose (utility relative to max(|U|, 1)).
Chosen indices must match wherever the decision is clear under that
tolerance: the oracle's best utility beats the runner-up (the best strictly
below it; exact ties are resolved by index on both sides) by more than the
tolerance, or with nothing feasible the latency margin does, and no latency
lies within the tolerance band of its query's SLO budget.  The remaining
choices must still be valid: at least as good, within tolerance, as every
surely feasible deployment.
"""
import numpy as np

import oracle as O
import workload as W

TOL = 2e-2


def check_against_oracle(p, got, idx=None, slo=None, lam=None, convex=False,
                         min_checked=0.5):
    """Compare GPU outputs for queries `idx` (all if None) with the fp64 oracle."""
    ch, lat, util = (np.asarray(a) for a in got)
    if idx is not None:
        sub = W.query_subset(p, idx)
        ch, lat, util = ch[idx], lat[idx], util[idx]
    else:
        sub = p
    slo = p["slo"] if slo is None else slo
    lam = p["lam"] if lam is None else lam
    orc = O.Problem(sub)
    C, U = orc.score_all(lam=lam, convex=convex, nthreads=16)
    if np.ndim(slo):                              # one budget per query
        slo = np.asarray(slo, np.float32)[idx] if idx is not None else np.asarray(slo, np.float32)
        wch, wlat, wutil, _ = orc.route_slo(slo, lam=lam, convex=convex)
        slo = slo.astype(np.float64)[:, None]
    else:
        wch, wlat, wutil, _ = orc.route(slo=slo, lam=lam, convex=convex, nthreads=16)
    ok = wch >= 0
    assert np.array_equal(ch >= 0, ok)
    # the chosen deployment may legitimately differ near ties, so compare the
    # GPU's outputs with the oracle's scores of the deployment the GPU chose
    qi = np.nonzero(ok)[0]
    glat = C[qi, ch[ok]]
    gutil = U[qi, ch[ok]]
    rl_own = np.abs(lat[ok] - glat) / np.maximum(np.abs(glat), 1e-3)
    ru_own = np.abs(util[ok] - gutil) / np.maximum(np.abs(gutil), 1.0)
    assert rl_own.max(initial=0) <= TOL, rl_own.max()
    assert ru_own.max(initial=0) <= TOL, ru_own.max()
    # decisions that are clear under the tolerance must match exactly
    with np.errstate(invalid="ignore"):
        band = np.where(np.isfinite(slo), TOL * np.maximum(np.abs(slo), 1e-3), 0.0)
    feas = C <= slo
    sure = C <= slo - band          # feasible under any in-tolerance latency
    maybe = C <= slo + band         # feasible under some in-tolerance latency
    near_slo = (sure != maybe).any(axis=1)
    with np.errstate(invalid="ignore"):
        Uf = np.where(feas, U, -np.inf)
        top1 = Uf.max(axis=1)
        # runner-up: the best utility strictly below the top.  Exact ties (the
        # GPU types of one model when lambda = 0) are resolved by index on both
        # sides, so they do not make a decision unclear.
        top2 = np.where(Uf < top1[:, None], Uf, -np.inf).max(axis=1)
        margin_u = (top1 - top2) > TOL * np.maximum(np.abs(top1), 1.0)
    Cs = np.sort(C, axis=1)
    margin_c = (Cs[:, 1] - Cs[:, 0]) > TOL * np.maximum(Cs[:, 0], 1e-3) if C.shape[1] > 1 \
        else np.ones(len(C), bool)
    any_feas = feas.any(axis=1)
    clear = np.where(any_feas, margin_u, margin_c) & ~near_slo
    bad = np.nonzero(clear & (ch != wch))[0]
    assert bad.size == 0, f"{bad.size} clear decisions differ, e.g. query {bad[:5]}"
    assert clear.mean() >= min_checked, clear.mean()
    # the rest must still be valid choices: a deployment the GPU may call
    # feasible is at least as good (within tolerance) as every surely feasible
    # one; a choice made as "nothing feasible" needs nothing surely feasible
    # and has the lowest latency within tolerance
    for q in np.nonzero(~clear & ok)[0]:
        c = ch[q]
        if maybe[q, c]:
            if sure[q].any():
                best = U[q][sure[q]].max()
                assert U[q, c] >= best - 2 * TOL * max(abs(best), 1.0), (q, c)
        else:
            assert not sure[q].any(), (q, c)
            assert C[q, c] <= C[q].min() * (1 + 2 * TOL), (q, c)
    return float(clear.mean())


