"""Pins for the CPU oracle: checks against what the paper and mathematics fix.

Every check takes the loaded oracle library (``lib``) so the same checks can
be re-run against deliberately broken oracle builds (test_oracle_mutants.py).
A check raises AssertionError when the oracle disagrees with the pin.

Kinds of pin used here
  * closed forms: hand-set weights for which TTFT, TPOT and the cost of
    Eq. 2 reduce to expressions like ln 5 + n ln(5/4) (golden file
    closed_form_predictor.json);
  * hand-worked selections under Eq. 3 (golden file selection_cases.json)
    and brute-force enumeration with a different algorithm (sort by key);
  * library routines as independent references: numpy.matmul in fp64 for
    the quality contraction;
  * special values: softplus(0) = ln 2, sigmoid(0) = 1/2, symmetry identities;
  * invariants: lambda = 0 picks the best-quality model, huge lambda picks the
    lowest cost, the choice is feasible whenever one is, permutation
    equivariance, sequential mode reducing to batch mode;
  * exact rational arithmetic: the canonical-fp32 mode recomputed with
    Fraction-based round-to-nearest-even fma on tiny inputs, bit for bit.
"""
from __future__ import annotations

import json
import math
import os
from fractions import Fraction

import numpy as np

import oracle as O
import workload as W

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


# ---------------------------------------------------------------------------
# exact float32 arithmetic (round to nearest, ties to even)

def round_f32(x: Fraction) -> float:
    if x == 0:
        return 0.0
    sign = -1.0 if x < 0 else 1.0
    a = abs(x)
    e = a.numerator.bit_length() - a.denominator.bit_length()
    while Fraction(2) ** e > a:
        e -= 1
    while Fraction(2) ** (e + 1) <= a:
        e += 1
    e = max(e, -126)
    q = Fraction(2) ** (e - 23)
    m = a / q
    n = m.numerator // m.denominator
    r = m - n
    if r > Fraction(1, 2) or (r == Fraction(1, 2) and n % 2 == 1):
        n += 1
    return sign * float(n * q)


def fma_f32(a, b, c) -> float:
    return round_f32(Fraction(float(a)) * Fraction(float(b)) + Fraction(float(c)))


def mul_f32(a, b) -> float:
    return round_f32(Fraction(float(a)) * Fraction(float(b)))


def f32(x) -> float:
    return float(np.float32(x))


# ---------------------------------------------------------------------------
# problem builders

def tiny(M=2, G=2, F=16, H1=4, H2=4, E=8, Q=4, dtype="f32", seed=11,
         bias_std=0.0, weight_std=0.1, lam=0.5, slo=5.0):
    return W.make_problem(Q=Q, M=M, G=G, F=F, H1=H1, H2=H2, E=E, dtype=dtype,
                          lam=lam, slo=slo, seed=seed, bias_std=bias_std,
                          weight_std=weight_std)


def blank(M=2, G=2, F=16, H1=4, H2=4, E=8, Q=1, n_heads=2):
    """A problem with zero weights, zero biases, identity transforms and
    (mu, sd) = (0, 1) on every slot, for hand-set closed-form cases."""
    p = W.make_problem(Q=Q, M=M, G=G, F=F, H1=H1, H2=H2, E=E, dtype="f32", lam=0.5,
                       slo=5.0, seed=11, n_heads=n_heads)
    for n in ("W1", "W2", "W3"):
        p[n] = np.zeros_like(p[n])
    for n in ("b1", "b2", "b3"):
        p[n] = np.zeros_like(p[n])
    p["mu"] = np.zeros(F, np.float32)
    p["sd"] = np.ones(F, np.float32)
    p["xform"] = np.zeros(F, np.uint8)
    return p


# ---------------------------------------------------------------------------
# special values of the output activations

def check_activations(lib):
    ln2 = math.log(2.0)
    sp = lambda z: O.softplus(z, O.F64, lib)
    sg = lambda s: O.sigmoid(s, O.F64, lib)
    assert abs(sp(0.0) - ln2) <= 2e-16, sp(0.0)
    assert abs(sg(0.0) - 0.5) == 0.0, sg(0.0)
    assert abs(sg(math.log(3.0)) - 0.75) <= 1e-15
    for z in (-30.0, -3.5, -0.25, 0.7, 4.0, 35.0):
        # log(1+e^z) - log(1+e^-z) = z, and log(1+e^z) >= max(z, 0)
        assert abs((sp(z) - sp(-z)) - z) <= 1e-13 * max(1.0, abs(z)), z
        assert sp(z) >= max(z, 0.0) and sp(z) > 0.0
        assert abs(sg(z) + sg(-z) - 1.0) <= 1e-15, z
    assert abs(sp(-40.0) / math.exp(-40.0) - 1.0) < 1e-12
    assert abs(sp(40.0) - 40.0 - math.exp(-40.0)) < 1e-15
    assert O.softplus(0.0, O.F32, lib) == f32(ln2)
    assert O.sigmoid(0.0, O.F32, lib) == 0.5


# ---------------------------------------------------------------------------
# closed-form predictor cases (golden/closed_form_predictor.json)

def _apply_case(p, case):
    lay = W.feature_layout(p["M"], p["G"], p["F"])
    if "slot_index" in case:
        k = case["slot_index"]
    elif case["slot"] == "pad":
        k = lay["tpot"] + 1
    else:
        k = lay[case["slot"]]
    p["W1"][0, k] = case["w1"]
    p["b1"][0] = case.get("b1", 0.0)
    p["W2"][0, 0] = case.get("w2", 1.0)
    p["b2"][0] = case.get("b2", 0.0)
    p["W3"][0, 0], p["W3"][1, 0] = case["w3"]
    p["b3"][:] = case.get("b3", [0.0, 0.0])
    p["mu"][k] = case.get("mu", 0.0)
    p["sd"][k] = case.get("sd", 1.0)
    p["xform"][k] = case.get("xform", 0)
    raw = case.get("raw")
    slot = case["slot"]
    if slot in ("running", "waiting", "kv", "gpu_util", "ttft", "tpot"):
        p["snap"][slot][:] = raw
    elif slot == "log10p":
        p["log10p"][:] = raw
    elif slot == "in_len":
        p["in_len"][:] = raw
    elif slot == "out_len":
        p["out_len"][:] = raw
    if "out_len" in case:
        p["out_len"][:] = case["out_len"]
    return k


def check_closed_form_predictor(lib):
    env = {"log": math.log, "exp": math.exp, "e": math.e}
    for case in _golden("closed_form_predictor.json")["cases"]:
        for mode, tol in ((O.F64, 1e-12), (O.F32, 2e-6)):
            p = blank()
            _apply_case(p, case)
            pr = O.Problem(p, lib=lib)
            C, _ = pr.score_all(lam=0.0, mode=mode)
            for d in range(p["D"]):
                if "expect_by_model" in case:
                    exp_ = case["expect_by_model"][str(int(p["dep_model"][d]))]
                elif "expect_by_gpu" in case:
                    exp_ = case["expect_by_gpu"][str(int(p["dep_gpu"][d]))]
                else:
                    exp_ = case["expect"]
                x = pr.features(d, p["in_len"][0], p["out_len"][0], mode)
                ttft, tpot = pr.predict(x, mode)
                want_ttft = eval(exp_["ttft"], env)
                want_tpot = eval(exp_["tpot"], env)
                want_c = want_ttft + float(p["out_len"][0]) * want_tpot
                assert abs(ttft - want_ttft) <= tol * abs(want_ttft), \
                    (case["name"], mode, d, ttft, want_ttft)
                assert abs(tpot - want_tpot) <= tol * abs(want_tpot), \
                    (case["name"], mode, d, tpot, want_tpot)
                assert abs(C[0, d] - want_c) <= tol * abs(want_c), \
                    (case["name"], mode, d, C[0, d], want_c)


# ---------------------------------------------------------------------------
# selection rule (Eq. 3)

def check_selection_golden(lib):
    nan = float("nan")
    for case in _golden("selection_cases.json")["cases"]:
        C = [nan if v is None else (float("-0.0") if v == "-0" else v)
             for v in case["C"]]
        U = [nan if v is None else (float("-0.0") if v == "-0" else v)
             for v in case["U"]]
        for mode in (O.F64, O.F32):
            got = O.select(C, U, case["slo"], mode, lib)
            assert got == case["chosen"], (case["name"], mode, got)


def _select_by_sort(C, U, slo):
    """Eq. 3 as a sort: feasible deployments first by (-U, d); else by (C, d)."""
    D = len(C)
    feas = [d for d in range(D) if C[d] <= slo and not math.isnan(U[d])]
    if feas:
        return sorted(feas, key=lambda d: (-U[d], d))[0]
    ok = [d for d in range(D) if not math.isnan(C[d])]
    if not ok:
        return -1
    return sorted(ok, key=lambda d: (C[d], d))[0]


def check_selection_bruteforce(lib, n=3000, seed=5):
    rng = np.random.default_rng(seed)
    levels = np.array([0.25, 0.5, 1.0, 2.0, 3.0])
    for _ in range(n):
        D = int(rng.integers(1, 6))
        C = [float(v) for v in rng.choice(levels, D)]
        U = [float(v) for v in rng.choice(levels - 1.0, D)]
        slo = float(rng.choice([0.1, 0.5, 1.0, 2.0, 5.0]))
        want = _select_by_sort(C, U, slo)
        for mode in (O.F64, O.F32):
            assert O.select(C, U, slo, mode, lib) == want, (C, U, slo)


# ---------------------------------------------------------------------------
# quality contraction (Sec. 3.2, hardware independent)

def check_quality_matmul(lib):
    for dtype in ("f32", "bf16"):
        p = tiny(dtype=dtype, E=24, M=3, G=2, Q=6, F=16)
        pr = O.Problem(p, lib=lib)
        emb = O._widen(p["emb"]).reshape(p["Q"], p["E"]).astype(np.float64)
        memb = O._widen(p["memb"]).reshape(p["E"], p["M"]).astype(np.float64)
        s = np.matmul(emb, memb)
        want = 1.0 / (1.0 + np.exp(-s))
        for q in range(p["Q"]):
            got = pr.quality(p["emb"][q], O.F64)
            assert np.allclose(got, want[q], rtol=1e-13, atol=0), (q, got, want[q])
            got32 = pr.quality(p["emb"][q], O.F32)
            assert np.allclose(got32, want[q], rtol=1e-6, atol=0)
    # an embedding orthogonal to every model column scores exactly 1/2
    p = blank(E=8, M=2, G=2)
    p["memb"] = np.zeros((8, 2), np.float32)
    p["memb"][0, 0] = 1.0
    p["memb"][1, 1] = -2.0
    pr = O.Problem(p, lib=lib)
    e = np.zeros(8, np.float32)
    e[2] = 1.0
    assert list(pr.quality(e, O.F64)) == [0.5, 0.5]
    e[0], e[1] = 0.5, 0.25
    got = pr.quality(e, O.F64)
    assert abs(got[0] - 1 / (1 + math.exp(-0.5))) < 1e-15
    assert abs(got[1] - 1 / (1 + math.exp(0.5))) < 1e-15


# ---------------------------------------------------------------------------
# invariants of the full route

def check_lambda_zero_picks_best_model(lib):
    for seed in (1, 2, 3):
        p = tiny(M=3, G=2, E=16, Q=40, seed=seed, F=16)
        pr = O.Problem(p, lib=lib)
        emb = O._widen(p["emb"]).reshape(p["Q"], p["E"]).astype(np.float64)
        s = emb @ O._widen(p["memb"]).reshape(p["E"], p["M"]).astype(np.float64)
        best_m = np.argmax(s, axis=1)
        for mode in (O.F64, O.F32):
            ch, _, util, _ = pr.route(slo=float("inf"), lam=0.0, mode=mode)
            # every GPU of the best model ties; the lowest index is m * G + 0
            assert np.array_equal(ch, best_m * p["G"]), (mode, ch, best_m)
            assert np.allclose(util, 1 / (1 + np.exp(-s.max(axis=1))), rtol=1e-6)


def check_huge_lambda_picks_cheapest(lib):
    p = tiny(M=3, G=3, Q=30, seed=4, F=16)
    pr = O.Problem(p, lib=lib)
    for mode in (O.F64, O.F32):
        C, _ = pr.score_all(lam=1e6, mode=mode)
        ch, lat, _, _ = pr.route(slo=float("inf"), lam=1e6, mode=mode)
        assert np.array_equal(ch, np.argmin(C, axis=1))
        assert np.array_equal(lat, C.min(axis=1))


def check_feasible_choice(lib):
    for seed in range(6):
        p = tiny(M=2, G=3, Q=50, seed=seed, F=16)
        pr = O.Problem(p, lib=lib)
        C, U = pr.score_all()
        for slo in (0.0, np.median(C), np.percentile(C, 90), 1e9):
            ch, lat, util, _ = pr.route(slo=slo)
            for q in range(p["Q"]):
                feas = C[q] <= slo
                if feas.any():
                    assert feas[ch[q]]
                    assert U[q, ch[q]] == U[q][feas].max()
                else:
                    assert C[q, ch[q]] == C[q].min()
                assert lat[q] == C[q, ch[q]] and util[q] == U[q, ch[q]]
                assert lat[q] > 0.0


def check_single_deployment(lib):
    p = tiny(M=1, G=1, Q=12, F=12)
    pr = O.Problem(p, lib=lib)
    for slo in (0.0, 1e9):
        ch, _, _, _ = pr.route(slo=slo)
        assert (ch == 0).all()


def check_permutation_equivariance(lib):
    p = tiny(M=3, G=2, Q=25, seed=9, F=16)
    pr = O.Problem(p, lib=lib)
    ch, lat, util, _ = pr.route()
    perm = np.array([3, 0, 5, 1, 4, 2])
    q = dict(p)
    q["dep_model"] = p["dep_model"][perm]
    q["dep_gpu"] = p["dep_gpu"][perm]
    q["snap"] = {k: v[perm] for k, v in p["snap"].items()}
    ch2, lat2, util2, _ = O.Problem(q, lib=lib).route()
    assert np.array_equal(perm[ch2], ch)
    assert np.array_equal(lat2, lat) and np.array_equal(util2, util)


def check_convex_score(lib):
    p = tiny(Q=20, seed=3)
    pr = O.Problem(p, lib=lib)
    lam = 0.25  # exactly representable: the route takes lambda as float32
    C, U = pr.score_all(lam=lam)
    _, Uc = pr.score_all(lam=lam, convex=True)
    qual = U + lam * C                       # U = Q - lam C
    assert np.allclose(Uc, (1 - lam) * qual - lam * C, rtol=1e-12, atol=1e-14)
    assert 0.0 < qual.min() and qual.max() < 1.0


def check_fp32_near_fp64(lib):
    for c, Q in ((0, 256), (1, 48), (2, 48)):
        p = W.make_config(c, Q=Q)
        pr = O.Problem(p, lib=lib)
        C64, U64 = pr.score_all(mode=O.F64)
        C32, U32 = pr.score_all(mode=O.F32)
        assert np.max(np.abs(C32 - C64) / np.abs(C64)) < 1e-5
        assert np.max(np.abs(U32 - U64) / np.maximum(np.abs(U64), 1.0)) < 1e-5


def check_sequential(lib):
    p = tiny(M=2, G=3, Q=30, seed=8, F=16, lam=0.5, slo=1e9)
    # make the running count matter
    lay = W.feature_layout(p["M"], p["G"], p["F"])
    p["W1"][:, lay["running"]] = 0.8
    pr = O.Problem(p, lib=lib)
    for mode in (O.F64, O.F32):
        # Q = 1: sequential == batch
        one = dict(in_len=p["in_len"][:1], out_len=p["out_len"][:1], emb=p["emb"][:1])
        a = pr.route(**one, mode=mode)
        b = pr.route(**one, mode=mode, sequential=True)
        assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])
        assert b[3][b[0][0]] == p["snap"]["running"][b[0][0]] + 1
        # query-by-query batch routing with a hand-updated snapshot
        ch_s, lat_s, ut_s, run_s = pr.route(mode=mode, sequential=True)
        run = p["snap"]["running"].copy()
        for q in range(p["Q"]):
            snap = dict(p["snap"])
            snap["running"] = run
            pq = O.Problem(p, snap=snap, lib=lib)
            c, l, u, _ = pq.route(p["in_len"][q:q + 1], p["out_len"][q:q + 1],
                                  p["emb"][q:q + 1], mode=mode)
            assert c[0] == ch_s[q] and l[0] == lat_s[q] and u[0] == ut_s[q]
            run = run.copy()
            run[c[0]] += 1
        assert np.array_equal(run, run_s)
        assert run_s.sum() == p["snap"]["running"].sum() + p["Q"]
    # with no weight on the running slot, sequential == batch
    p["W1"][:, lay["running"]] = 0.0
    pr = O.Problem(p, lib=lib)
    a = pr.route()
    b = pr.route(sequential=True)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])


# ---------------------------------------------------------------------------
# canonical fp32 mode, bit for bit, with exact rational arithmetic

def _canon_pair(p, d, q, lam, convex):
    """Canonical-fp32 evaluation of one (query, deployment) pair in exact
    rational arithmetic rounded to float32 after every operation."""
    M, G, F = p["M"], p["G"], p["F"]
    lay = W.feature_layout(M, G, F)
    W1 = O._widen(p["W1"]).reshape(p["H1"], F)
    W2 = O._widen(p["W2"]).reshape(p["H2"], p["H1"])
    W3 = O._widen(p["W3"]).reshape(2, p["H2"])
    memb = O._widen(p["memb"]).reshape(p["E"], M)
    emb = O._widen(p["emb"]).reshape(p["Q"], p["E"])
    m, g, s = int(p["dep_model"][d]), int(p["dep_gpu"][d]), p["snap"]
    raw = [0.0] * F
    raw[m] = 1.0
    raw[M + g] = 1.0
    raw[lay["log10p"]] = float(p["log10p"][m])
    for key in ("running", "waiting", "kv", "gpu_util", "ttft", "tpot"):
        raw[lay[key]] = float(s[key][d])
    raw[F - 2] = float(p["in_len"][q])
    raw[F - 1] = float(p["out_len"][q])
    x = []
    for k in range(F):
        t = raw[k]
        code = int(p["xform"][k])
        t = math.log1p(t) if code == 1 else (math.log(t) if code == 2 else t)
        x.append(f32((t - float(p["mu"][k])) / float(p["sd"][k])))
    h1 = []
    for j in range(p["H1"]):
        acc = float(p["b1"][j])
        for k in range(F):
            acc = fma_f32(W1[j, k], x[k], acc)
        h1.append(acc if acc > 0 else 0.0)
    h2 = []
    for i in range(p["H2"]):
        acc = float(p["b2"][i])
        for j in range(p["H1"]):
            acc = fma_f32(W2[i, j], h1[j], acc)
        h2.append(acc if acc > 0 else 0.0)
    z = []
    for o in range(2):
        acc = float(p["b3"][o])
        for i in range(p["H2"]):
            acc = fma_f32(W3[o, i], h2[i], acc)
        z.append(acc)
    sp = lambda v: f32(max(v, 0.0) + math.log1p(math.exp(-abs(v))))
    ttft, tpot = sp(z[0]), sp(z[1])
    C = fma_f32(p["out_len"][q], tpot, ttft)
    acc = 0.0
    for k in range(p["E"]):
        acc = fma_f32(emb[q, k], memb[k, m], acc)
    qual = f32(1.0 / (1.0 + math.exp(-acc)))
    lam32 = f32(lam)
    wq = f32(1.0 - lam32) if convex else 1.0
    U = fma_f32(-lam32, C, mul_f32(wq, qual))
    return C, U, x


def check_canonical_fp32_exact(lib):
    for seed, dtype, convex in ((21, "f32", False), (22, "bf16", True)):
        p = tiny(M=2, G=2, F=14, H1=5, H2=3, E=6, Q=3, seed=seed,
                 bias_std=0.2, weight_std=0.7, dtype=dtype)
        pr = O.Problem(p, lib=lib)
        C, U = pr.score_all(mode=O.F32, convex=convex)
        for q in range(p["Q"]):
            for d in range(p["D"]):
                c, u, x = _canon_pair(p, d, q, p["lam"], convex)
                assert C[q, d] == c and U[q, d] == u, (seed, q, d, C[q, d], c,
                                                        U[q, d], u)
                got_x = pr.features(d, p["in_len"][q], p["out_len"][q], O.F32)
                assert list(got_x) == x, (seed, q, d)
    # hand cases that separate fused from unfused and fix the order
    p = blank(F=12, H1=1, H2=1, M=1, G=1, E=1)
    lay = W.feature_layout(1, 1, 12)
    k1, k2, k3 = lay["kv"], lay["gpu_util"], lay["log10p"]
    tiny_ = 2.0 ** -24
    # bias first, then k ascending: 1 + 2^-24 rounds back to 1 twice
    p["b1"][0] = 1.0
    p["W1"][0, k1] = 1.0
    p["W1"][0, k2] = 1.0
    p["snap"]["kv"][:] = tiny_
    p["snap"]["gpu_util"][:] = tiny_
    p["W2"][0, 0] = 1.0
    p["W3"][0, 0] = 1.0
    p["W3"][1, 0] = 1.0
    pr = O.Problem(p, lib=lib)
    x = pr.features(0, p["in_len"][0], p["out_len"][0], O.F32)
    t, _ = pr.predict(x, O.F32)
    assert t == f32(math.log1p(math.exp(-1.0)) + 1.0), t  # z0 == 1 exactly
    # fused multiply-add: (1 + 2^-12)^2 - 1 keeps its 2^-24 term
    p = blank(F=12, H1=1, H2=1, M=1, G=1, E=1)
    a = 1.0 + 2.0 ** -12
    p["b1"][0] = -1.0
    p["W1"][0, k3] = a
    p["log10p"][:] = a
    p["W2"][0, 0] = 1.0
    p["W3"][0, 0] = 1.0
    pr = O.Problem(p, lib=lib)
    x = pr.features(0, p["in_len"][0], p["out_len"][0], O.F32)
    t, _ = pr.predict(x, O.F32)
    z = 2.0 ** -11 + 2.0 ** -24
    assert t == f32(z + math.log1p(math.exp(-z))), t


# ---------------------------------------------------------------------------
# third output head N_out (Eq. 1) entering the cost (Eq. 2)

def check_three_heads(lib):
    p = blank(n_heads=3)
    lay = W.feature_layout(p["M"], p["G"], p["F"])
    k = lay["running"]
    p["W1"][0, k] = 1.0
    p["xform"][k] = 1                      # log1p
    p["snap"]["running"][:] = 3            # x = ln 4
    p["W2"][0, 0] = 1.0
    p["W3"][:, 0] = [1.0, -1.0, 1.0]       # TTFT = log 5, TPOT = log 1.25, N_out = log 5
    for mode, tol in ((O.F64, 1e-12), (O.F32, 2e-6)):
        for out_len in (7.0, 700.0):       # the given length must not enter Eq. 2
            p["out_len"][:] = out_len
            pr = O.Problem(p, lib=lib)
            x = pr.features(0, p["in_len"][0], p["out_len"][0], mode)
            t, tp, n = pr.predict(x, mode, heads=True)
            assert abs(n - math.log(5.0)) <= tol * math.log(5.0), n
            C, _ = pr.score_all(lam=0.0, mode=mode)
            want = math.log(5.0) + math.log(5.0) * math.log(1.25)
            assert np.all(np.abs(C - want) <= tol * want), (C, want)
    # with a constant third head equal to every query's length, three heads
    # reduce to two
    q2 = tiny(Q=10, seed=6)
    q3 = tiny(Q=10, seed=6)
    q3["n_heads"] = 3
    q3["W3"] = np.concatenate([q2["W3"], np.zeros((1, q2["H2"]), np.float32)])
    n = 150.0
    q3["b3"] = np.concatenate([q2["b3"], [np.float32(math.log(math.expm1(n)))]])
    q2["out_len"][:] = n
    q3["out_len"][:] = n
    C2, U2 = O.Problem(q2, lib=lib).score_all()
    C3, U3 = O.Problem(q3, lib=lib).score_all()
    assert np.allclose(C3, C2, rtol=1e-5), (C2, C3)


# ---------------------------------------------------------------------------
# per-query SLO budgets (Sec. 4.4, Eq. 4-5)

def check_slo_budget(lib):
    # TTFT_SLO(p) = slack (a + b p); budget = TTFT_SLO(p) + d TPOT_SLO
    # (b = 2^-10 per token and TPOT_SLO = 2^-6 s are exact in float32)
    got = O.slo_budget(0.5, 2.0 ** -10, 1.25, 2.0 ** -6, [1024.0, 0.0], [64.0, 32.0], O.F64, lib)
    assert got[0] == 1.25 * (0.5 + 1.0) + 1.0, got
    assert got[1] == 1.25 * 0.5 + 0.5, got
    # fp32 order: t = fma(b, p, a); s = slack * t; B = fma(tpot, d, s)
    # values for which computing b * p + a unfused changes the final budget
    a, b, sl, tp = 0.4524623453617096, 0.000643032428342849, f32(1.2), f32(0.021)
    p_, d_ = 31701.0, 110.3285903930664
    assert fma_f32(tp, d_, mul_f32(sl, f32(f32(b * p_) + a))) != \
        fma_f32(tp, d_, mul_f32(sl, fma_f32(b, p_, a)))
    t = fma_f32(b, p_, a)
    want = fma_f32(tp, d_, mul_f32(sl, t))
    got = O.slo_budget(a, b, sl, tp, [p_], [d_], O.F32, lib)[0]
    assert got == want, (got, want)


def check_per_query_slo(lib):
    p = tiny(M=2, G=3, Q=60, seed=12, F=16)
    pr = O.Problem(p, lib=lib)
    C, U = pr.score_all()
    rng = np.random.default_rng(3)
    budgets = np.quantile(C, rng.uniform(0.0, 1.0, p["Q"])).astype(np.float32)
    budgets[:5] = np.inf
    budgets[5:10] = 0.0
    for mode in (O.F64, O.F32):
        ch, lat, util, _ = pr.route_slo(budgets, mode=mode)
        Cm, Um = pr.score_all(mode=mode)
        for q in range(p["Q"]):
            feas = Cm[q] <= budgets[q]
            if feas.any():
                assert feas[ch[q]] and Um[q, ch[q]] == Um[q][feas].max(), q
            else:
                assert Cm[q, ch[q]] == Cm[q].min(), q
        # one budget per query: equal to routing that query alone with it
        for q in (0, 7, 33):
            c1, l1, u1, _ = pr.route(p["in_len"][q:q + 1], p["out_len"][q:q + 1],
                                     p["emb"][q:q + 1], slo=float(budgets[q]), mode=mode)
            assert c1[0] == ch[q] and l1[0] == lat[q]
    # sequential with per-query budgets equals the query-by-query replay
    ch_s, _, _, run_s = pr.route_slo(budgets, sequential=True)
    run = p["snap"]["running"].copy()
    for q in range(p["Q"]):
        snap = dict(p["snap"])
        snap["running"] = run
        c, _, _, _ = O.Problem(p, snap=snap, lib=lib).route(
            p["in_len"][q:q + 1], p["out_len"][q:q + 1], p["emb"][q:q + 1],
            slo=float(budgets[q]))
        assert c[0] == ch_s[q], q
        run = run.copy()
        run[c[0]] += 1
    assert np.array_equal(run, run_s)


ALL_CHECKS = [
    check_activations,
    check_closed_form_predictor,
    check_selection_golden,
    check_selection_bruteforce,
    check_quality_matmul,
    check_lambda_zero_picks_best_model,
    check_huge_lambda_picks_cheapest,
    check_feasible_choice,
    check_single_deployment,
    check_permutation_equivariance,
    check_convex_score,
    check_fp32_near_fp64,
    check_sequential,
    check_canonical_fp32_exact,
    check_slo_budget,
    check_per_query_slo,
    check_three_heads,
]
