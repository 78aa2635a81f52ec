"""Several values of lambda in one pass (the lambda sweep of HW-Router Sec. 5, RQ1).

hwr_route_batch_multi evaluates the predictor and the quality scores once and
applies the decision maker (Eq. 3) for each lambda.  Row k of its outputs must
equal a single-lambda route with lambdas[k]: bit for bit against the oracle's
canonical-fp32 route on the SIMT paths, bit for bit against the single-lambda
tensor route on the tensor path (both select from the same stored scores with
the same arithmetic), and within the bf16 tolerance of the fp64 oracle there.
"""
import numpy as np
import pytest

import oracle as O
import workload as W
import paper_2608_14575_gb300 as H
from tc_check import check_against_oracle

pytestmark = pytest.mark.gpu
LAMS = np.array([0.0, 0.25, 0.5, 1.0, 4.0, 0.125, 2.0 ** -7], np.float32)


@pytest.fixture(scope="module", autouse=True)
def built():
    H.build()


def _exact_row(got, k, want, what):
    ch, lat, util = (a[k] for a in got)
    bad = np.nonzero(ch != want[0])[0]
    assert bad.size == 0, f"{what}: chosen differs at {bad[:8]}"
    assert np.array_equal(lat, want[1].astype(np.float32), equal_nan=True), what
    assert np.array_equal(util, want[2].astype(np.float32), equal_nan=True), what


# (config, Q, flags): small batches, the fused SIMT kernel, bf16
# contexts on the SIMT kernels, and the score-convex utility
@pytest.mark.parametrize("c,Q,flags", [
    (0, 1, 0), (0, 97, 0), (0, 256, 0), (0, 1000, 0),
    (1, 40, H.HWR_PATH_SIMT), (1, 300, H.HWR_PATH_SIMT),
    (0, 300, H.HWR_SCORE_CONVEX), (4, 20, H.HWR_PATH_SIMT),
])
def test_simt_rows_equal_oracle_single_lambda(c, Q, flags):
    p = W.make_config(c, Q=Q)
    r = H.Router(p)
    lams = LAMS if not flags & H.HWR_SCORE_CONVEX else np.array([0.0, 0.25, 0.5, 1.0], np.float32)
    got = r.route_multi(lams, flags=flags)
    assert got[0].shape == (len(lams), Q)
    orc = O.Problem(p)
    conv = bool(flags & H.HWR_SCORE_CONVEX)
    for k, lam in enumerate(lams):
        want = orc.route(lam=float(lam), mode=O.F32, convex=conv, nthreads=8)
        _exact_row(got, k, want, f"cfg{c} Q={Q} lambda={lam}")
    # lambda = 0 picks by quality alone, a large lambda by latency alone:
    # the sweep's two ends must differ somewhere
    if Q >= 97 and not conv:
        assert not np.array_equal(got[0][0], got[0][4])
    r.close()


def test_three_heads_rows_exact():
    p = W.make_config(0, Q=200, n_heads=3)
    r = H.Router(p)
    got = r.route_multi(LAMS[:3])
    orc = O.Problem(p)
    for k, lam in enumerate(LAMS[:3]):
        _exact_row(got, k, orc.route(lam=float(lam), mode=O.F32, nthreads=8), f"lambda={lam}")
    r.close()


def test_max_lambdas_and_degenerate_budgets():
    p = W.make_config(0, Q=130)
    r = H.Router(p)
    lams = np.linspace(0.0, 3.0, 16).astype(np.float32)
    orc = O.Problem(p)
    for slo in (0.0, float("inf"), 5.0):
        got = r.route_multi(lams, slo=slo)
        for k in (0, 7, 15):
            _exact_row(got, k, orc.route(slo=slo, lam=float(lams[k]), mode=O.F32, nthreads=8),
                       f"slo={slo} k={k}")
    r.close()


def test_tensor_rows_equal_single_lambda_tensor():
    p = W.make_config(3, Q=3000)
    r = H.Router(p)
    lams = np.array([0.0, 0.1, 0.3, 1.0, 3.0], np.float32)
    got = r.route_multi(lams, flags=H.HWR_PATH_TENSOR)
    for k, lam in enumerate(lams):
        one = r.route(lam=float(lam), flags=H.HWR_PATH_TENSOR)
        for a, b in zip(one, (g[k] for g in got)):
            assert np.array_equal(a, b, equal_nan=True), f"lambda={lam}"
        check_against_oracle(p, (g[k] for g in got), lam=float(lam), min_checked=0.2)
    r.close()


def test_pipelined_host_equals_device():
    import torch
    p = W.make_config(3, Q=20_000)
    r = H.Router(p, stream=torch.cuda.current_stream().cuda_stream)
    lams = np.array([0.05, 0.3, 2.0], np.float32)
    host = r.route_multi(lams)                      # chunked host copies
    dev = torch.device("cuda:0")
    il = torch.from_numpy(p["in_len"]).to(dev)
    ol = torch.from_numpy(p["out_len"]).to(dev)
    em = torch.from_numpy(p["emb"].view(np.int16)).to(dev)
    K, Q = len(lams), p["Q"]
    ch = torch.empty((K, Q), dtype=torch.int32, device=dev)
    lat = torch.empty((K, Q), dtype=torch.float32, device=dev)
    ut = torch.empty((K, Q), dtype=torch.float32, device=dev)
    r.route_device_multi(lams, il, ol, em, ch, lat, ut, slo=p["slo"])
    torch.cuda.synchronize()
    assert np.array_equal(ch.cpu().numpy(), host[0])
    assert np.array_equal(lat.cpu().numpy(), host[1])
    assert np.array_equal(ut.cpu().numpy(), host[2])
    # and row by row the same as single-lambda routes of the default path
    for k, lam in enumerate(lams):
        one = r.route(lam=float(lam))
        assert np.array_equal(one[0], host[0][k])
    r.close()


def test_argument_errors():
    p = W.make_config(0, Q=8)
    r = H.Router(p)
    for bad in (np.zeros(0, np.float32), np.zeros(17, np.float32),
                np.array([0.5, np.nan], np.float32), np.array([np.inf], np.float32)):
        with pytest.raises(H.HwrError) as e:
            r.route_multi(bad)
        assert e.value.status == 1
    with pytest.raises(H.HwrError) as e:
        r.route_multi(LAMS[:2], flags=H.HWR_SEQUENTIAL)
    assert e.value.status == 7
    assert r.route_multi(LAMS[:2])[0].shape == (2, 8)     # still usable
    r.close()


@pytest.mark.parametrize("c,Q", [(0, 97), (2, 40)])
def test_pair_kernel_rows_equal_oracle(monkeypatch, c, Q):
    """The pair-parallel kernel's stored scores feed the multi-lambda selection."""
    monkeypatch.setenv("HWR_PAIRS_MAX_PAIRS", "2048")
    p = W.make_config(c, Q=Q)
    r = H.Router(p)
    got = r.route_multi(LAMS)
    C, qual = r.score()
    r.close()
    orc = O.Problem(p)
    for k, lam in enumerate(LAMS):
        _exact_row(got, k, orc.route(lam=float(lam), mode=O.F32, nthreads=8), f"cfg{c} lambda={lam}")
    Cw, _ = orc.score_all(mode=O.F32, nthreads=8)
    assert np.array_equal(C, Cw.astype(np.float32))


# the selection kernel's lane map (lane l: deployments l and l + 32) on
# clusters of 1, 15, 33 and 64 deployments, and exact ties (every model's
# quality 0.5 and only the GPU one-hot and the query lengths feeding layer 1:
# deployments of one GPU type tie exactly and the lowest index must win)
@pytest.mark.parametrize("shape", [
    dict(M=1, G=1, F=12, H1=8, H2=8, E=8),
    dict(M=5, G=3, F=24, H1=40, H2=24, E=16),
    dict(M=11, G=3, F=24, H1=32, H2=36, E=24),
    dict(M=16, G=4, F=48, H1=32, H2=32, E=16),
])
def test_selection_lane_map_rows_exact(shape):
    p = W.make_problem(Q=150, dtype="f32", lam=0.3, slo=3.0, seed=53, bias_std=0.2, **shape)
    r = H.Router(p)
    got = r.route_multi(LAMS)
    r.close()
    orc = O.Problem(p)
    for k, lam in enumerate(LAMS):
        _exact_row(got, k, orc.route(lam=float(lam), mode=O.F32, nthreads=8), f"{shape} lambda={lam}")


@pytest.mark.parametrize("slo", [float("inf"), float("-inf")])
def test_selection_exact_ties_rows(slo):
    M, G, F = 16, 4, 48
    p = W.make_problem(Q=60, dtype="f32", M=M, G=G, F=F, H1=32, H2=32, E=16, seed=9,
                       lam=0.4, slo=2.0, bias_std=0.3)
    keep = np.zeros(F, bool)
    keep[M:M + G] = True
    keep[F - 2:] = True
    p["W1"] = np.where(keep[None, :], p["W1"], 0.0).astype(p["W1"].dtype)
    p["memb"] = np.zeros_like(p["memb"])
    r = H.Router(p)
    got = r.route_multi(LAMS, slo=slo)
    r.close()
    orc = O.Problem(p)
    for k, lam in enumerate(LAMS):
        _exact_row(got, k, orc.route(slo=slo, lam=float(lam), mode=O.F32, nthreads=8),
                   f"ties slo={slo} lambda={lam}")
        assert np.all((got[0][k] >= 0) & (got[0][k] < G))
