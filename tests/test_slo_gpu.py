"""Per-query SLO budgets (HW-Router Sec. 4.4, Eq. 4-5) on the GPU.

hwr_route_batch_slo takes one budget per query, or the paper's SLO model
B_q = slack * (a + b * p_q) + d_q * TPOT_SLO evaluated on the device.  The
SIMT kernels must equal the oracle's canonical-fp32 route bit for bit; the
tensor path must meet the bf16 tolerance (tests/tc_check.py).
"""
import numpy as np
import pytest

import oracle as O
import workload as W
import paper_2608_14575_gb300 as H
from tc_check import check_against_oracle

pytestmark = pytest.mark.gpu
MODEL = (0.35, 2.0 ** -9, 1.2, 0.0119)          # a (s), b (s/token), slack, TPOT_SLO (s)


@pytest.fixture(scope="module", autouse=True)
def built():
    H.build()


def _budgets(p, seed=0):
    C, _ = O.Problem(p).score_all(nthreads=16)
    rng = np.random.default_rng(seed)
    b = np.quantile(C, rng.uniform(0.0, 1.0, p["Q"])).astype(np.float32)
    b[::17] = np.inf
    b[5::23] = 0.0
    return b


def _exact(got, want):
    assert np.array_equal(got[0], want[0])
    assert np.array_equal(got[1], want[1].astype(np.float32), equal_nan=True)
    assert np.array_equal(got[2], want[2].astype(np.float32), equal_nan=True)


@pytest.mark.parametrize("c,Q", [(0, 97), (0, 256), (1, 40), (1, 300)])
def test_budget_array_simt_exact(c, Q):
    p = W.make_config(c, Q=Q)
    b = _budgets(p)
    r = H.Router(p)
    got = r.route_slo(budgets=b, flags=H.HWR_PATH_SIMT)
    _exact(got, O.Problem(p).route_slo(b, mode=O.F32))
    r.close()


# (0, 256): the fused kernel; (2, 64): the small-batch kernel, which reads the
# lengths from the mapped host staging
@pytest.mark.parametrize("c,Q", [(0, 256), (2, 64)])
def test_budget_model_simt_exact(c, Q):
    p = W.make_config(c, Q=Q)
    want_b = O.slo_budget(*MODEL, p["in_len"], p["out_len"], mode=O.F32).astype(np.float32)
    r = H.Router(p)
    got = r.route_slo(model=MODEL)
    _exact(got, O.Problem(p).route_slo(want_b, mode=O.F32))
    # the same budgets given as an array route identically
    got2 = r.route_slo(budgets=want_b)
    assert all(np.array_equal(a, b) for a, b in zip(got, got2))
    r.close()


def test_budget_model_sequential_exact():
    p = W.make_config(2, Q=70)
    want_b = O.slo_budget(*MODEL, p["in_len"], p["out_len"], mode=O.F32).astype(np.float32)
    r = H.Router(p)
    got = r.route_slo(model=MODEL, flags=H.HWR_SEQUENTIAL)
    want = O.Problem(p).route_slo(want_b, mode=O.F32, sequential=True)
    _exact(got, want)
    assert np.array_equal(r.get_snapshot(), want[3])
    r.close()


def test_budget_array_sequential_exact():
    p = W.make_config(2, Q=150)
    b = _budgets(p, seed=4)
    r = H.Router(p)
    got = r.route_slo(budgets=b, flags=H.HWR_SEQUENTIAL)
    want = O.Problem(p).route_slo(b, mode=O.F32, sequential=True)
    _exact(got, want)
    assert np.array_equal(r.get_snapshot(), want[3])
    r.close()


def test_budget_tensor_within_tolerance():
    p = W.make_config(3, Q=3000)
    b = _budgets(p, seed=2)
    r = H.Router(p)
    got = r.route_slo(budgets=b, flags=H.HWR_PATH_TENSOR)
    check_against_oracle(p, got, slo=b, min_checked=0.2)
    gm = r.route_slo(model=MODEL, flags=H.HWR_PATH_TENSOR)
    bm = O.slo_budget(*MODEL, p["in_len"], p["out_len"], mode=O.F32).astype(np.float32)
    check_against_oracle(p, gm, slo=bm, min_checked=0.2)
    r.close()


def test_budget_pipelined_host_and_device_agree():
    import torch
    p = W.make_config(3, Q=20_000)
    b = _budgets(p, seed=3)
    r = H.Router(p, stream=torch.cuda.current_stream().cuda_stream)
    host = r.route_slo(budgets=b)                      # chunked copies
    dev = torch.device("cuda:0")
    il = torch.from_numpy(p["in_len"]).to(dev)
    ol = torch.from_numpy(p["out_len"]).to(dev)
    em = torch.from_numpy(p["emb"].view(np.int16)).to(dev)
    bd = torch.from_numpy(b).to(dev)
    ch = torch.empty(p["Q"], dtype=torch.int32, device=dev)
    lat = torch.empty(p["Q"], dtype=torch.float32, device=dev)
    ut = torch.empty(p["Q"], dtype=torch.float32, device=dev)
    r.route_device_slo(il, ol, em, ch, lat, ut, budgets=bd, lam=p["lam"])
    torch.cuda.synchronize()
    assert np.array_equal(ch.cpu().numpy(), host[0])
    assert np.array_equal(lat.cpu().numpy(), host[1])
    r.close()


def test_budget_spec_validation():
    p = W.make_config(0, Q=8)
    r = H.Router(p)
    with pytest.raises(H.HwrError) as e:
        r.route_slo(model=(0.1, float("nan"), 1.2, 0.01))
    assert e.value.status == 1
    r.close()
