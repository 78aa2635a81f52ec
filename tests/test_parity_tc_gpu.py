"""GPU parity of the bf16 tensor-core path (tcgen05 + TMA) against the oracle.

The tensor path rounds the layer-1 activations to bf16 for the layer-2 MMA and
accumulates in fp32, so it is held to the bf16 tolerance against the fp64
oracle: predicted latency and utility within 2e-2 relative (utility relative
to max(|U|, 1)).  Chosen indices must match wherever the decision is not
within that tolerance of a tie: the oracle's top-2 utility margin (or, with
no feasible deployment, the top-2 latency margin) exceeds 2e-2 and no
deployment's latency is within 2e-2 of the SLO.  For the remaining queries
the chosen deployment must still be a valid near-optimal choice.
"""
import numpy as np
import pytest

import oracle as O  # noqa: F401
import workload as W
import paper_2608_14575_gb300 as H
from tc_check import TOL, check_against_oracle

pytestmark = pytest.mark.gpu
TC = H.HWR_PATH_TENSOR


@pytest.fixture(scope="module", autouse=True)
def built():
    H.build()


def test_mid_bf16_full():
    p = W.make_config(1)                   # Q = 4096, D = 12, H = 128, E = 768
    r = H.Router(p)
    got = r.route(flags=TC)
    frac = check_against_oracle(p, got)
    auto = r.route()                        # a batch this large takes the tensor path
    assert all(np.array_equal(a, b) for a, b in zip(got, auto))
    st = r.stats()
    assert st["launches"]["mlp_tc"] == 2 and st["launches"]["qual_tc"] == 2
    r.close()
    assert frac > 0.6


def test_large_bf16_full_size_sampled():
    p = W.make_config(3)                   # Q = 65,536, D = 64, H = 256, E = 1024
    r = H.Router(p)
    got = r.route()                         # host buffers: copied in chunks
    st = r.stats()["launches"]
    assert st["mlp_tc"] == st["qual_tc"] >= 2
    idx = np.arange(0, p["Q"], 61)          # sampled outputs, spanning every tile
    check_against_oracle(p, got, idx=idx)
    r.close()


@pytest.mark.parametrize("Q", [1, 5, 127, 128, 129, 300, 1000])
def test_forced_tensor_ragged_batches(Q):
    p = W.make_config(1, Q=Q)
    r = H.Router(p)
    check_against_oracle(p, r.route(flags=TC), min_checked=0.0 if Q < 10 else 0.5)
    r.close()


@pytest.mark.parametrize("shape", [
    dict(M=1, G=1, F=12, H1=64, H2=32, E=40),        # D = 1, E not a multiple of 64
    dict(M=5, G=3, F=24, H1=192, H2=96, E=1000),     # odd M, Epad > E
    dict(M=17, G=2, F=40, H1=128, H2=160, E=64),     # Mpad = 32
    dict(M=32, G=2, F=48, H1=256, H2=256, E=256),    # D = 64, M = 32
    dict(M=7, G=1, F=24, H1=64, H2=256, E=128),      # D = 7
])
def test_tensor_shapes_with_biases(shape):
    p = W.make_problem(Q=700, dtype="bf16", lam=0.3, slo=4.0, seed=77, bias_std=0.3,
                       **shape)
    r = H.Router(p)
    check_against_oracle(p, r.route(flags=TC), min_checked=0.3)
    r.close()


@pytest.mark.parametrize("slo,lam,convex", [(0.0, 0.3, False), (float("inf"), 0.3, False),
                                            (10.0, 0.0, False), (10.0, 0.25, True)])
def test_tensor_budgets(slo, lam, convex):
    p = W.make_config(3, Q=3000)
    r = H.Router(p)
    got = r.route(flags=TC | (H.HWR_SCORE_CONVEX if convex else 0), slo=slo, lam=lam)
    check_against_oracle(p, got, slo=slo, lam=lam, convex=convex, min_checked=0.3)
    r.close()


def test_tensor_matches_simt_within_tolerance_and_is_deterministic():
    p = W.make_config(3, Q=2048)
    r = H.Router(p)
    tc = r.route(flags=TC)
    simt = r.route(flags=H.HWR_PATH_SIMT)
    same = tc[0] == simt[0]
    assert same.mean() > 0.95
    assert np.all(np.abs(tc[1] - simt[1])[same] <= TOL * np.abs(simt[1])[same])
    for _ in range(3):
        again = r.route(flags=TC)
        assert all(np.array_equal(a, b) for a, b in zip(tc, again))
    r.close()


def test_tensor_device_pointers():
    import torch
    p = W.make_config(4, Q=4096)
    r = H.Router(p, stream=torch.cuda.current_stream().cuda_stream)
    host = r.route(flags=TC)
    dev = torch.device("cuda:0")
    il = torch.from_numpy(p["in_len"]).to(dev)
    ol = torch.from_numpy(p["out_len"]).to(dev)
    em = torch.from_numpy(p["emb"].view(np.int16)).to(dev)
    ch = torch.empty(p["Q"], dtype=torch.int32, device=dev)
    lat = torch.empty(p["Q"], dtype=torch.float32, device=dev)
    ut = torch.empty(p["Q"], dtype=torch.float32, device=dev)
    r.route_device(il, ol, em, ch, lat, ut, slo=p["slo"], lam=p["lam"], flags=TC)
    torch.cuda.synchronize()
    assert np.array_equal(ch.cpu().numpy(), host[0])
    assert np.array_equal(lat.cpu().numpy(), host[1])
    r.close()


def _dev_batch(p, lo, hi, dev):
    import torch
    return (torch.from_numpy(p["in_len"][lo:hi].copy()).to(dev),
            torch.from_numpy(p["out_len"][lo:hi].copy()).to(dev),
            torch.from_numpy(p["emb"][lo:hi].view(np.int16).copy()).to(dev))


def _outs(n, dev):
    import torch
    return (torch.empty(n, dtype=torch.int32, device=dev), torch.empty(n, device=dev),
            torch.empty(n, device=dev))


@pytest.mark.parametrize("cfg,Q", [(4, 4096), (4, 1024), (3, 8192)])
def test_back_to_back_routes_keep_stream_order(cfg, Q):
    """Routes queued back to back overlap (a predictor starts while the
    quality kernel and the previous predictor still run); each must still
    equal the same route run alone, and a later route writing the same
    output arrays must leave its own results there."""
    import torch
    dev = torch.device("cuda:0")
    p = W.make_config(cfg, Q=2 * Q)
    r = H.Router(p, stream=torch.cuda.current_stream().cuda_stream)
    A, B = _dev_batch(p, 0, Q, dev), _dev_batch(p, Q, 2 * Q, dev)
    ref = []
    for batch in (A, B):
        o = _outs(Q, dev)
        r.route_device(*batch, *o, slo=p["slo"], lam=p["lam"], flags=TC)
        torch.cuda.synchronize()
        ref.append([t.cpu().numpy() for t in o])
    X, Y = _outs(Q, dev), _outs(Q, dev)
    for _ in range(3):
        r.route_device(*A, *X, slo=p["slo"], lam=p["lam"], flags=TC | H.HWR_ASYNC)
        r.route_device(*B, *X, slo=p["slo"], lam=p["lam"], flags=TC | H.HWR_ASYNC)
        r.route_device(*A, *Y, slo=p["slo"], lam=p["lam"], flags=TC | H.HWR_ASYNC)
    r.synchronize()
    for got, want in ((X, ref[1]), (Y, ref[0])):
        for a, b in zip(got, want):
            assert np.array_equal(a.cpu().numpy(), b, equal_nan=True)
    r.close()


def test_inputs_that_are_the_previous_routes_outputs():
    """A route queued right behind another whose outputs it reads as inputs
    (here the first route's latencies as the second's output lengths) must
    see them complete: the predictor then waits for the previous one before
    it reads anything."""
    import torch
    dev = torch.device("cuda:0")
    p = W.make_config(4, Q=4096)
    r = H.Router(p, stream=torch.cuda.current_stream().cuda_stream)
    il, ol, em = _dev_batch(p, 0, p["Q"], dev)
    o1, o2 = _outs(p["Q"], dev), _outs(p["Q"], dev)
    for _ in range(3):
        r.route_device(il, ol, em, *o1, slo=p["slo"], lam=p["lam"], flags=TC | H.HWR_ASYNC)
        r.route_device(il, o1[1], em, *o2, slo=p["slo"], lam=p["lam"], flags=TC | H.HWR_ASYNC)
    r.synchronize()
    lat1 = o1[1].clone()
    o3 = _outs(p["Q"], dev)
    r.route_device(il, lat1, em, *o3, slo=p["slo"], lam=p["lam"], flags=TC)
    torch.cuda.synchronize()
    for a, b in zip(o2, o3):
        assert np.array_equal(a.cpu().numpy(), b.cpu().numpy(), equal_nan=True)
    r.close()


@pytest.mark.parametrize("Q", [1, 16, 256, 4096, 65_536])
def test_batch_sweep_d32(Q):
    p = W.make_config(4, Q=Q)
    r = H.Router(p)
    got = r.route()
    idx = None if Q <= 4096 else np.arange(0, Q, 67)
    check_against_oracle(p, got, idx=idx, min_checked=0.0 if Q < 100 else 0.5)
    r.close()


@pytest.mark.slow
def test_batch_sweep_d32_one_million():
    p = W.make_config(4, Q=1_048_576)
    r = H.Router(p)
    got = r.route()
    check_against_oracle(p, got, idx=np.arange(0, p["Q"], 1021))
    # every query got a defined choice
    assert (got[0] >= 0).all() and (got[0] < p["D"]).all()
    r.close()


def test_pipelined_host_batch_matches_device_path():
    # a large host-pointer batch is copied in chunks that overlap the kernels;
    # the decisions must be those of the one-shot device-pointer call
    import torch
    p = W.make_config(3, Q=40_000)
    r = H.Router(p, stream=torch.cuda.current_stream().cuda_stream)
    host = r.route()                                   # pipelined (>= 2 chunks)
    dev = torch.device("cuda:0")
    il = torch.from_numpy(p["in_len"]).to(dev)
    ol = torch.from_numpy(p["out_len"]).to(dev)
    em = torch.from_numpy(p["emb"].view(np.int16)).to(dev)
    ch = torch.empty(p["Q"], dtype=torch.int32, device=dev)
    lat = torch.empty(p["Q"], dtype=torch.float32, device=dev)
    ut = torch.empty(p["Q"], dtype=torch.float32, device=dev)
    r.route_device(il, ol, em, ch, lat, ut, slo=p["slo"], lam=p["lam"])
    torch.cuda.synchronize()
    assert np.array_equal(ch.cpu().numpy(), host[0])
    assert np.array_equal(lat.cpu().numpy(), host[1])
    assert np.array_equal(ut.cpu().numpy(), host[2])
    # a small call between two large ones reuses the staging buffer safely
    small = r.route(p["in_len"][:100], p["out_len"][:100], p["emb"][:100])
    again = r.route()
    assert all(np.array_equal(a, b) for a, b in zip(host, again))
    assert np.array_equal(small[0], host[0][:100])
    r.close()


@pytest.mark.parametrize("c,Q", [(1, 2000), (3, 3000)])
def test_three_heads_tensor(c, Q):
    p = W.make_config(c, Q=Q, n_heads=3)
    r = H.Router(p)
    check_against_oracle(p, r.route(flags=TC), min_checked=0.3)
    r.close()


def test_repeated_routes_and_scores_are_bitwise_identical():
    """Every route and score of the same batch gives the same bits.

    The predictor kernel streams its operands through shared-memory rings
    that producer and copy engines reuse as soon as they are released; a
    release that came too early would corrupt a few rows now and then.  This
    repeats both entry points on one large batch, through the pipelined host
    path and the device path, and demands bit-identical results.
    """
    import torch
    p = W.make_config(3, Q=20_000)
    dev = torch.device("cuda:0")
    r = H.Router(p, stream=torch.cuda.current_stream().cuda_stream)
    il = torch.from_numpy(p["in_len"]).to(dev)
    ol = torch.from_numpy(p["out_len"]).to(dev)
    em = torch.from_numpy(p["emb"].view(np.int16)).to(dev)
    C0, Q0 = r.score(flags=TC)
    R0 = r.route(flags=TC)
    Cd = torch.empty((p["Q"], p["D"]), dtype=torch.float32, device=dev)
    Qd = torch.empty((p["Q"], p["M"]), dtype=torch.float32, device=dev)
    for _ in range(6):
        C, Qm = r.score(flags=TC)
        assert np.array_equal(C, C0) and np.array_equal(Qm, Q0)
        r.score_device(il, ol, em, Cd, Qd, flags=TC)
        torch.cuda.synchronize()
        assert np.array_equal(Cd.cpu().numpy(), C0)
        R = r.route(flags=TC)
        for a, b in zip(R, R0):
            assert np.array_equal(a, b, equal_nan=True)
    r.close()


def test_tensor_route_after_sequential_sees_the_increments():
    """A sequential call raises the running counts and refreshes the layer-1
    prefix, fp32 and bf16; a tensor-core batch route afterwards must score
    against the raised counts (and a new snapshot must undo them)."""
    p = W.make_config(1, Q=600)                    # bf16, D = 12
    r = H.Router(p)
    seq_q = 64
    got_seq = r.route(p["in_len"][:seq_q], p["out_len"][:seq_q], p["emb"][:seq_q],
                      flags=H.HWR_SEQUENTIAL)
    orc = O.Problem(p)
    want = orc.route(p["in_len"][:seq_q], p["out_len"][:seq_q], p["emb"][:seq_q],
                     mode=O.F32, sequential=True, nthreads=8)
    assert np.array_equal(got_seq[0], want[0])
    raised = r.get_snapshot()
    assert np.array_equal(raised, want[3]) and not np.array_equal(raised, p["snap"]["running"])
    after = r.route(flags=H.HWR_PATH_TENSOR)
    snap = dict(p["snap"])
    snap["running"] = raised
    check_against_oracle(dict(p, snap=snap), after)
    # a fresh snapshot restores the original counts for the tensor path too
    r.update_snapshot(p["snap"])
    check_against_oracle(p, r.route(flags=H.HWR_PATH_TENSOR))
    r.close()


# ---------------------------------------------------------------------------
# sequential mode with the score table on the tensor cores (HWR_SEQUENTIAL |
# HWR_PATH_TENSOR): every query's choice is checked against the fp64 oracle
# at the running counts the GPU's own earlier picks imply (a near tie may go
# the other way, after which the counts legitimately differ from the
# canonical run), and the persisted counts must be exactly those picks

def _replay_check(p, got):
    ch, lat, util = got
    D = p["D"]
    r0 = np.asarray(p["snap"]["running"], np.int64)
    clear = []
    for i in range(len(ch)):
        prev = ch[:i][ch[:i] >= 0]
        snap = dict(p["snap"])
        snap["running"] = (r0 + np.bincount(prev, minlength=D)).astype(np.int32)
        pi = dict(W.query_subset(p, [i]), snap=snap)
        clear.append(check_against_oracle(pi, (ch[i:i + 1], lat[i:i + 1], util[i:i + 1]),
                                          min_checked=0.0))
    return float(np.mean(clear))


@pytest.mark.parametrize("c,Q", [(1, 150), (4, 70), (4, 64), (3, 45), (3, 64)])
def test_sequential_tensor_table_valid(c, Q):
    p = W.make_config(c, Q=Q)
    r = H.Router(p)
    got = r.route(flags=H.HWR_SEQUENTIAL | H.HWR_PATH_TENSOR)
    final = r.get_snapshot()
    r.update_snapshot(p["snap"])
    canon = r.route(flags=H.HWR_SEQUENTIAL)           # canonical fp32 order
    r.close()
    ch = got[0]
    assert np.array_equal(final, np.asarray(p["snap"]["running"]) +
                          np.bincount(ch[ch >= 0], minlength=p["D"]))
    assert _replay_check(p, got) >= 0.5
    # most decisions agree with the canonical run
    assert np.mean(ch == canon[0]) >= 0.5


@pytest.mark.parametrize("c,Q,step", [(1, None, 1), (3, 8192, 7)])
def test_tensor_scores_match_the_oracle_elementwise(c, Q, step):
    """hwr_score_batch on the tensor path: every cost C = TTFT + N_out TPOT
    (Eq. 1-2) and every quality score (Sec. 3.2 (3)) against the fp64 oracle,
    element by element (all of the mid workload; every 7th query of 8,192 on
    the large one)."""
    p = W.make_config(c, Q=Q)
    r = H.Router(p)
    C, Qm = r.score(flags=TC)
    r.close()
    idx = np.arange(0, p["Q"], step)
    sub = W.query_subset(p, idx)
    orc = O.Problem(sub)
    Co, _ = orc.score_all(nthreads=16)
    rel = np.abs(C[idx] - Co) / np.maximum(np.abs(Co), 1e-3)
    assert rel.max() <= TOL, rel.max()
    Qo = np.stack([orc.quality(sub["emb"][i]) for i in range(idx.size)])
    relq = np.abs(Qm[idx] - Qo) / np.maximum(np.abs(Qo), 1e-3)
    assert relq.max() <= TOL, relq.max()


@pytest.mark.parametrize("c,bound,bound999", [(1, 5e-3, 3e-3), (3, 8e-3, 4e-3)])
def test_tensor_latency_error_stays_at_its_bf16_level(c, bound, bound999):
    """The tensor path rounds the layer-1 activations to bf16 (fp32
    accumulation); its cost error against the fp64 oracle is measured at
    2.4e-3 (mid workload) and 4.8e-3 (large; 3.0e-3 at the 99.9th
    percentile), far inside the 2e-2 tolerance.  These bounds catch a
    precision regression that the tolerance would let through."""
    p = W.make_config(c, Q=4096)
    r = H.Router(p)
    C, _ = r.score(flags=TC, quality=False)
    r.close()
    Co, _ = O.Problem(p).score_all(nthreads=16)
    rel = np.abs(C - Co) / np.maximum(np.abs(Co), 1e-3)
    print(f"workload {c}: max relative cost error {rel.max():.3e}, "
          f"99.9th percentile {np.quantile(rel, 0.999):.3e}")
    assert rel.max() <= bound, rel.max()
    assert np.quantile(rel, 0.999) <= bound999
