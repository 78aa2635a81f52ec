"""GPU parity: the CUDA path against the CPU oracle on the same seeded inputs.

fp32 SIMT kernels follow the canonical fp32 order, so their latency, utility
and chosen index must equal the oracle's canonical-fp32 mode bit for bit (and
sit within 1e-5 relative of the fp64 oracle).  bf16 contexts routed through
the SIMT kernels are the same computation on bf16-valued inputs and are held
to the same bit-exact bar.
"""
import numpy as np
import pytest

import oracle as O
import workload as W
import paper_2608_14575_gb300 as H

pytestmark = pytest.mark.gpu

SIMT = H.HWR_PATH_SIMT


@pytest.fixture(scope="module", autouse=True)
def built():
    H.build()


def _f32(a):
    return np.asarray(a, np.float64).astype(np.float32)


def assert_exact(got, want, what=""):
    ch, lat, util = got
    wch, wlat, wutil = want[:3]
    bad = np.nonzero(ch != wch)[0]
    assert bad.size == 0, f"{what}: chosen differs at {bad[:10]} ({ch[bad[:5]]} vs {wch[bad[:5]]})"
    assert np.array_equal(lat, _f32(wlat), equal_nan=True), what
    assert np.array_equal(util, _f32(wutil), equal_nan=True), what


def assert_close_f64(got, want, tol=1e-5):
    _, lat, util = got
    _, wlat, wutil = want[:3]
    ok = np.isfinite(wlat)
    assert np.all(np.abs(lat[ok] - wlat[ok]) <= tol * np.maximum(np.abs(wlat[ok]), 1e-3))
    assert np.all(np.abs(util[ok] - wutil[ok]) <= tol * np.maximum(np.abs(wutil[ok]), 1.0))


def route_both(p, flags=0, **kw):
    r = H.Router(p)
    got = r.route(flags=flags, **kw)
    orc = O.Problem(p)
    conv = bool(flags & H.HWR_SCORE_CONVEX)
    want = orc.route(mode=O.F32, convex=conv, nthreads=8, **kw)
    r.close()
    return got, want, orc


@pytest.mark.parametrize("Q", [1, 2, 17, 31, 33, 255, 256])
def test_tiny_fp32_exact(Q):
    p = W.make_config(0, Q=Q)
    got, want, orc = route_both(p)
    assert_exact(got, want, f"cfg0 Q={Q}")
    assert_close_f64(got, orc.route(mode=O.F64))


@pytest.mark.parametrize("slo,lam", [(0.0, 0.5), (float("inf"), 0.5), (5.0, 0.0),
                                     (1.0, 4.0), (float("-inf"), 0.5)])
def test_tiny_fp32_degenerate_budgets(slo, lam):
    p = W.make_config(0, Q=97)
    got, want, _ = route_both(p, slo=slo, lam=lam)
    assert_exact(got, want, f"slo={slo} lam={lam}")


def test_convex_score_exact():
    p = W.make_config(0, Q=129)
    got, want, _ = route_both(p, flags=H.HWR_SCORE_CONVEX, lam=0.25)
    assert_exact(got, want, "convex")


@pytest.mark.parametrize("c,Q", [(1, 300), (3, 40), (4, 65)])
def test_bf16_contexts_simt_exact(c, Q):
    p = W.make_config(c, Q=Q)
    got, want, orc = route_both(p, flags=SIMT)
    assert_exact(got, want, f"cfg{c} simt")
    assert_close_f64(got, orc.route(mode=O.F64, nthreads=8))


@pytest.mark.parametrize("shape", [
    dict(M=1, G=1, F=12, H1=8, H2=8, E=8),      # D = 1
    dict(M=3, G=1, F=16, H1=40, H2=24, E=16),   # odd widths, K not a chunk multiple
    dict(M=5, G=3, F=24, H1=96, H2=200, E=40),  # D = 15, H2 not a multiple of 32
    dict(M=16, G=4, F=48, H1=256, H2=256, E=64),  # D = 64, widest tile
])
def test_shapes_with_biases_exact(shape):
    p = W.make_problem(Q=77, dtype="f32", lam=0.4, slo=2.0, seed=31, bias_std=0.3,
                       **shape)
    got, want, _ = route_both(p)
    assert_exact(got, want, str(shape))


def test_device_pointers_match_host():
    import torch
    p = W.make_config(0, Q=200)
    stream = torch.cuda.current_stream().cuda_stream
    r = H.Router(p, stream=stream)
    host = r.route()
    dev = torch.device("cuda:0")
    il = torch.from_numpy(p["in_len"]).to(dev)
    ol = torch.from_numpy(p["out_len"]).to(dev)
    em = torch.from_numpy(p["emb"]).to(dev)
    ch = torch.empty(200, dtype=torch.int32, device=dev)
    lat = torch.empty(200, dtype=torch.float32, device=dev)
    ut = torch.empty(200, dtype=torch.float32, device=dev)
    r.route_device(il, ol, em, ch, lat, ut, slo=p["slo"], lam=p["lam"])
    torch.cuda.synchronize()
    assert np.array_equal(ch.cpu().numpy(), host[0])
    assert np.array_equal(lat.cpu().numpy(), host[1])
    assert np.array_equal(ut.cpu().numpy(), host[2])
    r.close()


def test_deterministic_reruns():
    p = W.make_config(1, Q=512)
    r = H.Router(p)
    first = r.route(flags=SIMT)
    for _ in range(5):
        again = r.route(flags=SIMT)
        for a, b in zip(first, again):
            assert np.array_equal(a, b)
    r.close()


def test_route_before_snapshot_and_bad_args():
    p = W.make_config(0, Q=8)
    r = H.Router(p)
    with pytest.raises(H.HwrError) as e:
        r.route(slo=float("nan"))
    assert e.value.status == 1
    with pytest.raises(H.HwrError) as e:
        r.route(flags=H.HWR_PATH_TENSOR)       # fp32 context has no tensor path
    assert e.value.status == 7
    # the context stays usable after argument errors
    got = r.route()
    assert got[0].shape == (8,)
    r.close()


# ---------------------------------------------------------------------------
# sequential mode

def test_sequential_single_call_exact():
    p = W.make_config(2, Q=200)     # several chunks of the sequential table
    r = H.Router(p)
    got = r.route(flags=H.HWR_SEQUENTIAL)
    orc = O.Problem(p)
    want = orc.route(mode=O.F32, sequential=True, nthreads=8)
    assert_exact(got, want, "sequential")
    assert np.array_equal(r.get_snapshot(), want[3])
    # increments persist until the next snapshot
    got2 = r.route(flags=H.HWR_SEQUENTIAL)
    want2 = orc.route(mode=O.F32, sequential=True, running=want[3], nthreads=8)
    assert_exact(got2, want2, "sequential, second call")
    # and a batch call afterwards sees the incremented counts
    snap = dict(p["snap"])
    snap["running"] = want2[3]
    got3 = r.route()
    want3 = O.Problem(p, snap=snap).route(mode=O.F32, nthreads=8)
    assert_exact(got3, want3, "batch after sequential")
    r.update_snapshot(p["snap"])
    assert np.array_equal(r.get_snapshot(), p["snap"]["running"])
    r.close()


def test_back_to_back_snapshots_last_one_wins():
    """Snapshot updates reuse one staging buffer; an update waits for the
    previous snapshot kernel only while the host has not yet seen later work
    on the stream complete.  Updates in a row, and an update after an
    asynchronous route, must each leave exactly their own snapshot in force."""
    p = W.make_config(0, Q=256)
    rng = np.random.default_rng(5)
    snaps = []
    for _ in range(3):
        s = {k: np.array(v, copy=True) for k, v in p["snap"].items()}
        s["running"] = rng.integers(0, 30, p["D"]).astype(np.int32)
        s["kv"] = rng.uniform(0, 1, p["D"]).astype(np.float32)
        snaps.append(s)
    r = H.Router(p)
    for s in snaps:
        r.update_snapshot(s)
    assert_exact(r.route(), O.Problem(p, snap=snaps[2]).route(mode=O.F32, nthreads=8), "last of three")
    r.route(flags=H.HWR_ASYNC)
    r.update_snapshot(snaps[0])
    assert_exact(r.route(), O.Problem(p, snap=snaps[0]).route(mode=O.F32, nthreads=8), "after async")
    r.close()


def _online(p, n):
    """Run the online micro-batch loop through the GPU and through the oracle."""
    r = H.Router(p)

    def gpu_route(snap, lo, hi):
        r.update_snapshot(snap)
        return r.route(p["in_len"][lo:hi], p["out_len"][lo:hi], p["emb"][lo:hi],
                       flags=H.HWR_SEQUENTIAL)[0]

    orc = O.Problem(p)

    def cpu_route(snap, lo, hi):
        orc.set_snapshot(snap)
        return orc.route(p["in_len"][lo:hi], p["out_len"][lo:hi], p["emb"][lo:hi],
                         mode=O.F32, sequential=True, running=snap["running"],
                         nthreads=8)[0]

    g, _ = W.simulate_online(p, gpu_route, n_requests=n)
    c, _ = W.simulate_online(p, cpu_route, n_requests=n)
    r.close()
    return g, c


def test_online_sequential_prefix_exact():
    p = W.make_config(2, Q=6_432)   # 100 full micro-batches and a ragged one
    g, c = _online(p, p["Q"])
    bad = np.nonzero(g != c)[0]
    assert bad.size == 0, f"first divergence at request {bad[:1]}"


@pytest.mark.slow
def test_online_sequential_full_100k_exact():
    p = W.make_config(2)
    g, c = _online(p, p["Q"])
    bad = np.nonzero(g != c)[0]
    assert bad.size == 0, f"first divergence at request {bad[:1]}"
    assert len(np.unique(g)) > 1


# ---------------------------------------------------------------------------
# three output heads: N_out predicted (Eq. 1) and used by the cost (Eq. 2)

@pytest.mark.parametrize("c,Q,flags", [(0, 50, 0), (0, 256, 0), (1, 300, SIMT),
                                       (2, 120, H.HWR_SEQUENTIAL)])
def test_three_heads_simt_exact(c, Q, flags):
    p = W.make_config(c, Q=Q, n_heads=3)
    r = H.Router(p)
    got = r.route(flags=flags)
    want = O.Problem(p).route(mode=O.F32, sequential=bool(flags & H.HWR_SEQUENTIAL),
                              nthreads=8)
    assert_exact(got, want, f"three heads cfg{c}")
    r.close()


# ---------------------------------------------------------------------------
# both small-batch kernels (pair-parallel and fused) at the same sizes: the
# threshold between them is a tuning choice, so each must be exact on its own

@pytest.mark.parametrize("pairs_max", ["0", "2048"])
@pytest.mark.parametrize("c,Q", [(0, 1), (0, 100), (0, 511), (2, 7), (2, 64), (2, 170)])
def test_small_batch_kernels_both_exact(monkeypatch, pairs_max, c, Q):
    monkeypatch.setenv("HWR_PAIRS_MAX_PAIRS", pairs_max)
    p = W.make_config(c, Q=Q)
    r = H.Router(p)
    got = r.route()
    C, qual = r.score()
    r.close()
    orc = O.Problem(p)
    assert_exact(got, orc.route(mode=O.F32, nthreads=8), f"cfg{c} Q={Q} pairs_max={pairs_max}")
    Cw, _ = orc.score_all(mode=O.F32, nthreads=8)
    assert np.array_equal(C, Cw.astype(np.float32))
    qw = np.array([orc.quality(p["emb"][i], mode=O.F32) for i in range(Q)])
    assert np.array_equal(qual, qw.astype(np.float32))


# the small-batch kernel groups 32 consecutive (query, deployment) pairs and
# splits their layer 2 by 32-column blocks: groups holding many queries
# (D = 1), queries straddling two groups (D = 15), every query spanning two
# groups (D = 33), ragged last column blocks (H2 = 200: 8 columns; H2 = 98: 2
# columns and 2 of padding), the largest batch the kernel takes (64 groups)
# and a bf16 context
@pytest.mark.parametrize("shape,Q", [
    (dict(M=1, G=1, F=12, H1=8, H2=8, E=8), 70),
    (dict(M=5, G=3, F=24, H1=96, H2=200, E=40), 37),
    (dict(M=11, G=3, F=24, H1=64, H2=98, E=24), 20),
    (dict(M=16, G=4, F=48, H1=40, H2=72, E=16), 32),      # D = 64: 2,048 pairs, the limit
    ("cfg4", 5),
])
def test_pairs_kernel_group_shapes_exact(monkeypatch, shape, Q):
    monkeypatch.setenv("HWR_PAIRS_MAX_PAIRS", "2048")
    if shape == "cfg4":
        p = W.make_config(4, Q=Q)
    else:
        p = W.make_problem(Q=Q, dtype="f32", lam=0.3, slo=3.0, seed=43, bias_std=0.2, **shape)
    r = H.Router(p)
    got = r.route()
    C, qual = r.score()
    r.close()
    orc = O.Problem(p)
    assert_exact(got, orc.route(mode=O.F32, nthreads=8), str(shape))
    Cw, _ = orc.score_all(mode=O.F32, nthreads=8)
    assert np.array_equal(C, Cw.astype(np.float32))


# the small-batch kernel's fused column blocks (8 columns, taken when every
# block of the grid has an SM of its own): H1 with a 4-wide tail (92), H1 not
# a multiple of 4 (37), H2 with a ragged last block and an odd head row (30,
# 45), a query straddling two groups (D = 15), every query spanning two groups
# (D = 64), and the sweep's cluster (D = 32, H = 256) at one and four queries
@pytest.mark.parametrize("shape,Q", [
    (dict(M=5, G=3, F=24, H1=92, H2=30, E=40), 3),
    (dict(M=3, G=2, F=20, H1=37, H2=45, E=16), 9),
    (dict(M=16, G=4, F=48, H1=64, H2=64, E=32), 2),
    ("cfg4", 1),
    ("cfg4", 4),
])
def test_pairs_kernel_fused_shapes_exact(monkeypatch, shape, Q):
    monkeypatch.setenv("HWR_PAIRS_MAX_PAIRS", "2048")
    if shape == "cfg4":
        p = W.make_config(4, Q=Q)
    else:
        p = W.make_problem(Q=Q, dtype="f32", lam=0.3, slo=3.0, seed=47, bias_std=0.2, **shape)
    r = H.Router(p)
    got = r.route()
    C, qual = r.score()
    r.close()
    orc = O.Problem(p)
    assert_exact(got, orc.route(mode=O.F32, nthreads=8), str(shape))
    Cw, _ = orc.score_all(mode=O.F32, nthreads=8)
    assert np.array_equal(C, Cw.astype(np.float32))


# ---------------------------------------------------------------------------
# sequential mode on more shapes: D > 32 (two deployments per lane of the
# chain's warp), odd D, D = 1, a bf16 context, several chunks each

@pytest.mark.parametrize("shape,Q", [
    (dict(M=16, G=4, F=48, H1=32, H2=32, E=16), 100),    # D = 64: chunks of 39
    (dict(M=5, G=3, F=24, H1=96, H2=200, E=40), 150),    # D = 15
    (dict(M=1, G=1, F=12, H1=8, H2=8, E=8), 70),         # D = 1
])
def test_sequential_shapes_exact(shape, Q):
    p = W.make_problem(Q=Q, dtype="f32", lam=0.3, slo=3.0, seed=41, bias_std=0.2, **shape)
    r = H.Router(p)
    got = r.route(flags=H.HWR_SEQUENTIAL)
    want = O.Problem(p).route(mode=O.F32, sequential=True, nthreads=8)
    assert_exact(got, want, str(shape))
    assert np.array_equal(r.get_snapshot(), want[3])
    r.close()


def test_sequential_bf16_context_exact():
    p = W.make_config(4, Q=90)      # D = 32, H = 256, bf16 inputs
    r = H.Router(p)
    got = r.route(flags=H.HWR_SEQUENTIAL)
    want = O.Problem(p).route(mode=O.F32, sequential=True, nthreads=8)
    assert_exact(got, want, "cfg4 sequential")
    r.close()


@pytest.mark.parametrize("slo", [0.0, float("-inf"), float("inf")])
def test_sequential_degenerate_budgets_exact(slo):
    p = W.make_config(2, Q=80)
    r = H.Router(p)
    got = r.route(slo=slo, flags=H.HWR_SEQUENTIAL)
    want = O.Problem(p).route(slo=slo, mode=O.F32, sequential=True, nthreads=8)
    assert_exact(got, want, f"slo={slo}")
    r.close()


# ---------------------------------------------------------------------------
# exact ties: only the GPU-type columns of W1 (and the query slots) carry
# weight and the model embeddings are zero, so deployments of one GPU type
# have bit-identical costs and utilities; the lowest index must win (that is
# d = g* for the best type g*, d = m G + g), on every path

def _tied_problem(Q):
    M, G, F = 16, 4, 48
    p = W.make_problem(Q=Q, dtype="f32", M=M, G=G, F=F, H1=32, H2=32, E=16, seed=9,
                       lam=0.4, slo=2.0, bias_std=0.3)
    keep = np.zeros(F, bool)
    keep[M:M + G] = True
    keep[F - 2:] = True
    p["W1"] = np.where(keep[None, :], p["W1"], 0.0).astype(p["W1"].dtype)
    p["memb"] = np.zeros_like(p["memb"])
    return p


@pytest.mark.parametrize("slo", [float("inf"), float("-inf")])
@pytest.mark.parametrize("mode", ["pairs", "fused", "sequential"])
def test_exact_ties_go_to_lowest_index(monkeypatch, slo, mode):
    Q = 40
    p = _tied_problem(Q)
    monkeypatch.setenv("HWR_PAIRS_MAX_PAIRS", "0" if mode == "fused" else "2048")
    flags = H.HWR_SEQUENTIAL if mode == "sequential" else 0
    r = H.Router(p)
    got = r.route(slo=slo, flags=flags)
    r.close()
    want = O.Problem(p).route(slo=slo, mode=O.F32, sequential=bool(flags), nthreads=8)
    assert_exact(got, want, f"ties {mode} slo={slo}")
    assert np.all((got[0] >= 0) & (got[0] < p["G"]))


# ---------------------------------------------------------------------------
# widths the SIMT tile pads: H2 not a multiple of 4 (padded rows of W2
# transposed), H1 not a multiple of the 32-wide K chunk, width 1, the widest
# columns, on the pair-parallel, fused and sequential paths

@pytest.mark.parametrize("shape", [
    dict(M=2, G=2, F=13, H1=37, H2=30, E=24),
    dict(M=3, G=2, F=16, H1=1, H2=1, E=8),
    dict(M=2, G=3, F=20, H1=250, H2=253, E=16),
])
@pytest.mark.parametrize("mode", ["pairs", "fused", "sequential"])
def test_odd_widths_exact(monkeypatch, shape, mode):
    Q = 45
    p = W.make_problem(Q=Q, dtype="f32", lam=0.35, slo=2.5, seed=77, bias_std=0.25, **shape)
    monkeypatch.setenv("HWR_PAIRS_MAX_PAIRS", "0" if mode == "fused" else "2048")
    flags = H.HWR_SEQUENTIAL if mode == "sequential" else 0
    r = H.Router(p)
    got = r.route(flags=flags)
    r.close()
    want = O.Problem(p).route(mode=O.F32, sequential=bool(flags), nthreads=8)
    assert_exact(got, want, f"{shape} {mode}")
