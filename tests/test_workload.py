"""The seeded input generator: determinism, shapes and value ranges (CPU)."""
import numpy as np
import pytest

import oracle
import workload as W


@pytest.mark.parametrize("c", [0, 1, 2, 3, 4])
def test_config_shapes_and_determinism(c):
    a = W.make_config(c, Q=64)
    b = W.make_config(c, Q=64)
    for k in ("W1", "W2", "W3", "memb", "emb", "in_len", "out_len", "mu", "sd"):
        assert np.array_equal(a[k], b[k]), k
    D, F, H, E, M = a["D"], a["F"], a["H1"], a["E"], a["M"]
    assert D == a["M"] * a["G"]
    assert a["W1"].shape == (H, F) and a["W2"].shape == (H, H)
    assert a["W3"].shape == (2, H) and a["memb"].shape == (E, M)
    assert a["emb"].shape == (64, E)
    bf16 = a["dtype"] == "bf16"
    assert a["emb"].dtype == (np.uint16 if bf16 else np.float32)
    e = W.bf16_bits_to_f32(a["emb"]).reshape(64, E) if bf16 else a["emb"]
    assert np.allclose(np.linalg.norm(e.astype(np.float64), axis=1), 1.0, atol=2e-2)
    lo, hi = W.CONFIGS[c]["in_len"][2:]
    assert a["in_len"].min() >= lo and a["in_len"].max() <= hi
    assert np.array_equal(a["in_len"], np.rint(a["in_len"]))
    assert (a["out_len"] > 0).all()
    assert (a["snap"]["running"] >= 0).all() and (a["snap"]["kv"] <= 1).all()


def test_bf16_rounding_nearest_even():
    x = np.array([1.0, 1 + 2 ** -8, 1 + 3 * 2 ** -8, -2.5, 3.0e38], np.float32)
    got = W.bf16_bits_to_f32(W.to_bf16_bits(x))
    assert list(got[:4]) == [1.0, 1.0, 1 + 2 ** -6, -2.5]


@pytest.mark.parametrize("c", [0, 1, 3, 4])
def test_feasible_fraction_not_degenerate(c):
    p = W.make_config(c, Q=256)
    C, _ = oracle.Problem(p).score_all(nthreads=4)
    frac = float((C <= p["slo"]).mean())
    assert 0.05 <= frac <= 0.97, frac


def test_online_simulation_bookkeeping():
    p = W.make_config(2, Q=640)
    seen = []

    def route(snap, lo, hi):
        seen.append(snap["running"].copy())
        return np.full(hi - lo, lo // 64 % p["D"], np.int32)

    ch, hist = W.simulate_online(p, route)
    assert len(hist) == 10 and ch.shape == (640,)
    for b in range(1, 10):
        prev = hist[b - 1]["running"].copy()
        prev[(b - 1) % p["D"]] += 64
        assert (hist[b]["running"] <= prev).all() and (hist[b]["running"] >= 0).all()
