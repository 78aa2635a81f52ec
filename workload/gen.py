"""Seeded synthetic inputs for HW-Router route scoring.

This module only draws numbers: deployment tables, predictor weights, model
and query embeddings, hardware snapshots, query lengths and the online
arrival/drain process.  It holds none of the routing method's arithmetic
(no feature assembly, no predictor, no quality score, no selection), so the
CPU oracle and the CUDA library can both be fed from it without sharing code.

The paper's workloads (MixInstruct short prompts mixed with LongBench long
contexts, Sec. 4.3 "Dataset"; vLLM-observed runtime signals, Table 2) are not
available here; the distributions below stand in for them.

Conventions
-----------
* Deployment index d = m * G + g (model-major): every model on every GPU type.
* Feature slots (P = M + G):
    [0, M)          one-hot model id            (Sec. 3.2, Eq. 1: one-hot ids)
    [M, P)          one-hot GPU type id
    P               log10(parameter count)      (model size)
    P+1 .. P+6      running, waiting, kv util, GPU util, recent TTFT, recent TPOT
                    (Table 2, plus GPU utilisation named in the abstract)
    P+7 .. F-3      zero padding
    F-2, F-1        input length, expected output length (query features)
* Per-slot transform codes: 0 = identity, 1 = log1p, 2 = natural log.
* bf16 tensors are returned as uint16 bit patterns (round-to-nearest-even of
  the float32 draw); fp32 tensors as float32.
"""
from __future__ import annotations

import functools

import numpy as np

XF_ID, XF_LOG1P, XF_LOG = 0, 1, 2

# One entry per workload.  Shapes and distributions follow the five workload
# descriptions the build is measured on; lambda / SLO per workload.
CONFIGS = {
    0: dict(name="tiny_fp32", Q=256, M=2, G=2, F=16, H=32, E=64, dtype="f32",
            lam=0.5, slo=5.0, log10p=(9.0, 10.5), run_mean=8.0, wait_mean=3.0,
            in_len=(5.5, 1.0, 16.0, 4096.0)),
    1: dict(name="mid_bf16", Q=4096, M=4, G=3, F=32, H=128, E=768, dtype="bf16",
            lam=0.5, slo=3.0, log10p=(9.0, 11.0), run_mean=8.0, wait_mean=3.0,
            in_len=(5.5, 1.0, 16.0, 4096.0)),
    2: dict(name="online_seq_fp32", Q=100_000, M=4, G=3, F=32, H=128, E=768,
            dtype="f32", lam=0.5, slo=3.0, log10p=(9.0, 11.0), run_mean=8.0,
            wait_mean=3.0, in_len=(5.5, 1.0, 16.0, 4096.0),
            batch=64, rate=200.0, drain_p=0.3, kv_walk=0.02,
            emb_bf16_values=True),
    3: dict(name="large_bf16", Q=65_536, M=16, G=4, F=48, H=256, E=1024,
            dtype="bf16", lam=0.3, slo=10.0, log10p=(9.0, 11.0), run_mean=16.0,
            wait_mean=6.0, in_len=(6.0, 1.2, 16.0, 32768.0)),
    4: dict(name="sweep_d32", Q=65_536, M=8, G=4, F=48, H=256, E=1024,
            dtype="bf16", lam=0.3, slo=10.0, log10p=(9.0, 11.0), run_mean=16.0,
            wait_mean=6.0, in_len=(6.0, 1.2, 16.0, 32768.0),
            sweep=(1, 16, 256, 4096, 65_536, 1_048_576)),
}

# Medians of the recent-TTFT / recent-TPOT priors (lognormal mu = -2 and -4).
TTFT_MEDIAN = float(np.exp(-2.0))
TPOT_MEDIAN = float(np.exp(-4.0))
CALIB_SEED = 7
CALIB_DRAWS = 1 << 20

# Substream order inside SeedSequence(base + cfg).spawn(8).
_S_TABLE, _S_WEIGHTS, _S_MEMB, _S_SNAP, _S_QLEN, _S_QEMB, _S_ARRIVE, _S_DRAIN = range(8)
BASE_SEED = 20261202


def to_bf16_bits(a) -> np.ndarray:
    """Round float32 values to bfloat16 (nearest-even), return uint16 bits."""
    f = np.ascontiguousarray(a, dtype=np.float32)
    u = f.view(np.uint32)
    rounded = (u + (np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1)))) >> np.uint32(16)
    return rounded.astype(np.uint16)


def bf16_bits_to_f32(b) -> np.ndarray:
    """Widen bfloat16 bit patterns to float32 (exact)."""
    b = np.ascontiguousarray(b, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


def feature_layout(M: int, G: int, F: int) -> dict:
    """Slot indices of the feature vector (see module docstring)."""
    P = M + G
    if F < P + 9:
        raise ValueError(f"F={F} too small for M={M}, G={G} (need >= {P + 9})")
    return dict(P=P, log10p=P, running=P + 1, waiting=P + 2, kv=P + 3,
                gpu_util=P + 4, ttft=P + 5, tpot=P + 6, in_len=F - 2,
                out_len=F - 1)


def _softplus_inv(y: float) -> float:
    # Bias that centres an output head on a prior median y (weights are drawn
    # zero-mean, so z ~ b3 and softplus(b3) = y).  Not part of the method.
    return float(np.log(np.expm1(y)))


def _draw_in_len(rng, n, mu, sigma, lo, hi):
    x = rng.lognormal(mu, sigma, size=n)
    return np.clip(np.rint(x), lo, hi).astype(np.float32)


def _draw_out_len(rng, n):
    return rng.lognormal(5.0, 0.8, size=n).astype(np.float32)


def _draw_snapshot(rng, D, run_mean, wait_mean):
    return dict(
        running=rng.poisson(run_mean, size=D).astype(np.int32),
        waiting=rng.poisson(wait_mean, size=D).astype(np.int32),
        kv=rng.beta(2.0, 3.0, size=D).astype(np.float32),
        gpu_util=rng.uniform(0.0, 1.0, size=D).astype(np.float32),
        ttft=rng.lognormal(-2.0, 0.5, size=D).astype(np.float32),
        tpot=rng.lognormal(-4.0, 0.4, size=D).astype(np.float32),
    )


def calibration(M, G, F, log10p, run_mean, wait_mean, in_len):
    """Copies of the cached per-slot calibration (see _calibration)."""
    mean, std, xf = _calibration(int(M), int(G), int(F), tuple(log10p),
                                 float(run_mean), float(wait_mean), tuple(in_len))
    return mean.copy(), std.copy(), xf.copy()


@functools.lru_cache(maxsize=64)
def _calibration(M, G, F, log10p, run_mean, wait_mean, in_len):
    """Per-slot (mean, std, transform) from a fixed calibration stream.

    Stands in for the statistics a trained predictor would ship with: each
    signal is drawn CALIB_DRAWS times from its workload distribution, passed
    through its slot's transform, and its sample mean / std recorded.
    One-hot and padding slots get (0, 1, identity).
    """
    lay = feature_layout(M, G, F)
    rng = np.random.Generator(np.random.PCG64(CALIB_SEED))
    n = CALIB_DRAWS
    mean = np.zeros(F, np.float64)
    std = np.ones(F, np.float64)
    xf = np.zeros(F, np.uint8)
    draws = {
        "log10p": (rng.uniform(log10p[0], log10p[1], n), XF_ID),
        "running": (rng.poisson(run_mean, n).astype(np.float64), XF_LOG1P),
        "waiting": (rng.poisson(wait_mean, n).astype(np.float64), XF_LOG1P),
        "kv": (rng.beta(2.0, 3.0, n), XF_ID),
        "gpu_util": (rng.uniform(0.0, 1.0, n), XF_ID),
        "ttft": (rng.lognormal(-2.0, 0.5, n), XF_LOG),
        "tpot": (rng.lognormal(-4.0, 0.4, n), XF_LOG),
        "in_len": (np.clip(np.rint(rng.lognormal(in_len[0], in_len[1], n)),
                           in_len[2], in_len[3]), XF_LOG1P),
        "out_len": (rng.lognormal(5.0, 0.8, n), XF_LOG1P),
    }
    for key, (v, code) in draws.items():
        k = lay[key]
        t = v if code == XF_ID else (np.log1p(v) if code == XF_LOG1P else np.log(v))
        mean[k] = t.mean()
        std[k] = t.std()
        xf[k] = code
    return mean.astype(np.float32), std.astype(np.float32), xf


OUT_LEN_MEDIAN = float(np.exp(5.0))   # median of the expected-output-length prior


def make_problem(*, Q, M, G, F, H1, H2, E, dtype, lam, slo, log10p=(9.0, 11.0),
                 run_mean=8.0, wait_mean=3.0, in_len=(5.5, 1.0, 16.0, 4096.0),
                 seed=BASE_SEED, weight_std=0.1, bias_std=0.0,
                 emb_bf16_values=False, name="custom", cfg=None, n_heads=2):
    """Draw one complete routing problem (table, predictor, state, queries)."""
    ss = np.random.SeedSequence(seed).spawn(8)
    rngs = [np.random.Generator(np.random.PCG64(s)) for s in ss]
    D = M * G
    bf16 = dtype == "bf16"

    r = rngs[_S_TABLE]
    dep_model = np.repeat(np.arange(M, dtype=np.int32), G)
    dep_gpu = np.tile(np.arange(G, dtype=np.int32), M)
    log10p_m = r.uniform(log10p[0], log10p[1], size=M).astype(np.float32)

    r = rngs[_S_WEIGHTS]
    W1 = r.normal(0.0, weight_std, size=(H1, F)).astype(np.float32)
    W2 = r.normal(0.0, weight_std, size=(H2, H1)).astype(np.float32)
    W3 = r.normal(0.0, weight_std, size=(2, H2)).astype(np.float32)
    if n_heads == 3:   # drawn after the others so two-head problems are unchanged
        W3 = np.concatenate([W3, r.normal(0.0, weight_std, size=(1, H2)).astype(np.float32)])
    if bias_std > 0:
        b1 = r.normal(0.0, bias_std, size=H1).astype(np.float32)
        b2 = r.normal(0.0, bias_std, size=H2).astype(np.float32)
    else:
        b1 = np.zeros(H1, np.float32)
        b2 = np.zeros(H2, np.float32)
    b3 = np.array([_softplus_inv(TTFT_MEDIAN), _softplus_inv(TPOT_MEDIAN)]
                  + ([_softplus_inv(OUT_LEN_MEDIAN)] if n_heads == 3 else []), np.float32)
    mu, sd, xf = calibration(M, G, F, log10p, run_mean, wait_mean, in_len)

    r = rngs[_S_MEMB]
    memb = r.normal(0.0, 1.0, size=(E, M)).astype(np.float32)

    snap = _draw_snapshot(rngs[_S_SNAP], D, run_mean, wait_mean)

    r = rngs[_S_QLEN]
    in_l = _draw_in_len(r, Q, *in_len)
    out_l = _draw_out_len(r, Q)

    emb = _draw_embeddings(rngs[_S_QEMB], Q, E, bf16 or emb_bf16_values,
                           as_bits=bf16)

    p = dict(name=name, cfg=cfg, Q=Q, M=M, G=G, D=D, F=F, H1=H1, H2=H2, E=E, n_heads=n_heads,
             dtype=dtype, lam=float(lam), slo=float(slo),
             dep_model=dep_model, dep_gpu=dep_gpu, log10p=log10p_m,
             b1=b1, b2=b2, b3=b3, mu=mu, sd=sd, xform=xf, snap=snap,
             in_len=in_l, out_len=out_l, emb=emb)
    if bf16:
        p.update(W1=to_bf16_bits(W1), W2=to_bf16_bits(W2), W3=to_bf16_bits(W3),
                 memb=to_bf16_bits(memb))
    else:
        p.update(W1=W1, W2=W2, W3=W3, memb=memb)
    p["_rng_arrive"] = rngs[_S_ARRIVE]
    p["_rng_drain"] = rngs[_S_DRAIN]
    return p


def _draw_embeddings(rng, Q, E, round_bf16, as_bits, chunk=65_536):
    """N(0,1) rows, L2-normalised; optionally rounded to bf16."""
    out = np.empty((Q, E), np.uint16 if as_bits else np.float32)
    for s in range(0, Q, chunk):
        n = min(chunk, Q - s)
        x = rng.standard_normal(size=(n, E), dtype=np.float32)
        x /= np.sqrt(np.einsum("ij,ij->i", x, x))[:, None]
        if as_bits:
            out[s:s + n] = to_bf16_bits(x)
        elif round_bf16:
            out[s:s + n] = bf16_bits_to_f32(to_bf16_bits(x)).reshape(n, E)
        else:
            out[s:s + n] = x
    return out


def make_config(c: int, Q: int | None = None, seed_offset: int = 0, **over):
    """Problem for workload `c` (0..4); Q overrides the query count."""
    k = dict(CONFIGS[c])
    k.update(over)
    q = k.pop("Q") if Q is None else Q
    k.pop("Q", None)
    H = k.pop("H")
    extra = {key: k.pop(key) for key in
             ("batch", "rate", "drain_p", "kv_walk", "sweep") if key in k}
    emb_bf16 = k.pop("emb_bf16_values", False)
    p = make_problem(Q=q, H1=H, H2=H, seed=BASE_SEED + c + seed_offset,
                     emb_bf16_values=emb_bf16, cfg=c, **k)
    p.update(extra)
    return p


def query_slice(p: dict, lo: int, hi: int) -> dict:
    """The same problem restricted to queries [lo, hi)."""
    s = dict(p)
    s["in_len"] = p["in_len"][lo:hi]
    s["out_len"] = p["out_len"][lo:hi]
    s["emb"] = p["emb"][lo:hi]
    s["Q"] = hi - lo
    return s


def query_subset(p: dict, idx) -> dict:
    """The same problem restricted to the queries at indices `idx`."""
    idx = np.asarray(idx)
    s = dict(p)
    s["in_len"] = p["in_len"][idx]
    s["out_len"] = p["out_len"][idx]
    s["emb"] = p["emb"][idx]
    s["Q"] = int(idx.size)
    return s


def arrivals(p: dict, n: int, rate: float) -> np.ndarray:
    """Poisson arrival times (s): exponential gaps with mean 1/rate."""
    return np.cumsum(p["_rng_arrive"].exponential(1.0 / rate, size=n))


def simulate_online(p: dict, route_fn, n_requests=None, batch=None):
    """Online micro-batch loop of the sequential workload.

    Requests are taken in arrival order in micro-batches of `batch`.  For
    each batch the current snapshot is handed to `route_fn(snapshot, lo, hi)`,
    which must return the chosen deployment per request (routing in sequential
    mode, so each decision already raised its deployment's running count).
    Then the environment moves on: the running counts take the batch's
    choices, queues drain by Binomial(running, drain_p) and KV utilisation
    random-walks with N(0, kv_walk), clipped to [0, 1].  Other signals are
    held.  Returns the chosen sequence (int32) and the per-batch snapshots.
    """
    n = p["Q"] if n_requests is None else n_requests
    b = p.get("batch", 64) if batch is None else batch
    rng = np.random.Generator(np.random.PCG64(
        np.random.SeedSequence(BASE_SEED + 1000 + (p.get("cfg") or 0))))
    snap = {k: v.copy() for k, v in p["snap"].items()}
    chosen = np.empty(n, np.int32)
    history = []
    D = p["D"]
    for lo in range(0, n, b):
        hi = min(n, lo + b)
        history.append({k: v.copy() for k, v in snap.items()})
        c = np.asarray(route_fn({k: v.copy() for k, v in snap.items()}, lo, hi),
                       dtype=np.int32)
        chosen[lo:hi] = c
        snap["running"] = snap["running"] + np.bincount(
            c[c >= 0], minlength=D).astype(np.int32)
        drained = rng.binomial(snap["running"], p.get("drain_p", 0.3))
        snap["running"] = (snap["running"] - drained).astype(np.int32)
        kv = snap["kv"].astype(np.float64) + rng.normal(0.0, p.get("kv_walk", 0.02), D)
        snap["kv"] = np.clip(kv, 0.0, 1.0).astype(np.float32)
    return chosen, history
