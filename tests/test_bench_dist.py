"""bench.py's multi-rank logic on CPU: two gloo ranks on 127.0.0.1.

Batch routing shards by queries with no data exchange; the only collective is
the max over ranks of the step time, and the reported value is the work of
all ranks over that time.  Each rank draws its own seeded batch.
"""
import os
import socket

import pytest


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import torch.distributed as dist

    import bench
    import workload as W
    dist.init_process_group("gloo", rank=rank, world_size=world)
    r, w, local = bench.dist_env()
    step = 0.010 * (rank + 1)                      # rank 1 is the slower one
    slowest = bench.max_over_ranks(step, dist, "cpu")
    value = bench.whole_job_rate(1000, w, slowest)
    batch = W.make_config(0, Q=16, seed_offset=rank)
    out.put((r, w, local, slowest, value, batch["in_len"].tolist()))
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_weak_scaling_aggregate():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=180) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, w0, l0, s0, v0, b0), (r1, w1, l1, s1, v1, b1) = res
    assert (r0, r1, w0, w1, l0, l1) == (0, 1, 2, 2, 0, 1)
    assert s0 == s1 == pytest.approx(0.020)
    assert v0 == v1 == pytest.approx(2 * 1000 / 0.020)
    assert b0 != b1                                 # each rank routes its own batch


def test_single_process_defaults(monkeypatch):
    import bench
    for k in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)
    assert bench.dist_env() == (0, 1, 0)
    assert bench.max_over_ranks(1.5) == 1.5
    assert bench.whole_job_rate(65_536, 1, 0.5) == 131_072


def _route_loop_worker(rank, world, port, out):
    """One CPU rank of bench.py's timed region: its own seeded batch, routed
    by a callable the test supplies (the oracle here; bench.py routes through
    the library), timed between barriers, max over ranks."""
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import time

    import numpy as np
    import torch.distributed as dist

    import bench
    import oracle as O
    import workload as W
    dist.init_process_group("gloo", rank=rank, world_size=world)
    r, w, _ = bench.dist_env()
    p = W.make_config(0, Q=64, seed_offset=r)
    orc = O.Problem(p)
    calls = []

    def route(k):
        calls.append(k)
        ch = orc.route(mode=O.F32)[0]
        if r == 1:
            time.sleep(0.02)                        # rank 1 is the slow one
        return ch

    sec = bench.timed_route_loop(route, steps=4, warmup=3, timer=bench.WallTimer(), dist=dist,
                                 device="cpu")
    value = bench.whole_job_rate(p["Q"], w, sec)
    seen = list(calls)
    chosen = route(0)
    out.put((r, sec, value, seen, chosen.tolist(),
             np.array_equal(chosen, O.Problem(p).route(mode=O.F32)[0])))
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_run_the_timed_route_loop():
    """Unmeasured on GPU hardware (one GPU per call here): this covers the
    rank logic of the timed region on CPU ranks."""
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_route_loop_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=180) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, s0, v0, c0, ch0, ok0), (r1, s1, v1, c1, ch1, ok1) = res
    assert (r0, r1) == (0, 1)
    assert c0 == c1 == [0, 1, 2, 0, 1, 2, 3]        # 3 warm-up calls, then 4 timed
    assert s0 == s1 >= 0.02                         # the slowest rank sets the step time
    assert v0 == v1 == pytest.approx(2 * 64 / s0)   # work of both ranks over that time
    assert ok0 and ok1 and ch0 != ch1               # each rank routed its own batch
