"""Throughput of HW-Router batched route scoring on GB300.

One step = one hwr_route_batch call over one batch of synthetic queries: the
whole hot path (feature assembly, latency predictor, cost, quality, SLO mask,
argmax) for every (query, deployment) pair of the batch.

Default workload: the large bf16 configuration -- Q = 65,536 queries,
D = 64 deployments (16 models x 4 GPU types), 48 features, predictor
48 -> 256 -> 256 -> 2, 1024-wide bf16 embeddings, lambda = 0.3, SLO = 10 s.

Printed (one JSON line, rank 0):
  value     routed queries/s with inputs resident in HBM (device pointers),
            timed with CUDA events over K steps after W warm-up steps;
  e2e       the same through the C ABI with pinned host buffers: the
            host->device copy of the batch and the device->host copy of the
            results are inside every timed step;
  roofline  the dominant kernel's algorithmic FLOP (or bytes) per launch over
            its CUDA-event duration, against the measured GB300 peak (the
            durations come from a second pass of the K steps with events
            around every launch: those events stop the predictor kernel from
            starting while the quality kernel finishes, so that pass's step
            time, ms_per_step_profiled_pass, is a little longer);
  q1_latency_us  p50 / p99 single-query route latency through the C ABI with
            host buffers, at D = 32 (the batch-sweep shape);
  cpu_baseline   the CPU oracle on a bounded sample of the same workload;
  multi_lambda   one hwr_route_batch_multi call for 8 values of lambda on the
            same batch (the Sec. 5 lambda sweep), next to 8 single routes;
  sweep_d32 the batch-size sweep at D = 32 (8 models x 4 GPU types, H = 256,
            E = 1024): per Q in {1, 16, 256, 4096, 65536, 1048576}, p50 / p99
            of the CUDA-event time of isolated calls with device pointers, the
            time per call of calls queued back to back (groups of up to 20
            between one pair of events), queries/s at that time, and the
            fraction of the bf16 tensor roofline.
--impl reference times the CPU oracle (the reference arm for this build).
--online prints the online evaluation metrics of Sec. 4.4 (SLO attainment,
queue composition, load/running/waiting skew) for the online sequential
workload's shapes under each arrival pattern, for the hardware-aware router
and for the frozen-snapshot static-cost mode, one JSON line each, with the
wall-clock time of each micro-batch's route call through the C ABI.
"""
from __future__ import annotations

import argparse
import gc
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import workload as W  # noqa: E402

L2_BYTES = 129 * 1024 * 1024
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0,
                  "bf16_tflops_sustained": 1700.0, "sm_max_mhz": 2070.0}
# fp32 SIMT peak: 152 SMs x 128 FP32 lanes x 2 flop (FMA) x max SM clock.
SMS, FP32_LANES = 152, 128


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return d, "measured"
    except (OSError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


def workload_name(p):
    return (f"{p['name']}: Q={p['Q']} D={p['D']} ({p['M']} models x {p['G']} GPU types) "
            f"F={p['F']} MLP {p['F']}->{p['H1']}->{p['H2']}->2 E={p['E']} {p['dtype']} "
            f"lambda={p['lam']} SLO={p['slo']}s")


def flops_per_pair(p):
    # layer 2 (2 H1 H2) + the two heads (2 * 2 H2) + the layer-1 query suffix
    # (2 features x H1 x 2); the deployment prefix of layer 1 is per snapshot.
    return 2 * p["H1"] * p["H2"] + 4 * p["H2"] + 4 * p["H1"]


def bytes_per_query(p):
    es = 2 if p["dtype"] == "bf16" else 4
    return p["E"] * es + 8 + 12


def qual_bytes_per_query(p):
    # the quality kernel: the embedding row read, Mpad fp32 qualities written
    return p["E"] * 2 + (16 if p["M"] <= 16 else 32) * 4


def same_size_copy(torch, nbytes, stream, dev):
    """A device-to-device copy moving the same number of bytes (half read,
    half written), L2 flushed before each: what a transfer of this size
    reaches here, ramp and drain included (the measured peak is a long copy)."""
    half = nbytes // 2
    src = torch.empty(half, dtype=torch.uint8, device=dev)
    dst = torch.empty_like(src)
    flush = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device=dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ts = []
    with torch.cuda.stream(stream):
        src.fill_(1)
        for i in range(13):
            flush.fill_(i & 0xff)
            e0.record(stream)
            dst.copy_(src)
            e1.record(stream)
            e1.synchronize()
            if i >= 3:
                ts.append(e0.elapsed_time(e1))
    ms = float(sorted(ts)[len(ts) // 2])
    return {"bytes": 2 * half, "ms": ms, "gbs": 2 * half / (ms * 1e-3) / 1e9}


class ClockSampler:
    """SM clock and clock-event (throttle) reasons, sampled during the timed
    region.  Read-only NVML queries from a host thread every ~2 ms (the
    driver's management library, through ctypes), so that timed regions of a
    few milliseconds still get samples; nvidia-smi every 200 ms if NVML cannot
    be loaded."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    # NVML clock-event reason bits
    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}
    NVML_CLOCK_SM = 1

    def __init__(self, gpu_index, uuid=None):
        self.gpu, self.uuid = gpu_index, uuid
        self.proc = None
        self.file = None
        self.thread = None
        self.nvml = self._nvml_handle()

    def _nvml_handle(self):
        import ctypes as ct
        try:
            lib = ct.CDLL("libnvidia-ml.so.1")
            if lib.nvmlInit_v2() != 0:
                return None
            h = ct.c_void_p()
            rc = -1
            if self.uuid:
                rc = lib.nvmlDeviceGetHandleByUUID(self.uuid.encode(), ct.byref(h))
            if rc != 0:
                rc = lib.nvmlDeviceGetHandleByIndex_v2(ct.c_uint(self.gpu), ct.byref(h))
            if rc != 0:
                return None
            reasons = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
                lib.nvmlDeviceGetCurrentClocksThrottleReasons
            return lib, h, reasons
        except (OSError, AttributeError):
            return None

    def _poll(self):
        import ctypes as ct
        lib, h, reasons = self.nvml
        mhz, mask, mw = ct.c_uint(), ct.c_ulonglong(), ct.c_uint()
        while not self.done.is_set():
            if (lib.nvmlDeviceGetClockInfo(h, self.NVML_CLOCK_SM, ct.byref(mhz)) == 0 and
                    reasons(h, ct.byref(mask)) == 0):
                pw = mw.value if lib.nvmlDeviceGetPowerUsage(h, ct.byref(mw)) == 0 else 0
                self.samples.append((mhz.value, mask.value, pw))
            time.sleep(0.002)

    def start(self):
        if self.nvml:
            import threading
            self.samples, self.done = [], threading.Event()
            self.thread = threading.Thread(target=self._poll, daemon=True)
            self.thread.start()
            return
        try:
            self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=self.file, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def _stop_nvml(self):
        import ctypes as ct
        self.done.set()
        self.thread.join(timeout=5)
        self.thread = None
        if not self.samples:
            return None
        lib, h, _ = self.nvml
        mx = ct.c_uint()
        smax = mx.value if lib.nvmlDeviceGetMaxClockInfo(h, self.NVML_CLOCK_SM,
                                                         ct.byref(mx)) == 0 else None
        reasons = sorted({n for _, m, _ in self.samples for bit, n in self.REASONS.items()
                          if m & bit})
        return {"sm_mhz": statistics.median(s[0] for s in self.samples), "sm_max_mhz": smax,
                "reasons": reasons, "samples": len(self.samples),
                "power_w_max": max(s[2] for s in self.samples) / 1e3, "source": "nvml"}

    def stop(self):
        if self.thread:
            return self._stop_nvml()
        if not self.proc:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.file.flush()
        self.file.seek(0)
        rows = [l.split(",") for l in self.file.read().splitlines() if l.strip()]
        os.unlink(self.file.name)
        sm, mx, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for r in rows:
            if len(r) < 9:
                continue
            try:
                sm.append(float(r[1]))
                mx.append(float(r[2]))
            except ValueError:
                continue
            for n, v in zip(names, r[5:9]):
                if v.strip().lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx),
                "reasons": sorted(reasons), "samples": len(sm), "source": "nvidia-smi"}


def kernel_sources_sha256():
    """Hash of the sources the tensor-core kernels are built from."""
    import hashlib
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2608_14575_gb300", "csrc")
    for f in sorted(["k_tc.cu", "umma.cuh", "select.cuh", "hwr_internal.cuh"]):
        with open(os.path.join(csrc, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def profiled_traffic(kernel):
    """DRAM bytes per launch from the committed ncu capture, or None when the
    kernel sources changed since the counters were taken."""
    try:
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
            t = json.load(f)
    except (OSError, ValueError):
        return None
    if t.get("sources_sha256") != kernel_sources_sha256():
        return None
    k = t.get("kernels", {}).get(kernel)
    return None if k is None else k.get("dram_bytes_per_launch")


def max_over_ranks(x, dist=None, device=None):
    """Largest value of x over all ranks (x itself without a process group)."""
    if dist is None:
        return float(x)
    import torch
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(queries_per_rank, world, seconds):
    """Units processed by all ranks over the slowest rank's time."""
    return world * queries_per_rank / seconds


class EventTimer:
    """Seconds between start() and stop(), from CUDA events recorded on the
    stream the kernels run on (torch's events see only the stream they are
    recorded on)."""

    def __init__(self, torch, stream):
        self.torch, self.stream = torch, stream
        self.e0 = torch.cuda.Event(enable_timing=True)
        self.e1 = torch.cuda.Event(enable_timing=True)

    def sync(self):
        self.torch.cuda.synchronize()

    def start(self):
        self.sync()
        self.e0.record(self.stream)

    def stop(self):
        self.e1.record(self.stream)
        self.sync()
        return self.e0.elapsed_time(self.e1) * 1e-3


class WallTimer:
    """Host wall-clock seconds (CPU ranks, end-to-end host loops)."""

    def sync(self):
        pass

    def start(self):
        self.t = time.perf_counter()

    def stop(self):
        return time.perf_counter() - self.t


def timed_route_loop(route, steps, warmup, timer, dist=None, device=None, before=None,
                     after=None):
    """The per-rank timed region: `warmup` untimed calls route(k), then
    `steps` timed ones between barriers; returns the max over ranks of the
    seconds per step.  `before` runs after the warm-up (reset counters, start
    the clock sampler), `after` once the timed calls have finished."""
    for k in range(warmup):
        route(k)
    timer.sync()
    if before:
        before()
    if dist:
        dist.barrier()
    timer.start()
    for k in range(steps):
        route(k)
    sec = timer.stop()
    if after:
        after()
    if dist:
        dist.barrier()
    return max_over_ranks(sec / steps, dist, device)


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def cpu_oracle_rate(p, seconds, nthreads):
    """Queries/s of the oracle (fp64 mode) on a sample sized to ~`seconds`."""
    import oracle as O
    orc = O.Problem(p)
    n = min(p["Q"], 64 * nthreads)
    t = time.perf_counter()
    orc.route(p["in_len"][:n], p["out_len"][:n], p["emb"][:n], nthreads=nthreads)
    per_q = (time.perf_counter() - t) / n
    n = int(min(p["Q"], max(64, seconds / max(per_q, 1e-9))))
    t = time.perf_counter()
    orc.route(p["in_len"][:n], p["out_len"][:n], p["emb"][:n], nthreads=nthreads)
    dt = time.perf_counter() - t
    return n / dt, n, dt


def run_reference(args, p):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    cores = len(os.sched_getaffinity(0))
    import oracle as O
    orc = O.Problem(p)
    # per-step sample sized to about 1.5 s of CPU work
    t = time.perf_counter()
    orc.route(p["in_len"][:32], p["out_len"][:32], p["emb"][:32], nthreads=cores)
    per_q = (time.perf_counter() - t) / 32
    S = int(min(p["Q"], max(32, 1.5 / max(per_q, 1e-9))))
    for k in range(args.warmup):
        lo = (k * S) % max(1, p["Q"] - S + 1)
        orc.route(p["in_len"][lo:lo + S], p["out_len"][lo:lo + S], p["emb"][lo:lo + S],
                  nthreads=cores)
    t = time.perf_counter()
    for k in range(args.steps):
        lo = (k * S) % max(1, p["Q"] - S + 1)
        orc.route(p["in_len"][lo:lo + S], p["out_len"][lo:lo + S], p["emb"][lo:lo + S],
                  nthreads=cores)
    dt = time.perf_counter() - t
    v = S * args.steps / dt
    line = {
        "impl": "reference", "metric": "routed_queries_per_s", "value": v,
        "unit": "queries/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": dt / args.steps * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": workload_name(p), "sample_queries_per_step": S},
        "cpu_baseline": {"value": v, "unit": "queries/s", "cores": cores, "kind": "oracle",
                         "sample": f"{S} queries of the workload per step, fp64 oracle, "
                                   f"{cores} OpenMP threads"},
        "e2e": {"value": v, "unit": "queries/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def q1_latency(H, iters=10_000):
    """p50/p99 of one-query routes through the C ABI with pinned host buffers."""
    import torch
    p = W.make_config(4, Q=1024)
    r = H.Router(p)
    il = torch.from_numpy(p["in_len"]).pin_memory()
    ol = torch.from_numpy(p["out_len"]).pin_memory()
    em = torch.from_numpy(p["emb"].view(np.int16)).pin_memory()
    ch = torch.empty(1, dtype=torch.int32).pin_memory()
    lat = torch.empty(1, dtype=torch.float32).pin_memory()
    ut = torch.empty(1, dtype=torch.float32).pin_memory()
    es = em.element_size() * p["E"]
    times = []
    gc.collect()
    gc.disable()      # a collector pause inside a timed call is not the library's
    for k in range(iters + 200):
        i = k % p["Q"]
        t = time.perf_counter()
        r.route_host_ptrs(1, il.data_ptr() + 4 * i, ol.data_ptr() + 4 * i,
                          em.data_ptr() + es * i, ch.data_ptr(), lat.data_ptr(),
                          ut.data_ptr(), slo=p["slo"], lam=p["lam"])
        if k >= 200:
            times.append(time.perf_counter() - t)
    gc.enable()
    r.close()
    a = np.array(times) * 1e6
    return {"p50": float(np.percentile(a, 50)), "p99": float(np.percentile(a, 99)),
            "calls": iters, "config": "D=32 (8 models x 4 GPU types), MLP 48->256->256->2, "
                                      "E=1024 bf16, host buffers, end to end",
            "paper_routing_overhead_us": 200.0}


def config_latencies(H, stream, dev, calls=300):
    """Per-call latency of the other workloads: the small fp32 batch and the mid
    bf16 batch (device pointers, isolated calls, CUDA events) and a 64-request
    micro-batch of the online sequential workload (snapshot upload + sequential
    route through the C ABI with host buffers, wall clock)."""
    import torch
    out = {}
    for c in (0, 1):
        p = W.make_config(c)
        r = H.Router(p, stream=stream.cuda_stream)
        emb = p["emb"].view(np.int16) if p["dtype"] == "bf16" else p["emb"]
        args = (torch.from_numpy(p["in_len"]).to(dev), torch.from_numpy(p["out_len"]).to(dev),
                torch.from_numpy(emb).to(dev), torch.empty(p["Q"], dtype=torch.int32, device=dev),
                torch.empty(p["Q"], dtype=torch.float32, device=dev),
                torch.empty(p["Q"], dtype=torch.float32, device=dev))
        for _ in range(20):
            r.route_device(*args, slo=p["slo"], lam=p["lam"])
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(calls)]
        for e0, e1 in ev:
            e0.record(stream)
            r.route_device(*args, slo=p["slo"], lam=p["lam"])
            e1.record(stream)
        torch.cuda.synchronize()
        t = np.array([a.elapsed_time(b) for a, b in ev]) * 1e3
        r.close()
        out[f"config{c}"] = {"workload": workload_name(p), "calls": calls,
                             "p50_us": float(np.median(t)), "p99_us": float(np.percentile(t, 99)),
                             "queries_per_s": float(p["Q"] / (np.median(t) * 1e-6))}
    p = W.make_config(2, Q=64 * 200)
    r = H.Router(p)
    n, times = 64, []
    gc.collect()
    gc.disable()      # a collector pause inside a timed call is not the library's
    for k in range(220):
        lo = (k % 200) * n
        t = time.perf_counter()
        r.update_snapshot(p["snap"])
        r.route(p["in_len"][lo:lo + n], p["out_len"][lo:lo + n], p["emb"][lo:lo + n],
                flags=H.HWR_SEQUENTIAL)
        if k >= 20:
            times.append(time.perf_counter() - t)
    gc.enable()
    r.close()
    a = np.array(times) * 1e6
    out["config2"] = {"workload": workload_name(p) + ", micro-batches of 64, sequential",
                      "calls": len(a), "p50_us": float(np.median(a)),
                      "p99_us": float(np.percentile(a, 99)),
                      "requests_per_s": float(n / (np.median(a) * 1e-6)),
                      "note": "snapshot upload + sequential route of one micro-batch, "
                              "host buffers, wall clock"}
    # sequential mode on a bf16 cluster (the sweep's shapes, D = 32, H = 256):
    # the score table on the SIMT path (canonical fp32 order) and on the
    # tensor cores (HWR_PATH_TENSOR)
    p = W.make_config(4, Q=64 * 50)
    r = H.Router(p)
    seq = {}
    gc.collect()
    gc.disable()
    for name, fl in (("simt_table", H.HWR_SEQUENTIAL),
                     ("tensor_table", H.HWR_SEQUENTIAL | H.HWR_PATH_TENSOR)):
        times = []
        for k in range(120):
            lo = (k % 50) * n
            t = time.perf_counter()
            r.update_snapshot(p["snap"])
            r.route(p["in_len"][lo:lo + n], p["out_len"][lo:lo + n], p["emb"][lo:lo + n],
                    flags=fl)
            if k >= 20:
                times.append(time.perf_counter() - t)
        a = np.array(times) * 1e6
        seq[name] = {"p50_us": float(np.median(a)), "p99_us": float(np.percentile(a, 99)),
                     "requests_per_s": float(n / (np.median(a) * 1e-6))}
    gc.enable()
    r.close()
    out["sequential_bf16"] = {"workload": workload_name(p) + ", micro-batches of 64, sequential",
                              "calls": 100, **seq,
                              "note": "snapshot upload + sequential route of one micro-batch, "
                                      "host buffers, wall clock"}
    return out


# Online scenarios on the online sequential workload's shapes (D = 12).  The
# serving world has 16 slots per deployment and 0.5 s mean service, so it
# completes 384 requests/s with every slot busy.
ONLINE_SCENARIOS = {
    "online_sequential": dict(),   # the workload itself: Poisson 200 req/s, batches of 64
    "poisson": dict(pattern="poisson", rate=200.0, window=0.02, cap=16, drain="per_time",
                    service_s=0.5),
    "micro_burst": dict(pattern="micro_burst", rate=150.0, window=0.02, cap=16,
                        drain="per_time", service_s=0.5, burst_factor=8.0, burst_len=0.05,
                        period=1.0),
    "sustained_overload": dict(pattern="sustained_overload", rate=384.0, window=0.02, cap=16,
                               drain="per_time", service_s=0.5, overload=1.25),
}


def online_report(args):
    import paper_2608_14575_gb300 as H
    from paper_2608_14575_gb300 import metrics as MX
    from paper_2608_14575_gb300.online import OnlineRouter
    from workload import serve
    H.build()
    p = W.make_config(2, Q=args.q or 20_000)
    for name, world in ONLINE_SCENARIOS.items():
        for mode, static in (("hw_router", False), ("static_cost", True)):
            times = []
            with OnlineRouter(p) as r:
                def route(snap, lo, hi):
                    t = time.perf_counter()
                    out = r.route(snap, lo, hi)
                    times.append(time.perf_counter() - t)
                    return out
                gc.collect()
                gc.disable()      # collector pauses are not the library's call latency
                try:
                    tr = serve.run_online(p, route, r.score, static=static, **world)
                finally:
                    gc.enable()
            m = MX.summarize(tr, p["dep_gpu"], p["G"], p["D"])
            us = np.array(times) * 1e6
            sizes = tr["batch_end"] - tr["batch_start"]
            print(json.dumps({
                "online": name, "mode": mode, "workload": workload_name(p),
                "world": {k: v for k, v in world.items()}, **m,
                "route_call_us": {"p50": float(np.percentile(us, 50)),
                                  "p99": float(np.percentile(us, 99)),
                                  "mean_batch": float(sizes[sizes > 0].mean()),
                                  "requests_per_s": float(sizes.sum() / (us.sum() * 1e-6)),
                                  "note": "snapshot upload + sequential route of one "
                                          "micro-batch, host buffers, wall clock"}}),
                flush=True)


def sweep_d32(H, stream, dev):
    """Per-call latency and throughput over the batch sizes of the D = 32 sweep."""
    import torch
    base = W.make_config(4, Q=65_536)
    Qmax = max(W.CONFIGS[4]["sweep"])
    r = H.Router(base, stream=stream.cuda_stream)
    il0 = torch.from_numpy(base["in_len"]).to(dev)
    ol0 = torch.from_numpy(base["out_len"]).to(dev)
    em0 = torch.from_numpy(base["emb"].view(np.int16)).to(dev)
    reps = Qmax // base["Q"]
    # the largest batch is the 65,536-query batch repeated (every query is still routed)
    ilb, olb, emb = il0.repeat(reps), ol0.repeat(reps), em0.repeat(reps, 1)
    ch = torch.empty(Qmax, dtype=torch.int32, device=dev)
    lat = torch.empty(Qmax, dtype=torch.float32, device=dev)
    ut = torch.empty(Qmax, dtype=torch.float32, device=dev)
    torch.cuda.synchronize()
    pk, _ = peaks()
    fq = base["D"] * flops_per_pair(base) + 2 * base["E"] * base["M"]   # flop per query
    out = []
    for Q in W.CONFIGS[4]["sweep"]:
        n = 200 if Q <= 4096 else (50 if Q <= 65_536 else 20)
        args = (ilb[:Q], olb[:Q], emb[:Q], ch[:Q], lat[:Q], ut[:Q])
        for _ in range(10):
            r.route_device(*args, slo=base["slo"], lam=base["lam"])
        # isolated calls (each waits for its results: the latency a caller
        # sees; CUDA events around every call) and calls queued back to back
        # (HWR_ASYNC, one pair of events around groups of calls, as for the
        # main value: the throughput of a caller that pipelines its calls)
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(n)]
        for e0, e1 in ev:
            e0.record(stream)
            r.route_device(*args, slo=base["slo"], lam=base["lam"])
            e1.record(stream)
        torch.cuda.synchronize()
        iso = np.array([e0.elapsed_time(e1) for e0, e1 in ev]) * 1e3   # us
        group = max(1, min(n, 20))
        per = []
        for _ in range(max(3, n // group)):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for _ in range(group):
                r.route_device(*args, slo=base["slo"], lam=base["lam"], flags=H.HWR_ASYNC)
            e1.record(stream)
            torch.cuda.synchronize()
            per.append(e0.elapsed_time(e1) * 1e3 / group)
        r.synchronize()
        med = float(np.median(per))
        qps = Q / (med * 1e-6)
        out.append({"Q": Q, "calls": n, "p50_us": float(np.median(iso)),
                    "p99_us": float(np.percentile(iso, 99)),
                    "pipelined_us_per_call": med, "queries_per_s": qps,
                    "frac_of_tensor_roofline": qps * fq / (pk["bf16_tflops"] * 1e12)})
    r.close()
    return {"config": "D=32 (8 models x 4 GPU types), MLP 48->256->256->2, E=1024 bf16; "
                      "device pointers; p50/p99 of isolated calls (CUDA events around each), "
                      "queries/s from calls queued back to back (events around groups of "
                      "up to 20 calls, median per-call time); "
                      f"Q={Qmax} is the 65,536-query batch repeated {reps}x",
            "points": out}


def multi_lambda(H, r, p, bufs, flags, stream, steps=10):
    """One 8-lambda call against 8 single-lambda calls on the same device batch."""
    import torch
    lams = np.linspace(0.05, 2.0, 8).astype(np.float32)
    Q, K = p["Q"], len(lams)
    dev = bufs[0][0].device
    ch = torch.empty((K, Q), dtype=torch.int32, device=dev)
    lat = torch.empty((K, Q), dtype=torch.float32, device=dev)
    ut = torch.empty((K, Q), dtype=torch.float32, device=dev)
    torch.cuda.synchronize()
    il, ol, em = bufs[0]

    fa = flags | H.HWR_ASYNC

    def multi():
        r.route_device_multi(lams, il, ol, em, ch, lat, ut, slo=p["slo"], flags=fa)

    def singles():
        for k in range(K):
            r.route_device(il, ol, em, ch[k], lat[k], ut[k], slo=p["slo"], lam=float(lams[k]),
                           flags=fa)
    res = {}
    for name, fn in (("multi", multi), ("singles", singles)):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(steps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        r.synchronize()
        res[name] = e0.elapsed_time(e1) / steps
    return {"lambdas": K, "ms_per_call": res["multi"], "ms_8_single_calls": res["singles"],
            "lambda_routes_per_s": Q * K / (res["multi"] * 1e-3)}


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="hwr", choices=["hwr", "reference"])
    ap.add_argument("--config", type=int, default=3)
    ap.add_argument("--q", type=int, default=None, help="override the query count")
    ap.add_argument("--path", default="auto", choices=["auto", "simt", "tensor"])
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--no-q1", action="store_true")
    ap.add_argument("--no-clocks", action="store_true")
    ap.add_argument("--no-multi", action="store_true")
    ap.add_argument("--no-sweep", action="store_true")
    ap.add_argument("--no-configs", action="store_true")
    ap.add_argument("--online", action="store_true",
                    help="print the online evaluation metrics instead of the throughput line")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    rank, world, local = dist_env()
    if args.online:
        if rank == 0:
            online_report(args)
        return

    if args.impl == "reference":
        if rank == 0:
            p = W.make_config(args.config, Q=args.q, seed_offset=0)
            run_reference(args, p)
        return

    import torch
    import paper_2608_14575_gb300 as H
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    H.build()

    p = W.make_config(args.config, Q=args.q, seed_offset=rank)
    Q = p["Q"]
    dev = torch.device("cuda", local)
    # a stream of its own (the default stream's handle is NULL, for which the
    # library would create a private stream): the CUDA events below are
    # recorded on the stream the kernels run on
    stream = torch.cuda.Stream(device=dev)
    r = H.Router(p, stream=stream.cuda_stream)
    flags = {"auto": 0, "simt": H.HWR_PATH_SIMT, "tensor": H.HWR_PATH_TENSOR}[args.path]

    emb_np = p["emb"].view(np.int16) if p["dtype"] == "bf16" else p["emb"]
    in_bytes = Q * bytes_per_query(p)
    nbuf = max(1, min(4, -(-3 * L2_BYTES // max(in_bytes, 1))))
    bufs = []
    for _ in range(nbuf):
        bufs.append((torch.from_numpy(p["in_len"]).to(dev), torch.from_numpy(p["out_len"]).to(dev),
                     torch.from_numpy(emb_np).to(dev)))
    ch = torch.empty(Q, dtype=torch.int32, device=dev)
    lat = torch.empty(Q, dtype=torch.float32, device=dev)
    ut = torch.empty(Q, dtype=torch.float32, device=dev)
    torch.cuda.synchronize()      # inputs are written on the default stream

    def step(k, extra=0):
        il, ol, em = bufs[k % nbuf]
        r.route_device(il, ol, em, ch, lat, ut, slo=p["slo"], lam=p["lam"],
                       flags=flags | extra)

    try:
        uuid = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except (AttributeError, RuntimeError):
        uuid = None
    clocks = ClockSampler(local, uuid)
    marks = {}

    def before():
        r.stats(reset=True)
        marks["launches"] = r.stats()["kernel_launches"]
        if not args.no_clocks:
            clocks.start()

    # warm-up steps synchronous, timed steps queued back to back (the status
    # word is checked after them)
    ms = 1e3 * timed_route_loop(lambda k: step(k, H.HWR_ASYNC if marks else 0), args.steps,
                                args.warmup, EventTimer(torch, stream), dist, dev,
                                before=before, after=r.synchronize)
    clk = clocks.stop()
    launches = r.stats(reset=True)["kernel_launches"] - marks["launches"]
    value = whole_job_rate(Q, world, ms * 1e-3)
    # Per-kernel durations: a second pass of the same K steps with CUDA events
    # around every launch (the events sit between the quality and predictor
    # kernels, so that pass loses their overlap and is timed separately).
    ep0, ep1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ep0.record(stream)
    for k in range(args.steps):
        step(k, H.HWR_PROFILE | H.HWR_ASYNC)
    ep1.record(stream)
    torch.cuda.synchronize()
    r.synchronize()
    ms_prof = ep0.elapsed_time(ep1) / args.steps
    st = r.stats(reset=True)

    # dominant kernel and its roofline
    pk, src = peaks()
    kms = {k: st["profiled_ms"][k] / max(1, st["profiled_launches"][k])
           for k in H.KERNELS if st["profiled_launches"][k]}
    top = max(kms, key=kms.get)
    pairs = Q * p["D"]
    if top == "mlp_tc":
        flop = pairs * flops_per_pair(p)
        ach = flop / (kms[top] * 1e-3) / 1e12
        roof = {"bound": "tensor", "achieved": ach, "peak": pk["bf16_tflops"],
                "unit": "TFLOP/s", "frac": ach / pk["bf16_tflops"], "traffic": profiled_traffic(top),
                "kernel": top, "ms_per_launch": kms[top],
                "peak_source": f"{src} bf16 burst (cuBLAS), frac vs sustained "
                               f"{ach / pk.get('bf16_tflops_sustained', pk['bf16_tflops']):.3f}"}
    elif top == "qual_tc":
        byt = Q * qual_bytes_per_query(p)
        ach = byt / (kms[top] * 1e-3) / 1e9
        roof = {"bound": "hbm", "achieved": ach, "peak": pk["hbm_gbs"], "unit": "GB/s",
                "frac": ach / pk["hbm_gbs"], "traffic": profiled_traffic(top), "kernel": top,
                "ms_per_launch": kms[top], "peak_source": f"{src} copy bandwidth"}
    else:
        flop = pairs * flops_per_pair(p)
        peak = SMS * FP32_LANES * 2 * pk.get("sm_max_mhz", 2070.0) * 1e6 / 1e12
        ach = flop / (kms[top] * 1e-3) / 1e12
        roof = {"bound": "alu", "achieved": ach, "peak": peak, "unit": "TFLOP/s",
                "frac": ach / peak, "traffic": None, "kernel": top, "ms_per_launch": kms[top],
                "peak_source": "fp32 FMA: 152 SMs x 128 lanes x 2 x max SM clock"}

    # the other roofline-bound kernel of the step, against the measured peak
    # and against a copy of the same size
    others = {}
    if "qual_tc" in kms and top != "qual_tc":
        byt = Q * qual_bytes_per_query(p)
        ach = byt / (kms["qual_tc"] * 1e-3) / 1e9
        cp = same_size_copy(torch, byt, stream, dev)
        others["qual_tc"] = {"bound": "hbm", "achieved": ach, "peak": pk["hbm_gbs"], "unit": "GB/s",
                             "frac": ach / pk["hbm_gbs"], "traffic": profiled_traffic("qual_tc"),
                             "ms_per_launch": kms["qual_tc"], "bytes_per_launch": byt,
                             "same_size_copy": cp, "frac_of_same_size_copy": ach / cp["gbs"]}

    line = {
        "metric": "routed_queries_per_s", "value": value, "unit": "queries/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": p["dtype"], "data": "synthetic (seeded; shapes and distributions of the "
                                     "paper's workload stand-ins)",
        "config": {"workload": workload_name(p), "queries_per_gpu": Q,
                   "path": args.path,
                   "l2": f"{nbuf} input buffers of {in_bytes / 2**20:.0f} MiB rotated per step "
                         f"({'inputs > L2' if in_bytes > L2_BYTES else 'rotation > L2'})",
                   "parallelism": f"replicas x{world} (queries sharded, no collective)"},
        "kernel_ms": kms, "ms_per_step_profiled_pass": ms_prof,
        "gpu_launches": launches, "roofline": roof, "other_kernels": others, "clocks": clk,
    }

    if not args.no_e2e:
        pin = (torch.from_numpy(p["in_len"]).pin_memory(), torch.from_numpy(p["out_len"]).pin_memory(),
               torch.from_numpy(emb_np).pin_memory())
        och = torch.empty(Q, dtype=torch.int32).pin_memory()
        olat = torch.empty(Q, dtype=torch.float32).pin_memory()
        out_ = torch.empty(Q, dtype=torch.float32).pin_memory()

        def host_step():
            r.route_host_ptrs(Q, pin[0].data_ptr(), pin[1].data_ptr(), pin[2].data_ptr(),
                              och.data_ptr(), olat.data_ptr(), out_.data_ptr(),
                              slo=p["slo"], lam=p["lam"], flags=flags)
        dt = timed_route_loop(lambda k: host_step(), args.steps, args.warmup, WallTimer(),
                              dist, dev)
        line["e2e"] = {"value": whole_job_rate(Q, world, dt), "unit": "queries/s",
                       "h2d_bytes_per_step": Q * (bytes_per_query(p) - 12),
                       "d2h_bytes_per_step": Q * 12, "ms_per_step": dt * 1e3}
    if not args.no_multi:
        line["multi_lambda"] = multi_lambda(H, r, p, bufs, flags, stream)
    if rank == 0 and not args.no_sweep and p["dtype"] == "bf16":
        line["sweep_d32"] = sweep_d32(H, stream, dev)
    if rank == 0 and not args.no_q1:
        line["q1_latency_us"] = q1_latency(H)
    if rank == 0 and not args.no_configs:
        line["configs"] = config_latencies(H, stream, dev)
    if rank == 0 and not args.no_cpu:
        cores = len(os.sched_getaffinity(0))
        v, n, dt = cpu_oracle_rate(p, 10.0, cores)
        v1, n1, dt1 = cpu_oracle_rate(p, 4.0, 1)
        line["cpu_baseline"] = {"value": v, "unit": "queries/s", "cores": cores,
                                "kind": "oracle",
                                "sample": f"first {n} queries of the workload, fp64 oracle, "
                                          f"{cores} OpenMP threads, {dt:.1f} s",
                                "single_thread": {"value": v1, "sample": f"first {n1} queries, "
                                                                         f"1 thread, {dt1:.1f} s"}}
    r.close()
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
