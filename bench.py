#!/usr/bin/env python3
"""Benchmark of progressive approximate-LSTM inference on GB300.

Workload (batch-1 latency workload): one LSTM layer, D=1024 (ReLU-distributed
CNN-feature-like inputs), H=512, T=20 timesteps, one stream per GPU, fp32
factors, keep 25% of each v (NZ=384 of C=1536), refinement depth K=256 with
intermediate outputs at depths 16 and 64 emitted in the same run.  One step
is one call of the library over the whole sequence: the hoisted input
projection, the persistent recurrence kernel (coefficients, sums over u,
cell update, intermediate outputs) -- every step of the path.

Metric: timesteps*streams per second (whole job over all GPUs) and the p50
per-timestep latency; a sweep over K = 16, 64, 256 is reported beside it.
Factor sets and inputs are seeded synthetic draws with the structure of the
method's factors (the timed cost does not depend on the values).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Under torchrun each rank drives its own GPU with its own stream (weak
scaling, no data-path collective); rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import time

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
if HERE not in sys.path:
    sys.path.insert(0, HERE)

from workloads import WORKLOADS, nz_from_keep, synthetic_layer_factors, workload_inputs  # noqa: E402

METRIC = "approx-LSTM timesteps·streams/sec vs rank K; p50 per-step latency at batch 1"
UNIT = "timesteps*streams/s"
WL = WORKLOADS["c2"]
KEEP = 0.25
K_MAIN = 256
CKPTS = (16, 64)
K_SWEEP = (16, 64, 256)
L2_FLUSH_BYTES = 256 << 20

# DRAM bytes (dram__bytes_read.sum + dram__bytes_write.sum) of one launch of
# the recurrence kernel on this workload, from the ncu capture summarised in
# profiles/persistent_kernel_lstm-d1024-h512-t20-b1-fp32.md.  The figure
# holds only for the kernel sources it was taken on: `captured_traffic`
# returns None once their SHA-256 differs.
TRAFFIC_SOURCES = ("k_persistent.cu", "ptx.cuh")
TRAFFIC_CAPTURE = {"sha256": "74b3043aed6800cc4782c7daec6ca4f72bc8c4a7bf4ec800d298c7eadca2fe73",
                   "bytes": 4345600}


def captured_traffic():
    csrc = os.path.join(HERE, "paper_1905_00689_gb300", "csrc")
    h = hashlib.sha256()
    for f in TRAFFIC_SOURCES:
        with open(os.path.join(csrc, f), "rb") as fh:
            h.update(fh.read())
    return TRAFFIC_CAPTURE["bytes"] if h.hexdigest() == TRAFFIC_CAPTURE["sha256"] else None


def _config(n_gpus: int) -> dict:
    C = WL.C()
    return {
        "workload": (f"{WL.name}: 1-layer LSTM D={WL.D} H={WL.H} T={WL.T}, {WL.B} stream per GPU, fp32 factors, "
                     f"keep {KEEP} -> NZ={nz_from_keep(KEEP, C)} of C={C}, K={K_MAIN}, "
                     f"intermediate outputs at K={','.join(map(str, CKPTS))}"),
        "streams_per_gpu": WL.B, "timesteps": WL.T, "K": K_MAIN, "checkpoints": list(CKPTS),
        "l2": "flushed between timed steps (256 MiB device write outside the step's events)",
        "parallelism": f"replicas x{n_gpus} (independent streams, no collective)",
    }


def p90(xs) -> float:
    """90th percentile (nearest rank) of a non-empty sequence."""
    ys = sorted(xs)
    return ys[min(len(ys) - 1, max(0, math.ceil(0.9 * len(ys)) - 1))]


def _dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


# --------------------------------------------------------------------------
# host-side helpers (also used by the CPU tests)
# --------------------------------------------------------------------------

def algorithmic_bytes_per_timestep(H: int, C: int, nz: int, K: int, s: int = 4) -> int:
    """Factor bytes one timestep of one stream must read: 4 gates x K terms x
    (NZ values + a 1-bit column mask + u + sigma)."""
    return 4 * K * (nz * s + (C + 7) // 8 + H * s + s)


def recurrence_bytes_per_timestep(H: int, nz_h: float, K: int, s: int = 4) -> float:
    """Factor bytes of the recurrent part alone (h columns of v, mask, u, sigma)."""
    return 4 * K * (nz_h * s + (H + 7) // 8 + H * s + s)


def aggregate(values_ms, world_size: int, units_per_rank: int):
    """Whole-job throughput from per-rank step times: units of all ranks over the slowest rank."""
    t = max(values_ms)
    return units_per_rank * world_size / (t / 1e3), t


def combine_ranks(times_ms, units_per_rank: int, dist=None, device="cpu"):
    """Max over ranks of each per-rank time (one all-reduce), and the whole-job
    throughput for each: the units all ranks processed over the slowest rank."""
    import torch
    vals = torch.tensor(list(times_ms), dtype=torch.float64, device=device)
    ws = 1
    if dist is not None:
        dist.all_reduce(vals, op=dist.ReduceOp.MAX)
        ws = dist.get_world_size()
    worst = [float(v) for v in vals.cpu()]
    return [units_per_rank * ws / (t / 1e3) for t in worst], worst


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = os.path.join("/tmp", f"bench_clocks_{os.getpid()}.csv")

    def __enter__(self):
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                          "-lms", "50", "-i", str(self.gpu)], stdout=self.fh,
                                         stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.fh.close()

    def summary(self):
        if self.proc is None or not os.path.exists(self.path):
            return None
        sm, mx, reasons = [], None, set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = float(parts[2])
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# --------------------------------------------------------------------------
# reference arm: the fp64 oracle on the host cores
# --------------------------------------------------------------------------

def _oracle_sample(reps_budget_s: float, K: int, checkpoints=CKPTS):
    """Time the oracle (as it stands) on the benchmark workload; returns (s per run, runs)."""
    import oracle
    layers = [synthetic_layer_factors(WL, 0, K, KEEP)]
    x = workload_inputs(WL).astype(np.float32).astype(np.float64)
    runs, t0 = 0, time.perf_counter()
    while True:
        oracle.run_lstm(layers, x, K, checkpoints=checkpoints)
        runs += 1
        el = time.perf_counter() - t0
        if el >= reps_budget_s:
            return el / runs, runs


def cpu_baseline(budget_s: float = 12.0) -> dict:
    """Oracle throughput on the host, single-threaded, in a child process."""
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
    code = (f"import sys; sys.path.insert(0, {HERE!r}); import bench; "
            f"s, n = bench._oracle_sample({budget_s}, {K_MAIN}); print(s, n)")
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env, timeout=600)
    if r.returncode != 0:
        return {"value": None, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": "failed: " + r.stderr[-200:]}
    s_per_run, runs = map(float, r.stdout.split())
    return {"value": WL.T * WL.B / s_per_run, "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": (f"{int(runs)} full runs of the benchmark workload (T={WL.T}, B={WL.B}, K={K_MAIN}, "
                       f"checkpoints {list(CKPTS)}) in {s_per_run * runs:.1f} s, fp64 NumPy, 1 thread")}


# the oracle on every workload: (workload, keep, K, intermediate depths, T and
# streams of the bounded sample); streams are independent, so the oracle's
# throughput on a few streams and steps is its throughput on the whole workload
ORACLE_CONFIGS = (("c1", 0.5, 64, (), None, 1), ("c2", 0.25, 256, (16, 64), None, 1),
                  ("c3", 0.5, 512, (), 4, 1), ("c4", 0.5, 512, (), 2, 1), ("c4", 0.1, 128, (), 4, 1),
                  ("c5", 0.3, 1024, (16, 64, 256, 1024), 2, 1))


def oracle_config_sweep(budget_s: float = 4.0) -> list:
    """The fp64 oracle (as it stands, one thread) timed on a bounded sample of
    every workload: timesteps*streams/s and the sample it was taken on."""
    import oracle
    out = []
    for name, keep, K, cps, T_s, B_s in ORACLE_CONFIGS:
        w = WORKLOADS[name]
        T_s = T_s or w.T
        layers = [synthetic_layer_factors(w, l, K, keep) for l in range(w.L)]
        x = workload_inputs(w, T=T_s, B=B_s).astype(np.float32).astype(np.float64)
        runs, t0 = 0, time.perf_counter()
        while True:
            oracle.run_lstm(layers, x, K, checkpoints=cps)
            runs += 1
            el = time.perf_counter() - t0
            if el >= budget_s:
                break
        out.append({"workload": w.name, "keep": keep, "K": K, "checkpoints": list(cps),
                    "value": T_s * B_s * runs / el, "unit": UNIT, "cores": 1,
                    "sample": f"{runs} runs of T={T_s}, B={B_s} in {el:.1f} s"})
    return out


def run_reference(args):
    ws, rank, _ = _dist_env()
    if rank != 0:
        return
    if args.all_configs:  # the oracle on every workload (one line per workload), then the usual line
        env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
        code = (f"import sys, json; sys.path.insert(0, {HERE!r}); import bench; "
                f"print(json.dumps(bench.oracle_config_sweep()))")
        r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env, timeout=1200)
        print(json.dumps({"impl": "reference", "oracle_by_workload": json.loads(r.stdout) if r.returncode == 0
                          else "failed: " + r.stderr[-300:]}), flush=True)
    import oracle
    layers = [synthetic_layer_factors(WL, 0, K_MAIN, KEEP)]
    x = workload_inputs(WL).astype(np.float32).astype(np.float64)
    for _ in range(args.warmup):
        oracle.run_lstm(layers, x, K_MAIN, checkpoints=CKPTS)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        oracle.run_lstm(layers, x, K_MAIN, checkpoints=CKPTS)
        times.append(time.perf_counter() - t0)
    ms = 1e3 * sum(times) / len(times)
    value = WL.T * WL.B / (ms / 1e3)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": _config(1),
        "p50_us_per_timestep": 1e3 * statistics.median(times) / WL.T * 1e3,
        "p90_us_per_timestep": 1e3 * p90(times) / WL.T * 1e3,
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                         "sample": f"{args.steps} full runs of the benchmark workload, fp64 NumPy, one thread"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------------------
# our arm
# --------------------------------------------------------------------------

def run_ours(args):
    import torch
    from paper_1905_00689_gb300 import (LSTMApprox, OPT_TIMING, Q_CLUSTER, Q_LAST_PATH, Q_LAUNCHES,
                                        Q_PERSISTENT_VARIANT)

    ws, rank, local = _dist_env()
    dist = None
    if ws > 1:
        import torch.distributed as dist_mod
        dist = dist_mod
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local if ws > 1 else 0)
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream(dev)

    H, D, T, B = WL.H, WL.D, WL.T, WL.B
    C = WL.C()
    nz = nz_from_keep(KEEP, C)
    factors = synthetic_layer_factors(WL, 0, K_MAIN, KEEP)
    nz_h = float(np.mean([np.count_nonzero(f["idx"] >= D) / f["idx"].shape[0] for f in factors]))
    m = LSTMApprox(1, [D], H, K_MAIN, B, "fp32", stream=stream)
    m.set_layer(0, factors)
    x_host = workload_inputs(WL).astype(np.float32)
    x = torch.from_numpy(x_host).to(dev)
    out_h = torch.empty((T, B, H), device=dev)
    out_c = torch.empty((1, B, H), device=dev)
    ck_h = torch.empty((len(CKPTS), T, B, H), device=dev)
    ck_c = torch.empty((len(CKPTS), T, B, H), device=dev)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)

    def step(K=K_MAIN, cps=CKPTS):
        m.run(x, K, out_h, out_c=out_c, checkpoints=list(cps), ckpt_h=ck_h if cps else None,
              ckpt_c=ck_c if cps else None)

    def timed_loop(nsteps, fn):
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(nsteps)]
        for i in range(nsteps):
            flush.fill_(float(i))
            evs[i][0].record(stream)
            fn()
            evs[i][1].record(stream)
        torch.cuda.synchronize(dev)
        return [a.elapsed_time(b) for a, b in evs]

    for _ in range(args.warmup):
        step()
    m.sync()

    # ---- main timed region -------------------------------------------------
    if dist:
        dist.barrier()
    torch.cuda.synchronize(dev)
    launches0 = m.query(Q_LAUNCHES)
    with ClockSampler(torch.cuda.current_device()) as clk:
        step_ms = timed_loop(args.steps, step)
    m.sync()
    launches = m.query(Q_LAUNCHES) - launches0
    if dist:
        dist.barrier()
    torch.cuda.synchronize(dev)
    ms_mean = sum(step_ms) / len(step_ms)
    p50_ms = statistics.median(step_ms)
    path = m.query(Q_LAST_PATH)
    cluster = m.query(Q_CLUSTER)
    variant = m.query(Q_PERSISTENT_VARIANT)

    # ---- per-phase device times (CUDA events on the library's stream) ------
    m.set_option(OPT_TIMING, 1)
    ph = []
    for i in range(3 if args.quick else max(10, min(args.steps, 50))):
        flush.fill_(float(i))
        step()
        ph.append(m.phase_times())
    m.set_option(OPT_TIMING, 0)
    xproj_ms = statistics.mean(p[0] for p in ph)
    rec_ms = statistics.mean(p[1] for p in ph)

    # ---- K sweep (separate runs, no intermediate outputs) ------------------
    sweep = []
    for K in (() if args.quick else K_SWEEP):
        for _ in range(3):
            step(K, ())
        t = timed_loop(max(10, min(args.steps, 50)), lambda K=K: step(K, ()))
        med = statistics.median(t)
        sweep.append({"K": K, "value": T * B / (statistics.mean(t) / 1e3), "unit": UNIT,
                      "p50_us_per_timestep": 1e3 * med / T, "p90_us_per_timestep": 1e3 * p90(t) / T,
                      "effective_factor_gbs": algorithmic_bytes_per_timestep(H, C, nz, K) * T / (med / 1e3) / 1e9})

    # ---- large-batch tensor-core path (bf16 factors) -------------------------
    large = [] if (args.quick or args.no_large) else large_batch_sweep(dev, stream, peaks_bf16())
    paper_case = None if (args.quick or args.no_large) else paper_case_sweep(dev, stream)
    dense = None if args.quick else dense_comparator(dev, stream, x)
    dense_kernel = None if args.quick else dense_kernel_comparator(dev, stream, flush, x, statistics.median(step_ms))
    k_sweeps = [] if (args.quick or args.no_large) else workload_k_sweeps(dev, flush)
    tau_layouts = [] if (args.quick or args.no_large) else tau_layout_comparison(dev, stream)
    tensor_launches = [] if (args.quick or args.no_large) else tensor_launch_comparison(dev, stream, flush)

    # ---- end to end through the host-buffer entry point ---------------------
    xh = torch.from_numpy(x_host).pin_memory()
    oh = torch.empty((T, B, H), dtype=torch.float32).pin_memory()
    kh = torch.empty((len(CKPTS), T, B, H), dtype=torch.float32).pin_memory()
    xh_np, oh_np, kh_np = xh.numpy(), oh.numpy(), kh.numpy()
    for _ in range(3):
        m.run_host(xh_np, K_MAIN, oh_np, checkpoints=list(CKPTS), ckpt_h=kh_np)
    e2e_t = []
    for i in range(2 if args.quick else args.steps):
        flush.fill_(float(i))
        torch.cuda.synchronize(dev)
        t0 = time.perf_counter()
        m.run_host(xh_np, K_MAIN, oh_np, checkpoints=list(CKPTS), ckpt_h=kh_np)
        e2e_t.append(time.perf_counter() - t0)
    e2e_ms = 1e3 * sum(e2e_t) / len(e2e_t)

    # ---- aggregate over ranks ----------------------------------------------
    (value, e2e_value), (ms_max, e2e_max) = combine_ranks([ms_mean, e2e_ms], T * B, dist, dev)

    if rank == 0:
        peaks = {}
        try:
            peaks = json.load(open(os.path.join(HERE, "MEASURED_PEAKS.json")))
        except (OSError, ValueError):
            pass
        hbm_peak = peaks.get("hbm_gbs")
        peak_note = "measured (MEASURED_PEAKS.json hbm_gbs)" if hbm_peak else "fallback 6800 GB/s"
        hbm_peak = hbm_peak or 6800.0
        rec_bytes = recurrence_bytes_per_timestep(H, nz_h, K_MAIN) * T
        achieved = rec_bytes / (rec_ms / 1e3) / 1e9
        path_bytes = algorithmic_bytes_per_timestep(H, C, nz, K_MAIN) * T
        clocks = clk.summary()
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_max, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic", "config": _config(ws),
            "p50_us_per_timestep": 1e3 * p50_ms / T, "p90_us_per_timestep": 1e3 * p90(step_ms) / T,
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": int(x_host.nbytes),
                    "d2h_bytes_per_step": int(oh.numel() * 4 + kh.numel() * 4)},
            "roofline": {"kernel": "persistent recurrence kernel", "bound": "hbm", "achieved": achieved,
                         "peak": hbm_peak, "peak_source": peak_note, "unit": "GB/s", "frac": achieved / hbm_peak,
                         "traffic": captured_traffic() if (path == 2 and variant == 1) else None,
                         "algorithmic_bytes_per_launch": rec_bytes, "launch_ms": rec_ms},
            "path_effective_gbs": path_bytes / (ms_max / 1e3) / 1e9,
            "phase_ms": {"input_projection": xproj_ms, "recurrence": rec_ms},
            "recurrence_path": {1: "simt", 2: "persistent", 3: "tensor"}.get(path, str(path)),
            "cluster_ctas": cluster, "persistent_kernel": {1: "per-unit-block", 2: "one-exchange"}.get(variant),
            "gpu_launches": launches, "sweep": sweep, "clocks": clocks,
            "large_batch": large,
            "k_sweeps": k_sweeps,
            "tau_layouts": tau_layouts,
            "tensor_launches": tensor_launches,
            "paper_case_study": paper_case,
            "dense_lstm_comparator": dense,
            "dense_kernel_comparator": dense_kernel,
        }
        if ws == 1 and not (args.no_cpu_baseline or args.quick):
            line["cpu_baseline"] = cpu_baseline()
        print(json.dumps(line), flush=True)
    if dist:
        dist.barrier()
        dist.destroy_process_group()


LARGE_BATCH = (("c3", 0.5, 512, ()), ("c4", 0.5, 512, ()), ("c4", 0.1, 128, ()),
               ("c5", 0.3, 1024, (16, 64, 256, 1024)))


# throughput against K on the other workloads: (workload, dtype, keep, K values);
# one model per row holds the largest K, and each smaller K runs its prefix
K_SWEEPS = (("c1", "fp32", 0.5, (1, 4, 16, 64)),
            ("c3", "bf16", 0.5, (32, 128, 512)),
            ("c4", "bf16", 0.5, (8, 32, 128, 512)),
            ("c4", "bf16", 0.1, (8, 32, 128, 512)))


def workload_k_sweeps(dev, flush):
    """Timesteps·streams/s and p50 per-timestep latency against K for each
    row of K_SWEEPS (no intermediate outputs, L2 flushed before every run),
    eager and replayed as a CUDA graph.  Runs on a stream of its own (the
    default stream cannot be captured)."""
    import torch
    from paper_1905_00689_gb300 import LSTMApprox, Q_LAST_PATH
    torch.cuda.synchronize(dev)  # the flush buffer was last written on another stream
    stream = torch.cuda.Stream(dev)
    out = []
    with torch.cuda.stream(stream):
        for name, dtype, keep, Ks in K_SWEEPS:
            out.append(_k_sweep_row(dev, stream, flush, WORKLOADS[name], dtype, keep, Ks, LSTMApprox, Q_LAST_PATH))
            torch.cuda.empty_cache()
    torch.cuda.synchronize(dev)
    return out


def _k_sweep_row(dev, stream, flush, w, dtype, keep, Ks, LSTMApprox, Q_LAST_PATH):
    import torch
    km = max(Ks)
    m = LSTMApprox(w.L, [w.D] + [w.H] * (w.L - 1), w.H, km, w.B, dtype, stream=stream)
    for l in range(w.L):
        m.set_layer(l, synthetic_layer_factors(w, l, km, keep))
    x = torch.from_numpy(workload_inputs(w).astype(np.float32)).to(dev)
    oh = torch.empty((w.T, w.B, w.H), device=dev)
    row = {"workload": w.name, "dtype": dtype, "keep": keep, "points": []}
    n = 50 if w.B == 1 else 10

    def timed(fn):
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
        for i, (a, b) in enumerate(evs):
            flush.fill_(float(i))
            a.record(stream)
            fn()
            b.record(stream)
        torch.cuda.synchronize(dev)
        return [a.elapsed_time(b) for a, b in evs]

    for K in Ks:
        for _ in range(3):
            m.run(x, K, oh)
        t = timed(lambda: m.run(x, K, oh))
        path = m.query(Q_LAST_PATH)
        # the same call captured once as a CUDA graph: the device time of its
        # launches without the host's enqueue between them
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            m.run(x, K, oh)
        g.replay()
        tg = timed(g.replay)
        del g
        row["points"].append({
            "K": K, "value": w.T * w.B / (statistics.mean(t) / 1e3), "unit": UNIT,
            "p50_us_per_timestep": 1e3 * statistics.median(t) / w.T,
            "p50_us_per_timestep_graph": 1e3 * statistics.median(tg) / w.T,
            "path": {1: "simt", 2: "persistent", 3: "tensor"}.get(path)})
    return row


def peaks_bf16():
    try:
        pk = json.load(open(os.path.join(HERE, "MEASURED_PEAKS.json")))
        return float(pk["bf16_tflops"]), "measured (MEASURED_PEAKS.json bf16_tflops)"
    except (OSError, ValueError, KeyError):
        return 1900.0, "fallback 1900 TFLOP/s"


def large_batch_sweep(dev, stream, peak):
    """The bf16 workloads on the tensor-core path: throughput, and the hoisted
    input projection (the large dense contraction) against the bf16 peak."""
    import torch
    from paper_1905_00689_gb300 import LSTMApprox, OPT_TIMING, Q_LAST_PATH
    peak_tf, peak_src = peak
    out = []
    for name, keep, K, cps in LARGE_BATCH:
        w = WORKLOADS[name]
        m = LSTMApprox(w.L, [w.D] + [w.H] * (w.L - 1), w.H, K, w.B, "bf16", stream=stream)
        for l in range(w.L):
            m.set_layer(l, synthetic_layer_factors(w, l, K, keep))
        x = torch.from_numpy(workload_inputs(w).astype(np.float32)).to(dev)
        oh = torch.empty((w.T, w.B, w.H), device=dev)
        ck = torch.empty((max(1, len(cps)), w.T, w.B, w.H), device=dev)
        run = lambda: m.run(x, K, oh, checkpoints=list(cps), ckpt_h=ck if cps else None)
        for _ in range(3):
            run()
        m.sync()
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(10)]
        for a, b in evs:
            a.record(stream)
            run()
            b.record(stream)
        torch.cuda.synchronize(dev)
        ms = statistics.median(a.elapsed_time(b) for a, b in evs)
        m.set_option(OPT_TIMING, 1)
        ph = []
        for _ in range(5):
            run()
            ph.append(m.phase_times())
        m.set_option(OPT_TIMING, 0)
        xp_ms = statistics.median(p[0] for p in ph)
        # MMA work as issued: masked-dense products, each activation operand
        # as its bf16 pair (two MMAs per factor tile)
        exec_fl = sum(2 * w.T * w.B * (2 * 4 * K * w.C(l) + 2 * 4 * K * w.H) for l in range(w.L))
        # the method's own operations (Sec. III): 4 gates x K (2R + 2NZ + 1) per stream-step
        alg_fl = sum(w.T * w.B * 4 * K * (2 * w.H + 2 * nz_from_keep(keep, w.C(l)) + 1) for l in range(w.L))
        xp_fl = sum(2 * w.T * w.B * 2 * 4 * K * w.input_dim(l) for l in range(w.L))
        xp_tf = xp_fl / (xp_ms / 1e3) / 1e12
        out.append({
            "workload": w.name, "keep": keep, "K": K, "checkpoints": list(cps),
            "path": {1: "simt", 2: "persistent", 3: "tensor"}.get(m.query(Q_LAST_PATH)),
            "ms_per_run": ms, "value": w.T * w.B / (ms / 1e3), "unit": UNIT,
            "executed_tflops": exec_fl / (ms / 1e3) / 1e12,
            "executed_frac": exec_fl / (ms / 1e3) / 1e12 / peak_tf,
            "algorithmic_tflops": alg_fl / (ms / 1e3) / 1e12,
            "input_projection": {"ms": xp_ms, "tflops": xp_tf, "peak": peak_tf, "frac": xp_tf / peak_tf,
                                 "peak_source": peak_src},
            "recurrence_ms": statistics.median(p[1] for p in ph),
        })
        del m, x, oh, ck
        torch.cuda.empty_cache()
    return out


def dense_comparator(dev, stream, x, steps: int = 200) -> dict:
    """A dense fp32 LSTM layer of the benchmark shape (torch.nn.LSTM, the
    library cuDNN/cuBLAS step) on the same input: the analogue of the paper's
    dense baselines, for the speed-up of the approximation.  Not part of the
    timed path."""
    import torch
    T, B, D = x.shape
    lstm = torch.nn.LSTM(D, WL.H).to(dev).float()
    with torch.no_grad(), torch.cuda.stream(stream):
        for _ in range(10):
            lstm(x)
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
        for a, b in evs:
            a.record(stream)
            lstm(x)
            b.record(stream)
    torch.cuda.synchronize(dev)
    ms = statistics.median(a.elapsed_time(b) for a, b in evs)
    return {"kind": "dense torch.nn.LSTM (cuDNN), fp32, same D/H/T/B, warm caches", "ms_per_run": ms,
            "value": T * B / (ms / 1e3), "unit": UNIT,
            "dense_weight_bytes": 4 * 4 * WL.H * (D + WL.H)}


def tensor_launch_comparison(dev, stream, flush) -> list:
    """The tensor path at the workloads' small depths as one launch per tile
    of streams for all timesteps (the default where the layer fits) against
    two launches per timestep (LSTM_APPROX_OPT_TENSOR_SEQ = 1): whole-run
    timesteps·streams/s and µs per timestep (CUDA events on the library's
    stream, L2 flushed before each run, median of 10)."""
    import torch
    from paper_1905_00689_gb300 import LSTMApprox, OPT_TENSOR_SEQ, Q_TENSOR_SEQ
    out = []
    for name, keep, Ks in (("c3", 0.5, (32,)), ("c4", 0.5, (8, 32)), ("c4", 0.1, (8, 32))):
        w = WORKLOADS[name]
        m = LSTMApprox(1, [w.D], w.H, max(Ks), w.B, "bf16", stream=stream)
        m.set_layer(0, synthetic_layer_factors(w, 0, max(Ks), keep))
        x = torch.from_numpy(workload_inputs(w).astype(np.float32)).to(dev)
        oh = torch.empty((w.T, w.B, w.H), device=dev)
        for K in Ks:
            row = {"workload": w.name, "keep": keep, "K": K}
            for seq, key in ((0, "one_launch"), (1, "per_timestep")):
                m.set_option(OPT_TENSOR_SEQ, seq)
                for _ in range(3):
                    m.run(x, K, oh)
                evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                       for _ in range(10)]
                torch.cuda.synchronize(dev)
                with torch.cuda.stream(stream):  # the flush on the timed stream, outside the events
                    for i, (a, b) in enumerate(evs):
                        flush.fill_(float(i))
                        a.record(stream)
                        m.run(x, K, oh)
                        b.record(stream)
                torch.cuda.synchronize(dev)
                ms = statistics.median(a.elapsed_time(b) for a, b in evs)
                row[key] = {"value": w.T * w.B / (ms / 1e3), "unit": UNIT, "us_per_timestep": 1e3 * ms / w.T,
                            "one_launch_taken": bool(m.query(Q_TENSOR_SEQ))}
            out.append(row)
        m.set_option(OPT_TENSOR_SEQ, 0)
        m.close()
        del x, oh
        torch.cuda.empty_cache()
    return out


def tau_layout_comparison(dev, stream) -> list:
    """The tensor path's recurrent projection with masked-dense v rows on the
    tensor cores against v's kept entries (compressed rows) on the CUDA cores
    (LSTM_APPROX_OPT_TAU_LAYOUT), D=2048 H=1024 T=64 B=1024 at both keep
    levels: recurrence milliseconds per run (CUDA events on the library's
    stream, median of 5) and per timestep."""
    import torch
    from paper_1905_00689_gb300 import LSTMApprox, OPT_TAU_LAYOUT, OPT_TIMING
    w = WORKLOADS["c4"]
    x = torch.from_numpy(workload_inputs(w).astype(np.float32)).to(dev)
    oh = torch.empty((w.T, w.B, w.H), device=dev)
    out = []
    for keep in (0.1, 0.5):
        m = LSTMApprox(1, [w.D], w.H, 512, w.B, "bf16", stream=stream)
        m.set_layer(0, synthetic_layer_factors(w, 0, 512, keep))
        for K in (128, 512):
            row = {"workload": w.name, "keep": keep, "K": K}
            for layout, name in ((0, "masked_dense_tensor"), (1, "compressed_cuda_cores")):
                m.set_option(OPT_TAU_LAYOUT, layout)
                for _ in range(2):
                    m.run(x, K, oh)
                m.set_option(OPT_TIMING, 1)
                rec = []
                for _ in range(5):
                    m.run(x, K, oh)
                    rec.append(m.phase_times()[1])
                m.set_option(OPT_TIMING, 0)
                ms = statistics.median(rec)
                row[name] = {"recurrence_ms": ms, "us_per_timestep": 1e3 * ms / w.T}
            row["faster"] = min(("masked_dense_tensor", "compressed_cuda_cores"),
                                key=lambda k: row[k]["recurrence_ms"])
            out.append(row)
        m.set_option(OPT_TAU_LAYOUT, 0)
        m.close()
        torch.cuda.empty_cache()
    return out


def dense_kernel_comparator(dev, stream, flush, x, approx_ms: float) -> list:
    """The library's dense LSTM kernel (lstm_approx_dense_run: the full gate
    matrices of Sec. II on the same persistent cluster design) timed like the
    approximate path: on the benchmark shape with the L2 flushed before every
    run (as the main timed loop), and on the paper's case-study shape
    (H = 64, C = 8320, one timestep) with warm caches (as paper_case_sweep):
    the like-for-like baseline of the approximation's speed-up (Sec. VI-B)."""
    import torch
    from paper_1905_00689_gb300 import dense_run, dense_workspace_bytes
    from workloads import draw_weight
    out = []
    f1 = WORKLOADS["f1"]
    for w, xin, ref_ms, flushed in ((WL, x, approx_ms, True), (f1, None, None, False)):
        D, H, T, B = w.D, w.H, w.T, w.B
        W = [draw_weight(H, D + H, 77 + g) for g in range(4)]
        Wx = torch.from_numpy(np.concatenate([m[:, :D] for m in W]).astype(np.float32)).to(dev)
        Wh = torch.from_numpy(np.concatenate([m[:, D:] for m in W]).astype(np.float32)).to(dev)
        xx = xin if xin is not None else torch.from_numpy(workload_inputs(w).astype(np.float32)).to(dev)
        oh = torch.empty((T, B, H), device=dev)
        ws = torch.empty(dense_workspace_bytes(H, T, B), dtype=torch.uint8, device=dev)
        run = lambda: dense_run(Wx, Wh, None, xx, oh, workspace=ws, stream=stream)
        for _ in range(5):
            run()
        n = 100
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
        for i, (a, b) in enumerate(evs):
            if flushed:
                flush.fill_(float(i))
            a.record(stream)
            run()
            b.record(stream)
        torch.cuda.synchronize(dev)
        ms = statistics.median(a.elapsed_time(b) for a, b in evs)
        row = {"workload": w.name, "kind": "dense LSTM kernel of this library (lstm_approx_dense_run), fp32, " +
                                          ("L2 flushed before each run" if flushed else "warm caches"),
               "ms_per_run": ms,
               "value": T * B / (ms / 1e3), "unit": UNIT, "dense_weight_bytes": 4 * 4 * H * (D + H)}
        if ref_ms is not None:
            row["approx_speedup"] = ms / ref_ms
        out.append(row)
    return out


# the paper's FPGA latencies for one timestep of its case-study LSTM (Table I),
# by kept entries per v; context only (another machine, K chosen by the paper)
PAPER_FPGA_MS = {4160: 0.36190, 130: 0.03924, 32: 0.00072}


def paper_case_sweep(dev, stream):
    """The paper's case-study shape (H=64, C=8320, one timestep, one stream,
    fp32): device time of one whole call (projection + recurrence) per K and
    NZ, warm caches.  Calls this short are bound by the host's launch path, so
    each call is also captured once as a CUDA graph and replayed: the graph
    time is the device time of the call's kernels alone."""
    import torch
    from paper_1905_00689_gb300 import LSTMApprox, Q_LAST_PATH
    w = WORKLOADS["f1"]
    cs = torch.cuda.Stream(dev)
    x = torch.from_numpy(workload_inputs(w).astype(np.float32)).to(dev)
    oh = torch.empty((w.T, w.B, w.H), device=dev)
    out = []

    def timed(fn, n):
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
        with torch.cuda.stream(cs):
            for a, b in evs:
                a.record(cs)
                fn()
                b.record(cs)
        torch.cuda.synchronize(dev)
        return 1e3 * statistics.median(a.elapsed_time(b) for a, b in evs)

    for keep in w.keeps:
        nz = nz_from_keep(keep, w.C())
        m = LSTMApprox(1, [w.D], w.H, max(w.Ks), w.B, "fp32", stream=cs)
        m.set_layer(0, synthetic_layer_factors(w, 0, max(w.Ks), keep))
        for K in w.Ks:
            call = lambda K=K: m.run(x, K, oh)
            for _ in range(10):
                call()
            m.sync()
            us_call = timed(call, 200)
            us_graph = None
            try:
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=cs):
                    call()
                g.replay()
                torch.cuda.synchronize(dev)
                us_graph = timed(g.replay, 200)
            except RuntimeError:
                pass
            out.append({"NZ": nz, "K": K, "us_per_timestep": us_call, "us_per_timestep_graph": us_graph,
                        "path": {1: "simt", 2: "persistent", 3: "tensor"}.get(m.query(Q_LAST_PATH)),
                        "paper_fpga_us_any_K": 1e3 * PAPER_FPGA_MS[nz]})
        m.sync()
        del m
    return {"workload": w.name, "dtype": "f32", "T": w.T, "B": w.B, "points": out,
            "note": "paper figure: Xilinx ZC706 FPGA at 100 MHz, K chosen per KL bound (Table I); context only"}


def run_profile(args):
    """Run one workload's path `--steps` times and print a short JSON line.

    Used as the target of ncu captures: c1/c2 take the fp32 persistent path,
    c3/c4/c5 the bf16 tensor-core path, at their largest listed K.
    """
    import torch
    from paper_1905_00689_gb300 import LSTMApprox, Q_LAST_PATH
    w = WORKLOADS[args.profile]
    if args.profile_dense:  # the dense comparator kernel on this workload's shape (fp32, one layer)
        from paper_1905_00689_gb300 import dense_run, dense_set_launch_order
        dense_set_launch_order(1)  # a profiler runs kernels one at a time: projection first
        from workloads import draw_weight
        dev = torch.device("cuda", 0)
        W = [draw_weight(w.H, w.D + w.H, 77 + g) for g in range(4)]
        Wx = torch.from_numpy(np.concatenate([m[:, :w.D] for m in W]).astype(np.float32)).to(dev)
        Wh = torch.from_numpy(np.concatenate([m[:, w.D:] for m in W]).astype(np.float32)).to(dev)
        x = torch.from_numpy(workload_inputs(w).astype(np.float32)).to(dev)
        oh = torch.empty((w.T, w.B, w.H), device=dev)
        for _ in range(args.warmup + args.steps):
            dense_run(Wx, Wh, None, x, oh)
        print(json.dumps({"profile": w.name, "dense": True, "runs": args.warmup + args.steps}), flush=True)
        return
    keep = w.keeps[0]
    K = max(w.Ks)
    cps = list(w.checkpoints)
    if w.name == WL.name:  # the configuration of the main timed loop
        keep, K, cps = KEEP, K_MAIN, list(CKPTS)
    if args.profile_k:
        K = args.profile_k
        cps = [c for c in cps if c < K] + [K] if cps else []
    if args.profile_keep:
        keep = args.profile_keep
    dev = torch.device("cuda", 0)
    m = LSTMApprox(w.L, [w.D] + [w.H] * (w.L - 1), w.H, K, w.B, w.dtype)
    for l in range(w.L):
        m.set_layer(l, synthetic_layer_factors(w, l, K, keep))
    # a profiler runs kernels one at a time: the projection first, the
    # recurrence after it (the default order needs them to overlap)
    from paper_1905_00689_gb300 import OPT_LAUNCH_ORDER
    m.set_option(OPT_LAUNCH_ORDER, 1)
    if args.profile_tau_compressed:
        from paper_1905_00689_gb300 import OPT_TAU_LAYOUT
        m.set_option(OPT_TAU_LAYOUT, 1)
    x = torch.from_numpy(workload_inputs(w).astype(np.float32)).to(dev)
    oh = torch.empty((w.T, w.B, w.H), device=dev)
    ck = torch.empty((max(1, len(cps)), w.T, w.B, w.H), device=dev)
    for _ in range(args.warmup + args.steps):
        m.run(x, K, oh, checkpoints=cps, ckpt_h=ck if cps else None)
    m.sync()
    print(json.dumps({"profile": w.name, "K": K, "keep": keep, "checkpoints": cps, "runs": args.warmup + args.steps,
                      "path": m.query(Q_LAST_PATH)}), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--all-configs", action="store_true",
                    help="with --impl reference: first time the oracle on every workload (a few seconds each)")
    ap.add_argument("--no-large", action="store_true", help="skip the large-batch tensor-core measurements")
    ap.add_argument("--profile", choices=sorted(WORKLOADS), default=None,
                    help="only run one workload's path (warmup + steps runs), for profilers")
    ap.add_argument("--profile-k", type=int, default=0, help="with --profile: this K instead of the workload's largest")
    ap.add_argument("--profile-keep", type=float, default=0.0, help="with --profile: this keep fraction")
    ap.add_argument("--profile-tau-compressed", action="store_true",
                    help="with --profile (bf16 workloads): the compressed layout of v's h part for tau'")
    ap.add_argument("--profile-dense", action="store_true",
                    help="with --profile: the dense comparator kernel on the workload's shape (fp32, one layer)")
    ap.add_argument("--quick", action="store_true",
                    help="main timed loop only (short side measurements, no K sweep, no CPU baseline)")
    args = ap.parse_args()
    if args.warmup < 3 and not args.profile:
        ap.error("--warmup must be >= 3")
    if args.profile:
        run_profile(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
