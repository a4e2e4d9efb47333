#!/usr/bin/env python3
"""Benchmark of the DBW parameter-server iteration on GB300 (one JSON line).

A step is one whole DBW iteration of the largest workload (MLP
4096-4096-4096-4096-1000, n = 256 workers x B = 32, bf16 GEMMs with fp32
accumulation and fp32 master weights, Pareto(2) round-trip times, b chosen by
the estimator every iteration): choose b -> worker gradients (G is [256, 54.4M]
fp32, 55.75 GB) -> selection -> fused aggregation + SGD + statistics ->
estimator bookkeeping.  The working set (G alone) is far larger than L2, so no
L2 flush is needed between steps.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl dbw|reference] [--no-extras]

--gpus N > 1 runs under torchrun: every rank simulates its own independent PS
(replicas; the method has no cross-GPU data path), value = all ranks' iterations
/ the slowest rank's time.  At N = 1 the same line also carries the other
workloads (``configs``: whole iterations of the smaller models, points of the
aggregation-only sweep, the push-and-wait fit) and the CPU oracle's time on a
bounded sample.  --impl reference times the fp64 CPU oracle on a bounded sample
of the same workload (rank 0 only).

Single pieces, for profiling (one JSON line per case, CUDA-event times after
warm-up; no clocks, oracle or extras):

    python bench.py --case aggregate --n 64 --d 4000000 --b 16 [--reps 5] [--all-row-norms]
    python bench.py --case sweep                  # the aggregation-only sweep
    python bench.py --case grads --workload mlp4096x3-1000_n256_B32
    python bench.py --case received --workload mlp4096x3-1000_n256_B32 --b 64
    python bench.py --case psw --n 256 --iters 60  # push-and-wait clock + Eq. (17) fit
    python bench.py --case iterate --workload mlp784-256-10_n64_B64 [--received] [--graph]
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

os.environ.setdefault("OPENBLAS_NUM_THREADS", str(os.cpu_count() or 1))

import numpy as np  # noqa: E402

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2004_14696_gb300 import inputs, workloads  # noqa: E402

METRIC = "simulated PS iterations/sec at n workers"
UNIT = "iter/s"

# dram bytes (read + write) of one full-size aggregation launch from an ncu capture
# (n = 256, d = 54,440,936, k = 142: 31.1411 GB read + 0.1717 GB written against
# 31.3580 GB algorithmic), as a ratio to the algorithmic bytes so that it scales to the
# bench's launches (traffic grows with k d); reported as null once aggregate.cu
# differs from the source the counters were taken on.
AGG_TRAFFIC = {"ratio_to_algorithmic": (31.141070 + 0.171713) / 31.357979,
               "source_sha256": "1d5f6bb0b751a7ad2fae28b88999146db77319f34bc6ba9bcc4d5be0abfcec09",
               "case": "n=256 d=54440936 k=142"}
# dram bytes (read + write) of the per-worker weight-gradient launches of one
# full-size pass (ncu on mlp4096x3-1000_n256_B32): 4.2158 + 17.2505 + 17.2508 +
# 17.2520 GB against 4.2778 + 3 x 17.3141 GB algorithmic; keyed to the dW kernel's
# own source (dw_source_sha).
DW_TRAFFIC = {"ratio_to_algorithmic": (4.2158 + 17.2505 + 17.2508 + 17.2520) / (4.2778 + 3 * 17.3141),
              "source_sha256": "bafb8a813d2b51c8c7e1921e5fa40487cfd5f74fde82f3e96748fb7521c6d77b",
              "case": "mlp4096x3-1000_n256_B32, one pass"}

CASES = ("aggregate", "sweep", "grads", "received", "psw", "iterate")


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=100)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", default="dbw", choices=["dbw", "reference"])
    p.add_argument("--workload", default=workloads.MLP4096.key, choices=list(workloads.ALL))
    p.add_argument("--no-extras", action="store_true", help="only the headline workload (no configs / oracle)")
    # single pieces
    p.add_argument("--case", choices=CASES)
    p.add_argument("--n", type=int, default=64)
    p.add_argument("--tol", type=float, default=1e-4, help="--case psw: stopping tolerance of the Eq. (17) fit")
    p.add_argument("--d", type=int, default=4_000_000)
    p.add_argument("--b", type=int, default=16)
    p.add_argument("--reps", type=int, default=5)
    p.add_argument("--all-row-norms", action="store_true")
    p.add_argument("--iters", type=int, default=60)
    p.add_argument("--received", action="store_true")
    p.add_argument("--graph", action="store_true")
    p.add_argument("--max-bytes", type=float, default=float(workloads.AGG_MAX_BYTES))
    return p.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            j = json.load(f)
        return {"hbm_gbs": j["hbm_gbs"], "bf16_tflops": j["bf16_tflops"],
                "bf16_tflops_sustained": j.get("bf16_tflops_sustained"), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


def bench_config(wl, world):
    """The workload a step runs, identical in both arms (no measured values in it)."""
    return {"workload": wl.key, "widths": list(wl.widths), "n_workers": wl.n, "batch_per_worker": wl.B,
            "d": wl.d, "G_bytes": wl.n * wl.ld * 4, "time_model": wl.time_model, "policy": wl.policy,
            "l2": "working set > L2 (G is %.1f GB), no flush" % (wl.n * wl.ld * 4 / 1e9),
            "parallelism": "replicas" if world > 1 else "single"}


class ClockSampler:
    """nvidia-smi clock / throttle samples while the timed region runs."""
    Q = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self.window = None       # (start, end) wall-clock seconds of the timed region

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except (FileNotFoundError, OSError):
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def mark(self, start, end):
        self.window = (start, end)

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        """Median SM clock and throttle reasons of the samples taken during the timed
        window (a sample's arrival time is within 100 ms of the window); if the window
        is shorter than the sampling period, the samples nearest to it."""
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        parsed = []
        for (arrival, line) in self.lines:
            f = [x.strip() for x in line.split(",")]
            if len(f) < 10:
                continue
            try:
                parsed.append((arrival, float(f[2]), float(f[3]), f[6:10]))
            except ValueError:
                continue
        if not parsed:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        chosen = parsed
        where = "whole run"
        if self.window:
            a, b = self.window
            inside = [p for p in parsed if a - 0.1 <= p[0] <= b + 0.1]
            if inside:
                chosen, where = inside, "timed region"
            else:
                mid = 0.5 * (a + b)
                chosen, where = sorted(parsed, key=lambda p: abs(p[0] - mid))[:2], "nearest to timed region"
        reasons = set()
        for p in chosen:
            for name, v in zip(names, p[3]):
                if v.lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(p[1] for p in chosen), "sm_max_mhz": chosen[-1][2],
                "reasons": sorted(reasons), "samples": len(chosen), "window": where}


def combine_over_ranks(values, world, device):
    """Max over ranks of each per-rank timing: the slowest rank sets the job's time."""
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    if world > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return t.tolist()


def job_value(world, steps, max_elapsed_ms):
    """Whole-job throughput: every rank ran ``steps`` independent iterations."""
    return world * steps / (max_elapsed_ms * 1e-3)


def sha256_of(path):
    with open(path, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()


DW_REGION = ("// ------------------------------------------------------------------ persistent dW kernel",
             "// ------------------------------------------------------------------ host side")


def dw_source_sha():
    """sha256 of the per-worker dW kernel's own source (its region of gemm_tc.cu and the
    PTX helpers it is built from), so that edits to other kernels of the file keep its
    traffic record."""
    csrc = os.path.join(ROOT, "paper_2004_14696_gb300", "csrc")
    with open(os.path.join(csrc, "gemm_tc.cu")) as f:
        text = f.read()
    a, b = text.find(DW_REGION[0]), text.find(DW_REGION[1])
    if a < 0 or b < a:
        return None
    with open(os.path.join(csrc, "tc_ptx.cuh")) as f:
        helpers = f.read()
    return hashlib.sha256((text[a:b] + helpers).encode()).hexdigest()


def layer_flops(widths, rows, forward=True, dX=True, dW=False, gbar=False):
    """GEMM flops of one pass over ``rows`` samples: forward 2 rows in out per layer, input
    gradient for every layer but the first, weight gradient (per worker or mean) per layer."""
    f = 0
    for l in range(len(widths) - 1):
        mac = rows * widths[l] * widths[l + 1]
        f += 2 * mac * ((1 if forward else 0) + (1 if (dX and l > 0) else 0) + (1 if dW else 0) +
                        (1 if gbar else 0))
    return f


# ====================================================================== DBW arm
def run_dbw(args, rank, world, local_rank):
    # nvidia-smi takes a moment to start: the sampler runs for the whole arm, and only
    # the samples that arrive during the timed region are used
    with ClockSampler(local_rank) as clk:
        return _run_dbw(args, rank, world, local_rank, clk)


def _run_dbw(args, rank, world, local_rank, clk):
    import torch
    import torch.distributed as dist

    import __graft_entry__
    from paper_2004_14696_gb300 import dbw
    from paper_2004_14696_gb300.pipeline import Iteration

    if rank == 0 or world == 1:
        __graft_entry__.build()
    if world > 1:
        dist.barrier()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    wl = workloads.ALL[args.workload]
    K, W = args.steps, args.warmup
    if W < 3:
        raise SystemExit("--warmup must be >= 3")
    config = bench_config(wl, world)
    # each rank simulates an independent PS with its own seed
    if rank:
        from dataclasses import replace
        wl = replace(wl, seed_offset=wl.seed_offset + 1000 * rank)
    it = Iteration(wl, device=dev)
    w_init = it.w.clone()
    n, B = wl.n, wl.B
    total = W + K
    idx_h = np.stack([inputs.minibatch_indices(wl.seed, t, n, B, wl.S) for t in range(total)])
    tim_h = np.stack([inputs.completion_times(wl.seed, t, n, wl.time_model, **wl.time_params) for t in range(total)])
    idx_d = torch.from_numpy(idx_h).to(dev)
    tim_d = torch.from_numpy(tim_h).to(dev)
    stream = torch.cuda.current_stream(dev)
    ks = torch.zeros(total, dtype=torch.int32, device=dev)
    names = ["choose_b", "worker_grads", "select", "aggregate", "grad_stats"]
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(len(names) + 1)] for _ in range(total)]

    def one(t, timed):
        e = ev[t]
        wlx = it.wl
        if timed:
            e[0].record(stream)
        if it.static_b is None:
            dbw.dbw_choose_b(it.state, wlx.lr, wlx.beta, it.b, it.ratio, 0, stream)
        if timed:
            e[1].record(stream)
        dbw.dbw_worker_grads(wlx.widths, wlx.prec, it.w, it.pool, it.labels, idx_d[t], n, B, it.G, it.loss, it.ws,
                             stream)
        if timed:
            e[2].record(stream)
        dbw.dbw_select_fastest(tim_d[t], it.b, it.order, it.mask, it.tsorted, it.k, stream)
        if timed:
            e[3].record(stream)
        dbw.dbw_aggregate_update(it.G, n, it.d, it.mask, wlx.lr, it.w, it.partials, None, stream)
        if timed:
            e[4].record(stream)
        dbw.dbw_grad_stats(it.partials, n, it.mask, it.loss, it.tsorted, wlx.lr, it.state, it.stats,
                           it.row_sqnorm, stream)
        if timed:
            e[5].record(stream)
        ks[t:t + 1].copy_(it.k)

    for t in range(W):
        one(t, False)
    torch.cuda.synchronize(dev)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    dbw.dbw_profile_dw(True)
    dbw.dbw_profile_gemm(True)
    wall0 = time.time()
    t_start.record(stream)
    for t in range(W, total):
        one(t, True)
    t_end.record(stream)
    torch.cuda.synchronize(dev)
    clk.mark(wall0, time.time())
    time.sleep(0.15)                # let the sampler deliver the samples of the window
    dw_ms, dw_launches, dw_bytes = dbw.dbw_profile_dw_read()
    dbw.dbw_profile_dw(False)
    gm_ms, gm_launches = dbw.dbw_profile_gemm_read()
    dbw.dbw_profile_gemm(False)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    elapsed_ms = t_start.elapsed_time(t_end)
    phase_ms = {nm: sum(ev[t][i].elapsed_time(ev[t][i + 1]) for t in range(W, total)) / K
                for i, nm in enumerate(names)}
    kvals = ks[W:].cpu().numpy().astype(np.int64)
    status = int(it.ws[:4].view(torch.int32).item())

    # ---------------------------------------------------------------- e2e
    # the same steps through the public API with host buffers: per step, pinned
    # host -> device copies of the minibatch indices and times, the iteration,
    # and a device -> host read of the step's statistics (loss, k, V, ...).
    # the e2e leg replays the very same iterations: parameters and estimator state restart
    it.w.copy_(w_init)
    dbw.dbw_state_init(it.state, n, wl.D, stream)
    idx_pin = torch.from_numpy(idx_h).pin_memory()
    tim_pin = torch.from_numpy(tim_h).pin_memory()
    stats_pin = torch.empty(dbw.STATS_LEN, dtype=torch.float64).pin_memory()

    def one_e2e(t):
        it.idx.copy_(idx_pin[t], non_blocking=True)
        it.times.copy_(tim_pin[t], non_blocking=True)
        it.step(stream=stream)
        stats_pin.copy_(it.stats, non_blocking=True)
        stream.synchronize()
        return float(stats_pin[dbw.STAT_F])

    for t in range(W):
        one_e2e(t)
    torch.cuda.synchronize(dev)
    if world > 1:
        dist.barrier()
    t0 = time.perf_counter()
    for t in range(W, total):
        one_e2e(t)
    e2e_s = time.perf_counter() - t0
    if world > 1:
        dist.barrier()
    h2d = idx_h[0].nbytes + tim_h[0].nbytes
    d2h = stats_pin.numel() * 8
    launches = it.launches_per_step() * K
    d, ld = it.d, it.ld
    del it, idx_d, tim_d
    torch.cuda.empty_cache()

    # ---------------------------------------------------------------- received form
    rx = _time_received(wl, dev, idx_h, tim_h, W, K, stream, world)

    # ---------------------------------------------------------------- gather over ranks
    elapsed_ms, e2e_s = combine_over_ranks([elapsed_ms, e2e_s], world, dev)
    if rank != 0:
        return None
    pk = peaks()
    agg_bytes = float(np.mean((kvals * d + 2 * d) * 4.0))
    agg_ms = phase_ms["aggregate"]
    achieved = agg_bytes / (agg_ms * 1e-3) / 1e9
    traffic = None
    src = os.path.join(ROOT, "paper_2004_14696_gb300", "csrc", "aggregate.cu")
    if AGG_TRAFFIC["ratio_to_algorithmic"] is not None and AGG_TRAFFIC["source_sha256"] == sha256_of(src):
        traffic = AGG_TRAFFIC["ratio_to_algorithmic"] * agg_bytes
    # the dominant kernel (by share of the step): the per-worker weight gradient writing G
    dw = None
    if dw_launches:
        per_bytes, per_ms = dw_bytes / dw_launches, dw_ms / dw_launches
        dw_ach = per_bytes / (per_ms * 1e-3) / 1e9
        dw_traffic = (DW_TRAFFIC["ratio_to_algorithmic"] * per_bytes
                      if DW_TRAFFIC["source_sha256"] == dw_source_sha() else None)
        dw = {"kernel": "tc_dw_kernel (per-worker dW GEMM writing G, in dbw_worker_grads)", "bound": "hbm",
              "achieved": dw_ach, "peak": pk["hbm_gbs"], "unit": "GB/s", "frac": dw_ach / pk["hbm_gbs"],
              "traffic": dw_traffic, "algorithmic_bytes_per_launch": per_bytes, "ms_per_launch": per_ms,
              "launches_timed": dw_launches, "share_of_step": dw_ms / K / (elapsed_ms / K),
              "peak_source": pk["source"]}
    ms_step = elapsed_ms / K
    value = job_value(world, K, elapsed_ms)
    wd = wl.widths
    M = n * B
    gemm_flop = layer_flops(wd, M, dW=True)           # forward, input gradient, per-worker dW
    tc_flop = layer_flops(wd, M)                       # forward + input gradient (the pair kernel)
    # the forward and input-gradient GEMMs (persistent tcgen05 kernel), timed live; the
    # timed region lasts about a second, so the burst peak is the denominator
    tensor = None
    if gm_launches:
        tf = tc_flop * K / (gm_ms * 1e-3) / 1e12
        tensor = {"kernel": "tc_gemm_pair_kernel (forward + input-gradient GEMMs, in dbw_worker_grads)",
                  "bound": "tensor", "achieved": tf, "peak": pk["bf16_tflops"], "unit": "TFLOP/s",
                  "frac": tf / pk["bf16_tflops"], "traffic": None,
                  "frac_of_sustained": tf / pk["bf16_tflops_sustained"] if pk.get("bf16_tflops_sustained") else None,
                  "algorithmic_flop_per_step": tc_flop, "ms_per_step": gm_ms / K,
                  "launches_timed": gm_launches, "share_of_step": gm_ms / elapsed_ms,
                  "peak_kind": "bf16 dense, burst", "peak_source": pk["source"]}
    out = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K, "warmup": W,
        "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16+f32" if wl.prec == workloads.PREC_BF16 else "f32", "data": "synthetic",
        "config": config,
        "mean_k": float(kvals.mean()),
        "roofline": dw,
        "roofline_aggregate": {"kernel": "aggregate_kernel (dbw_aggregate_update)", "bound": "hbm",
                               "achieved": achieved, "peak": pk["hbm_gbs"], "unit": "GB/s",
                               "frac": achieved / pk["hbm_gbs"], "traffic": traffic,
                               "algorithmic_bytes_per_launch": agg_bytes, "peak_source": pk["source"]},
        "roofline_tensor": tensor,
        "phases_ms": phase_ms,
        "gemm": {"flop_per_step": gemm_flop, "worker_grads_tflops": gemm_flop / (phase_ms["worker_grads"] * 1e-3) / 1e12},
        "gpu_launches": launches,
        "device_status": status,
        "e2e": {"value": job_value(world, K, e2e_s * 1e3), "unit": UNIT, "h2d_bytes_per_step": int(h2d),
                "d2h_bytes_per_step": int(d2h)},
        "clocks": clk.summary(),
    }
    if rx is not None:
        kk = rx.pop("_k")
        flop = layer_flops(wd, kk * B, gbar=True)      # forward, mean-gradient GEMM, input gradient
        t_upd = rx["phases_ms"]["received_update"] * 1e-3
        rx["tensor"] = {"flop_per_step": flop, "tflops": flop / t_upd / 1e12,
                        "frac_of_burst": flop / t_upd / 1e12 / pk["bf16_tflops"],
                        "peak_burst": pk["bf16_tflops"], "peak_source": pk["source"]}
        gms, gl = rx.pop("_gemm")
        if gl:
            tf = flop / (gms * 1e-3) / 1e12
            rx["roofline"] = {"kernel": "tc_gemm_pair_kernel (forward, mean-gradient and input-gradient "
                                        "GEMMs, in dbw_received_grads_update)",
                              "bound": "tensor", "achieved": tf, "peak": pk["bf16_tflops"],
                              "unit": "TFLOP/s", "frac": tf / pk["bf16_tflops"], "traffic": None,
                              "algorithmic_flop_per_step": flop, "ms_per_step": gms, "launches_timed": gl * K,
                              "share_of_step": gms / rx["ms_per_step"], "peak_kind": "bf16 dense, burst",
                              "peak_source": pk["source"]}
        out["received_form"] = rx
    return out


def _time_received(wl, dev, idx_h, tim_h, W, K, stream, world):
    """The same iterations in the received-workers form (dbw_received_grads_update: no
    [n, d] matrix, gradients of the k received workers only), timed the same way."""
    import torch
    import torch.distributed as dist

    from paper_2004_14696_gb300 import dbw
    from paper_2004_14696_gb300.pipeline import Iteration

    if dbw.dbw_received_grads_workspace_bytes(wl.widths, wl.n, wl.B, wl.prec) == 0:
        return None
    it = Iteration(wl, device=dev, received=True)
    n, B = wl.n, wl.B
    total = W + K
    idx_d = torch.from_numpy(idx_h).to(dev)
    tim_d = torch.from_numpy(tim_h).to(dev)
    names = ["choose_b", "select", "received_update", "grad_stats"]
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(len(names) + 1)] for _ in range(total)]
    ks = torch.zeros(total, dtype=torch.int32, device=dev)

    def one(t, timed):
        e = ev[t]
        if timed:
            e[0].record(stream)
        dbw.dbw_choose_b(it.state, wl.lr, wl.beta, it.b, it.ratio, 0, stream)
        if timed:
            e[1].record(stream)
        dbw.dbw_select_fastest(tim_d[t], it.b, it.order, it.mask, it.tsorted, it.k, stream)
        if timed:
            e[2].record(stream)
        dbw.dbw_received_grads_update(wl.widths, wl.prec, it.w, it.pool, it.labels, idx_d[t], n, B, it.mask, wl.lr,
                                      it.loss, it.partials, it.ws, None, stream)
        if timed:
            e[3].record(stream)
        dbw.dbw_grad_stats(it.partials, n, it.mask, it.loss, it.tsorted, wl.lr, it.state, it.stats, it.row_sqnorm,
                           stream)
        if timed:
            e[4].record(stream)
        ks[t:t + 1].copy_(it.k)

    for t in range(W):
        one(t, False)
    torch.cuda.synchronize(dev)
    if world > 1:
        dist.barrier()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    dbw.dbw_profile_gemm(True)
    t0.record(stream)
    for t in range(W, total):
        one(t, True)
    t1.record(stream)
    torch.cuda.synchronize(dev)
    gm_ms, gm_launches = dbw.dbw_profile_gemm_read()
    dbw.dbw_profile_gemm(False)
    ms = t0.elapsed_time(t1)
    (ms,) = combine_over_ranks([ms], world, dev)
    phase = {nm: sum(ev[t][i].elapsed_time(ev[t][i + 1]) for t in range(W, total)) / K for i, nm in enumerate(names)}
    kv = ks[W:].cpu().numpy().astype(np.float64)
    status = int(it.ws[:4].view(torch.int32).item())
    out = {"call": "dbw_received_grads_update", "value": job_value(world, K, ms), "unit": UNIT,
           "ms_per_step": ms / K, "phases_ms": phase, "mean_k": float(kv.mean()), "device_status": status,
           "gpu_launches": it.launches_per_step() * K, "_k": float(kv.mean()),
           "_gemm": (gm_ms / K, gm_launches // K)}
    del it
    torch.cuda.empty_cache()
    return out


# ====================================================================== single pieces
def _events(reps):
    import torch
    return [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]


def _timed(fn, reps, warmup=2):
    """Mean and min CUDA-event time (ms) of fn() on the current stream, after warm-up."""
    import torch
    for _ in range(warmup):
        fn()
    st = torch.cuda.current_stream()
    evs = _events(reps)
    torch.cuda.synchronize()
    for e0, e1 in evs:
        e0.record(st)
        fn()
        e1.record(st)
    torch.cuda.synchronize()
    ms = [e0.elapsed_time(e1) for e0, e1 in evs]
    return float(np.mean(ms)), float(min(ms))


def aggregate_case(n, d, b, reps, flags=0, seed=workloads.AGG_SEED, G=None):
    """dbw_aggregate_update alone on G ~ N(0,1) [n, d] (filled on the device with torch's
    seeded generator: input generation only) with the n - b fastest of Exp(1) times."""
    import torch
    from paper_2004_14696_gb300 import dbw
    ld = inputs.round_up(d, 32)          # rows start on 128-byte boundaries, as in the workloads
    g = torch.Generator(device="cuda")
    g.manual_seed(seed + n)
    if G is None:
        G = torch.randn((n, ld), generator=g, device="cuda", dtype=torch.float32)
    w = torch.randn(d, generator=g, device="cuda", dtype=torch.float32)
    times = torch.from_numpy(inputs.completion_times(seed, 0, n, "shifted_exp", shift=0.0, rate=1.0)).cuda()
    bt = torch.tensor([b], dtype=torch.int32, device="cuda")
    order = torch.empty(n, dtype=torch.int32, device="cuda")
    mask = torch.empty(n, dtype=torch.uint8, device="cuda")
    ts = torch.empty(n, dtype=torch.float64, device="cuda")
    dbw.dbw_select_fastest(times, bt, order, mask, ts)
    part = torch.empty(dbw.dbw_aggregate_partials_bytes(n, d), dtype=torch.uint8, device="cuda")
    avg, mn = _timed(lambda: dbw.dbw_aggregate_update(G, n, d, mask, 1e-3, w, part, flags=flags), reps)
    k = n - b
    rows_read = n if flags & dbw.ALL_ROW_NORMS else k
    nbytes = (rows_read * d + 2 * d) * 4
    pk = peaks()
    gbs = nbytes / (avg * 1e-3) / 1e9
    return {"case": "aggregate", "n": n, "d": d, "b": b, "k": k,
            "flags": "DBW_ALL_ROW_NORMS" if flags & dbw.ALL_ROW_NORMS else 0, "G_bytes": n * ld * 4,
            "bytes": nbytes, "ms": avg, "ms_min": mn, "GB_s": gbs, "frac_of_peak": gbs / pk["hbm_gbs"],
            "frac_of_8TBs": gbs / 8000.0, "peak_GB_s": pk["hbm_gbs"], "peak_source": pk["source"], "reps": reps,
            "l2": "G > L2" if n * ld * 4 > 129e6 else "G fits in L2 (reads may hit L2)"}


def sweep_points(points, reps):
    """Aggregation-only cases; points sharing (n, d) share one device matrix."""
    import torch
    out = []
    for (n, d), group in _group_points(points).items():
        ld = inputs.round_up(d, 32)
        g = torch.Generator(device="cuda")
        g.manual_seed(workloads.AGG_SEED + n)
        G = torch.randn((n, ld), generator=g, device="cuda", dtype=torch.float32)
        for (b, flags) in group:
            out.append(aggregate_case(n, d, b, reps, flags=flags, G=G))
        del G
        torch.cuda.empty_cache()
    return out


def _group_points(points):
    groups = {}
    for (n, d, b, flags) in points:
        groups.setdefault((n, d), []).append((b, flags))
    return groups


def grads_case(key, reps):
    import torch
    from paper_2004_14696_gb300 import dbw
    from paper_2004_14696_gb300.pipeline import Iteration
    wl = workloads.ALL[key]
    it = Iteration(wl, static_b=0)
    it.load_inputs(0)
    avg, mn = _timed(lambda: dbw.dbw_worker_grads(wl.widths, wl.prec, it.w, it.pool, it.labels, it.idx, wl.n, wl.B,
                                                  it.G, it.loss, it.ws), reps)
    flop = layer_flops(wl.widths, wl.M, dW=True)
    out = {"case": "worker_grads", "workload": key, "ms": avg, "ms_min": mn, "flop": flop,
           "TFLOP_s": flop / (avg * 1e-3) / 1e12, "G_write_GB_s": wl.n * wl.ld * 4 / (avg * 1e-3) / 1e9,
           "status": int(it.ws[:4].view(torch.int32).item())}
    del it
    torch.cuda.empty_cache()
    return out


def received_case(key, b, reps):
    """dbw_received_grads_update alone (after one selection with static b): the received
    workers' gradients, mean, SGD step and norms without the [n, d] matrix."""
    import torch
    from paper_2004_14696_gb300 import dbw
    from paper_2004_14696_gb300.pipeline import Iteration
    wl = workloads.ALL[key]
    it = Iteration(wl, static_b=b, received=True)
    it.load_inputs(0)
    dbw.dbw_select_fastest(it.times, it.b, it.order, it.mask, it.tsorted, it.k)
    avg, mn = _timed(lambda: dbw.dbw_received_grads_update(wl.widths, wl.prec, it.w, it.pool, it.labels, it.idx,
                                                           wl.n, wl.B, it.mask, wl.lr, it.loss, it.partials, it.ws),
                     reps)
    k = wl.n - b
    flop = layer_flops(wl.widths, k * wl.B, gbar=True)
    pk = peaks()
    out = {"case": "received_update", "workload": key, "b": b, "k": k, "ms": avg, "ms_min": mn, "flop": flop,
           "TFLOP_s": flop / (avg * 1e-3) / 1e12, "frac_of_burst": flop / (avg * 1e-3) / 1e12 / pk["bf16_tflops"],
           "status": int(it.ws[:4].view(torch.int32).item())}
    del it
    torch.cuda.empty_cache()
    return out


def psw_case(n, iters, seed=2004146971, model="pareto", tol=1e-4):
    """The push-and-wait clock and the Eq. (17) fit alone, per iteration: arrivals,
    selection, record and the warm-started fit, with k_t drawn uniformly from 1..n
    (every row of the cell table gets samples, the hardest case for the fit)."""
    import torch
    from paper_2004_14696_gb300 import dbw
    psw = dbw.new_psw(n)
    e = torch.empty(n, dtype=torch.float64, device="cuda")
    T = torch.empty(n, dtype=torch.float64, device="cuda")
    bt = torch.zeros(1, dtype=torch.int32, device="cuda")
    order = torch.empty(n, dtype=torch.int32, device="cuda")
    mask = torch.empty(n, dtype=torch.uint8, device="cuda")
    ts = torch.empty(n, dtype=torch.float64, device="cuda")
    kk = torch.empty(1, dtype=torch.int32, device="cuda")
    rng = np.random.default_rng(seed)
    om = torch.from_numpy(np.stack([inputs.completion_times(seed, t, n, model, alpha=2.0, xm=1.0)
                                    for t in range(iters)])).cuda()
    bs = torch.from_numpy(np.array([0] + [n - int(rng.integers(1, n + 1)) for _ in range(iters - 1)],
                                   dtype=np.int32)).cuda()
    st = torch.cuda.current_stream()
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(iters)]
    sweeps = []
    for t in range(iters):
        ev[t][0].record(st)
        dbw.dbw_psw_arrivals(psw, n, om[t], e)
        bt.copy_(bs[t:t + 1])
        dbw.dbw_select_fastest(e, bt, order, mask, ts, kk)
        dbw.dbw_psw_record(psw, n, order, ts, kk)
        ev[t][1].record(st)
        dbw.dbw_psw_estimate(psw, n, T, tol=tol)
        ev[t][2].record(st)
        sweeps.append(psw[8:12].clone())   # dbw_psw_header.sweeps (int32 at byte 8)
    torch.cuda.synchronize()
    clock_ms = [ev[t][0].elapsed_time(ev[t][1]) for t in range(iters)]
    fit_ms = [ev[t][1].elapsed_time(ev[t][2]) for t in range(iters)]
    sw = [int(x.view(torch.int32).item()) for x in sweeps]
    h = dbw.read_psw(psw, n)
    rows = int((h["cnts"].sum(axis=1) > 0).sum())
    tail = slice(iters // 2, iters)
    return {"case": "psw", "n": n, "iters": iters, "tol": tol, "data_rows_at_end": rows,
            "clock_ms_mean": float(np.mean(clock_ms)), "fit_ms_mean": float(np.mean(fit_ms)),
            "fit_ms_mean_second_half": float(np.mean(fit_ms[tail])), "fit_ms_max": float(np.max(fit_ms)),
            "sweeps_mean": float(np.mean(sw)), "sweeps_mean_second_half": float(np.mean(sw[tail])),
            "sweeps_max": int(np.max(sw)), "flags": int(h["flags"])}


def iterate_case(key, iters, warmup, received=False, graph=False):
    """Whole DBW iterations of a workload (choose b, gradients, selection, aggregation,
    statistics; static-b workloads use their b = n/4), inputs resident on the device,
    CUDA events around the loop.  ``graph``: each iteration is one replay of a captured
    CUDA graph (its inputs copied into the captured buffers first)."""
    import torch
    from paper_2004_14696_gb300.pipeline import Iteration
    wl = workloads.ALL[key]
    static_b = wl.n // 4 if wl.policy == "static" else None
    it = Iteration(wl, static_b=static_b, received=received)
    total = warmup + iters
    idx = torch.from_numpy(np.stack([inputs.minibatch_indices(wl.seed, t, wl.n, wl.B, wl.S)
                                     for t in range(total)])).cuda()
    tim = torch.from_numpy(np.stack([inputs.completion_times(wl.seed, t, wl.n, wl.time_model, **wl.time_params)
                                     for t in range(total)])).cuda()
    if graph:
        it.idx.copy_(idx[0])
        it.times.copy_(tim[0])
        it.capture()

    def one(t):
        if graph:
            it.idx.copy_(idx[t])
            it.times.copy_(tim[t])
            it.replay()
        else:
            it.step(idx[t], tim[t])
    for t in range(warmup):
        one(t)
    st = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record(st)
    for t in range(warmup, total):
        one(t)
    e1.record(st)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / iters
    out = {"case": "iterate", "workload": key, "received": received, "graph": graph, "static_b": static_b,
           "iters": iters, "ms_per_iter": ms, "iter_per_s": 1e3 / ms,
           "status": int(it.ws[:4].view(torch.int32).item()), "launches_per_iter": it.launches_per_step()}
    del it
    torch.cuda.empty_cache()
    return out


def extras():
    """The other workloads, for the N = 1 line: whole iterations of the smaller models
    (captured CUDA graphs), points of the aggregation-only sweep (with and without every
    row's norm) and the push-and-wait fit."""
    import torch
    torch.cuda.empty_cache()
    cfg = {}
    cfg[workloads.SOFTMAX784.key] = iterate_case(workloads.SOFTMAX784.key, 300, 10, graph=True)
    cfg[workloads.MLP784.key] = iterate_case(workloads.MLP784.key, 300, 10, graph=True)
    cfg[workloads.MLP3072.key] = {"two_call": iterate_case(workloads.MLP3072.key, 200, 10, graph=True),
                                  "received": iterate_case(workloads.MLP3072.key, 200, 10, received=True, graph=True)}
    from paper_2004_14696_gb300 import dbw
    # the small matrix first: measured right after the 102 GB one it read slower
    pts = [(64, 10 ** 7, 0, 0), (64, 10 ** 7, 16, 0),
           (256, 10 ** 8, 0, 0), (256, 10 ** 8, 64, 0), (256, 10 ** 8, 64, dbw.ALL_ROW_NORMS)]
    cfg["aggregation_sweep"] = sweep_points(pts, reps=10)
    cfg["psw_fit"] = {str(n): psw_case(n, 60) for n in (16, 256)}
    return cfg


# ====================================================================== CPU oracle
def ref_agg_slices(wl):
    """Column slices of the oracle's aggregation sample: the whole width when n d is small
    (up to 2^24 entries), else about 2^24 entries per slice, at most 128 slices."""
    return int(min(128, max(1, -(-wl.n * wl.d // (1 << 24)))))


def oracle_step_seconds(wl, t, pool, labels, w, agg=True, threads=1):
    """One bounded sample of a DBW iteration on the CPU oracle, scaled to a full
    iteration; returns (seconds, parts).

    Sample: the Eq. (2) gradients of 2 of the n workers (each worker's gradient is an
    independent Eq. (2) over its own B samples; scaled by n/2), selection and the
    estimator in full, and the aggregation + statistics of every worker's row over
    column slice t mod S of S = ref_agg_slices(wl) (n distinct seeded rows drawn outside
    the timed part; scaled by S).  k = n: the estimator's choice from a fresh state
    (k_0 = n, Sect. 3), kept for every sampled step."""
    from oracle import dbw_oracle as O
    n, B = wl.n, wl.B
    idx = inputs.minibatch_indices(wl.seed, t, n, B, wl.S)
    times = inputs.completion_times(wl.seed, t, n, wl.time_model, **wl.time_params)
    bf16 = wl.prec == workloads.PREC_BF16
    t0 = time.perf_counter()
    for i in (0, 1):
        r = idx[i * B:(i + 1) * B]
        O.single_worker_grad(wl.widths, w, pool[r], labels[r], B, bf16=bf16)
    t_grad = (time.perf_counter() - t0) * (n / 2.0)
    t0 = time.perf_counter()
    st = O.State(n=n, D=wl.D)
    k, _ = O.choose_k(st, wl.lr, wl.beta)
    _, mask, ts = O.select_fastest(times, n - k)
    t_sel = time.perf_counter() - t0
    t_agg = 0.0
    if agg:
        S = ref_agg_slices(wl)
        s = t % S
        c0, c1 = s * wl.d // S, (s + 1) * wl.d // S
        Gs = inputs.gradient_columns(wl.seed, range(n), c0, c1, threads=threads)
        t0 = time.perf_counter()
        gbar = O.aggregate(Gs, mask)
        O.sgd_update(w[c0:c1], gbar, wl.lr)
        O.deviation_sumsq(Gs, mask, gbar)
        O.row_sqnorms(Gs, mask)
        t_agg = (time.perf_counter() - t0) * S
        del Gs
    return t_grad + t_sel + t_agg, {"grads_s": t_grad, "select_estimator_s": t_sel, "aggregation_s": t_agg}


def _oracle_inputs(wl):
    pool = inputs.feature_pool(wl.seed, wl.S, wl.widths[0], wl.feature_dist)
    labels = inputs.label_pool(wl.seed, wl.S, wl.classes)
    w = inputs.kaiming_uniform_params(wl.seed, wl.widths)
    return pool, labels, w


def _oracle_sample_text(wl, steps):
    S = ref_agg_slices(wl)
    return ("%d sampled iterations, each: Eq. (2) for 2 of the %d workers (x%d), selection and estimator in full, "
            "aggregation + statistics of all %d distinct seeded rows over one 1/%d column slice (x%d; the slices "
            "of the steps differ), k = n; fp64 numpy" % (steps, wl.n, wl.n // 2, wl.n, S, S))


def run_reference(args, rank, world):
    if rank != 0:
        return None
    wl = workloads.ALL[args.workload]
    pool, labels, w = _oracle_inputs(wl)
    threads = os.cpu_count() or 1
    for t in range(args.warmup):
        oracle_step_seconds(wl, t, pool, labels, w, agg=False)
    wall0 = time.perf_counter()
    per, parts = [], []
    for t in range(args.warmup, args.warmup + args.steps):
        s, p = oracle_step_seconds(wl, t, pool, labels, w, threads=threads)
        per.append(s)
        parts.append(p)
    wall = time.perf_counter() - wall0
    sec = float(np.mean(per))
    cores = int(os.environ.get("OPENBLAS_NUM_THREADS", os.cpu_count() or 1))
    value = 1.0 / sec
    extrap = {"grads": wl.n / 2.0, "aggregation": float(ref_agg_slices(wl)), "select_estimator": 1.0}
    mean_parts = {k2: float(np.mean([p[k2] for p in parts])) for k2 in parts[0]}
    return {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": sec * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": bench_config(wl, world),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": _oracle_sample_text(wl, args.steps), "extrapolated": extrap,
                             "seconds_per_step_by_part": mean_parts,
                             "wall_s_of_timed_steps": wall,
                             "note": "per-step seconds are the sampled parts scaled by the factors in "
                                     "'extrapolated', so they exceed the run's wall time"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def cpu_baseline_for(wl, budget_s=25.0):
    """The oracle on the host cores, bounded to about budget_s seconds of work."""
    pool, labels, w = _oracle_inputs(wl)
    threads = os.cpu_count() or 1
    oracle_step_seconds(wl, 0, pool, labels, w, agg=False)
    per, parts, t0 = [], [], time.perf_counter()
    while (time.perf_counter() - t0 < budget_s or len(per) < 2) and len(per) < 10:
        s, p = oracle_step_seconds(wl, 1 + len(per), pool, labels, w, threads=threads)
        per.append(s)
        parts.append(p)
    cores = int(os.environ.get("OPENBLAS_NUM_THREADS", os.cpu_count() or 1))
    return {"value": 1.0 / float(np.mean(per)), "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": _oracle_sample_text(wl, len(per)),
            "extrapolated": {"grads": wl.n / 2.0, "aggregation": float(ref_agg_slices(wl)), "select_estimator": 1.0},
            "seconds_per_step_by_part": {k2: float(np.mean([p[k2] for p in parts])) for k2 in parts[0]}}


# ====================================================================== main
def run_case(args):
    import torch
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)
    from paper_2004_14696_gb300 import dbw
    if args.case == "aggregate":
        print(json.dumps(aggregate_case(args.n, args.d, args.b, args.reps,
                                        flags=dbw.ALL_ROW_NORMS if args.all_row_norms else 0)), flush=True)
    elif args.case == "sweep":
        pts = [(n, d, b, 0) for n in workloads.AGG_NS for d in workloads.AGG_DS
               if n * inputs.round_up(d, 4) * 4 <= args.max_bytes for b in sorted({0, n // 4})]
        for r in sweep_points(pts, args.reps):
            print(json.dumps(r), flush=True)
    elif args.case == "grads":
        print(json.dumps(grads_case(args.workload, args.reps)), flush=True)
    elif args.case == "received":
        print(json.dumps(received_case(args.workload, args.b, args.reps)), flush=True)
    elif args.case == "psw":
        print(json.dumps(psw_case(args.n, args.iters, tol=args.tol)), flush=True)
    else:
        print(json.dumps(iterate_case(args.workload, args.iters, args.warmup, args.received, args.graph)), flush=True)


def main():
    args = parse()
    if args.case:
        run_case(args)
        return
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch
        import torch.distributed as dist
        if args.impl == "reference":
            if rank != 0:
                return
        else:
            torch.cuda.set_device(local_rank)
            dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    if args.impl == "reference":
        out = run_reference(args, rank, world)
    else:
        out = run_dbw(args, rank, world, local_rank)
        if out is not None and world == 1 and not args.no_extras:
            out["configs"] = extras()
            out["cpu_baseline"] = cpu_baseline_for(workloads.ALL[args.workload])
    if world > 1 and args.impl != "reference":
        import torch.distributed as dist
        dist.destroy_process_group()
    if out is not None:
        print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
