#!/usr/bin/env python3
"""Benchmark of the DBW parameter-server iteration on GB300 (one JSON line).

A step is one whole DBW iteration of the largest workload (MLP
4096-4096-4096-4096-1000, n = 256 workers x B = 32, bf16 GEMMs with fp32
accumulation and fp32 master weights, Pareto(2) round-trip times, b chosen by
the estimator every iteration): choose b -> worker gradients (G is [256, 54.4M]
fp32, 55.75 GB) -> selection -> fused aggregation + SGD + statistics ->
estimator bookkeeping.  The working set (G alone) is far larger than L2, so no
L2 flush is needed between steps.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl dbw|reference]

--gpus N > 1 runs under torchrun: every rank simulates its own independent PS
(replicas; the method has no cross-GPU data path), value = all ranks' iterations
/ the slowest rank's time.  --impl reference times the fp64 CPU oracle on a
bounded sample of the same workload (rank 0 only).
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

# dram bytes (read + write) of one aggregation launch from the ncu capture
# summarised in profiles/aggregate_kernel_n64_d4e6_ncu.md (n = 64, d = 4e6, k = 48:
# 792.1 MB against 800 MB algorithmic), as a ratio to the algorithmic bytes so it
# scales to the bench's launches (traffic grows with k d); reported as null once
# aggregate.cu differs from the source the counters were taken on.
AGG_TRAFFIC = {"ratio_to_algorithmic": 792.06e6 / 800.0e6,
               "source_sha256": "e243d8095142453e2c54ea9def1a971b7a4d25fa82962af0340eeaa9d779b39c",
               "case": "n=64 d=4e6 k=48"}
# dram bytes (read + write) of the per-worker weight-gradient launches of one
# full-size step (ncu on mlp4096x3-1000_n256_B32, profiles/tc_dw_kernel_mlp4096_ncu.md):
# 4.2130 + 17.2599 + 17.2596 + 17.2583 GB against 4.2778 + 3 x 17.3141 GB algorithmic;
# keyed to the dW kernel's own source (dw_source_sha).
DW_TRAFFIC = {"ratio_to_algorithmic": (4.2130 + 17.2599 + 17.2596 + 17.2583) / (4.2778 + 3 * 17.3141),
              "source_sha256": "49652b56fb1338974566dcb78b1b940bb43688a603dfa846f820898c31d62839",
              "case": "mlp4096x3-1000_n256_B32, one step"}


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", default="dbw", choices=["dbw", "reference"])
    p.add_argument("--workload", default=workloads.MLP4096.key, choices=list(workloads.ALL))
    return p.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            j = json.load(f)
        return {"hbm_gbs": j["hbm_gbs"], "bf16_tflops": j["bf16_tflops"],
                "bf16_tflops_sustained": j.get("bf16_tflops_sustained"), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


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

    # ---------------------------------------------------------------- e2e
    # the same steps through the public API with host buffers: per step, pinned
    # host -> device copies of the minibatch indices and times, the iteration,
    # and a device -> host read of the step's statistics (loss, k, V, ...).
    # the e2e leg replays the very same iterations: parameters and estimator state restart
    it2 = it
    it2.w.copy_(w_init)
    dbw.dbw_state_init(it2.state, n, wl.D, stream)
    idx_pin = torch.from_numpy(idx_h).pin_memory()
    tim_pin = torch.from_numpy(tim_h).pin_memory()
    stats_pin = torch.empty(dbw.STATS_LEN, dtype=torch.float64).pin_memory()

    def one_e2e(t):
        it2.idx.copy_(idx_pin[t], non_blocking=True)
        it2.times.copy_(tim_pin[t], non_blocking=True)
        it2.step(stream=stream)
        stats_pin.copy_(it2.stats, non_blocking=True)
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

    # ---------------------------------------------------------------- received form
    rx = _time_received(wl, dev, idx_d, tim_d, W, K, stream, world)

    # ---------------------------------------------------------------- gather over ranks
    elapsed_ms, e2e_s = combine_over_ranks([elapsed_ms, e2e_s], world, dev)
    if rank != 0:
        return None
    pk = peaks()
    d = it.d
    agg_bytes = float(np.mean((kvals * d + 2 * d) * 4.0))
    agg_ms = phase_ms["aggregate"]
    achieved = agg_bytes / (agg_ms * 1e-3) / 1e9
    traffic = None
    src = os.path.join(ROOT, "paper_2004_14696_gb300", "csrc", "aggregate.cu")
    if AGG_TRAFFIC["source_sha256"] == sha256_of(src):
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
    gemm_flop = 0
    tc_flop = 0
    wd = wl.widths
    M = n * B
    for l in range(len(wd) - 1):
        gemm_flop += 2 * M * wd[l] * wd[l + 1] * 2          # forward + per-worker dW
        tc_flop += 2 * M * wd[l] * wd[l + 1]                # forward
        if l > 0:
            gemm_flop += 2 * M * wd[l] * wd[l + 1]          # input gradient
            tc_flop += 2 * M * wd[l] * wd[l + 1]
    # the forward and input-gradient GEMMs (persistent tcgen05 kernel), timed live
    tensor = None
    if gm_launches:
        tf = tc_flop * K / (gm_ms * 1e-3) / 1e12
        tensor = {"kernel": "tc_gemm_pair_kernel (forward + input-gradient GEMMs, in dbw_worker_grads)",
                  "bound": "tensor", "achieved": tf, "peak": pk["bf16_tflops_sustained"], "unit": "TFLOP/s",
                  "frac": tf / pk["bf16_tflops_sustained"], "traffic": None,
                  "algorithmic_flop_per_step": tc_flop, "ms_per_step": gm_ms / K,
                  "launches_timed": gm_launches, "share_of_step": gm_ms / elapsed_ms,
                  "peak_kind": "bf16 dense, sustained", "peak_source": pk["source"]}
    out = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K, "warmup": W,
        "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16+f32" if wl.prec == workloads.PREC_BF16 else "f32", "data": "synthetic",
        "config": {"workload": wl.key, "widths": list(wd), "n_workers": n, "batch_per_worker": B,
                   "d": d, "G_bytes": n * it.ld * 4, "time_model": wl.time_model, "policy": "dbw",
                   "mean_k": float(kvals.mean()), "l2": "working set > L2 (G is %.1f GB), no flush"
                   % (n * it.ld * 4 / 1e9), "parallelism": "replicas" if world > 1 else "single"},
        "roofline": dw,
        "roofline_aggregate": {"kernel": "aggregate_kernel (dbw_aggregate_update)", "bound": "hbm",
                               "achieved": achieved, "peak": pk["hbm_gbs"], "unit": "GB/s",
                               "frac": achieved / pk["hbm_gbs"], "traffic": traffic,
                               "algorithmic_bytes_per_launch": agg_bytes, "peak_source": pk["source"]},
        "roofline_tensor": tensor,
        "phases_ms": phase_ms,
        "gemm": {"flop_per_step": gemm_flop, "worker_grads_tflops": gemm_flop / (phase_ms["worker_grads"] * 1e-3) / 1e12},
        "gpu_launches": None,
        "e2e": {"value": job_value(world, K, e2e_s * 1e3), "unit": UNIT, "h2d_bytes_per_step": int(h2d),
                "d2h_bytes_per_step": int(d2h)},
        "clocks": clk.summary(),
    }
    out["gpu_launches"] = it.launches_per_step() * K
    if rx is not None:
        kk = rx.pop("_k")
        flop = 0
        for l in range(len(wd) - 1):
            flop += 2 * kk * B * wd[l] * wd[l + 1] * (3 if l > 0 else 2)   # forward, g_t GEMM, input gradient
        t_upd = rx["phases_ms"]["received_update"] * 1e-3
        rx["tensor"] = {"flop_per_step": flop, "tflops": flop / t_upd / 1e12,
                        "frac_of_sustained": flop / t_upd / 1e12 / pk["bf16_tflops_sustained"]
                        if pk.get("bf16_tflops_sustained") else None,
                        "peak_sustained": pk.get("bf16_tflops_sustained"), "peak_source": pk["source"]}
        gms, gl = rx.pop("_gemm")
        if gl:
            tf = flop / (gms * 1e-3) / 1e12
            rx["roofline"] = {"kernel": "tc_gemm_pair_kernel (forward, mean-gradient and input-gradient "
                                        "GEMMs, in dbw_received_grads_update)",
                              "bound": "tensor", "achieved": tf, "peak": pk["bf16_tflops_sustained"],
                              "unit": "TFLOP/s", "frac": tf / pk["bf16_tflops_sustained"], "traffic": None,
                              "algorithmic_flop_per_step": flop, "ms_per_step": gms, "launches_timed": gl * K,
                              "share_of_step": gms / rx["ms_per_step"], "peak_kind": "bf16 dense, sustained",
                              "peak_source": pk["source"]}
        out["received_form"] = rx
    return out


def _time_received(wl, dev, idx_d, tim_d, W, K, stream, world):
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


# ====================================================================== CPU oracle
def oracle_sample_step(wl, t, pool, labels, w, rng_cols):
    """One bounded sample of a DBW iteration on the CPU oracle; returns seconds per full iteration.

    Sample: the gradients of 2 of the n workers (each worker's gradient is an
    independent Eq. (2) over its own B samples), selection and the estimator in
    full, and the aggregation + statistics over a 1/64 column slice of the
    sampled rows broadcast to n rows.  Scaled up by n/2 (gradients) and 64
    (aggregation columns).
    """
    from oracle import dbw_oracle as O
    n, B = wl.n, wl.B
    idx = inputs.minibatch_indices(wl.seed, t, n, B, wl.S)
    times = inputs.completion_times(wl.seed, t, n, wl.time_model, **wl.time_params)
    bf16 = wl.prec == workloads.PREC_BF16
    t0 = time.perf_counter()
    rows = []
    for i in (0, 1):
        r = idx[i * B:(i + 1) * B]
        g, _ = O.single_worker_grad(wl.widths, w, pool[r], labels[r], B, bf16=bf16)
        rows.append(g)
    t_grad = (time.perf_counter() - t0) * (n / 2.0)
    t0 = time.perf_counter()
    st = O.State(n=n, D=wl.D)
    k, _ = O.choose_k(st, wl.lr, wl.beta)
    _, mask, ts = O.select_fastest(times, n - k)
    c0 = int(rng_cols.integers(0, 64)) * (wl.d // 64)
    sl = slice(c0, c0 + wl.d // 64)
    Gs = np.stack([rows[i % 2][sl] for i in range(n)])
    gbar = O.aggregate(Gs, mask)
    O.sgd_update(w[sl], gbar, wl.lr)
    O.deviation_sumsq(Gs, mask, gbar)
    O.row_sqnorms(Gs, mask)
    t_agg = (time.perf_counter() - t0) * 64.0
    return t_grad + t_agg


def run_reference(args, rank, world):
    if rank != 0:
        return None
    wl = workloads.ALL[args.workload]
    pool = inputs.feature_pool(wl.seed, wl.S, wl.widths[0], wl.feature_dist)
    labels = inputs.label_pool(wl.seed, wl.S, wl.classes)
    w = inputs.kaiming_uniform_params(wl.seed, wl.widths)
    rng = np.random.default_rng(0)
    for t in range(args.warmup):
        oracle_sample_step(wl, t, pool, labels, w, rng)
    per = [oracle_sample_step(wl, args.warmup + t, pool, labels, w, rng) for t in range(args.steps)]
    sec = float(np.mean(per))
    cores = int(os.environ.get("OPENBLAS_NUM_THREADS", os.cpu_count() or 1))
    value = 1.0 / sec
    sample = ("per step: Eq. (2) gradients of 2 of the %d workers (scaled x%d) + selection, estimator and the "
              "aggregation/statistics on a 1/64 column slice (scaled x64); fp64 numpy" % (wl.n, wl.n // 2))
    return {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": sec * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": wl.key, "n_workers": wl.n, "batch_per_worker": wl.B, "d": wl.d},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def cpu_baseline_for(wl, budget_s=20.0):
    """The oracle on the host cores, bounded to about budget_s seconds of work."""
    pool = inputs.feature_pool(wl.seed, wl.S, wl.widths[0], wl.feature_dist)
    labels = inputs.label_pool(wl.seed, wl.S, wl.classes)
    w = inputs.kaiming_uniform_params(wl.seed, wl.widths)
    rng = np.random.default_rng(0)
    per, t0 = [], time.perf_counter()
    while time.perf_counter() - t0 < budget_s or len(per) < 2:
        per.append(oracle_sample_step(wl, len(per), pool, labels, w, rng))
        if len(per) >= 10:
            break
    cores = int(os.environ.get("OPENBLAS_NUM_THREADS", os.cpu_count() or 1))
    return {"value": 1.0 / float(np.mean(per[1:] if len(per) > 1 else per)), "unit": UNIT, "cores": cores,
            "kind": "oracle",
            "sample": "%d sampled iterations: Eq. (2) for 2 of %d workers (scaled x%d) + selection/estimator + "
                      "aggregation on a 1/64 column slice (scaled x64), fp64 numpy" % (len(per), wl.n, wl.n // 2)}


def main():
    args = parse()
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
        if out is not None and world == 1:
            out["cpu_baseline"] = cpu_baseline_for(workloads.ALL[args.workload])
    if world > 1 and args.impl != "reference":
        import torch.distributed as dist
        dist.destroy_process_group()
    if out is not None:
        print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
