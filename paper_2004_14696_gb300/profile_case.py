"""Run single pieces of the DBW iteration on chosen sizes, for timing and ncu captures.

    python -m paper_2004_14696_gb300.profile_case aggregate --n 64 --d 4000000 --b 16 --reps 3
    python -m paper_2004_14696_gb300.profile_case sweep            # the aggregation-only sweep
    python -m paper_2004_14696_gb300.profile_case grads --workload mlp4096x3-1000_n256_B32 --reps 3
    python -m paper_2004_14696_gb300.profile_case received --workload mlp4096x3-1000_n256_B32 --b 64
    python -m paper_2004_14696_gb300.profile_case psw --n 256 --iters 60     # push-and-wait clock + Eq. (17)
    python -m paper_2004_14696_gb300.profile_case iterate --workload mlp784-256-10_n64_B64   # whole iterations

Each prints one JSON line per case with CUDA-event times (on the launching
stream, after warm-up).  Large gradient matrices are filled on the device with
torch's seeded normal generator (input generation only); times come from the
same seeded host models as everywhere else.
"""
from __future__ import annotations

import argparse
import json
import os

import numpy as np
import torch

from . import dbw, inputs, workloads
from .pipeline import Iteration


def _peak_hbm():
    path = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            return json.load(f)["hbm_gbs"], "measured"
    return 6800.0, "fallback"


def aggregate_case(n, d, b, reps, seed=2004146963, warmup=2):
    ld = inputs.round_up(d, 4)
    g = torch.Generator(device="cuda")
    g.manual_seed(seed + n)
    G = torch.randn((n, ld), generator=g, device="cuda", dtype=torch.float32)
    w = torch.randn(d, generator=g, device="cuda", dtype=torch.float32)
    times = torch.from_numpy(inputs.completion_times(seed, 0, n, "shifted_exp", shift=0.0, rate=1.0)).cuda()
    bt = torch.tensor([b], dtype=torch.int32, device="cuda")
    order = torch.empty(n, dtype=torch.int32, device="cuda")
    mask = torch.empty(n, dtype=torch.uint8, device="cuda")
    ts = torch.empty(n, dtype=torch.float64, device="cuda")
    dbw.dbw_select_fastest(times, bt, order, mask, ts)
    part = torch.empty(dbw.dbw_aggregate_partials_bytes(n, d), dtype=torch.uint8, device="cuda")
    for _ in range(warmup):
        dbw.dbw_aggregate_update(G, n, d, mask, 1e-3, w, part)
    st = torch.cuda.current_stream()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
    torch.cuda.synchronize()
    for e0, e1 in evs:
        e0.record(st)
        dbw.dbw_aggregate_update(G, n, d, mask, 1e-3, w, part)
        e1.record(st)
    torch.cuda.synchronize()
    ms = [e0.elapsed_time(e1) for e0, e1 in evs]
    k = n - b
    nbytes = (k * d + 2 * d) * 4
    avg = float(np.mean(ms))
    peak, src = _peak_hbm()
    gbs = nbytes / (avg * 1e-3) / 1e9
    l2_note = "G > L2" if n * ld * 4 > 129e6 else "G fits in L2 (reads may hit L2)"
    return {"case": "aggregate", "n": n, "d": d, "b": b, "k": k, "G_bytes": n * ld * 4, "bytes": nbytes,
            "ms": avg, "ms_min": min(ms), "GB_s": gbs, "frac_of_peak": gbs / peak, "peak_GB_s": peak,
            "peak_source": src, "reps": reps, "l2": l2_note}


def grads_case(key, reps, warmup=2):
    wl = workloads.ALL[key]
    it = Iteration(wl, static_b=0)
    it.load_inputs(0)
    for _ in range(warmup):
        dbw.dbw_worker_grads(wl.widths, wl.prec, it.w, it.pool, it.labels, it.idx, wl.n, wl.B, it.G, it.loss, it.ws)
    st = torch.cuda.current_stream()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
    torch.cuda.synchronize()
    for e0, e1 in evs:
        e0.record(st)
        dbw.dbw_worker_grads(wl.widths, wl.prec, it.w, it.pool, it.labels, it.idx, wl.n, wl.B, it.G, it.loss, it.ws)
        e1.record(st)
    torch.cuda.synchronize()
    ms = [e0.elapsed_time(e1) for e0, e1 in evs]
    M = wl.n * wl.B
    flop = 0
    for l in range(len(wl.widths) - 1):
        flop += 4 * M * wl.widths[l] * wl.widths[l + 1] + (2 * M * wl.widths[l] * wl.widths[l + 1] if l else 0)
    avg = float(np.mean(ms))
    return {"case": "worker_grads", "workload": key, "ms": avg, "ms_min": min(ms), "flop": flop,
            "TFLOP_s": flop / (avg * 1e-3) / 1e12, "G_write_GB_s": wl.n * wl.ld * 4 / (avg * 1e-3) / 1e9}


def received_case(key, b, reps, warmup=2):
    """dbw_received_grads_update alone (after one selection with static b): the received
    workers' gradients, mean, SGD step and norms without the [n, d] matrix."""
    wl = workloads.ALL[key]
    it = Iteration(wl, static_b=b, received=True)
    it.load_inputs(0)
    dbw.dbw_select_fastest(it.times, it.b, it.order, it.mask, it.tsorted, it.k)

    def call():
        dbw.dbw_received_grads_update(wl.widths, wl.prec, it.w, it.pool, it.labels, it.idx, wl.n, wl.B, it.mask,
                                      wl.lr, it.loss, it.partials, it.ws)
    for _ in range(warmup):
        call()
    st = torch.cuda.current_stream()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
    torch.cuda.synchronize()
    for e0, e1 in evs:
        e0.record(st)
        call()
        e1.record(st)
    torch.cuda.synchronize()
    ms = [e0.elapsed_time(e1) for e0, e1 in evs]
    k = wl.n - b
    Mk = k * wl.B
    flop = 0
    for l in range(len(wl.widths) - 1):
        flop += 2 * Mk * wl.widths[l] * wl.widths[l + 1] * (3 if l else 2)
    avg = float(np.mean(ms))
    return {"case": "received_update", "workload": key, "b": b, "k": k, "ms": avg, "ms_min": min(ms),
            "flop": flop, "TFLOP_s": flop / (avg * 1e-3) / 1e12,
            "status": int(it.ws[:4].view(torch.int32).item())}


def psw_case(n, iters, seed=2004146971, model="pareto", tol=1e-6):
    """The push-and-wait clock and the Eq. (17) fit alone, per iteration: arrivals,
    selection, record and the warm-started fit, with k_t drawn uniformly from 1..n
    (every row of the cell table gets samples, the hardest case for the fit)."""
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
    """Whole DBW iterations of a workload (the bench's step: choose b, gradients, selection,
    aggregation, statistics; static-b workloads use their b = n/4), inputs resident on the
    device, CUDA events around the loop.  ``graph``: each iteration is one replay of a
    captured CUDA graph (its inputs copied into the captured buffers first)."""
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
    return {"case": "iterate", "workload": key, "received": received, "graph": graph, "static_b": static_b,
            "iters": iters, "ms_per_iter": ms, "iter_per_s": 1e3 / ms,
            "status": int(it.ws[:4].view(torch.int32).item()), "launches_per_iter": it.launches_per_step()}


def main(argv=None):
    p = argparse.ArgumentParser()
    sub = p.add_subparsers(dest="cmd", required=True)
    a = sub.add_parser("aggregate")
    a.add_argument("--n", type=int, default=64)
    a.add_argument("--d", type=int, default=4_000_000)
    a.add_argument("--b", type=int, default=16)
    a.add_argument("--reps", type=int, default=5)
    s = sub.add_parser("sweep")
    s.add_argument("--reps", type=int, default=10)
    s.add_argument("--max-bytes", type=float, default=float(workloads.AGG_MAX_BYTES))
    gr = sub.add_parser("grads")
    gr.add_argument("--workload", default=workloads.MLP4096.key, choices=list(workloads.ALL))
    gr.add_argument("--reps", type=int, default=3)
    rc = sub.add_parser("received")
    rc.add_argument("--workload", default=workloads.MLP4096.key, choices=list(workloads.ALL))
    rc.add_argument("--b", type=int, default=64)
    rc.add_argument("--reps", type=int, default=3)
    pw = sub.add_parser("psw")
    pw.add_argument("--n", type=int, default=256)
    pw.add_argument("--iters", type=int, default=60)
    pw.add_argument("--tol", type=float, default=1e-6)
    itp = sub.add_parser("iterate")
    itp.add_argument("--workload", default=workloads.MLP784.key, choices=list(workloads.ALL))
    itp.add_argument("--iters", type=int, default=50)
    itp.add_argument("--warmup", type=int, default=5)
    itp.add_argument("--received", action="store_true")
    itp.add_argument("--graph", action="store_true", help="replay each iteration as a captured CUDA graph")
    args = p.parse_args(argv)
    torch.cuda.set_device(0)
    if args.cmd == "aggregate":
        print(json.dumps(aggregate_case(args.n, args.d, args.b, args.reps)), flush=True)
    elif args.cmd == "sweep":
        for n in workloads.AGG_NS:
            for d in workloads.AGG_DS:
                if n * inputs.round_up(d, 4) * 4 > args.max_bytes:
                    continue
                for b in sorted({0, n // 4}):
                    print(json.dumps(aggregate_case(n, d, b, args.reps)), flush=True)
                    torch.cuda.empty_cache()
    elif args.cmd == "iterate":
        print(json.dumps(iterate_case(args.workload, args.iters, args.warmup, args.received, args.graph)),
              flush=True)
    elif args.cmd == "psw":
        print(json.dumps(psw_case(args.n, args.iters, tol=args.tol)), flush=True)
    elif args.cmd == "received":
        print(json.dumps(received_case(args.workload, args.b, args.reps)), flush=True)
    else:
        print(json.dumps(grads_case(args.workload, args.reps)), flush=True)


if __name__ == "__main__":
    main()
