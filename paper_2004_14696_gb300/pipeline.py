"""One DBW parameter-server iteration as a sequence of libdbw calls.

``Iteration`` owns the device buffers of one workload (G, w, workspace,
partials, estimator state) and issues, per step, the five C-ABI calls in the
paper's order (Sect. 3: b_t is chosen right after w_t is available):

    dbw_choose_b -> dbw_worker_grads -> dbw_select_fastest
                 -> dbw_aggregate_update -> dbw_grad_stats

or, with ``received=True`` (the same iteration without the [n, d] gradient
matrix, for the k received workers only):

    dbw_choose_b -> dbw_select_fastest -> dbw_received_grads_update -> dbw_grad_stats

Python only sequences the calls and owns memory through torch; every step of
the computation runs in libdbw's kernels on the current CUDA stream.
"""
from __future__ import annotations

import numpy as np
import torch

from . import dbw, inputs
from .workloads import Workload


class Iteration:
    def __init__(self, wl: Workload, device="cuda", static_b=None, blind=False, keep_gbar=False,
                 pool=None, labels=None, w0=None, received=False, clock="psi", psw_tol=1e-4,
                 psw_max_sweeps=100000):
        self.wl = wl
        self.device = torch.device(device)
        n, d, ld = wl.n, wl.d, wl.ld
        self.n, self.d, self.ld = n, d, ld
        self.static_b = static_b
        self.blind = blind
        self.received = received
        if clock not in ("psi", "psw"):
            raise ValueError("clock must be 'psi' (push-and-interrupt) or 'psw' (push-and-wait)")
        self.clock = clock
        self.psw_tol, self.psw_max_sweeps = psw_tol, psw_max_sweeps
        if pool is None:
            pool = inputs.feature_pool(wl.seed, wl.S, wl.widths[0], wl.feature_dist)
        if labels is None:
            labels = inputs.label_pool(wl.seed, wl.S, wl.classes)
        if w0 is None:
            w0 = inputs.kaiming_uniform_params(wl.seed, wl.widths)
        self.pool = torch.as_tensor(pool).to(self.device)
        self.labels = torch.as_tensor(labels).to(self.device)
        self.w = torch.as_tensor(w0).to(self.device).clone()
        self.loss = torch.empty(n, dtype=torch.float32, device=self.device)
        if received:
            wsb = dbw.dbw_received_grads_workspace_bytes(wl.widths, n, wl.B, wl.prec)
            if wsb == 0:
                raise ValueError(f"{wl.key}: the received-workers pass needs bf16, B % 32 == 0, B | 128 or 128 | B")
            self.G = None
            self.ws = torch.empty(wsb, dtype=torch.uint8, device=self.device)
            self.partials = torch.empty(dbw.dbw_received_partials_bytes(n), dtype=torch.uint8, device=self.device)
        else:
            self.G = torch.empty((n, ld), dtype=torch.float32, device=self.device)
            self.ws = torch.empty(dbw.dbw_worker_grads_workspace_bytes(wl.widths, n, wl.B, wl.prec),
                                  dtype=torch.uint8, device=self.device)
            self.partials = torch.empty(dbw.dbw_aggregate_partials_bytes(n, d), dtype=torch.uint8,
                                        device=self.device)
        self.state = dbw.new_state(n, wl.D, self.device)
        self.b = torch.zeros(1, dtype=torch.int32, device=self.device)
        if static_b is not None:
            self.b.fill_(int(static_b))
        self.k = torch.zeros(1, dtype=torch.int32, device=self.device)
        self.order = torch.empty(n, dtype=torch.int32, device=self.device)
        self.mask = torch.empty(n, dtype=torch.uint8, device=self.device)
        self.tsorted = torch.empty(n, dtype=torch.float64, device=self.device)
        self.ratio = torch.empty(n, dtype=torch.float64, device=self.device)
        self.stats = torch.empty(dbw.STATS_LEN, dtype=torch.float64, device=self.device)
        self.row_sqnorm = torch.empty(n, dtype=torch.float64, device=self.device)
        self.gbar = torch.empty(d, dtype=torch.float32, device=self.device) if keep_gbar else None
        if clock == "psw":
            self.psw = dbw.new_psw(n, self.device)
            self.T_hat = torch.full((n,), float("nan"), dtype=torch.float64, device=self.device)
            self.arrivals = torch.empty(n, dtype=torch.float64, device=self.device)
        # per-step inputs (device copies written by the caller or by load_inputs)
        self.idx = torch.empty(n * wl.B, dtype=torch.int32, device=self.device)
        self.times = torch.empty(n, dtype=torch.float64, device=self.device)

    # ------------------------------------------------------------ inputs
    def host_inputs(self, t):
        wl = self.wl
        idx = inputs.minibatch_indices(wl.seed, t, wl.n, wl.B, wl.S)
        times = inputs.completion_times(wl.seed, t, wl.n, wl.time_model, **wl.time_params)
        return idx, times

    def load_inputs(self, t):
        idx, times = self.host_inputs(t)
        self.idx.copy_(torch.from_numpy(idx))
        self.times.copy_(torch.from_numpy(times))

    # ------------------------------------------------------------ one iteration
    def step(self, idx=None, times=None, stream=None):
        """Issue one iteration; idx / times default to the buffers self.idx / self.times."""
        wl = self.wl
        idx = self.idx if idx is None else idx
        times = self.times if times is None else times
        psw = self.clock == "psw"
        if self.static_b is None:
            if psw:
                dbw.dbw_choose_b_times(self.state, self.T_hat, wl.lr, wl.beta, self.b, self.ratio,
                                       dbw.CHOOSE_BLIND if self.blind else 0, stream)
            else:
                dbw.dbw_choose_b(self.state, wl.lr, wl.beta, self.b, self.ratio,
                                 dbw.CHOOSE_BLIND if self.blind else 0, stream)
        # static b is known on the host: its learning-rate rule applies; DBW uses lr
        lr = wl.lr if self.static_b is None else wl.lr_for(wl.n - int(self.static_b))
        if psw:
            # push-and-wait: the gradients of w_t arrive at the residual busy time plus the round trip
            dbw.dbw_psw_arrivals(self.psw, wl.n, times, self.arrivals, stream)
            times = self.arrivals
        if self.received:
            dbw.dbw_select_fastest(times, self.b, self.order, self.mask, self.tsorted, self.k, stream)
            dbw.dbw_received_grads_update(wl.widths, wl.prec, self.w, self.pool, self.labels, idx, wl.n, wl.B,
                                          self.mask, lr, self.loss, self.partials, self.ws, self.gbar, stream)
        else:
            dbw.dbw_worker_grads(wl.widths, wl.prec, self.w, self.pool, self.labels, idx, wl.n, wl.B, self.G,
                                 self.loss, self.ws, stream)
            dbw.dbw_select_fastest(times, self.b, self.order, self.mask, self.tsorted, self.k, stream)
            dbw.dbw_aggregate_update(self.G, wl.n, self.d, self.mask, lr, self.w, self.partials, self.gbar, stream)
        dbw.dbw_grad_stats(self.partials, wl.n, self.mask, self.loss, self.tsorted, lr, self.state, self.stats,
                           self.row_sqnorm, stream)
        if psw:
            dbw.dbw_psw_record(self.psw, wl.n, self.order, self.tsorted, self.k, stream)
            dbw.dbw_psw_estimate(self.psw, wl.n, self.T_hat, self.psw_tol, self.psw_max_sweeps, stream)

    # ------------------------------------------------------------ CUDA graph
    def capture(self, warmup=2):
        """Record one whole iteration (on self.idx / self.times) as a CUDA graph.

        Every call of the iteration is asynchronous and reads nothing back to the
        host, so the iteration captures as is; replay() then costs one launch
        instead of one per kernel, which is what bounds the small workloads.  The
        inputs of each step go into self.idx / self.times before replay()."""
        s = torch.cuda.Stream(self.device)
        s.wait_stream(torch.cuda.current_stream(self.device))
        with torch.cuda.stream(s):
            for _ in range(warmup):   # first calls: lazy library setup happens outside the capture
                self.step()
        torch.cuda.current_stream(self.device).wait_stream(s)
        self.graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(self.graph):
            self.step()
        return self.graph

    def replay(self):
        self.graph.replay()

    # ------------------------------------------------------------ checkpoint
    def checkpoint(self):
        """Host copy of everything an iteration carries over: w and the estimator state.

        The gradient matrix, workspace and partials are scratch that each
        iteration rewrites, so (w, state) restores the run exactly.
        """
        torch.cuda.synchronize(self.device)
        ck = {"w": self.w.detach().cpu().clone(), "state": self.state.detach().cpu().clone(),
              "b": self.b.detach().cpu().clone(), "key": self.wl.key}
        if self.clock == "psw":
            ck["psw"] = self.psw.detach().cpu().clone()
            ck["T_hat"] = self.T_hat.detach().cpu().clone()
        return ck

    def restore(self, ckpt):
        if ckpt["key"] != self.wl.key:
            raise ValueError("checkpoint of another workload")
        self.w.copy_(ckpt["w"])
        self.state.copy_(ckpt["state"])
        self.b.copy_(ckpt["b"])
        if self.clock == "psw":
            self.psw.copy_(ckpt["psw"])
            self.T_hat.copy_(ckpt["T_hat"])

    def record(self, t, wall_ms=None):
        """One iteration's log record (reads the statistics back: synchronises)."""
        s = self.stats.cpu().numpy()
        st = dbw.read_state(self.state)
        k = int(s[dbw.STAT_K])
        rec = {"t": t, "b": self.n - k, "k": k, "T_k": float(self.tsorted[k - 1].item()),
               "vclock": float(s[dbw.STAT_VCLOCK]), "F": float(s[dbw.STAT_F]),
               "gbar_sq": float(s[dbw.STAT_GBAR_SQ]), "V": float(s[dbw.STAT_V]), "N": float(s[dbw.STAT_N]),
               "L": float(s[dbw.STAT_L]), "flags": int(s[dbw.STAT_FLAGS]), "k_next_state": int(st.k_next)}
        if wall_ms is not None:
            rec["wall_ms"] = wall_ms
        return rec

    def launches_per_step(self):
        """Kernels libdbw launches per step (for the bench's launch count); the status-word
        memsets are copies, not kernels."""
        L = len(self.wl.widths) - 1
        choose = (0 if self.static_b is not None else 1) + (3 if self.clock == "psw" else 0)   # + arrivals, record, fit
        # loss + dZ (+ dZ^T, written by the same kernel when its transposing tile fits)
        loss = 1 if self.wl.B * (self.wl.widths[-1] + 8) * 2 <= 160 * 1024 else 2
        if self.received:
            # select; compaction, the weight cast-transposes of all layers (1), X and X^T, L forward
            # GEMMs, loss + dZ^T, per layer the mean-gradient GEMM (with the dX GEMM in the same
            # launch when l > 0); bias row sums and bias mean of all layers (2), Gram norms of all
            # layers (1), finish; grad_stats (2)
            return choose + 1 + (1 + 1 + 1 + L + loss + L + 2 + 1 + 1) + 2
        if self.wl.prec == dbw.PREC_BF16 and self.wl.B % 32 == 0:
            # tcgen05 pass: the weight cast-transposes of all layers (1), X and X^T, L forward GEMMs,
            # loss + dZ^T, L dW GEMMs, L bias gradients, L-1 dX GEMMs
            grads = 1 + 1 + L + loss + L + L + (L - 1)
        else:
            grads = 1 + L + 1 + L + L + (L - 1)    # gather, forward, loss, dW, bias, dX
            if self.wl.prec == dbw.PREC_BF16:
                grads += 1                          # bf16 weight cast
            grads += self._simt_extra_launches()
        return choose + grads + 1 + 1 + 2

    def _simt_extra_launches(self):
        """Launches beyond one per GEMM on the SIMT pass: a GEMM in three tf32 passes splits
        its two operands first (2), a split-K GEMM sums its splits (1); the skinny kernels
        are one launch.  Mirrors the plan's rules in csrc/grads.cu."""
        wd, M = self.wl.widths, self.wl.n * self.wl.B
        sms = torch.cuda.get_device_properties(self.device).multi_processor_count

        def split_launch(m, n, k):
            tiles = -(-n // 128) * -(-m // 128)
            s = min(-(-2 * sms // tiles), k // 64)
            if s <= 1:
                return 0
            kps = -(-(-(-k // s)) // 16) * 16
            return 1 if -(-k // kps) > 1 else 0

        def skinny_n(n, k, off):     # the forward GEMM with few outputs (W_l at offset off of w)
            vec = self.wl.prec == dbw.PREC_FP32 and k % 4 == 0 and off % 4 == 0
            return n <= 16 and (vec or n * k * 4 <= 48 * 1024)

        def skinny_k(n, k):     # the input-gradient GEMM with a short inner dimension
            return k <= 32 and (n + 16) * k * 4 <= 48 * 1024

        B, n, off = self.wl.B, self.wl.n, 0
        extra = 0
        for l in range(len(wd) - 1):
            fin, fout = wd[l], wd[l + 1]
            if (self.wl.prec == dbw.PREC_FP32 and B % 32 == 0 and B <= 256 and fin % 4 == 0 and off % 4 == 0
                    and fout >= 32 and n * fout * fin * B >= 1 << 25):
                extra += 1 if l == 0 else 2     # transposed parts of dZ_l (and of the input above layer 1)
            if self.wl.prec == dbw.PREC_FP32 and fout >= 32 and M * fout * fin >= 1 << 27:
                extra += 1 if l == 0 else 2     # the gather writes the first layer's input parts
            elif not skinny_n(fout, fin, off):
                extra += split_launch(M, fout, fin)
            off += fin * fout + fout
            if l > 0 and not skinny_k(fin, fout):
                extra += split_launch(M, fin, fout)
        return extra


def agg_case(n, d, seed, b, device="cuda", mean=0.0, std=1.0):
    """Inputs of an aggregation-only case: G [n, ld] ~ N(mean, std^2), w, Exp(1) times."""
    ld = inputs.round_up(d, 4)
    G = inputs.gradient_matrix(seed, n, d, ld, mean, std)
    w = inputs.rng(seed, inputs.STREAM_INIT).standard_normal(d, dtype=np.float32)
    times = inputs.completion_times(seed, 0, n, "shifted_exp", shift=0.0, rate=1.0)
    return G, w, times


def run(wl: Workload, iters, log=None, static_b=None, blind=False, device="cuda", start=0, it=None,
        received=False, clock="psi"):
    """Run ``iters`` iterations of a workload; returns (and optionally writes as JSON
    lines to the file object ``log``) one record per iteration: b_t, k_t, the k_t-th
    arrival time T_(k_t) (the iteration's virtual duration), the virtual clock, F^_t,
    ||g_t||^2, V^+, ||grad F||^2^+, L^+ and the flags raised."""
    import json
    import time
    if it is None:
        it = Iteration(wl, device=device, static_b=static_b, blind=blind, received=received, clock=clock)
    out = []
    for t in range(start, start + iters):
        it.load_inputs(t)
        t0 = time.perf_counter()
        it.step()
        torch.cuda.synchronize(it.device)
        rec = it.record(t, (time.perf_counter() - t0) * 1e3)
        out.append(rec)
        if log is not None:
            log.write(json.dumps(rec) + "\n")
    return out, it


def _main(argv=None):
    import argparse
    import sys
    from . import workloads
    p = argparse.ArgumentParser(description="Run a DBW workload and log one JSON line per iteration.")
    p.add_argument("--workload", default=workloads.MLP784.key, choices=list(workloads.ALL))
    p.add_argument("--iters", type=int, default=None)
    p.add_argument("--static-b", type=int, default=None)
    p.add_argument("--blind", action="store_true", help="B-DBW: the gain of k is k itself")
    p.add_argument("--received", action="store_true",
                   help="received workers only, without the [n, d] gradient matrix")
    p.add_argument("--clock", default="psi", choices=["psi", "psw"],
                   help="push-and-interrupt (fresh times) or push-and-wait (residual times, Eq. (17) estimator)")
    p.add_argument("--log", default="-")
    a = p.parse_args(argv)
    wl = workloads.ALL[a.workload]
    f = sys.stdout if a.log == "-" else open(a.log, "w")
    try:
        run(wl, a.iters or wl.iters, f, a.static_b, a.blind, received=a.received, clock=a.clock)
    finally:
        if f is not sys.stdout:
            f.close()


if __name__ == "__main__":
    _main()
