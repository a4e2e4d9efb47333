"""GPU parity on the workloads themselves, at their full sizes: the static-b sweep
of the softmax-regression workload as independent trajectories, and the largest
point of the aggregation-only sweep (n = 256, d = 1e8, a 102 GB gradient matrix)
checked on sampled columns and rows against the oracle and through identities
that hold at any size."""
import math

import numpy as np
import pytest
import torch

from oracle import dbw_oracle as O
from paper_2004_14696_gb300 import dbw, inputs, workloads
from paper_2004_14696_gb300.pipeline import Iteration
from gpu_util import RTOL_FP32, assert_close_rows, assert_close_scalar, assert_worker_grads_match

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


@pytest.mark.parametrize("b,rule", [(0, "fixed"), (5, "fixed"), (15, "fixed"), (8, "proportional")])
def test_softmax_static_b_trajectory(b, rule):
    """Softmax regression (784 -> 10, n = 16, B = 32) with a static number of backup
    workers (and, for one case, the proportional learning-rate rule lr * k / n of
    Sect. 4): GPU and oracle run 12 iterations each from the same seeds."""
    from dataclasses import replace
    wl = replace(workloads.SOFTMAX784, lr_rule=rule)
    it = Iteration(wl, static_b=b, keep_gbar=True)
    pool, labels = it.pool.cpu().numpy(), it.labels.cpu().numpy()
    ost = O.State(n=wl.n, D=wl.D)
    w_or = inputs.kaiming_uniform_params(wl.seed, wl.widths).astype(np.float64)
    for t in range(12):
        idx, times = it.host_inputs(t)
        it.load_inputs(t)
        it.step()
        torch.cuda.synchronize()
        ref = O.step(ost, wl.widths, w_or, pool[idx], labels[idx], times, wl.B, wl.lr_for(wl.n - b), wl.beta, b=b)
        assert np.array_equal(it.mask.cpu().numpy(), ref["mask"])
        assert_worker_grads_match(it.G.cpu().numpy()[:, :wl.d], it.loss.cpu().numpy(), wl.widths, w_or, pool[idx],
                                  labels[idx], wl.B, False, range(wl.n), RTOL_FP32)
        assert_close_rows(it.w.cpu().numpy(), ref["w"], RTOL_FP32, "w")
        s = it.stats.cpu().numpy()
        assert_close_scalar(s[dbw.STAT_F], ref["F"], RTOL_FP32, "F")
        if ref["k"] >= 2:
            assert_close_scalar(s[dbw.STAT_SS], ref["SS"], RTOL_FP32, "SS")
        assert s[dbw.STAT_VCLOCK] == ref["vclock"]
        w_or = ref["w"]


def test_aggregation_largest_sweep_point_sampled():
    """n = 256, d = 1e8 (G is 102.4 GB), b = n/4: the masked mean and SGD step on
    sampled column blocks (and the ragged tail) against the oracle, two received
    rows' squared norms against the oracle, and the identity
    sum_j ||g_j||^2 - k ||g_t||^2 = sum of squared deviations at full size."""
    n, d, b = 256, 10**8, 64
    ld = inputs.round_up(d, 4)
    lr = 0.05
    gen = torch.Generator(device="cuda")
    gen.manual_seed(inputs.BASE_SEED + 3)
    G = torch.randn((n, ld), generator=gen, device="cuda", dtype=torch.float32)
    G.add_(0.25)                                    # a nonzero column mean
    w = torch.randn(d, generator=gen, device="cuda", dtype=torch.float32)
    times = inputs.completion_times(inputs.BASE_SEED + 3, 0, n, "shifted_exp", shift=0.0, rate=1.0)
    rng = np.random.default_rng(5)
    blocks = [int(c) for c in rng.integers(0, d // 4096 - 1, size=4) * 4096] + [d - 3001]
    w_before = {c: w[c:c + 4096].cpu().numpy() for c in blocks}
    G_blocks = {c: G[:, c:min(c + 4096, d)].cpu().numpy() for c in blocks}

    tdev = torch.from_numpy(times).cuda()
    bt = torch.tensor([b], dtype=torch.int32, device="cuda")
    order = torch.empty(n, dtype=torch.int32, device="cuda")
    mask = torch.empty(n, dtype=torch.uint8, device="cuda")
    ts = torch.empty(n, dtype=torch.float64, device="cuda")
    dbw.dbw_select_fastest(tdev, bt, order, mask, ts)
    part = torch.empty(dbw.dbw_aggregate_partials_bytes(n, d), dtype=torch.uint8, device="cuda")
    gbar = torch.empty(d, dtype=torch.float32, device="cuda")
    dbw.dbw_aggregate_update(G, n, d, mask, lr, w, part, gbar)
    state = dbw.new_state(n, 5)
    stats = torch.empty(dbw.STATS_LEN, dtype=torch.float64, device="cuda")
    rn = torch.empty(n, dtype=torch.float64, device="cuda")
    dbw.dbw_grad_stats(part, n, mask, torch.zeros(n, dtype=torch.float32, device="cuda"), ts, lr, state, stats, rn)
    torch.cuda.synchronize()

    _, mask_or, _ = O.select_fastest(times, b)
    assert np.array_equal(mask.cpu().numpy(), mask_or)
    for c in blocks:
        gb_ref = O.aggregate(G_blocks[c], mask_or)
        width = gb_ref.shape[0]
        assert_close_rows(gbar[c:c + width].cpu().numpy(), gb_ref, RTOL_FP32, f"g_t[{c}:]")
        assert_close_rows(w[c:c + width].cpu().numpy(), O.sgd_update(w_before[c][:width], gb_ref, lr), RTOL_FP32,
                          f"w[{c}:]")
    sel = np.flatnonzero(mask_or)
    for j in (int(sel[0]), int(sel[-1])):
        row = G[j, :d].cpu().numpy().astype(np.float64)
        assert_close_scalar(rn[j].item(), float(row @ row), RTOL_FP32, f"||g_{j}||^2")
    s = stats.cpu().numpy()
    k = n - b
    r = rn.cpu().numpy()
    lhs = float(np.nansum(r)) - k * s[dbw.STAT_GBAR_SQ]
    assert math.isclose(lhs, s[dbw.STAT_SS], rel_tol=1e-6)
    assert s[dbw.STAT_K] == k
    del G, w, gbar
    torch.cuda.empty_cache()


def test_checkpoint_resume_is_bit_exact_and_run_is_deterministic():
    """Resuming from (w, estimator state) reproduces the uninterrupted run bit for bit,
    which also shows that every kernel of the iteration is deterministic."""
    from paper_2004_14696_gb300.pipeline import run
    wl = workloads.Workload(key="ckpt_bf16", widths=(256, 128, 64, 10), n=8, B=32, prec=workloads.PREC_BF16,
                            S=500, feature_dist="normal", time_model="pareto", time_params={"alpha": 2.0},
                            lr=0.01, seed_offset=81)
    recs, it = run(wl, 4)
    ck = it.checkpoint()
    later, it = run(wl, 3, start=4, it=it)
    w_end = it.w.cpu().clone()
    it.restore(ck)
    again, it = run(wl, 3, start=4, it=it)
    assert torch.equal(it.w.cpu(), w_end)
    for a, b in zip(later, again):
        a.pop("wall_ms")
        b.pop("wall_ms")
        assert a.keys() == b.keys()
        for key in a:
            assert (a[key] == b[key]) or (a[key] != a[key] and b[key] != b[key]), key
    assert [r["t"] for r in recs] == [0, 1, 2, 3]


@pytest.mark.parametrize("form", ["fp32", "bf16", "received", "psw"])
def test_graph_replay_is_the_same_iteration(form):
    """One iteration captured as a CUDA graph and replayed gives, step after step, the
    bits eager launches give from the same state (every kernel is deterministic and
    nothing in an iteration reads back to the host)."""
    from paper_2004_14696_gb300.pipeline import Iteration
    if form == "fp32":
        wl, kw = workloads.MLP784, {}
    else:
        wl = workloads.Workload(key="graph_bf16", widths=(256, 128, 64, 10), n=16, B=32, prec=workloads.PREC_BF16,
                                S=900, feature_dist="normal", time_model="pareto", time_params={"alpha": 2.0},
                                lr=0.01, seed_offset=97)
        kw = {"received": form == "received", "clock": "psw" if form == "psw" else "psi"}
    eager = Iteration(wl, **kw)
    graphed = Iteration(wl, **kw)
    graphed.load_inputs(0)
    ck = eager.checkpoint()
    graphed.capture()              # its warm-up steps moved graphed's state: restart both from ck
    graphed.restore(ck)
    if form == "psw":
        dbw.dbw_psw_init(graphed.psw, wl.n)
        graphed.T_hat.fill_(float("nan"))
    for t in range(5):
        eager.load_inputs(t)
        eager.step()
        graphed.load_inputs(t)
        graphed.replay()
        torch.cuda.synchronize()
        assert torch.equal(eager.w, graphed.w), t
        assert torch.equal(eager.stats.view(torch.int64), graphed.stats.view(torch.int64)), t
        assert torch.equal(eager.b, graphed.b) and torch.equal(eager.mask, graphed.mask), t
        if form == "psw":
            assert torch.equal(eager.psw, graphed.psw), t


def test_debug_sync_mode():
    """DBW_DEBUG_SYNC=1 (read once per process): every call synchronises its stream
    before returning, except while the stream is being captured into a graph; eager
    steps and a captured, replayed iteration both still run clean."""
    import os
    import subprocess
    import sys
    code = r'''
import torch
import __graft_entry__
__graft_entry__.build()
from paper_2004_14696_gb300 import workloads
from paper_2004_14696_gb300.pipeline import Iteration
wl = workloads.Workload(key="dbgsync", widths=(256, 128, 10), n=8, B=32, prec=workloads.PREC_BF16, S=300,
                        feature_dist="normal", time_model="pareto", time_params={"alpha": 2.0}, lr=0.01,
                        seed_offset=96)
for received in (False, True):
    it = Iteration(wl, received=received)
    for t in range(3):
        it.load_inputs(t)
        it.step()
    it.capture()
    it.load_inputs(3)
    it.replay()
    torch.cuda.synchronize()
    assert int(it.ws[:4].view(torch.int32).item()) == 0
print("ok")
'''
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = dict(os.environ, DBW_DEBUG_SYNC="1", PYTHONPATH=root)
    out = subprocess.run([sys.executable, "-c", code], cwd=root, env=env, capture_output=True, text=True, timeout=600)
    assert out.returncode == 0 and out.stdout.strip().endswith("ok"), out.stderr[-3000:]
