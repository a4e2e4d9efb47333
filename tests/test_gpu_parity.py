"""GPU parity of every libdbw entry point against the fp64 CPU oracle, called
through the C ABI on seeded inputs: bit-exact selection and b, fp32 results
within 1e-5 and bf16-GEMM results within 2e-2 (row-rms relative)."""
import math

import numpy as np
import pytest
import torch

from oracle import dbw_oracle as O
from paper_2004_14696_gb300 import dbw, inputs, workloads
from paper_2004_14696_gb300.pipeline import Iteration, agg_case
from gpu_util import RTOL_BF16, RTOL_FP32, assert_close_rows, assert_close_scalar

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def dev(x):
    return torch.as_tensor(np.ascontiguousarray(x)).cuda()


def gpu_select(times, b):
    n = len(times)
    out = dict(order=torch.empty(n, dtype=torch.int32, device="cuda"),
               mask=torch.empty(n, dtype=torch.uint8, device="cuda"),
               tsorted=torch.empty(n, dtype=torch.float64, device="cuda"),
               k=torch.empty(1, dtype=torch.int32, device="cuda"))
    dbw.dbw_select_fastest(dev(times), dev(np.int32([b])), out["order"], out["mask"], out["tsorted"], out["k"])
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in out.items()}


def to_oracle_state(s: dbw.DbwState) -> O.State:
    st = O.State(n=s.n, D=s.D)
    for f in ("t", "k_last", "c", "cntV", "cntN", "cntL", "flags", "has_last"):
        setattr(st, f, int(getattr(s, f)))
    for f in ("F_last", "F_prev", "N_last", "V_last", "vclock"):
        setattr(st, f, float(getattr(s, f)))
    st.ringV, st.ringN, st.ringL = list(s.ringV), list(s.ringN), list(s.ringL)
    st.S = list(s.S)[: s.n]
    return st


def bits(x):
    return np.float64(x).view(np.uint64)


def assert_state_equal(g: dbw.DbwState, o: O.State):
    for f in ("t", "k_last", "c", "cntV", "cntN", "cntL", "flags", "has_last"):
        assert int(getattr(g, f)) == getattr(o, f), f
    for f in ("F_last", "F_prev", "N_last", "V_last", "vclock"):
        assert bits(getattr(g, f)) == bits(getattr(o, f)), (f, getattr(g, f), getattr(o, f))
    for name in ("ringV", "ringN", "ringL"):
        assert np.array_equal(np.array(getattr(g, name)).view(np.uint64),
                              np.array(getattr(o, name), dtype=np.float64).view(np.uint64)), name
    assert np.array_equal(np.array(g.S[: g.n]).view(np.uint64), np.array(o.S, dtype=np.float64).view(np.uint64))


# ================================================================ selection
@pytest.mark.parametrize("n", [1, 2, 3, 16, 33, 64, 255, 256, 1000, 1024])
def test_select_bit_exact(n):
    rng = np.random.default_rng(n)
    for times in (rng.exponential(size=n), rng.integers(0, max(2, n // 4), size=n).astype(np.float64)):
        for b in sorted({0, 1 % n, n // 4, n - 1}):
            got = gpu_select(times, b)
            order, mask, ts = O.select_fastest(times, b)
            assert np.array_equal(got["order"], order)
            assert np.array_equal(got["mask"], mask)
            assert np.array_equal(got["tsorted"].view(np.uint64), ts.view(np.uint64))
            assert int(got["k"][0]) == n - b


def test_select_clamps_out_of_range_b():
    times = np.random.default_rng(0).exponential(size=10)
    assert int(gpu_select(times, -3)["k"][0]) == 10
    got = gpu_select(times, 99)
    assert int(got["k"][0]) == 1 and got["mask"].sum() == 1


# ================================================================ aggregation
AGG_CASES = [(1, 5, 0), (2, 7, 1), (5, 3, 2), (16, 1000, 0), (16, 1000, 4), (16, 1000, 15),
             (64, 12345, 16), (256, 4099, 0), (256, 4099, 255), (7, 256 * 37 + 1, 3), (3, 100003, 1)]


def run_agg(G, w, times, b, lr, loss=None, gbar=True):
    n, ld = G.shape
    d = w.shape[0]
    sel = gpu_select(times, b)
    Gd, wd, maskd = dev(G), dev(w), dev(sel["mask"])
    part = torch.empty(dbw.dbw_aggregate_partials_bytes(n, d), dtype=torch.uint8, device="cuda")
    gb = torch.empty(d, dtype=torch.float32, device="cuda") if gbar else None
    dbw.dbw_aggregate_update(Gd, n, d, maskd, lr, wd, part, gb)
    state = dbw.new_state(n, 5)
    stats = torch.empty(dbw.STATS_LEN, dtype=torch.float64, device="cuda")
    rn = torch.empty(n, dtype=torch.float64, device="cuda")
    loss = np.zeros(n, np.float32) if loss is None else loss
    dbw.dbw_grad_stats(part, n, maskd, dev(loss), dev(sel["tsorted"]), lr, state, stats, rn)
    torch.cuda.synchronize()
    return sel, wd.cpu().numpy(), (gb.cpu().numpy() if gbar else None), stats.cpu().numpy(), rn.cpu().numpy()


@pytest.mark.parametrize("n,d,b", AGG_CASES)
def test_aggregate_parity(n, d, b):
    G, w, times = agg_case(n, d, seed=1000 + n + d, b=b, mean=0.3)
    lr = 0.05
    sel, w_gpu, gbar_gpu, stats, rn = run_agg(G, w, times, b, lr)
    _, mask, _ = O.select_fastest(times, b)
    Gd = G[:, :d]
    gbar = O.aggregate(Gd, mask)
    assert_close_rows(gbar_gpu, gbar, RTOL_FP32, "g_t")
    assert_close_rows(w_gpu, O.sgd_update(w, gbar, lr), RTOL_FP32, "w_{t+1}")
    k = n - b
    SS = O.deviation_sumsq(Gd, mask, gbar)
    assert stats[dbw.STAT_K] == k
    assert_close_scalar(stats[dbw.STAT_GBAR_SQ], float(gbar @ gbar), RTOL_FP32, "||g_t||^2")
    if k >= 2:
        assert_close_scalar(stats[dbw.STAT_SS], SS, RTOL_FP32, "SS")
    else:
        assert stats[dbw.STAT_SS] == 0.0 and math.isnan(stats[dbw.STAT_V])
    r = O.row_sqnorms(Gd, mask)
    assert np.array_equal(np.isnan(rn), np.isnan(r))
    assert_close_rows(rn[~np.isnan(r)], r[~np.isnan(r)], RTOL_FP32, "row norms")


def test_aggregate_is_permutation_invariant_on_gpu():
    n, d = 32, 5000
    G, w, times = agg_case(n, d, seed=7, b=8)
    perm = np.random.default_rng(3).permutation(n)
    _, w1, g1, s1, _ = run_agg(G, w, times, 8, 0.1)
    _, w2, g2, s2, _ = run_agg(G[perm], w, times[perm], 8, 0.1)
    assert_close_rows(g1, g2, RTOL_FP32, "permuted g_t")
    assert_close_scalar(s1[dbw.STAT_SS], s2[dbw.STAT_SS], RTOL_FP32, "permuted SS")


def test_aggregate_does_not_read_padding_or_unselected_rows():
    n, d = 8, 1001
    G, w, times = agg_case(n, d, seed=5, b=3)      # padding columns are NaN
    _, mask, _ = O.select_fastest(times, 3)
    G[mask == 0, :] = np.nan                          # unselected rows poisoned too
    _, w_gpu, g_gpu, stats, _ = run_agg(G, w, times, 3, 0.1)
    assert np.isfinite(w_gpu).all() and np.isfinite(g_gpu).all()
    assert np.isfinite(stats[dbw.STAT_SS]) and np.isfinite(stats[dbw.STAT_GBAR_SQ])


# ================================================================ estimator
def test_estimator_sequence_teacher_forced_bit_exact():
    """Every iteration: GPU b_t equals the oracle's on the GPU's own state (bit for bit,
    ratios included), and the state after dbw_grad_stats equals the oracle's bookkeeping
    applied to the GPU's reduced sums."""
    n, d, D, lr, beta = 16, 3001, 5, 0.05, 1.01
    rng = np.random.default_rng(42)
    state = dbw.new_state(n, D)
    b = torch.zeros(1, dtype=torch.int32, device="cuda")
    ratio = torch.empty(n, dtype=torch.float64, device="cuda")
    part = torch.empty(dbw.dbw_aggregate_partials_bytes(n, d), dtype=torch.uint8, device="cuda")
    stats = torch.empty(dbw.STATS_LEN, dtype=torch.float64, device="cuda")
    w = dev(rng.standard_normal(d).astype(np.float32))
    decisions = set()
    F, prev = 50.0, None
    for t in range(60):
        ost = to_oracle_state(dbw.read_state(state))
        dbw.dbw_choose_b(state, lr, beta, b, ratio)
        torch.cuda.synchronize()
        k_or, ratio_or = O.choose_k(ost, lr, beta)
        assert n - int(b.item()) == k_or, t
        assert np.array_equal(ratio.cpu().numpy().view(np.uint64), np.array(ratio_or).view(np.uint64)), t
        decisions.add(k_or)
        # gradients whose mean shrinks over time (N falls towards V/k, so k_t should grow);
        # losses fall by the gain Eq. (9) predicts for L = 5, with a bump every 9 iterations
        # that trips the guard of Eq. (19)
        mu = 0.5 * math.exp(-t / 12.0)
        G = (mu + rng.standard_normal((n, d))).astype(np.float32)
        G = np.pad(G, ((0, 0), (0, inputs.round_up(d, 4) - d)))
        times = np.round(1.0 + rng.exponential(size=n), 1)     # ties happen
        if prev is not None:
            N, V, kk = prev
            F = F - ((lr - 5 * lr * lr / 2) * N - (5 * lr * lr / 2) * V / kk) + (0.5 if t % 9 == 4 else 0.0)
        loss = (F + 0.01 * rng.standard_normal(n)).astype(np.float32)
        sel = gpu_select(times, int(b.item()))
        dbw.dbw_aggregate_update(dev(G), n, d, dev(sel["mask"]), lr, w, part)
        dbw.dbw_grad_stats(part, n, dev(sel["mask"]), dev(loss), dev(sel["tsorted"]), lr, state, stats)
        torch.cuda.synchronize()
        s = stats.cpu().numpy()
        k = int(s[dbw.STAT_K])
        prev = (float(s[dbw.STAT_N]), float(s[dbw.STAT_V]), k) if k >= 2 else None
        O.record_iteration(ost, k, float(s[dbw.STAT_SS]), float(s[dbw.STAT_GBAR_SQ]), loss,
                           sel["mask"], sel["tsorted"], lr)
        assert_state_equal(dbw.read_state(state), ost)
    assert len(decisions) > 5, decisions      # the estimator actually moved


def test_blind_variant_bit_exact():
    n = 12
    state = dbw.new_state(n, 5)
    part = torch.empty(dbw.dbw_aggregate_partials_bytes(n, 64), dtype=torch.uint8, device="cuda")
    b = torch.zeros(1, dtype=torch.int32, device="cuda")
    ratio = torch.empty(n, dtype=torch.float64, device="cuda")
    rng = np.random.default_rng(1)
    w = dev(np.zeros(64, np.float32))
    for t in range(5):
        times = 1.0 + rng.exponential(size=n)
        sel = gpu_select(times, 0)
        G = rng.standard_normal((n, 64)).astype(np.float32)
        dbw.dbw_aggregate_update(dev(G), n, 64, dev(sel["mask"]), 0.1, w, part)
        dbw.dbw_grad_stats(part, n, dev(sel["mask"]), dev(np.ones(n, np.float32)), dev(sel["tsorted"]), 0.1, state)
    ost = to_oracle_state(dbw.read_state(state))
    dbw.dbw_choose_b(state, 0.1, 1.01, b, ratio, flags=dbw.CHOOSE_BLIND)
    torch.cuda.synchronize()
    k, r = O.choose_k(ost, 0.1, 1.01, blind=True)
    assert n - int(b.item()) == k
    assert np.array_equal(ratio.cpu().numpy().view(np.uint64), np.array(r).view(np.uint64))


def test_empty_mask_and_bad_state_raise_flags_without_fault():
    n, d = 4, 16
    state = dbw.new_state(n, 5)
    part = torch.empty(dbw.dbw_aggregate_partials_bytes(n, d), dtype=torch.uint8, device="cuda")
    w = dev(np.ones(d, np.float32))
    mask = dev(np.zeros(n, np.uint8))
    dbw.dbw_aggregate_update(dev(np.ones((n, d), np.float32)), n, d, mask, 0.1, w, part)
    dbw.dbw_grad_stats(part, n, mask, dev(np.ones(n, np.float32)), dev(np.arange(n, dtype=np.float64)), 0.1, state)
    torch.cuda.synchronize()
    s = dbw.read_state(state)
    assert s.flags & dbw.FLAG_EMPTY_MASK and s.t == 0
    assert np.array_equal(w.cpu().numpy(), np.ones(d, np.float32))
    dbw.dbw_grad_stats(part, n + 1, dev(np.ones(n + 1, np.uint8)), dev(np.ones(n + 1, np.float32)),
                       dev(np.arange(n + 1, dtype=np.float64)), 0.1, state)
    torch.cuda.synchronize()
    assert dbw.read_state(state).flags & dbw.FLAG_BAD_STATE


# ================================================================ worker gradients
SMALL_BF16 = workloads.Workload(
    key="small_bf16", widths=(256, 128, 64, 10), n=8, B=16, prec=workloads.PREC_BF16, S=500,
    feature_dist="normal", time_model="exp_slow", time_params={"rate": 1.0, "frac": 0.25, "factor": 10.0},
    lr=0.01, seed_offset=77)
SMALL_FP32_RAGGED = workloads.Workload(
    key="small_fp32", widths=(132, 200, 70, 7), n=5, B=3, prec=workloads.PREC_FP32, S=50,
    feature_dist="uniform", time_model="pareto", time_params={"alpha": 2.0, "xm": 1.0}, lr=0.05, seed_offset=78)


def grads_case(wl, t=0):
    it = Iteration(wl, static_b=0)
    idx, times = it.host_inputs(t)
    it.load_inputs(t)
    dbw.dbw_worker_grads(wl.widths, wl.prec, it.w, it.pool, it.labels, it.idx, wl.n, wl.B, it.G, it.loss, it.ws)
    torch.cuda.synchronize()
    return it, idx


@pytest.mark.parametrize("wl", [workloads.SOFTMAX784, workloads.MLP784, SMALL_FP32_RAGGED, SMALL_BF16],
                         ids=lambda w: w.key)
def test_worker_grads_parity_full(wl):
    it, idx = grads_case(wl)
    pool, labels, w = it.pool.cpu().numpy(), it.labels.cpu().numpy(), it.w.cpu().numpy()
    G, loss = O.worker_grads(wl.widths, w, pool[idx], labels[idx], wl.n, wl.B, bf16=wl.prec == workloads.PREC_BF16)
    rtol = RTOL_BF16 if wl.prec == workloads.PREC_BF16 else RTOL_FP32
    assert_close_rows(it.G.cpu().numpy()[:, :wl.d], G, rtol, "G")
    assert_close_rows(it.loss.cpu().numpy(), loss, rtol, "loss")


@pytest.mark.parametrize("wl", [workloads.MLP3072], ids=lambda w: w.key)
def test_worker_grads_parity_sampled_workers(wl):
    """Full-size bf16 config: the oracle recomputes a few sampled workers from their own minibatch."""
    it, idx = grads_case(wl)
    pool, labels, w = it.pool.cpu().numpy(), it.labels.cpu().numpy(), it.w.cpu().numpy()
    for i in (0, wl.n - 1, 37):
        rows = idx[i * wl.B:(i + 1) * wl.B]
        g, l = O.single_worker_grad(wl.widths, w, pool[rows], labels[rows], wl.B, bf16=True)
        assert_close_rows(it.G[i, :wl.d].cpu().numpy(), g, RTOL_BF16, f"G row {i}")
        assert_close_scalar(it.loss[i].item(), l, RTOL_BF16, f"loss {i}")


def test_bad_sample_index_poisons_only_that_worker():
    wl = SMALL_FP32_RAGGED
    it = Iteration(wl, static_b=0)
    idx, _ = it.host_inputs(0)
    idx[wl.B + 1] = wl.S + 7          # worker 1 gets an out-of-range sample
    it.idx.copy_(torch.from_numpy(idx))
    dbw.dbw_worker_grads(wl.widths, wl.prec, it.w, it.pool, it.labels, it.idx, wl.n, wl.B, it.G, it.loss, it.ws)
    torch.cuda.synchronize()
    loss = it.loss.cpu().numpy()
    assert np.isnan(loss[1]) and np.isfinite(np.delete(loss, 1)).all()
    G = it.G.cpu().numpy()[:, :wl.d]
    assert np.isnan(G[1]).all() and np.isfinite(np.delete(G, 1, axis=0)).all()


# ================================================================ whole iterations
@pytest.mark.parametrize("wl,iters", [(workloads.MLP784, 6), (SMALL_BF16, 8)], ids=["mlp784", "small_bf16"])
def test_dbw_iterations_teacher_forced(wl, iters):
    """Whole DBW iterations through the pipeline; each is compared with the oracle
    started from the GPU's own w_t and state (teacher forcing)."""
    it = Iteration(wl, keep_gbar=True)
    pool, labels = it.pool.cpu().numpy(), it.labels.cpu().numpy()
    bf16 = wl.prec == workloads.PREC_BF16
    rtol = RTOL_BF16 if bf16 else RTOL_FP32
    for t in range(iters):
        w0 = it.w.cpu().numpy().copy()
        ost = to_oracle_state(dbw.read_state(it.state))
        idx, times = it.host_inputs(t)
        it.load_inputs(t)
        it.step()
        torch.cuda.synchronize()
        k_or, _ = O.choose_k(ost, wl.lr, wl.beta)
        b = int(it.b.item())
        assert wl.n - b == k_or, t
        ref = O.step(ost, wl.widths, w0, pool[idx], labels[idx], times, wl.B, wl.lr, wl.beta, bf16=bf16, b=b)
        assert np.array_equal(it.mask.cpu().numpy(), ref["mask"])
        assert np.array_equal(it.order.cpu().numpy(), ref["order"])
        assert_close_rows(it.G.cpu().numpy()[:, :wl.d], ref["G"], rtol, "G")
        assert_close_rows(it.gbar.cpu().numpy(), ref["gbar"], rtol, "g_t")
        assert_close_rows(it.w.cpu().numpy(), ref["w"], rtol, "w")
        s = it.stats.cpu().numpy()
        assert_close_scalar(s[dbw.STAT_GBAR_SQ], ref["gbar_sq"], rtol, "||g_t||^2")
        if ref["k"] >= 2:
            assert_close_scalar(s[dbw.STAT_SS], ref["SS"], rtol, "SS")
        assert_close_scalar(s[dbw.STAT_F], ref["F"], rtol, "F")
