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
from gpu_util import (RTOL_BF16, RTOL_FP32, assert_close_rows, assert_close_scalar, assert_close_to_magnitude,
                      assert_worker_grads_match, gpu_active_sets, param_blocks, tensor_scale)

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


def same_f64(a, b):
    """Bit-identical fp64 arrays, except that any NaN matches any NaN (payload and sign
    of a NaN carry no meaning here and differ between the CUDA and numpy defaults)."""
    a = np.atleast_1d(np.asarray(a, dtype=np.float64))
    b = np.atleast_1d(np.asarray(b, dtype=np.float64))
    if a.shape != b.shape:
        return False
    na, nb = np.isnan(a), np.isnan(b)
    return bool(np.array_equal(na, nb) and np.array_equal(a[~na].view(np.uint64), b[~nb].view(np.uint64)))


def assert_state_equal(g: dbw.DbwState, o: O.State):
    for f in ("t", "k_last", "c", "cntV", "cntN", "cntL", "flags", "has_last"):
        assert int(getattr(g, f)) == getattr(o, f), f
    for f in ("F_last", "F_prev", "N_last", "V_last", "vclock"):
        assert same_f64(getattr(g, f), getattr(o, f)), (f, getattr(g, f), getattr(o, f))
    for name in ("ringV", "ringN", "ringL"):
        assert same_f64(list(getattr(g, name)), getattr(o, name)), name
    assert same_f64(list(g.S[: g.n]), o.S)


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
            assert same_f64(got["tsorted"], ts)
            assert int(got["k"][0]) == n - b


def test_select_negative_times_and_signed_zeros():
    """The comparisons order the doubles themselves: negative times, subnormals, and -0
    equal to +0 (so their tie goes to the lower index), as the oracle's sort does."""
    times = np.array([0.0, -0.0, -1.5, 2.0, -5e-324, 5e-324, -0.0, 0.0, 3.0, -2.0, -1.5, 1e300, -1e300, 2.0],
                     dtype=np.float64)
    for b in range(len(times)):
        got = gpu_select(times, b)
        order, mask, ts = O.select_fastest(times, b)
        assert np.array_equal(got["order"], order)
        assert np.array_equal(got["mask"], mask)
        assert same_f64(got["tsorted"], ts)


def test_select_clamps_out_of_range_b():
    times = np.random.default_rng(0).exponential(size=10)
    assert int(gpu_select(times, -3)["k"][0]) == 10
    got = gpu_select(times, 99)
    assert int(got["k"][0]) == 1 and got["mask"].sum() == 1


# ================================================================ aggregation
AGG_CASES = [(1, 5, 0), (2, 7, 1), (5, 3, 2), (16, 1000, 0), (16, 1000, 4), (16, 1000, 15),
             (64, 12345, 16), (256, 4099, 0), (256, 4099, 255), (7, 256 * 37 + 1, 3), (3, 100003, 1)]


def run_agg(G, w, times, b, lr, loss=None, gbar=True, flags=0):
    n, ld = G.shape
    d = w.shape[0]
    sel = gpu_select(times, b)
    Gd, wd, maskd = dev(G), dev(w), dev(sel["mask"])
    part = torch.empty(dbw.dbw_aggregate_partials_bytes(n, d), dtype=torch.uint8, device="cuda")
    gb = torch.empty(d, dtype=torch.float32, device="cuda") if gbar else None
    dbw.dbw_aggregate_update(Gd, n, d, maskd, lr, wd, part, gb, flags=flags)
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


@pytest.mark.parametrize("n,d,b", [(2, 7, 1), (16, 1000, 4), (16, 1000, 15), (64, 12345, 16), (256, 4099, 0),
                                   (256, 4099, 255), (7, 256 * 37 + 1, 3), (3, 100003, 2)])
def test_aggregate_all_row_norms(n, d, b):
    """DBW_ALL_ROW_NORMS (R12): the rows the mask leaves out are read for their
    squared norms, against the oracle; g_t, w_{t+1}, SS, ||g_t||^2 and the received
    rows' norms are bit for bit those of the default call (the received rows go
    through the same arithmetic in the same order)."""
    G, w, times = agg_case(n, d, seed=2000 + n + d, b=b, mean=0.3)
    lr = 0.05
    _, w0, g0, s0, rn0 = run_agg(G, w, times, b, lr)
    _, w1, g1, s1, rn1 = run_agg(G, w, times, b, lr, flags=dbw.ALL_ROW_NORMS)
    assert np.array_equal(w0, w1) and np.array_equal(g0, g1)
    assert same_f64(s0, s1)
    _, mask, _ = O.select_fastest(times, b)
    m = mask.astype(bool)
    assert np.array_equal(rn0[m], rn1[m]) and np.all(np.isnan(rn0[~m]))
    r = O.row_sqnorms(G[:, :d], mask, all_rows=True)
    assert np.all(np.isfinite(rn1))
    assert_close_rows(rn1, r, RTOL_FP32, "every row's squared norm")


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
# The estimator is checked on seeded inputs handed identically to both sides:
# states built on the host, and partial sums made of dyadic values so that every
# summation order gives the same exact fp64 totals.  Nothing flows from the GPU
# into the oracle.
def fill_state(n, D, rng):
    """A random but consistent estimator state, as (ctypes mirror, oracle State)."""
    g = dbw.DbwState()
    o = O.State(n=n, D=D)
    g.n, g.D = n, D
    vals = dict(t=int(rng.integers(0, 30)), k_last=int(rng.integers(1, n + 1)), c=int(rng.integers(0, 12)),
                cntV=int(rng.integers(0, 3 * D)), cntN=int(rng.integers(0, 3 * D)),
                cntL=int(rng.integers(0, 3 * D)), has_last=int(rng.integers(0, 2)))
    if rng.random() < 0.7:
        vals["cntV"] = max(vals["cntV"], 1)
        vals["cntN"] = max(vals["cntN"], 1)
        vals["cntL"] = max(vals["cntL"], 1)
        vals["c"] = max(vals["c"], 1)
    for k, v in vals.items():
        setattr(g, k, v)
        setattr(o, k, v)
    F_prev = float(rng.uniform(0.5, 3.0))
    F_last = F_prev * float(rng.choice([0.98, 1.0, 1.01, 1.02, 1.3]))
    fl = dict(F_last=F_last, F_prev=F_prev, N_last=float(rng.uniform(0, 2)), V_last=float(rng.uniform(0, 9)),
              vclock=float(rng.uniform(0, 100)))
    for k, v in fl.items():
        setattr(g, k, v)
        setattr(o, k, v)
    ringV = rng.uniform(0, 10, O.DMAX) * rng.choice([0.0, 1.0], O.DMAX, p=[0.1, 0.9])
    ringN = rng.uniform(0, 2, O.DMAX) * rng.choice([0.0, 1.0], O.DMAX, p=[0.2, 0.8])
    ringL = rng.uniform(-2, 40, O.DMAX)
    for name, arr in (("ringV", ringV), ("ringN", ringN), ("ringL", ringL)):
        getattr(g, name)[:] = arr.tolist()
        setattr(o, name, arr.tolist())
    times = np.sort(np.round(rng.exponential(size=n), 2)) * max(vals["c"], 1)
    S = np.zeros(dbw.NMAX)
    S[:n] = times
    g.S[:] = S.tolist()
    o.S = times.tolist()
    return g, o


def test_choose_b_bit_exact_on_seeded_states():
    rng = np.random.default_rng(2024)
    b = torch.zeros(1, dtype=torch.int32, device="cuda")
    for trial in range(400):
        n = int(rng.choice([1, 2, 3, 7, 16, 64, 256, 1024]))
        D = int(rng.choice([1, 3, 5, 64]))
        g, o = fill_state(n, D, rng)
        lr = float(rng.choice([0.01, 0.05, 0.1]))
        beta = float(rng.choice([1.0, 1.01, 1.05]))
        blind = bool(rng.random() < 0.15)
        state = torch.empty(dbw.STATE_BYTES, dtype=torch.uint8, device="cuda")
        dbw.write_state(state, g)
        ratio = torch.empty(n, dtype=torch.float64, device="cuda")
        dbw.dbw_choose_b(state, lr, beta, b, ratio, flags=dbw.CHOOSE_BLIND if blind else 0)
        torch.cuda.synchronize()
        k, r = O.choose_k(o, lr, beta, blind=blind)
        assert n - int(b.item()) == k, trial
        assert same_f64(ratio.cpu().numpy(), r), trial
        assert dbw.read_state(state).k_next == k


def seeded_partials(n, blocks, SS, g2, rows, device="cuda"):
    """A partials buffer (layout of include/dbw.h) whose per-block pieces sum exactly to SS, g2, rows."""
    vals = np.zeros((n + 2, blocks))
    for q, total in list(enumerate(rows)) + [(n, SS), (n + 1, g2)]:
        units = int(round(total * 1024))           # dyadic: multiples of 2^-10
        cuts = np.sort(np.random.default_rng(q).integers(0, units + 1, blocks - 1)) if units > 0 else \
            np.zeros(blocks - 1, dtype=np.int64)
        parts = np.diff(np.concatenate([[0], cuts, [units]]))
        vals[q] = parts / 1024.0
    head = np.array([dbw.PARTIALS_MAGIC, blocks, n, 0], dtype=np.int64).view(np.uint8)
    body = np.concatenate([np.zeros(n + 2), vals.ravel()]).view(np.uint8)
    return dev(np.concatenate([head, body]))


def test_estimator_trajectory_bit_exact():
    """60 DBW iterations of the estimator alone, both sides fed the same seeded sums,
    losses and times: every b_t, ratio vector and state is identical bit for bit, and
    k_t moves the way Sect. 4 describes (small while ||grad F||^2 dominates, growing
    as it falls), with the loss-increase guard tripping on the loss bumps."""
    n, d, D, lr, beta = 16, 3001, 5, 0.05, 1.01
    rng = np.random.default_rng(42)
    state = dbw.new_state(n, D)
    ost = O.State(n=n, D=D)
    b = torch.zeros(1, dtype=torch.int32, device="cuda")
    ratio = torch.empty(n, dtype=torch.float64, device="cuda")
    stats = torch.empty(dbw.STATS_LEN, dtype=torch.float64, device="cuda")
    rn = torch.empty(n, dtype=torch.float64, device="cuda")
    ks = []
    F, prev = 50.0, None
    for t in range(60):
        dbw.dbw_choose_b(state, lr, beta, b, ratio)
        torch.cuda.synchronize()
        k, r = O.choose_k(ost, lr, beta)
        assert n - int(b.item()) == k, t
        assert same_f64(ratio.cpu().numpy(), r), t
        ks.append(k)
        # sums of k rows ~ N(mu_t, 1) in d columns: SS ~ (k-1) d, ||g_t||^2 ~ d mu_t^2 + d / k
        mu = 0.5 * math.exp(-t / 12.0)
        SS = (k - 1) * d * float(rng.uniform(0.95, 1.05))
        g2 = d * mu * mu + d / k * float(rng.uniform(0.9, 1.1))
        times = np.round(1.0 + rng.exponential(size=n), 1)
        if prev is not None:
            N, V, kk = prev
            F = F - ((lr - 5 * lr * lr / 2) * N - (5 * lr * lr / 2) * V / kk) + (0.5 if t % 9 == 4 else 0.0)
        loss = (F + 0.01 * rng.standard_normal(n)).astype(np.float32)
        sel = gpu_select(times, n - k)
        _, mask, ts = O.select_fastest(times, n - k)
        assert np.array_equal(sel["mask"], mask)
        rows = [float(rng.integers(1, 1 << 20)) / 1024.0 if mask[j] else 0.0 for j in range(n)]
        SSq, g2q = round(SS * 1024) / 1024.0, round(g2 * 1024) / 1024.0
        part = seeded_partials(n, 3, SSq, g2q, rows)
        dbw.dbw_grad_stats(part, n, dev(mask), dev(loss), dev(ts), lr, state, stats, rn)
        torch.cuda.synchronize()
        rec = O.record_iteration(ost, k, SSq, g2q, loss, mask, ts, lr)
        assert_state_equal(dbw.read_state(state), ost)
        st = stats.cpu().numpy()
        for key, idx in (("V", dbw.STAT_V), ("N", dbw.STAT_N), ("F", dbw.STAT_F), ("L", dbw.STAT_L),
                         ("SS", dbw.STAT_SS), ("gbar_sq", dbw.STAT_GBAR_SQ), ("vclock", dbw.STAT_VCLOCK)):
            assert same_f64(st[idx], rec[key]), (t, key)
        assert same_f64(rn.cpu().numpy(), [rows[j] if mask[j] else math.nan for j in range(n)])
        prev = (rec["N"], rec["V"], k) if k >= 2 else None
    assert len(set(ks)) > 5 and min(ks) < 8 and ks[-1] == n, ks


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
# B = 32: runs the tcgen05 pass (ragged last layer of 10 classes, partial tiles everywhere)
SMALL_BF16 = workloads.Workload(
    key="small_bf16", widths=(256, 128, 64, 10), n=8, B=32, prec=workloads.PREC_BF16, S=500,
    feature_dist="normal", time_model="exp_slow", time_params={"rate": 1.0, "frac": 0.25, "factor": 10.0},
    lr=0.01, seed_offset=77)
# B = 16 is not whole 32-deep K blocks: the bf16 SIMT pass
SMALL_BF16_SIMT = workloads.Workload(
    key="small_bf16_simt", widths=(200, 96, 10), n=6, B=16, prec=workloads.PREC_BF16, S=300,
    feature_dist="uniform", time_model="shifted_exp", time_params={"shift": 1.0, "rate": 1.0}, lr=0.01,
    seed_offset=79)
# tcgen05 pass with widths that are not multiples of 8 (padded leading dimensions) and several
# K blocks per worker (B = 96 = 3 x 32)
ODD_BF16 = workloads.Workload(
    key="odd_bf16", widths=(300, 200, 100, 7), n=3, B=96, prec=workloads.PREC_BF16, S=400,
    feature_dist="normal", time_model="lognormal", time_params={"mu": 0.0, "sigma": 0.5}, lr=0.01,
    seed_offset=80)
# tcgen05 pass whose second weight block starts off a 16-byte boundary of the G row
# (offset 36*18 + 18 = 666 floats, row length 18): that layer's dW takes the
# one-CTA-per-tile kernel with scalar stores
UNALIGNED_BF16 = workloads.Workload(
    key="unaligned_bf16", widths=(36, 18, 10), n=2, B=32, prec=workloads.PREC_BF16, S=200,
    feature_dist="normal", time_model="shifted_exp", time_params={"shift": 1.0, "rate": 1.0}, lr=0.01,
    seed_offset=81)
# B (C + 8) bf16 larger than the softmax kernel's transposing tile: dZ_L^T by the separate
# transpose kernel
WIDE_BF16 = workloads.Workload(
    key="wide_bf16", widths=(64, 320), n=2, B=256, prec=workloads.PREC_BF16, S=600,
    feature_dist="normal", time_model="shifted_exp", time_params={"shift": 1.0, "rate": 1.0}, lr=0.01,
    seed_offset=82)
# one layer, 7 classes, 132 features: the 16-byte logits kernel on a ragged one-layer shape
SMALL_FP32_LINEAR = workloads.Workload(
    key="small_fp32_linear", widths=(132, 7), n=5, B=3, prec=workloads.PREC_FP32, S=50,
    feature_dist="uniform", time_model="pareto", time_params={"alpha": 2.0, "xm": 1.0}, lr=0.05, seed_offset=85)
SMALL_FP32_RAGGED = workloads.Workload(
    key="small_fp32", widths=(132, 200, 70, 7), n=5, B=3, prec=workloads.PREC_FP32, S=50,
    feature_dist="uniform", time_model="pareto", time_params={"alpha": 2.0, "xm": 1.0}, lr=0.05, seed_offset=78)
# fp32 forward GEMMs of at least 2^27 multiply-adds run in three tf32 passes on the tensor
# cores: M = 11 x 131 = 1441 rows (a partial 128-row tile); layer 1 with K = 1028 (a partial
# 32-deep K block) and 322 outputs (a partial 64-column tile); layer 2, its input from the
# first, with K = 322 (operand rows padded to 324 floats) and 330 outputs; the logits
# layer stays on SIMT
# per-worker weight gradients in three tf32 passes (B = 96: three 32-deep K blocks per
# worker): layer 1 with 200 outputs (a partial 128-row tile) and 516 inputs (a partial
# 128-column tile of 4 columns), layer 2 on the hidden activations (G offset 103,400)
TF32_DW = workloads.Workload(
    key="tf32_dw", widths=(516, 200, 136, 12), n=21, B=96, prec=workloads.PREC_FP32, S=4000,
    feature_dist="uniform", time_model="shifted_exp", time_params={"shift": 1.0, "rate": 1.0}, lr=0.01,
    seed_offset=84)
TF32_RAGGED = workloads.Workload(
    key="tf32_ragged", widths=(1028, 322, 330, 5), n=11, B=131, prec=workloads.PREC_FP32, S=3000,
    feature_dist="normal", time_model="lognormal", time_params={"mu": 0.0, "sigma": 0.5}, lr=0.01,
    seed_offset=83)


def grads_case(wl, t=0):
    it = Iteration(wl, static_b=0)
    idx, times = it.host_inputs(t)
    it.load_inputs(t)
    dbw.dbw_worker_grads(wl.widths, wl.prec, it.w, it.pool, it.labels, it.idx, wl.n, wl.B, it.G, it.loss, it.ws)
    torch.cuda.synchronize()
    assert int(it.ws[:4].view(torch.int32).item()) == 0, "device status word set"
    return it, idx


@pytest.mark.parametrize("wl", [workloads.SOFTMAX784, SMALL_FP32_LINEAR, workloads.MLP784, SMALL_FP32_RAGGED,
                                TF32_RAGGED, TF32_DW, SMALL_BF16, SMALL_BF16_SIMT, ODD_BF16, UNALIGNED_BF16,
                                WIDE_BF16],
                         ids=lambda w: w.key)
def test_worker_grads_parity_full(wl):
    it, idx = grads_case(wl)
    pool, labels, w = it.pool.cpu().numpy(), it.labels.cpu().numpy(), it.w.cpu().numpy()
    bf16 = wl.prec == workloads.PREC_BF16
    rtol = RTOL_BF16 if bf16 else RTOL_FP32
    assert_worker_grads_match(it.G.cpu().numpy()[:, :wl.d], it.loss.cpu().numpy(), wl.widths, w, pool[idx],
                              labels[idx], wl.B, bf16, range(wl.n), rtol,
                              gpu_active_sets(it.ws, wl.widths, wl.n, wl.B, wl.prec))


@pytest.mark.parametrize("wl", [workloads.MLP3072, workloads.MLP4096], ids=lambda w: w.key)
def test_worker_grads_parity_sampled_workers(wl):
    """Full-size bf16 configs, in the launch configuration the bench uses: the oracle
    recomputes sampled workers from their own minibatch (a worker's gradient depends
    only on its B samples and w)."""
    it, idx = grads_case(wl)
    pool, labels, w = it.pool.cpu().numpy(), it.labels.cpu().numpy(), it.w.cpu().numpy()
    workers = (0, 37, wl.n - 1) if wl.n <= 128 else (0, wl.n - 1)
    rows = {i: it.G[i, :wl.d].cpu().numpy() for i in workers}
    assert_worker_grads_match(rows, it.loss.cpu().numpy(), wl.widths, w, pool[idx], labels[idx], wl.B, True,
                              workers, RTOL_BF16, gpu_active_sets(it.ws, wl.widths, wl.n, wl.B, wl.prec))


def test_tf32_forward_on_eight_decades_of_magnitude():
    """The fp32 forward GEMMs in three tf32 passes keep fp32 accuracy whatever the
    operands' exponents: features of random sign and magnitude 10^U(-4, 4), every hidden
    activation of layers 1 and 2 (both in three passes) within 1e-6 of the sum of
    |terms| of its dot product, against the oracle's fp64 pre-activations (the level
    measured on N(0,1) features is about 1e-7)."""
    wl = TF32_RAGGED
    it = Iteration(wl, static_b=0)
    it.load_inputs(0)
    rng = np.random.default_rng(4242)
    S, F = it.pool.shape
    pool = (rng.choice([-1.0, 1.0], size=(S, F)) * 10.0 ** rng.uniform(-4.0, 4.0, size=(S, F))).astype(np.float32)
    it.pool.copy_(torch.from_numpy(pool))
    dbw.dbw_worker_grads(wl.widths, wl.prec, it.w, it.pool, it.labels, it.idx, wl.n, wl.B, it.G, it.loss, it.ws)
    torch.cuda.synchronize()
    assert int(it.ws[:4].view(torch.int32).item()) == 0
    acts = [dbw.hidden_activations(it.ws, wl.widths, wl.n, wl.B, wl.prec, h).cpu().numpy().astype(np.float64)
            for h in (1, 2)]
    idx, labels, w = it.idx.cpu().numpy(), it.labels.cpu().numpy(), it.w.cpu().numpy()
    off1 = wl.widths[0] * wl.widths[1] + wl.widths[1]   # where layer 2's parameters start in w
    worst = 0.0
    for i in range(wl.n):
        rows = slice(i * wl.B, (i + 1) * wl.B)
        y = labels[idx[rows]]
        # layer 1 from the features; layer 2 from the GPU's own layer-1 activations (the
        # oracle's forward of the network above layer 1), so each GEMM is checked alone
        _, _, z1, s1, _ = O.worker_grads(wl.widths, w, pool[idx[rows]].astype(np.float64), y, 1, wl.B, False,
                                         return_preact=True, return_magnitude=True)
        _, _, z2, s2, _ = O.worker_grads(wl.widths[1:], w[off1:], acts[0][rows], y, 1, wl.B, False,
                                         return_preact=True, return_magnitude=True)
        for z, sc, a in ((z1[0], s1[0], acts[0][rows]), (z2[0], s2[0], acts[1][rows])):
            ratio = np.abs(np.maximum(z, 0.0) - a) / (1e-6 * sc)
            worst = max(worst, float(ratio.max()))
    assert worst <= 1.0, f"worst activation error {worst:.3g} x 1e-6 of its sum of |terms|"


@pytest.mark.parametrize("wl", [SMALL_FP32_RAGGED, SMALL_FP32_LINEAR], ids=lambda w: w.key)
def test_bad_sample_index_poisons_only_that_worker(wl):
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
def decision_margin(st: O.State, lr, beta):
    """How far the oracle's b_t is from flipping: the relative gap between the best and
    the runner-up ratio of Eq. (18), and of the guard comparison of Eq. (19)."""
    gains = O.gain_estimates(st, lr)
    gaps = [math.inf]
    if gains is not None:
        T = O.time_estimates(st)
        r = sorted((g / t for g, t in zip(gains, T) if g > 0), reverse=True)
        if len(r) >= 2:
            gaps.append((r[0] - r[1]) / abs(r[0]))
        gaps.append(min(abs(g) for g in gains) / max(abs(g) for g in gains) if max(abs(g) for g in gains) > 0
                    else math.inf)
    if st.t >= 2 and st.k_last < st.n:
        gaps.append(abs(st.F_last - beta * st.F_prev) / abs(st.F_last))
    return min(gaps)


@pytest.mark.parametrize("wl,iters", [(workloads.MLP784, 6), (SMALL_BF16, 8)], ids=["mlp784", "small_bf16"])
def test_dbw_iterations_independent(wl, iters):
    """Whole DBW iterations: the GPU pipeline and the oracle each run their own
    trajectory from the same seeds.  b_t must agree exactly unless the oracle's own
    decision is within 1e-3 of flipping (then both choices are valid at fp32 input
    precision and the trajectories part; the comparison stops there)."""
    it = Iteration(wl, keep_gbar=True)
    pool, labels = it.pool.cpu().numpy(), it.labels.cpu().numpy()
    bf16 = wl.prec == workloads.PREC_BF16
    rtol = RTOL_BF16 if bf16 else RTOL_FP32
    ost = O.State(n=wl.n, D=wl.D)
    w_or = inputs.kaiming_uniform_params(wl.seed, wl.widths).astype(np.float64)
    compared = 0
    for t in range(iters):
        idx, times = it.host_inputs(t)
        margin = decision_margin(ost, wl.lr, wl.beta)
        k_or, _ = O.choose_k(ost, wl.lr, wl.beta)
        it.load_inputs(t)
        it.step()
        torch.cuda.synchronize()
        b = int(it.b.item())
        if wl.n - b != k_or:
            assert margin < 1e-3, (t, b, k_or, margin)
            break
        blocks = param_blocks(wl.widths)
        matched = assert_worker_grads_match(it.G.cpu().numpy()[:, :wl.d], it.loss.cpu().numpy(), wl.widths, w_or,
                                            pool[idx], labels[idx], wl.B, bf16, range(wl.n), rtol,
                                            gpu_active_sets(it.ws, wl.widths, wl.n, wl.B, wl.prec))
        G_ref = np.stack([matched[i][0] for i in range(wl.n)])
        loss_ref = np.array([matched[i][1] for i in range(wl.n)])
        G_mag = np.stack([np.maximum(matched[i][2], tensor_scale(matched[i][0], blocks)) for i in range(wl.n)])
        order, mask, ts = O.select_fastest(times, b)
        assert np.array_equal(it.mask.cpu().numpy(), mask)
        assert np.array_equal(it.order.cpu().numpy(), order)
        gbar = O.aggregate(G_ref, mask)
        w_new = O.sgd_update(w_or, gbar, wl.lr)
        SS = O.deviation_sumsq(G_ref, mask, gbar)
        rec = O.record_iteration(ost, wl.n - b, SS, float(gbar @ gbar), loss_ref, mask, ts, wl.lr)
        # g_t is a mean of rows each within rtol * magnitude: the mean is within rtol * mean magnitude
        mag = O.aggregate(G_mag, mask)
        assert_close_to_magnitude(it.gbar.cpu().numpy(), gbar, mag, rtol, "g_t")
        # w is stored in fp32 on the GPU and in fp64 by the oracle: allow 2^-20 |w| of storage drift
        assert_close_to_magnitude(it.w.cpu().numpy(), w_new, wl.lr * mag, rtol, "w", extra=2.0 ** -20 * np.abs(w_new))
        s = it.stats.cpu().numpy()
        assert_close_scalar(s[dbw.STAT_GBAR_SQ], rec["gbar_sq"], rtol, "||g_t||^2")
        if rec["k"] >= 2:
            assert_close_scalar(s[dbw.STAT_SS], rec["SS"], rtol, "SS")
        assert_close_scalar(s[dbw.STAT_F], rec["F"], rtol, "F")
        w_or = w_new
        compared += 1
    assert compared >= 3


def test_slowdown_estimator_trajectory_settles_at_half():
    """Sect. 4.3: all round-trip times equal, then half of the 16 workers 5x slower.
    Both sides get the same seeded statistics (a loss that falls as Eq. (9) predicts
    for L = 5, gradient variance small next to the gradient norm) and the slowdown
    times; b_t is bit-exact on every iteration, k_t = 16 while the times are equal
    and k_t = n/2 = 8 once the slow half is visible in the time estimates."""
    n, d, D, lr, beta, t_switch = 16, 4001, 5, 0.05, 1.01, 20
    rng = np.random.default_rng(7)
    state = dbw.new_state(n, D)
    ost = O.State(n=n, D=D)
    b = torch.zeros(1, dtype=torch.int32, device="cuda")
    ratio = torch.empty(n, dtype=torch.float64, device="cuda")
    stats = torch.empty(dbw.STATS_LEN, dtype=torch.float64, device="cuda")
    ks, F, prev = [], 50.0, None
    for t in range(60):
        dbw.dbw_choose_b(state, lr, beta, b, ratio)
        torch.cuda.synchronize()
        k, r = O.choose_k(ost, lr, beta)
        assert n - int(b.item()) == k, t
        assert same_f64(ratio.cpu().numpy(), r), t
        ks.append(k)
        SS = (k - 1) * 0.05 * float(rng.uniform(0.95, 1.05))        # V ~ 0.05 per unit of d
        g2 = 4.0 + 0.05 / k
        times = inputs.completion_times(0, t, n, "slowdown", value=1.0, factor=5.0, t_switch=t_switch)
        if prev is not None:
            N, V, kk = prev
            F = F - ((lr - 5 * lr * lr / 2) * N - (5 * lr * lr / 2) * V / kk)
        loss = np.full(n, F, dtype=np.float32)
        _, mask, ts = O.select_fastest(times, n - k)
        SSq, g2q = round(SS * 1024) / 1024.0, round(g2 * 1024) / 1024.0
        part = seeded_partials(n, 2, SSq, g2q, [1.0 if mask[j] else 0.0 for j in range(n)])
        dbw.dbw_grad_stats(part, n, dev(mask), dev(loss), dev(ts), lr, state, stats)
        torch.cuda.synchronize()
        rec = O.record_iteration(ost, k, SSq, g2q, loss, mask, ts, lr)
        assert_state_equal(dbw.read_state(state), ost)
        prev = (rec["N"], rec["V"], k) if k >= 2 else None
    assert all(k == n for k in ks[2:t_switch]), ks
    assert all(k == n // 2 for k in ks[t_switch + 2:]), ks
