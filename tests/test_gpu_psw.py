"""GPU parity of the push-and-wait clock (Sect. 2, 3.2) and the time estimator of Eq. (17)
against oracle/psw_oracle.py: the clock bit for bit (arrivals, residuals, pending
samples, counts, virtual time), the cell sums to their fixed-point rounding, the
fitted T^_k to the solver tolerance, b_t with given times bit for bit, and whole
DBW iterations under push-and-wait as independent trajectories."""
import math

import numpy as np
import pytest
import torch

from oracle import dbw_oracle as O
from oracle import psw_oracle as P
from paper_2004_14696_gb300 import dbw, inputs, workloads
from paper_2004_14696_gb300.pipeline import Iteration
from gpu_util import RTOL_BF16, assert_bf16_close, gpu_active_sets, oracle_rows_with_decisions, param_blocks, \
    tensor_scale

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def dev(x):
    return torch.from_numpy(np.ascontiguousarray(x)).cuda()


class Clock:
    """The GPU clock driven through the C ABI, step by step beside the oracle's."""

    def __init__(self, n):
        self.n = n
        self.psw = dbw.new_psw(n)
        self.ps = P.psw_init(n)
        self.e = torch.empty(n, dtype=torch.float64, device="cuda")
        self.b = torch.zeros(1, dtype=torch.int32, device="cuda")
        self.order = torch.empty(n, dtype=torch.int32, device="cuda")
        self.mask = torch.empty(n, dtype=torch.uint8, device="cuda")
        self.ts = torch.empty(n, dtype=torch.float64, device="cuda")
        self.k = torch.empty(1, dtype=torch.int32, device="cuda")

    def step(self, omega, k):
        n = self.n
        om = dev(np.asarray(omega, dtype=np.float64))
        dbw.dbw_psw_arrivals(self.psw, n, om, self.e)
        e_ref = P.arrivals(self.ps, omega)
        self.b.fill_(n - k)
        dbw.dbw_select_fastest(self.e, self.b, self.order, self.mask, self.ts, self.k)
        dbw.dbw_psw_record(self.psw, n, self.order, self.ts, self.k)
        out = P.record(self.ps, omega, k)
        torch.cuda.synchronize()
        assert np.array_equal(self.e.cpu().numpy(), e_ref), "arrivals"
        assert np.array_equal(self.order.cpu().numpy(), out["order"]), "arrival order"
        assert np.array_equal(self.mask.cpu().numpy().astype(bool), out["received"]), "received set"
        self.check()
        return out

    def check(self):
        n, ps = self.n, self.ps
        g = dbw.read_psw(self.psw, n)
        assert g["h"] == ps.h and g["flags"] == 0
        assert np.array_equal(g["r"], ps.r), "residuals"
        assert g["vclock"] == ps.vclock, "virtual clock"
        want_pend = np.zeros((n, 2), np.int32)
        want_v = {}
        for j, (h, i, v) in ps.pend.items():
            want_pend[j] = (h, i)
            want_v[j] = v
        assert np.array_equal(g["pend"][:, 0] != 0, want_pend[:, 0] != 0), "pending workers"
        for j, v in want_v.items():
            assert tuple(g["pend"][j]) == tuple(want_pend[j]) and g["pendv"][j] == v, ("pending sample", j)
        assert np.array_equal(g["cnts"], ps.cnts[1:, 1:]), "cell counts"
        # int64 fixed point (2^-32 units) against fp64 sums: one rounding per sample
        lim = (ps.cnts[1:, 1:] + 1) * 2.0 ** -32 + 1e-15 * np.abs(ps.sums[1:, 1:])
        assert np.all(np.abs(g["sums"] - ps.sums[1:, 1:]) <= lim), "cell sums"
        return g


def k_sequence(n, steps, seed):
    rng = np.random.default_rng(seed)
    return [n] + [int(rng.integers(1, n + 1)) for _ in range(steps - 1)]


@pytest.mark.parametrize("n,model,params", [
    (16, "shifted_exp", {"shift": 0.2, "rate": 1.0}),
    (64, "pareto", {"alpha": 2.0, "xm": 1.0}),
    (300, "exp_slow", {"rate": 1.0, "frac": 0.05, "factor": 10.0}),
    (1024, "lognormal", {"mu": 0.0, "sigma": 0.5}),
])
def test_push_and_wait_clock_bit_exact(n, model, params):
    c = Clock(n)
    ks = k_sequence(n, 30, n)
    for t in range(30):
        c.step(inputs.completion_times(7 + n, t, n, model, **params), ks[t])


def test_push_and_wait_clock_hand_worked_on_gpu():
    """The three-worker example of the oracle pins, on the GPU."""
    c = Clock(3)
    c.step([1.0, 2.0, 3.0], 2)
    c.step([2.0, 0.5, 1.0], 1)
    c.step([1.0, 1.0, 1.0], 3)
    g = dbw.read_psw(c.psw, 3)
    assert g["vclock"] == 5.0 and g["cnts"].sum() == 8


RTOL_FIT = 1e-5   # elementwise |x - r| <= 1e-5 |r|, the fp32 tolerance


def assert_fit_close(got, ref, what):
    got, ref = np.asarray(got, dtype=np.float64), np.asarray(ref, dtype=np.float64)
    assert np.array_equal(np.isnan(got), np.isnan(ref)), what
    ok = ~np.isnan(ref)
    err = np.abs(got[ok] - ref[ok])
    lim = RTOL_FIT * np.abs(ref[ok])
    assert np.all(err <= lim), (what, float(np.max(err / np.where(lim > 0, lim, np.inf))))


@pytest.mark.parametrize("tol", [1e-6, 1e-4])
@pytest.mark.parametrize("n,steps", [(16, 40), (64, 30), (256, 12)])
def test_time_estimates_match_the_oracle(n, steps, tol):
    """T^_k after several iterations (the GPU fit is warm-started from the previous
    one, the oracle's is not) against the oracle's, element by element within 1e-5 of
    each value.  The fp32 sweeps find the blocks of the solution; their values are
    the exact fp64 means of the blocks' samples.  So a looser stopping tolerance
    (1e-4, the pipeline's) gives the same values once the sweeps have found the blocks."""
    c = Clock(n)
    ks = k_sequence(n, steps, 3)
    T = torch.empty(n, dtype=torch.float64, device="cuda")
    for t in range(steps):
        c.step(inputs.completion_times(11, t, n, "pareto", alpha=2.0, xm=1.0), ks[t])
        dbw.dbw_psw_estimate(c.psw, n, T, tol=tol, max_sweeps=200000)
        if t in (0, 1, 4, steps // 2, steps - 1):
            torch.cuda.synchronize()
            ref = np.array(P.time_estimates(c.ps))
            got = T.cpu().numpy()
            g = dbw.read_psw(c.psw, n)
            assert not (g["flags"] & (dbw.PSW_NOT_CONVERGED | dbw.PSW_UNPOLISHED)), g["flags"]
            assert_fit_close(got, ref, f"T^ at t={t}")
            assert np.all(np.diff(got) >= 0.0), "T^ nondecreasing (Appendix A)"


def test_waiting_for_all_workers_is_push_and_interrupt_on_gpu():
    """k_t = n: T^ from the fit equals the per-k mean of the sorted times."""
    n = 32
    c = Clock(n)
    T = torch.empty(n, dtype=torch.float64, device="cuda")
    sums = np.zeros(n)
    for t in range(20):
        om = inputs.completion_times(5, t, n, "shifted_exp", shift=1.0, rate=1.0)
        c.step(om, n)
        sums += np.sort(om)
    dbw.dbw_psw_estimate(c.psw, n, T)
    torch.cuda.synchronize()
    # exact block means from the fixed-point cell sums (2^-32 units)
    assert np.allclose(T.cpu().numpy(), sums / 20, rtol=1e-9, atol=0)


def test_no_sample_and_cap_on_sweeps():
    """Before any sample T^ is NaN (and b = 0); max_sweeps = 1 on a fit that needs more
    raises DBW_PSW_NOT_CONVERGED and still returns finite, ordered estimates."""
    n = 24
    c = Clock(n)
    T = torch.empty(n, dtype=torch.float64, device="cuda")
    dbw.dbw_psw_estimate(c.psw, n, T)
    torch.cuda.synchronize()
    assert torch.isnan(T).all()
    state = dbw.new_state(n, 5)
    b = torch.full((1,), 7, dtype=torch.int32, device="cuda")
    dbw.dbw_choose_b_times(state, T, 0.05, 1.01, b)
    torch.cuda.synchronize()
    assert int(b.item()) == 0
    ks = k_sequence(n, 12, 9)
    for t in range(12):
        c.step(inputs.completion_times(3, t, n, "pareto", alpha=1.5, xm=1.0), ks[t])
    dbw.dbw_psw_estimate(c.psw, n, T, tol=1e-6, max_sweeps=1)
    torch.cuda.synchronize()
    g = dbw.read_psw(c.psw, n)
    assert g["flags"] & dbw.PSW_NOT_CONVERGED and g["sweeps"] == 1
    assert torch.isfinite(T).all()


def test_choose_b_times_bit_exact_on_seeded_states():
    from test_gpu_parity import fill_state, same_f64
    rng = np.random.default_rng(77)
    b = torch.zeros(1, dtype=torch.int32, device="cuda")
    for trial in range(300):
        n = int(rng.choice([1, 2, 5, 16, 64, 256, 1024]))
        g, o = fill_state(n, int(rng.choice([1, 5, 64])), rng)
        T = np.sort(rng.exponential(size=n)) + 0.1
        if rng.random() < 0.1:
            T[:] = math.nan
        lr = float(rng.choice([0.01, 0.05]))
        beta = float(rng.choice([1.0, 1.01]))
        blind = bool(rng.random() < 0.15)
        state = torch.empty(dbw.STATE_BYTES, dtype=torch.uint8, device="cuda")
        dbw.write_state(state, g)
        ratio = torch.empty(n, dtype=torch.float64, device="cuda")
        dbw.dbw_choose_b_times(state, dev(T), lr, beta, b, ratio, flags=dbw.CHOOSE_BLIND if blind else 0)
        torch.cuda.synchronize()
        k, r = O.choose_k(o, lr, beta, blind=blind, T=list(T))
        assert n - int(b.item()) == k, trial
        assert same_f64(ratio.cpu().numpy(), r), trial


def test_dbw_trajectory_under_push_and_wait():
    """Whole DBW iterations with the push-and-wait clock (received-workers form, bf16):
    the GPU pipeline and the oracle run their own trajectories; b_t agrees unless the
    oracle's decision is within 1e-3 of flipping, and the clock stays bit-exact."""
    wl = workloads.Workload(key="psw_b32", widths=(256, 128, 64, 10), n=16, B=32, prec=workloads.PREC_BF16, S=900,
                            feature_dist="normal", time_model="shifted_exp", time_params={"shift": 0.2, "rate": 1.0},
                            lr=0.01, seed_offset=95)
    it = Iteration(wl, keep_gbar=True, received=True, clock="psw")
    pool, labels = it.pool.cpu().numpy(), it.labels.cpu().numpy()
    ost = O.State(n=wl.n, D=wl.D)
    ps = P.psw_init(wl.n)
    w_or = inputs.kaiming_uniform_params(wl.seed, wl.widths).astype(np.float64)
    blocks = param_blocks(wl.widths)
    compared = 0
    for t in range(10):
        idx, omega = it.host_inputs(t)
        T_or = P.time_estimates(ps)
        k_or, _ = O.choose_k(ost, wl.lr, wl.beta, T=T_or)
        margin = psw_margin(ost, wl.lr, wl.beta, T_or)
        it.load_inputs(t)
        it.step()
        torch.cuda.synchronize()
        b = int(it.b.item())
        if wl.n - b != k_or:
            assert margin < 1e-3, (t, b, k_or, margin)
            break
        out = P.record(ps, omega, k_or)
        g = dbw.read_psw(it.psw, wl.n)
        assert np.array_equal(g["r"], ps.r) and g["vclock"] == ps.vclock
        mask = out["received"]
        assert np.array_equal(it.mask.cpu().numpy().astype(bool), mask)
        received = [int(j) for j in np.flatnonzero(mask)]
        slot = {j: s for s, j in enumerate(received)}
        rows = oracle_rows_with_decisions(wl.widths, w_or, pool[idx], labels[idx], wl.B, True, received,
                                          gpu_active_sets(it.ws, wl.widths, wl.n, wl.B, wl.prec),
                                          rows_of=lambda j: slice(slot[j] * wl.B, (slot[j] + 1) * wl.B))
        G_ref = np.zeros((wl.n, wl.d))
        G_mag = np.zeros((wl.n, wl.d))
        loss_ref = np.zeros(wl.n)
        for j in received:
            G_ref[j], loss_ref[j] = rows[j][0], rows[j][1]
            G_mag[j] = np.maximum(rows[j][2], tensor_scale(rows[j][0], blocks))
        gbar = O.aggregate(G_ref, mask)
        assert_bf16_close(it.gbar.cpu().numpy(), gbar, O.aggregate(G_mag, mask), blocks, RTOL_BF16, f"g_t at t={t}")
        ts = np.sort(out["arrivals"])
        O.record_iteration(ost, wl.n - b, O.deviation_sumsq(G_ref, mask, gbar), float(gbar @ gbar), loss_ref, mask,
                           ts, wl.lr)
        w_or = O.sgd_update(w_or, gbar, wl.lr)
        compared += 1
    assert compared >= 4


def psw_margin(st, lr, beta, T):
    """Relative gap between the best and the runner-up ratio of Eq. (18) with given T^."""
    gains = O.gain_estimates(st, lr)
    if gains is None or math.isnan(T[0]):
        return math.inf
    r = sorted((g / t for g, t in zip(gains, T) if g > 0), reverse=True)
    gaps = [math.inf]
    if len(r) >= 2:
        gaps.append((r[0] - r[1]) / abs(r[0]))
    if st.t >= 2 and st.k_last < st.n:
        gaps.append(abs(st.F_last - beta * st.F_prev) / abs(st.F_last))
    return min(gaps)


@pytest.mark.parametrize("tol", [1e-6, 1e-4])
@pytest.mark.parametrize("n", [96, 200])
def test_fit_on_planted_tables(n, tol):
    """Eq. (17) on cell tables written straight into the state, shaped so that the split
    chains pool across their parts: group rows whose cell means fall along the whole row
    (one block absorbs every part), rise (nothing pools), or zig-zag, with random counts;
    rows outside the group feed only the pooled column means.  Against the oracle's fit
    of the same table."""
    rng = np.random.default_rng(n)
    psw = dbw.new_psw(n)
    ps = P.psw_init(n)
    unit = 2.0 ** -32
    sums = np.zeros((n, n), np.uint64)
    cnts = np.zeros((n, n), np.int32)
    group = sorted(rng.choice(np.arange(2, n - 2), size=5, replace=False).tolist())
    shapes = ["fall", "rise", "zigzag", "fall", "random"]
    for h, shape in zip(group, shapes):           # 1-based row h, observed prefix 1..M_h
        M = int(rng.integers(h, n + 1))
        i = np.arange(M)
        if shape == "fall":
            mean = 50.0 - 40.0 * i / M
        elif shape == "rise":
            mean = 5.0 + 40.0 * i / M
        elif shape == "zigzag":
            mean = 20.0 + 10.0 * (i % 7) - 0.05 * i
        else:
            mean = rng.uniform(1.0, 40.0, size=M)
        c = rng.integers(1, 6, size=M)
        q = np.round(mean * c / unit)             # cell sums in 2^-32 units, as the clock stores them
        sums[h - 1, :M] = q.astype(np.uint64)
        cnts[h - 1, :M] = c
    for h in rng.choice([r for r in range(1, n) if r not in group], size=4, replace=False):
        M = int(rng.integers(1, h))                # below the diagonal: not in the fitted group
        c = rng.integers(1, 4, size=M)
        sums[h - 1, :M] = np.round(rng.uniform(1.0, 40.0, size=M) * c / unit).astype(np.uint64)
        cnts[h - 1, :M] = c
    write_table(psw, n, sums, cnts)
    ps.sums[1:, 1:] = sums.astype(np.float64) * unit
    ps.cnts[1:, 1:] = cnts
    T = torch.empty(n, dtype=torch.float64, device="cuda")
    dbw.dbw_psw_estimate(psw, n, T, tol=tol, max_sweeps=200000)
    torch.cuda.synchronize()
    g = dbw.read_psw(psw, n)
    assert not (g["flags"] & (dbw.PSW_NOT_CONVERGED | dbw.PSW_UNPOLISHED)), g["flags"]
    ref = np.array(P.time_estimates(ps, tol=1e-11))
    assert_fit_close(T.cpu().numpy(), ref, "T^")
    # the fitted group cells themselves (fp32 copies of the exact block means)
    H, fit, _ = P.solve(ps, tol=1e-11)
    for (h, i), v in fit.items():
        assert abs(float(g["x"][h - 1, i - 1]) - v) <= RTOL_FIT * abs(v), (h, i, float(g["x"][h - 1, i - 1]), v)


def write_table(psw, n, sums, cnts):
    """Cell sums ([n, n] uint64, 2^-32 units) and counts ([n, n] int32) straight into a GPU state."""
    import ctypes
    hdr = dbw.PswHeader.from_buffer_copy(psw[:ctypes.sizeof(dbw.PswHeader)].cpu().numpy().tobytes())
    assert hdr.n == n
    psw[hdr.off_sum:hdr.off_sum + 8 * n * n] = torch.from_numpy(sums.reshape(-1).view(np.uint8)).cuda()
    psw[hdr.off_cnt:hdr.off_cnt + 4 * n * n] = torch.from_numpy(cnts.reshape(-1).view(np.uint8)).cuda()


@pytest.mark.parametrize("name", ["clipped_above", "clipped_below", "two_group_rows"])
def test_free_diagonal_cells_hand_worked_on_gpu(name):
    """The hand-worked cell tables of the oracle pins (reading P3 (b)), on the GPU:
    T^ equals the values worked out by hand, to fp64 rounding."""
    from test_oracle_psw import HAND_TABLES
    n, cells, want = HAND_TABLES[name]
    unit = 2.0 ** -32
    sums = np.zeros((n, n), np.uint64)
    cnts = np.zeros((n, n), np.int32)
    for (h, i), (sm, c) in cells.items():
        sums[h - 1, i - 1] = np.uint64(round(sm / unit))
        cnts[h - 1, i - 1] = c
    psw = dbw.new_psw(n)
    write_table(psw, n, sums, cnts)
    T = torch.empty(n, dtype=torch.float64, device="cuda")
    dbw.dbw_psw_estimate(psw, n, T, tol=1e-6, max_sweeps=200000)
    torch.cuda.synchronize()
    g = dbw.read_psw(psw, n)
    assert not (g["flags"] & (dbw.PSW_NOT_CONVERGED | dbw.PSW_UNPOLISHED)), g["flags"]
    assert np.allclose(T.cpu().numpy(), want, rtol=1e-14, atol=0), (T.cpu().numpy(), want)

