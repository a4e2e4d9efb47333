"""Pins of the push-and-wait oracle (oracle/psw_oracle.py) against facts fixed by the
paper and by mathematics, independent of the oracle's own code paths:

* PAVA: brute force over all block partitions of short chains, and the
  isotonic-regression routine of scikit-learn.
* Eq. (17) solver: a general-purpose constrained minimiser on tiny grids; the
  optimality conditions of a projection onto a convex cone (feasibility,
  <y - x*, x*>_W = 0, <y - x*, z>_W <= 0 for the cone's generators: constants and
  indicators of up-sets of the order); feasible targets returned unchanged; a
  planted wrong constraint direction is caught.
* The estimator on sparse cells (rows and cells without samples): the order rule
  it relies on equals the transitive closure of Eq. (17)'s constraints (brute
  force); its estimate extends to a feasible point of (17) whose objective equals
  the general minimiser's.
* The clock: a hand-worked three-worker example of Sect. 2's push-and-wait rule;
  with k_t = n every worker is idle at every start, so the clock and the estimator
  reduce to the push-and-interrupt ones (per-k means of sorted time vectors).
* Appendix A and Sect. 3.2: waiting for more gradients makes iterations longer
  on average, and more idle workers at the start make the i-th arrival earlier.
"""
import itertools
import math

import numpy as np
import pytest

from oracle import dbw_oracle as O
from oracle import psw_oracle as P
from paper_2004_14696_gb300 import inputs


# ---------------------------------------------------------------- PAVA
def brute_isotonic(y, w):
    """Minimum of sum w (y - x)^2 over nondecreasing x: the optimum is piecewise constant,
    equal to the weighted block mean on each block of some partition into consecutive
    blocks; enumerate every partition whose block means are nondecreasing."""
    n = len(y)
    best, arg = math.inf, None
    for cuts in itertools.product([0, 1], repeat=n - 1):
        bounds = [0] + [i + 1 for i, c in enumerate(cuts) if c] + [n]
        x = np.empty(n)
        for a, b in zip(bounds, bounds[1:]):
            x[a:b] = np.dot(w[a:b], y[a:b]) / w[a:b].sum()
        if np.all(np.diff(x) >= -1e-15):
            f = float(np.dot(w, (y - x) ** 2))
            if f < best:
                best, arg = f, x
    return arg


def test_pava_equals_brute_force():
    rng = np.random.default_rng(11)
    for n in range(1, 9):
        for _ in range(20):
            y = rng.normal(size=n)
            w = rng.uniform(0.1, 3.0, size=n)
            assert np.allclose(P.pava(y, w), brute_isotonic(y, w), rtol=0, atol=1e-12)


def test_pava_matches_library_isotonic_regression():
    iso = pytest.importorskip("sklearn.isotonic")
    rng = np.random.default_rng(12)
    for n in (5, 40, 300):
        y = np.cumsum(rng.normal(size=n)) + rng.normal(scale=3.0, size=n)
        w = rng.uniform(0.05, 5.0, size=n)
        ref = iso.IsotonicRegression(increasing=True).fit(np.arange(n), y, sample_weight=w).predict(np.arange(n))
        assert np.allclose(P.pava(y, w), ref, rtol=1e-12, atol=1e-12)


# ---------------------------------------------------------------- Eq. (17)
def relations(n):
    """The pairs (a, b) of cells with x_a <= x_b required by Eq. (17) (0-based (h, k))."""
    rel = []
    for h in range(n):
        for k in range(n - 1):
            rel.append(((h, k), (h, k + 1)))          # increasing in k
    for h in range(n - 1):
        for k in range(n):
            rel.append(((h + 1, k), (h, k)))          # decreasing in h
    for k in range(n - 1):
        rel.append(((k, k), (k + 1, k + 1)))          # increasing diagonal
    return rel


def feasible(x, tol):
    n = x.shape[0]
    return all(x[a] <= x[b] + tol for a, b in relations(n))


def random_feasible(rng, n):
    """x_{h,k} = a_k - b_h with a increasing faster than b: increasing in k, decreasing in
    h, and x_{k,k} = a_k - b_k increasing."""
    db = rng.uniform(0, 1, size=n)
    da = db + rng.uniform(0, 1, size=n)
    a, b = np.cumsum(da), np.cumsum(db)
    return a[None, :] - b[:, None] + rng.normal()


def upset_indicator(rng, n):
    """Indicator of an up-set of the order (if a cell is in, every cell required to be
    >= it is in): the cells where a random feasible matrix exceeds a threshold."""
    z = random_feasible(rng, n)
    return (z > rng.uniform(z.min(), z.max())).astype(np.float64)


def check_projection(x, y, w, tol=1e-9):
    """Optimality of x as the W-weighted projection of y onto the cone of Eq. (17)."""
    scale = float(np.max(np.abs(y))) + 1.0
    assert feasible(x, tol * scale), "infeasible"
    r = w * (y - x)
    assert abs(float(np.sum(r * x))) <= tol * scale * scale * w.sum(), "<y - x, x>_W != 0"
    assert abs(float(np.sum(r))) <= tol * scale * w.sum(), "<y - x, 1>_W != 0"
    rng = np.random.default_rng(5)
    for _ in range(300):
        z = upset_indicator(rng, x.shape[0])
        assert float(np.sum(r * z)) <= tol * scale * w.sum(), "<y - x, 1_U>_W > 0 for an up-set U"


@pytest.mark.parametrize("n", [2, 5, 8])
def test_isotonic_2d_satisfies_projection_conditions(n):
    rng = np.random.default_rng(20 + n)
    for trial in range(6):
        y = rng.normal(size=(n, n)) * 2.0 + np.arange(n)[None, :] * 0.3
        w = rng.uniform(0.2, 4.0, size=(n, n))
        if trial % 2:                        # very unequal weights (sample counts)
            w = np.floor(np.exp(rng.uniform(0, 6, size=(n, n))))
        x, _ = P.isotonic_2d(y, w)
        check_projection(x, y, w)


def test_isotonic_2d_matches_general_constrained_minimiser():
    opt = pytest.importorskip("scipy.optimize")
    rng = np.random.default_rng(31)
    for n in (2, 3, 4):
        for _ in range(4):
            y = rng.normal(size=(n, n))
            w = rng.uniform(0.3, 3.0, size=(n, n))
            rel = relations(n)
            cons = [{"type": "ineq", "fun": (lambda v, a=a, b=b: v.reshape(n, n)[b] - v.reshape(n, n)[a])}
                    for a, b in rel]
            res = opt.minimize(lambda v: float(np.sum(w * (v.reshape(n, n) - y) ** 2)), y.ravel(),
                               jac=lambda v: (2 * w * (v.reshape(n, n) - y)).ravel(), constraints=cons,
                               method="SLSQP", options={"ftol": 1e-15, "maxiter": 2000})
            x, _ = P.isotonic_2d(y, w)
            assert np.allclose(x, res.x.reshape(n, n), atol=1e-6), (x, res.x.reshape(n, n))


def test_isotonic_2d_returns_feasible_targets_unchanged():
    rng = np.random.default_rng(41)
    for n in (3, 7, 12):
        y = random_feasible(rng, n)
        w = rng.uniform(0.5, 2.0, size=(n, n))
        x, sweeps = P.isotonic_2d(y, w)
        assert np.array_equal(x, y) and sweeps == 1


def test_planted_wrong_constraint_direction_is_caught(monkeypatch):
    """Columns made increasing in h (the wrong direction) must fail the optimality check."""
    right = P.grid_families

    def wrong(n):
        rows, cols, diag = right(n)
        return [rows, [list(reversed(c)) for c in cols], diag]
    monkeypatch.setattr(P, "grid_families", wrong)
    rng = np.random.default_rng(43)
    y = rng.normal(size=(5, 5))
    w = rng.uniform(0.5, 2.0, size=(5, 5))
    x, _ = P.isotonic_2d(y, w, max_sweeps=2000)
    with pytest.raises(AssertionError):
        check_projection(x, y, w)


# ---------------------------------------------------------------- the estimator on sparse cells
def order_rule(a, b):
    """(h, j) <= (h', k') in the order Eq. (17) imposes (0-based cells): through the grid
    (h >= h', j <= k') or through the diagonal (j <= h, h' <= k', j <= k')."""
    (h, j), (h2, k2) = a, b
    return (h >= h2 and j <= k2) or (j <= h and h2 <= k2 and j <= k2)


def test_order_rule_is_the_transitive_closure_of_eq17():
    for n in range(1, 6):
        cells = [(h, k) for h in range(n) for k in range(n)]
        idx = {c: i for i, c in enumerate(cells)}
        R = np.eye(len(cells), dtype=bool)
        for a, b in relations(n):
            R[idx[a], idx[b]] = True
        for m in range(len(cells)):                    # Floyd-Warshall closure
            R |= R[:, m:m + 1] & R[m:m + 1, :]
        for a in cells:
            for b in cells:
                assert R[idx[a], idx[b]] == order_rule(a, b), (n, a, b)


def sparse_state(rng, n):
    """A cell table shaped like the clock's: each row with samples has observed a prefix
    of ranks 1..M_h, some rows have none, and some stop before their diagonal cell."""
    ps = P.psw_init(n)
    rows = sorted(rng.choice(np.arange(1, n + 1), size=int(rng.integers(1, n + 1)), replace=False))
    for h in rows:
        M = int(rng.integers(1, n + 1))
        for i in range(1, M + 1):
            c = int(rng.integers(1, 5))
            ps.cnts[h, i] = c
            ps.sums[h, i] = c * float(rng.uniform(0.5, 3.0) + 0.4 * i - 0.2 * h)
    return ps


@pytest.mark.parametrize("n", [2, 3, 4])
def test_estimator_is_an_optimum_of_eq17(n):
    """Group (a)'s fitted cells plus all diagonal estimates respect the order of Eq. (17),
    extend to a feasible point of (17), and reach the minimum a general constrained
    minimiser finds for (17) over the samples of group (a)'s rows."""
    opt = pytest.importorskip("scipy.optimize")
    rng = np.random.default_rng(100 + n)
    checked = 0
    for _ in range(12):
        ps = sparse_state(rng, n)
        H, fit, _ = P.solve(ps)
        T = P.time_estimates(ps)
        if not H:
            assert all(math.isnan(v) for v in T)
            continue
        known = {(h - 1, i - 1): v for (h, i), v in fit.items()}
        for k in range(n):
            if (k, k) in known:
                assert known[(k, k)] == T[k]
            known[(k, k)] = T[k]
        for a in known:                                 # the determined values respect the order
            for b in known:
                if order_rule(a, b):
                    assert known[a] <= known[b] + 1e-9, (a, b)
        base = min(known.values())
        x = np.array([[max([base] + [v for c, v in known.items() if order_rule(c, (h, k))]) for k in range(n)]
                      for h in range(n)])
        assert feasible(x, 1e-9)
        for c, v in known.items():
            assert abs(x[c] - v) <= 1e-12
        C = np.zeros((n, n))
        for h in H:
            C[h - 1] = ps.cnts[h, 1:]
        Y = np.divide(ps.sums[1:, 1:], np.maximum(ps.cnts[1:, 1:], 1))
        f_est = float(np.sum(C * (x - Y) ** 2))
        cons = [{"type": "ineq", "fun": (lambda v, a=a, b=b: v.reshape(n, n)[b] - v.reshape(n, n)[a])}
                for a, b in relations(n)]
        res = opt.minimize(lambda v: float(np.sum(C * (v.reshape(n, n) - Y) ** 2)), x.ravel(),
                           jac=lambda v: (2 * C * (v.reshape(n, n) - Y)).ravel(), constraints=cons,
                           method="SLSQP", options={"ftol": 1e-15, "maxiter": 2000})
        assert f_est <= res.fun + 1e-7 * (1 + res.fun), (f_est, res.fun)
        checked += 1
    assert checked >= 6


def test_stage_one_satisfies_projection_conditions_on_its_rows():
    """Group (a) is the count-weighted projection onto the order restricted to its
    observed cells: optimality against the up-sets of that order."""
    rng = np.random.default_rng(7)
    done = 0
    for n in (5, 8, 8, 12):
        ps = sparse_state(rng, n)
        H, fit, _ = P.solve(ps)
        if not H:
            continue
        cells = sorted(fit)
        x = np.array([fit[c] for c in cells])
        y = np.array([ps.sums[c] / ps.cnts[c] for c in cells])
        w = np.array([float(ps.cnts[c]) for c in cells])
        le = lambda c, d: order_rule((c[0] - 1, c[1] - 1), (d[0] - 1, d[1] - 1))
        for a, c in enumerate(cells):
            for b, d in enumerate(cells):
                if le(c, d):
                    assert x[a] <= x[b] + 1e-9
        r = w * (y - x)
        scale = float(np.max(np.abs(y))) + 1.0
        assert abs(float(np.sum(r))) <= 1e-9 * scale * w.sum()
        assert abs(float(np.sum(r * x))) <= 1e-9 * scale * scale * w.sum()
        for _ in range(200):
            th = rng.uniform(x.min(), x.max())
            U = np.array([1.0 if any(le(cells[a], d) and x[a] > th for a in range(len(cells))) else 0.0
                          for d in cells])
            assert float(np.sum(r * U)) <= 1e-8 * scale * w.sum()
        done += 1
    assert done >= 2


# ---------------------------------------------------------------- the clock
def test_push_and_wait_clock_hand_worked():
    """n = 3.  t = 0 (h = 3, all idle): times 1, 2, 3 and k = 2 -> T = 2, worker 2's
    gradient (rank 3, value 3) is late and worker 2 stays busy for 1.  t = 1 (h = 2):
    times 2, 0.5, 1 and k = 1 -> arrivals 2, 0.5, 2; worker 2 is busy past T = 0.5 and
    does not compute; worker 1 arrives first (sample (2, 1, 0.5)), worker 0 second but
    late (pending (2, 2, 2)).  t = 2 (h = 1): times 1, 1, 1 and k = 3 -> arrivals
    2.5, 1, 1.5; both pending samples arrive; ranks 1, 2, 3 = workers 1, 2, 0."""
    ps = P.psw_init(3)
    out = P.record(ps, [1.0, 2.0, 3.0], 2)
    assert out["T"] == 2.0 and list(out["received"]) == [True, True, False]
    assert list(ps.r) == [0.0, 0.0, 1.0] and ps.pend == {2: (3, 3, 3.0)}
    out = P.record(ps, [2.0, 0.5, 1.0], 1)
    assert out["T"] == 0.5 and list(out["received"]) == [False, True, False]
    assert list(ps.r) == [1.5, 0.0, 0.5] and ps.pend == {2: (3, 3, 3.0), 0: (2, 2, 2.0)}
    out = P.record(ps, [1.0, 1.0, 1.0], 3)
    assert out["T"] == 2.5 and list(out["arrivals"]) == [2.5, 1.0, 1.5]
    assert list(ps.r) == [0.0, 0.0, 0.0] and ps.pend == {} and ps.vclock == 5.0
    expect = {(3, 1): 1.0, (3, 2): 2.0, (3, 3): 3.0, (2, 1): 0.5, (2, 2): 2.0, (1, 1): 1.0, (1, 2): 1.5,
              (1, 3): 2.5}
    for (h, i), v in expect.items():
        assert ps.cnts[h, i] == 1 and ps.sums[h, i] == v, (h, i)
    assert ps.cnts.sum() == len(expect)


def test_waiting_for_all_workers_reduces_to_push_and_interrupt():
    """k_t = n: every worker is idle at every start, each iteration contributes the n
    sorted times to row h = n, and T^_k is the per-k mean of the sorted vectors, the
    push-and-interrupt estimator S_k / c."""
    n, seed = 6, 77
    ps = P.psw_init(n)
    st = O.State(n=n, D=5)
    st.S = [0.0] * n
    for t in range(25):
        om = inputs.completion_times(seed, t, n, "pareto", alpha=2.0, xm=1.0)
        out = P.record(ps, om, n)
        assert np.all(ps.r == 0.0) and out["T"] == np.max(om)
        ts = np.sort(om)
        st.S = [a + b for a, b in zip(st.S, ts)]
        st.c += 1
    T = P.time_estimates(ps)
    assert np.allclose(T, O.time_estimates(st), rtol=1e-12, atol=0)


def test_no_sample_means_no_estimate():
    ps = P.psw_init(4)
    assert all(math.isnan(v) for v in P.time_estimates(ps))
    st = O.State(n=4, D=5)
    k, _ = O.choose_k(st, 0.05, 1.01, T=P.time_estimates(ps))
    assert k == 4


def test_external_times_equal_to_push_and_interrupt_give_the_same_choice():
    """choose_k with T given as S_k / c is the push-and-interrupt choice itself."""
    rng = np.random.default_rng(3)
    for _ in range(20):
        n = 12
        st = O.State(n=n, D=5)
        st.t, st.c = 6, 5
        for ring, cnt in ((st.ringV, "cntV"), (st.ringN, "cntN"), (st.ringL, "cntL")):
            for i in range(5):
                ring[i] = float(rng.uniform(0.1, 5.0))
            setattr(st, cnt, 5)
        st.S = list(np.cumsum(rng.uniform(0.1, 1.0, size=n)) * 5)
        st.F_last, st.F_prev, st.k_last = 1.0, 1.0, n
        assert O.choose_k(st, 0.05, 1.01, T=O.time_estimates(st)) == O.choose_k(st, 0.05, 1.01)


def mean_durations(n, k_of_t, iters, seed):
    ps = P.psw_init(n)
    Ts = []
    for t in range(iters):
        om = inputs.completion_times(seed, t, n, "shifted_exp", shift=0.0, rate=1.0)
        Ts.append(P.record(ps, om, k_of_t(t))["T"])
    return ps, float(np.mean(Ts[50:]))


def test_appendix_a_waiting_for_more_gradients_is_slower():
    """Appendix A: E[T_{i,i}] <= E[T_{i+1,i+1}] (exponential times, static k)."""
    means = [mean_durations(8, lambda t, k=k: k, 3000, 90 + k)[1] for k in range(1, 9)]
    assert all(a < b for a, b in zip(means, means[1:])), means


def test_more_idle_workers_at_start_is_faster():
    """Sect. 3.2: E[T_{h+1,i}] <= E[T_{h,i}].  k alternates between 3 and 6, so rows h = 3
    and h = 6 both collect samples; the i-th arrival (i <= 3) is earlier after h = 6."""
    ps, _ = mean_durations(8, lambda t: 3 if t % 2 else 6, 4000, 5)
    for i in (1, 2, 3):
        m3 = ps.sums[3, i] / ps.cnts[3, i]
        m6 = ps.sums[6, i] / ps.cnts[6, i]
        assert m6 < m3, (i, m6, m3)


# ---------------------------------------------------------------- P3 (b): diagonal cells outside group (a)
# Hand-worked cell tables: every expected T^_k below is worked out by hand from P3's
# rule (pooled column means, the nearest sampled column before else after for an
# empty column, PAVA with unit weights over the cells outside group (a), clipped to
# the bounds the order of Eq. (17) puts on them), not by the oracle's code.
def table(n, cells):
    """A push-and-wait state whose cell (h, i) holds samples summing to s, c of them."""
    ps = P.psw_init(n)
    for (h, i), (s, c) in cells.items():
        ps.sums[h, i] = s
        ps.cnts[h, i] = c
    return ps


# n = 5.  Group (a) = row 3 alone: cells 1, 2, 3 already increasing, so the fit
# keeps them.  Row 5 has no diagonal sample.  Column means: col 1 = (1 + 27)/4 = 7,
# col 2 = (2 + 1)/2 = 1.5, col 4 = 3.5, col 5 empty -> col 4's 3.5.  PAVA over the
# cells k = 1, 2, 4, 5 of [7, 1.5, 3.5, 3.5]: 7 > 1.5 pools to 4.25 (2 cells), then
# 4.25 > 3.5 pools to 4 (3 cells), then 4 > 3.5 pools to 3.875 (4 cells).  Bounds
# from row 3: k = 1: [x31, x33] = [1, 3] -> 3 (clipped from above); k = 2:
# [x32, x33] = [2, 3] -> 3 (from above); k = 4, 5: [x33, inf) = [3, inf) -> 3.875.
TABLE_ABOVE = (5, {(3, 1): (1.0, 1), (3, 2): (2.0, 1), (3, 3): (3.0, 1),
                   (5, 1): (27.0, 3), (5, 2): (1.0, 1), (5, 3): (2.5, 1), (5, 4): (3.5, 1)},
               [3.0, 3.0, 3.0, 3.875, 3.875])
# n = 5.  Group (a) = row 2 with the single cell (2, 2), mean 8/2 = 4.  Column 1 is
# empty with no sampled column before it -> col 2's 4; col 3 = 3; col 4 empty ->
# col 3's 3 (the column before it, not col 5's 6); col 5 = 6.  PAVA over k = 1, 3, 4, 5
# of [4, 3, 3, 6]: 4 > 3 pools to 3.5, then 3.5 > 3 pools to 10/3; 6 stays.  Bounds
# from (2, 2): k = 1: (-inf, 4] -> 10/3; k = 3, 4, 5: [4, inf) -> 4, 4 (clipped from
# below), 6.
TABLE_BELOW = (5, {(2, 2): (8.0, 2), (5, 3): (3.0, 1), (4, 5): (6.0, 1)},
               [10.0 / 3.0, 4.0, 4.0, 4.0, 6.0])
# n = 4.  Group (a) = rows 2 and 4.  Cells a = (2,1) = 1, b = (2,2) = 4, c = (4,1) = 2,
# d = (4,2) = 1, e = (4,3) = 3, f = (4,4) = 5.  Eq. (17): a <= b, c <= d <= e <= f
# (rows), c <= a, d <= b (columns), b <= f (diagonal).  The projection pools
# {a, c, d} to (1 + 2 + 1)/3 = 4/3: every lower part of that block has a mean >= 4/3
# ({c} 2, {c, d} 1.5, {c, a} 1.5) and every upper part <= 4/3 ({a} 1, {d} 1), and
# the result is feasible.  So T^_2 = 4 and T^_4 = 5.  Row 3 has no diagonal sample.
# Col 1 = (1 + 2 + 0.5)/3 = 7/6, col 3 = 3.  PAVA over k = 1, 3: unchanged.  k = 1:
# lo = max(x21, x41) = 4/3, hi = min(x22, x44) = 4 -> 4/3 (clipped from below by a
# pooled value); k = 3: lo = max over row 2 (j <= 2) and row 4 (j <= 3) = 4,
# hi = x44 = 5 -> 4.
TABLE_TWO_ROWS = (4, {(2, 1): (1.0, 1), (2, 2): (4.0, 1), (4, 1): (2.0, 1), (4, 2): (1.0, 1), (4, 3): (3.0, 1),
                      (4, 4): (5.0, 1), (3, 1): (0.5, 1), (3, 2): (6.0, 1)},
                  [4.0 / 3.0, 4.0, 4.0, 5.0])
HAND_TABLES = {"clipped_above": TABLE_ABOVE, "clipped_below": TABLE_BELOW, "two_group_rows": TABLE_TWO_ROWS}


@pytest.mark.parametrize("name", sorted(HAND_TABLES))
def test_free_diagonal_cells_hand_worked(name):
    n, cells, want = HAND_TABLES[name]
    got = P.time_estimates(table(n, cells))
    assert np.allclose(got, want, rtol=1e-12, atol=0), (got, want)


def test_planted_next_column_fallback_is_caught(monkeypatch):
    """An empty column that takes the next sampled column's mean instead of the previous one's."""
    def wrong(ps):
        n = ps.n
        col_sum, col_cnt = ps.sums[1:, 1:].sum(axis=0), ps.cnts[1:, 1:].sum(axis=0)
        mu = np.full(n, math.nan)
        for i in range(n - 1, -1, -1):
            if col_cnt[i] > 0:
                mu[i] = col_sum[i] / col_cnt[i]
            elif i < n - 1:
                mu[i] = mu[i + 1]
        return mu
    monkeypatch.setattr(P, "column_means", wrong)
    n, cells, want = TABLE_BELOW
    assert not np.allclose(P.time_estimates(table(n, cells)), want, rtol=1e-12, atol=0)


def test_planted_missing_pava_over_free_cells_is_caught(monkeypatch):
    """Skipping the PAVA pass (each free cell keeps its own column mean).  Group (a) of
    this table is one increasing row, which PAVA leaves as it is either way."""
    monkeypatch.setattr(P, "pava", lambda y, w: np.array(y, dtype=np.float64))
    n, cells, want = TABLE_ABOVE
    assert not np.allclose(P.time_estimates(table(n, cells)), want, rtol=1e-12, atol=0)


def test_planted_wrong_lower_bound_is_caught(monkeypatch):
    """A lower bound taken over j <= max(h, k) instead of j <= min(h, k)."""
    def wrong(fit, k):
        lo, hi = -math.inf, math.inf
        for (h, j), xv in fit.items():
            if j <= max(h, k):
                lo = max(lo, xv)
            if j >= max(h, k):
                hi = min(hi, xv)
        return lo, hi
    monkeypatch.setattr(P, "diagonal_bounds", wrong)
    n, cells, want = TABLE_TWO_ROWS
    assert not np.allclose(P.time_estimates(table(n, cells)), want, rtol=1e-12, atol=0)
