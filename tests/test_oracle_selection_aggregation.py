"""Pins of the oracle's selection (Eq. (4)), aggregation (Eqs. (3)/(4)) and the
gradient statistics of Sect. 3.1 (Eqs. (8), (10), (11)) against facts that do not
come from the oracle itself: library sorts, brute force over permutations,
special cases the paper states, closed forms and Monte-Carlo expectations."""
import itertools
import math

import numpy as np
import pytest

from oracle import dbw_oracle as O


def _tie_heavy_times(rng, n):
    return rng.integers(0, max(2, n // 3), size=n).astype(np.float64)


@pytest.mark.parametrize("n", [1, 2, 5, 16, 64, 256])
def test_select_matches_stable_library_sort(n):
    rng = np.random.default_rng(n)
    for times in (rng.exponential(size=n), _tie_heavy_times(rng, n)):
        expected = np.argsort(times, kind="stable")     # stable: lower index first on ties
        for b in sorted({0, n // 4, n // 2, n - 1}):
            order, mask, tsorted = O.select_fastest(times, b)
            assert np.array_equal(order, expected)
            assert np.array_equal(tsorted, times[expected])
            k = n - b
            assert mask.sum() == k
            assert set(np.flatnonzero(mask)) == set(expected[:k].tolist())


def test_select_brute_force_over_permutations():
    rng = np.random.default_rng(7)
    for n in range(1, 7):
        for _ in range(20):
            times = rng.integers(0, 3, size=n).astype(np.float64)
            valid = [p for p in itertools.permutations(range(n))
                     if all((times[p[r]], p[r]) < (times[p[r + 1]], p[r + 1]) for r in range(n - 1))]
            assert len(valid) == 1
            order, _, _ = O.select_fastest(times, 0)
            assert tuple(order.tolist()) == valid[0]


def test_select_special_cases():
    times = np.array([3.0, 1.0, 1.0, 2.0])
    order, mask, tsorted = O.select_fastest(times, 3)     # b = n-1: single fastest, lowest index on tie
    assert mask.tolist() == [0, 1, 0, 0]
    order, mask, _ = O.select_fastest(times, 0)           # b = 0: everybody
    assert mask.tolist() == [1, 1, 1, 1]
    with pytest.raises(ValueError):
        O.select_fastest(times, 4)


def _rows(n, d, seed=0):
    return np.random.default_rng(seed).standard_normal((n, d))


def test_b_zero_is_full_synchronous_mean_and_b_max_is_fastest_row():
    n, d = 9, 33
    G = _rows(n, d)
    times = np.random.default_rng(1).exponential(size=n)
    _, mask, _ = O.select_fastest(times, 0)
    # Eq. (3) with b = 0: the mean over all n rows (numpy's mean is an independent routine)
    np.testing.assert_allclose(O.aggregate(G, mask), G.mean(axis=0), rtol=1e-14, atol=1e-15)
    _, mask, _ = O.select_fastest(times, n - 1)
    fastest = int(np.argmin(times))
    assert np.array_equal(O.aggregate(G, mask), G[fastest])   # exactly that row


def test_aggregation_is_permutation_invariant():
    n, d = 12, 50
    G = _rows(n, d, 3)
    times = np.random.default_rng(4).exponential(size=n)
    perm = np.random.default_rng(5).permutation(n)
    for b in (0, 3, 11):
        _, m1, _ = O.select_fastest(times, b)
        _, m2, _ = O.select_fastest(times[perm], b)
        g1 = O.aggregate(G, m1)
        g2 = O.aggregate(G[perm], m2)
        np.testing.assert_allclose(g1, g2, rtol=1e-13, atol=1e-15)
        np.testing.assert_allclose(O.deviation_sumsq(G, m1, g1), O.deviation_sumsq(G[perm], m2, g2),
                                   rtol=1e-12)


def test_sgd_update_direction():
    w = np.array([1.0, -2.0, 0.5])
    g = np.array([0.5, 0.5, -1.0])
    # one step against the gradient: w - 0.1 g, checked element by element by hand
    assert np.allclose(O.sgd_update(w, g, 0.1), [0.95, -2.05, 0.6], rtol=0, atol=1e-15)


def test_statistics_closed_forms():
    d = 40
    rng = np.random.default_rng(8)
    mu, a = rng.standard_normal(d), rng.standard_normal(d)
    G = np.stack([mu + a, mu - a])                         # two rows mu +- a
    mask = np.array([1, 1], dtype=np.uint8)
    gbar = O.aggregate(G, mask)
    np.testing.assert_allclose(gbar, mu, rtol=1e-14, atol=1e-14)
    SS = O.deviation_sumsq(G, mask, gbar)
    assert math.isclose(SS, 2 * float(a @ a), rel_tol=1e-13)
    assert math.isclose(O.variance_plus(SS, 2), 2 * float(a @ a), rel_tol=1e-13)
    # identical rows: no spread
    G = np.tile(mu, (5, 1))
    m5 = np.ones(5, dtype=np.uint8)
    assert O.deviation_sumsq(G, m5, O.aggregate(G, m5)) < 1e-24
    # k = 1 (R1): no variance
    assert math.isnan(O.variance_plus(3.0, 1))


def test_deviation_identity_with_row_norms():
    # sum_j ||g_j - gbar||^2 = sum_j ||g_j||^2 - k ||gbar||^2 (algebraic identity)
    G = _rows(17, 64, 9) + 0.3
    mask = (np.random.default_rng(10).random(17) < 0.6).astype(np.uint8)
    mask[0] = 1
    gbar = O.aggregate(G, mask)
    r = O.row_sqnorms(G, mask)
    k = int(mask.sum())
    lhs = O.deviation_sumsq(G, mask, gbar)
    rhs = np.nansum(r) - k * float(gbar @ gbar)
    assert math.isclose(lhs, rhs, rel_tol=1e-10)
    assert np.all(np.isnan(r[mask == 0]))


def test_row_norms_of_every_row_closed_form():
    """R12 with every row's norm: row j filled with +-(j+1) has ||g_j||^2 = d (j+1)^2,
    received or not; the received rows' values are those of the default form."""
    n, d = 6, 40
    signs = np.where(np.random.default_rng(11).random((n, d)) < 0.5, -1.0, 1.0)
    G = signs * (np.arange(n) + 1.0)[:, None]
    mask = np.array([1, 0, 0, 1, 1, 0], dtype=np.uint8)
    full = O.row_sqnorms(G, mask, all_rows=True)
    assert np.array_equal(full, d * (np.arange(n) + 1.0) ** 2)
    part = O.row_sqnorms(G, mask)
    assert np.array_equal(part[mask == 1], full[mask == 1]) and np.all(np.isnan(part[mask == 0]))


@pytest.mark.parametrize("k", [2, 3, 8])
def test_variance_estimator_unbiased_and_second_moment(k):
    """Eq. (10) is unbiased (E V^+ = d sigma^2) and Eq. (8): E||g_t||^2 = ||mu||^2 + V/k."""
    d, sigma, trials = 16, 0.7, 6000
    rng = np.random.default_rng(100 + k)
    mu = rng.standard_normal(d) * 0.5
    Vtrue = d * sigma ** 2
    mask = np.ones(k, dtype=np.uint8)
    Vs, g2s, Ns = [], [], []
    for _ in range(trials):
        G = mu + sigma * rng.standard_normal((k, d))
        gbar = O.aggregate(G, mask)
        V = O.variance_plus(O.deviation_sumsq(G, mask, gbar), k)
        Vs.append(V)
        g2 = float(gbar @ gbar)
        g2s.append(g2)
        Ns.append(g2 - V / k)                      # Eq. (11) before the clamp
    # V^+ * (k-1) / sigma^2 ~ chi^2 with d (k-1) dof: sd(V^+) = Vtrue * sqrt(2 / (d (k-1)))
    se = Vtrue * math.sqrt(2.0 / (d * (k - 1))) / math.sqrt(trials)
    assert abs(np.mean(Vs) - Vtrue) < 5 * se
    mu2 = float(mu @ mu)
    se2 = np.std(g2s) / math.sqrt(trials)
    assert abs(np.mean(g2s) - (mu2 + Vtrue / k)) < 5 * se2
    seN = np.std(Ns) / math.sqrt(trials)
    assert abs(np.mean(Ns) - mu2) < 5 * seN       # the unclamped Eq. (11) is unbiased for ||mu||^2


def test_norm_plus_clamps_at_zero():
    assert O.norm_plus(1.0, 10.0, 2) == 0.0
    assert O.norm_plus(3.0, 2.0, 2) == 2.0


def test_planted_wrong_denominator_is_caught(monkeypatch):
    """A variance divided by k instead of k-1 must fail the unbiasedness pin."""
    monkeypatch.setattr(O, "variance_plus", lambda SS, k: SS / float(k))
    with pytest.raises(AssertionError):
        test_variance_estimator_unbiased_and_second_moment(2)
