"""Pins of the oracle's DBW estimator (Sect. 3.1-3.3): the behaviours the paper
states for special cases, the algebraic link between Eq. (9) and Eq. (12), the
window rule, the order-statistic closed form for T^_k, monotonicity (Appendix A)
and brute-force enumeration of Eq. (18) on small n."""
import json
import math
import os

import numpy as np
import pytest

from oracle import dbw_oracle as O
from paper_2004_14696_gb300 import inputs


def _state_with(n, D=5, V=1.0, N=1.0, L=1.0, T=None, t=5, k_last=None, F_last=1.0, F_prev=1.0):
    st = O.State(n=n, D=D)
    for _ in range(D):
        st.cntV = O._push(st.ringV, st.cntV, V)
        st.cntN = O._push(st.ringN, st.cntN, N)
        st.cntL = O._push(st.ringL, st.cntL, L)
    T = np.arange(1, n + 1, dtype=float) if T is None else np.asarray(T, dtype=float)
    st.c = 4
    st.S = [4.0 * x for x in T]
    st.t = t
    st.k_last = n if k_last is None else k_last
    st.F_last, st.F_prev = F_last, F_prev
    return st


@pytest.fixture(scope="module")
def paper(golden_dir):
    with open(os.path.join(golden_dir, "paper_settings.json")) as f:
        return json.load(f)


def test_L_plus_inverts_the_gain_formula():
    """Eq. (12) is Eq. (9) solved for L: feed it the gain Eq. (9) predicts, get L back."""
    rng = np.random.default_rng(0)
    for _ in range(200):
        L, N, V = rng.uniform(0.1, 10), rng.uniform(0, 5), rng.uniform(0, 50)
        eta, k = rng.uniform(1e-3, 0.2), int(rng.integers(2, 64))
        gain = (eta - L * eta ** 2 / 2) * N - (L * eta ** 2 / 2) * V / k     # Eq. (9)
        F_prev = 3.0
        num, den = O.L_plus(eta, N, V, k, F_prev, F_prev - gain)
        assert math.isclose(num / den, L, rel_tol=1e-9)


def test_window_rule():
    ring = [0.0] * O.DMAX
    cnt = 0
    for v in range(1, 11):
        cnt = O._push(ring, cnt, float(v))
    assert O.window_mean(ring, cnt, 5) == 8.0           # mean of 6..10
    assert O.window_mean(ring, 3, 5) == 2.0             # only 1, 2, 3 recorded
    for v in range(11, 11 + 2 * O.DMAX):                 # ring wraps
        cnt = O._push(ring, cnt, float(v))
    assert O.window_mean(ring, cnt, 1) == float(10 + 2 * O.DMAX)


def test_gain_increases_with_k_for_nonnegative_L():
    st = _state_with(12, V=3.0, N=0.5, L=2.0)
    g = O.gain_estimates(st, 0.1)
    assert all(g[i] < g[i + 1] for i in range(len(g) - 1))


def test_equal_times_choose_all_workers(paper):
    """alpha = 0 (all times equal): the PS should aggregate all gradients (Sect. 4.1)."""
    case = paper["equal_times_all_workers"]
    n = case["n"]
    st = _state_with(n, V=5.0, N=1.0, L=1.0, T=[1.0] * n)
    k, _ = O.choose_k(st, 0.05, paper["beta"]["value"])
    assert k == case["expected_k"]


def test_half_workers_five_times_slower_choose_half(paper):
    """Half of the workers 5x slower, times otherwise deterministic: k = n/2 (Sect. 4.3)."""
    case = paper["slowdown_half_workers"]
    n = case["n"]
    st = O.State(n=n, D=paper["D"]["value"])
    # record the deterministic order statistics of a few slowed-down iterations
    for t in range(6):
        times = inputs.completion_times(0, 100 + t, n, "slowdown", value=1.0,
                                        factor=case["slow_factor"], t_switch=0)
        _, mask, ts = O.select_fastest(times, 0)
        O.record_iteration(st, n, SS=float(n - 1), gbar_sq=2.0, loss=np.full(n, 1.0 - 0.01 * t),
                           mask=mask, tsorted=ts, lr=0.05)
    k, ratio = O.choose_k(st, 0.05, paper["beta"]["value"])
    assert k == case["expected_k"]


def test_zero_variance_strictly_increasing_times_choose_one():
    st = _state_with(10, V=0.0, N=1.0, L=1.0)
    k, _ = O.choose_k(st, 0.05, 1.01)
    assert k == 1


def test_all_gains_negative_choose_n(paper):
    st = _state_with(10, V=1.0, N=0.0, L=5.0)      # G_k = -q V / k < 0 for all k
    assert all(g < 0 for g in O.gain_estimates(st, 0.1))
    k, _ = O.choose_k(st, 0.1, 1.01)
    assert k == 10


def test_startup_waits_for_all():
    st = O.State(n=8, D=5)
    assert O.choose_k(st, 0.05, 1.01)[0] == 8
    # one iteration recorded: V and N exist but no L yet (R3)
    _, mask, ts = O.select_fastest(np.arange(8.0), 0)
    O.record_iteration(st, 8, 7.0, 1.0, np.ones(8), mask, ts, 0.05)
    assert st.cntL == 0 and O.choose_k(st, 0.05, 1.01)[0] == 8


def test_loss_increase_guard():
    """Eq. (19): if F^_{t-1} > beta F^_{t-2}, k_t >= k_{t-1} + 1 (capped at n)."""
    n = 10
    base = dict(V=0.0, N=1.0, L=1.0)                     # Eq. (18) alone picks k = 1
    st = _state_with(n, k_last=4, F_last=1.02, F_prev=1.0, **base)
    assert O.choose_k(st, 0.05, 1.01)[0] == 5
    st = _state_with(n, k_last=4, F_last=1.005, F_prev=1.0, **base)
    assert O.choose_k(st, 0.05, 1.01)[0] == 1            # rise below beta: no guard
    st = _state_with(n, k_last=n, F_last=2.0, F_prev=1.0, **base)
    assert O.choose_k(st, 0.05, 1.01)[0] == 1            # k_{t-1} = n: indicator is 0
    st = _state_with(n, k_last=4, F_last=2.0, F_prev=1.0, t=1, **base)
    assert O.choose_k(st, 0.05, 1.01)[0] == 1            # F^_{t-2} does not exist yet (R8)


@pytest.mark.parametrize("n", [1, 2, 3, 5, 8])
def test_brute_force_enumeration_of_greedy_choice(n):
    rng = np.random.default_rng(n)
    for trial in range(300):
        T = np.sort(rng.choice([0.5, 1.0, 1.5, 2.0], size=n))    # ties in T make ties in ratio
        st = _state_with(n, V=float(rng.choice([0.0, 1.0, 4.0])), N=float(rng.choice([0.0, 0.5, 2.0])),
                         L=float(rng.choice([-1.0, 0.0, 2.0, 40.0])), T=T, k_last=int(rng.integers(1, n + 1)),
                         F_last=float(rng.choice([1.0, 1.2])), F_prev=1.0)
        lr = 0.1
        gains = O.gain_estimates(st, lr)
        ratios = [gains[k - 1] / (st.S[k - 1] / st.c) for k in range(1, n + 1)]
        pos = [k for k in range(1, n + 1) if gains[k - 1] > 0]
        if pos:
            best = max(ratios[k - 1] for k in pos)
            k18 = max(k for k in pos if ratios[k - 1] == best)
        else:
            k18 = n
        guard = st.F_last > 1.01 * st.F_prev and st.k_last < n
        expect = max(k18, st.k_last + 1) if guard else k18
        assert O.choose_k(st, lr, 1.01)[0] == min(expect, n)


def test_time_estimate_matches_exponential_order_statistics():
    """Shifted Exp(1): E[T_(k)] = shift + sum_{j=n-k+1}^{n} 1/j (Renyi); T^_k is monotone."""
    n, iters, shift = 8, 20000, 1.0
    st = O.State(n=n, D=5)
    mask = np.ones(n, dtype=np.uint8)
    sq = np.zeros(n)
    for t in range(iters):
        times = inputs.completion_times(11, t, n, "shifted_exp", shift=shift, rate=1.0)
        ts = np.sort(times)
        sq += (ts - shift) ** 2
        for i in range(n):
            st.S[i] += float(ts[i])
        st.c += 1
    T = O.time_estimates(st)
    assert all(T[i] <= T[i + 1] for i in range(n - 1))          # Appendix A ordering
    for k in range(1, n + 1):
        mean = sum(1.0 / j for j in range(n - k + 1, n + 1))
        var = sum(1.0 / j ** 2 for j in range(n - k + 1, n + 1))
        assert abs(T[k - 1] - (shift + mean)) < 5 * math.sqrt(var / iters)


def test_blind_variant_uses_k_over_time():
    n = 6
    st = _state_with(n, T=[1.0, 1.0, 1.0, 5.0, 5.0, 5.0])
    k, ratio = O.choose_k(st, 0.05, 1.01, blind=True)
    assert k == 3 and ratio[2] == 3.0


def test_record_iteration_bookkeeping():
    n = 4
    st = O.State(n=n, D=5)
    times = np.array([2.0, 1.0, 4.0, 3.0])
    _, mask, ts = O.select_fastest(times, 1)
    rec = O.record_iteration(st, 3, SS=6.0, gbar_sq=5.0, loss=np.array([1.0, 2.0, 9.0, 3.0]),
                             mask=mask, tsorted=ts, lr=0.1)
    assert rec["V"] == 3.0 and rec["N"] == 4.0 and rec["F"] == 2.0   # (1+2+3)/3
    assert st.vclock == 3.0 and st.S == [1.0, 2.0, 3.0, 4.0] and st.c == 1 and st.t == 1
    assert math.isnan(rec["L"]) and st.cntL == 0
    # second iteration: observed gain F^0 - F^1 = 0.5 gives L^+ by Eq. (12)
    rec2 = O.record_iteration(st, 3, SS=6.0, gbar_sq=5.0, loss=np.array([1.5, 1.5, 9.0, 1.5]),
                              mask=mask, tsorted=ts, lr=0.1)
    assert math.isclose(rec2["L"], 2 * (0.1 * 4.0 - 0.5) / (0.01 * (4.0 + 3.0 / 3)), rel_tol=1e-12)
    assert st.cntL == 1 and st.F_prev == 2.0 and st.F_last == 1.5 and st.vclock == 6.0


def test_planted_sign_error_in_gain_is_caught(monkeypatch, paper):
    """A flipped sign on the variance term of Eq. (16) must fail the equal-times pin."""
    def flipped(st, lr):
        Vh = O.window_mean(st.ringV, st.cntV, st.D)
        Nh = O.window_mean(st.ringN, st.cntN, st.D)
        Lh = O.window_mean(st.ringL, st.cntL, st.D)
        q = ((Lh * lr) * lr) / 2.0
        return [((lr - q) * Nh) + (q * (Vh / float(k))) for k in range(1, st.n + 1)]
    monkeypatch.setattr(O, "gain_estimates", flipped)
    with pytest.raises(AssertionError):
        test_equal_times_choose_all_workers(paper)


def test_zero_time_estimate_follows_ieee_division():
    """A time estimate of 0 gives an infinite ratio (IEEE), which Eq. (18) then prefers."""
    st = _state_with(4, V=1.0, N=1.0, L=1.0, T=[0.0, 1.0, 2.0, 3.0])
    k, ratio = O.choose_k(st, 0.05, 1.01)
    assert ratio[0] == math.inf and k == 1
