"""Plain, slow fp64 CPU oracle of one Dynamic Backup Workers (DBW) iteration.

TEST INFRASTRUCTURE.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import or call
anything here.  The product path (the CUDA library and its Python binding) never
does, and this module imports nothing from it: inputs arrive as numpy arrays.

What it computes, in the paper's order and notation (Xu, Neglia, Sebastianelli,
"Dynamic Backup Workers for Parallel Machine Learning"):

* Eq. (2)   per-worker minibatch gradient g_i = (1/B) sum_{x in B_i} grad f(x, w)
            of a ReLU MLP with softmax cross-entropy loss f (Sect. 4).
* Eq. (4)   the PS keeps the k = n - b first arrivals and averages them;
            b = 0 is Eq. (3)'s full synchronous mean.
* Eq. (3)   SGD update w <- w - eta * g_t.
* Eq. (10)  unbiased variance estimate V^+ over the k received rows (two-pass).
* Eq. (11)  ||grad F||^2^+ = max(||g_t||^2 - V^+/k, 0).
* Sect. 3.1 loss estimate F^_t = mean of the received workers' minibatch losses,
            observed gain G^+ = F^_{t-1} - F^_t and Eq. (12) for L^+.
* Eqs. (13)-(15)  window means of the last D "+" estimates.
* Eq. (16)  gain estimate G^_{k,t} for every k.
* Sect. 3.2 / Eq. (17)  time estimate T^_k.  Under the push-and-interrupt model
            used here every iteration draws fresh times and all n arrivals are
            observed, so every k has the same number of samples and the per-k
            means of sorted vectors are already monotone: the constrained
            least-squares problem (17) returns the plain per-k means.
* Eqs. (18)-(19)  greedy choice of k_t with the loss-increase guard.

Readings of points the paper leaves open (each also listed in the design notes):

 R1  k = 1: Eq. (10) divides by k-1 = 0.  V^+ is NaN, and neither V^+,
     ||grad F||^2^+ nor the next L^+ is recorded; g_t and w are still updated.
 R2  "the first t-1 if t <= D": each window averages the min(D, #recorded)
     most recent recorded values, summed newest first and divided by the count.
 R3  k_0 = n; L^+ needs two losses, so k_1 = n too: DBW chooses only when all
     three windows hold at least one value.
 R4  Eq. (12): a value whose denominator is <= 0 or that is not finite is not
     recorded; negative finite values are kept.
 R5  the symbol in the loss estimate of Sect. 3.1 is read as f (cross-entropy).
 R6  argmax ties in Eq. (18) go to the largest k.
 R7  "all G^ < 0 => k = n": k_t = n if no k has G^_k > 0, else the argmax over
     the k with G^_k > 0.
 R8  the guard of Eq. (19) applies only when F^_{t-1} and F^_{t-2} exist; the
     result is capped at n.
 R9  L^+_t uses the "+" estimates and k of iteration t-1 and F^_{t-1} - F^_t.
 R10 arrival order: (time, worker index) lexicographic, lower index first.
 R11 push-and-interrupt time model, see Eq. (17) above.
 R12 the statistics use the k received rows only.
 R13 ReLU'(0) = 0; numerically stable log-softmax; sampling with replacement.
     Where a pre-activation lies within rounding of 0 the derivative's value is a
     decision the kernel's precision may take either way; ``worker_grads`` can
     evaluate the other side (``relu_flip``) so that a check can accept either.
 R14 bf16 operands (the two large MLPs): every GEMM operand -- X, the weight
     matrices, the hidden activations and the backpropagated dZ -- is rounded to
     bf16 (round to nearest even) as it enters a product; everything else is fp64.

Scalar estimator arithmetic (F^, V^+, Eq. (11), Eq. (12), the windows, Eq. (16),
T^_k, the ratio of Eq. (18)) is written as plain Python float operations in a
fixed order; the device estimator performs the same IEEE operations in the same
order, which is what makes the chosen b comparable bit for bit.
"""
from __future__ import annotations

from dataclasses import dataclass, field
import math

import numpy as np

DMAX = 64          # capacity of the history rings (window D must be <= DMAX)


# =============================================================== model layout
def param_layout(widths):
    """Offsets of each layer in the flat vector: W_l [out, in] row-major, then b_l [out]."""
    layers = []
    off = 0
    for l in range(len(widths) - 1):
        fin, fout = int(widths[l]), int(widths[l + 1])
        layers.append((off, fout, fin, off + fout * fin))
        off += fout * fin + fout
    return layers, off


def unflatten(w, widths):
    layers, d = param_layout(widths)
    assert w.shape[0] == d
    out = []
    for (offW, fout, fin, offb) in layers:
        out.append((w[offW:offW + fout * fin].reshape(fout, fin), w[offb:offb + fout]))
    return out


def bf16_round(x):
    """Round fp32 values to the nearest bf16 (ties to even); returned as fp64.

    bf16 keeps the top 16 bits of an IEEE binary32 word; rounding adds half an
    ulp of the kept part (0x7FFF) plus the lowest kept bit (for ties to even)
    before truncating.  Inputs must be finite.
    """
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    lsb = (u >> np.uint64(16)) & np.uint64(1)
    r = ((u + np.uint64(0x7FFF) + lsb) & np.uint64(0xFFFF0000)).astype(np.uint32)
    return r.view(np.float32).astype(np.float64)


# ================================================== Eq. (2): worker gradients
def _log_softmax(Z):
    m = Z.max(axis=1, keepdims=True)
    s = Z - m
    return s - np.log(np.exp(s).sum(axis=1, keepdims=True))


def sample_losses(widths, w, X, y, bf16=False):
    """Per-sample cross-entropy f(x, w) of the ReLU MLP (forward pass only)."""
    params = unflatten(np.asarray(w, dtype=np.float64), widths)
    if bf16:
        A = bf16_round(X)
        params = [(bf16_round(np.asarray(W, dtype=np.float32)), b) for (W, b) in params]
    else:
        A = np.asarray(X, dtype=np.float64)
    L = len(params)
    for l, (W, b) in enumerate(params):
        Z = A @ W.T + b
        A = np.maximum(Z, 0.0) if l < L - 1 else Z
    lsm = _log_softmax(A)
    return -lsm[np.arange(A.shape[0]), np.asarray(y, dtype=np.int64)]


def worker_grads(widths, w, X, y, n, B, bf16=False, relu_flip=None, return_preact=False, return_magnitude=False):
    """Eq. (2) for every worker: G [n, d] fp64 and the minibatch mean losses [n].

    Rows ``i*B .. i*B+B-1`` of X / y are worker i's minibatch.  Backpropagation
    through Z_l = A_{l-1} W_l^T + b_l, A_l = ReLU(Z_l), softmax cross-entropy on
    the last Z.  Each worker's gradient is the mean over its own B samples, so
    dL/dZ_last = (softmax - onehot) / B and the per-worker weight gradient is
    dZ_l[i]^T A_{l-1}[i].

    bf16 (R14): every GEMM operand is rounded to bf16 before it is used -- X, the
    weight matrices, the hidden activations A_l and the backpropagated dZ_l --
    and all arithmetic is fp64.

    relu_flip (R13): optional list, one boolean [n*B, width] array per hidden
    layer; where True the ReLU derivative takes the other one-sided value
    (1[Z > 0] is replaced by 1[Z >= 0] semantics at that entry, i.e. the mask
    bit is inverted).  Only meaningful where Z is within rounding of 0.
    return_preact: also return the hidden pre-activations Z_l and their scale
    sum_k |A_{l-1}[r,k] W_l[u,k]| + |b_l[u]| (the size a rounding error of Z is
    relative to).
    return_magnitude: also return, for every entry of G, the sum of the absolute
    values of the products it is made of (|dZ_l|^T |A_{l-1}| for weights, the sum
    of |dZ_l| for biases): the scale a floating-point error of that entry is
    relative to.  Returned last.
    """
    rnd = (lambda a: bf16_round(np.asarray(a, dtype=np.float32))) if bf16 else (lambda a: a)
    w64 = np.asarray(w, dtype=np.float64)
    params = unflatten(w64, widths)
    if bf16:
        params = [(rnd(W), b) for (W, b) in params]
    A0 = rnd(np.asarray(X, dtype=np.float64))
    M = n * B
    assert A0.shape[0] == M
    L = len(params)
    acts = [A0]          # A_0 .. A_{L-1} as the GEMMs consume them
    zs, scales = [], []
    A = A0
    for l, (W, b) in enumerate(params):
        Z = A @ W.T + b
        if l < L - 1:
            zs.append(Z)
            if return_preact:
                scales.append(np.abs(A) @ np.abs(W).T + np.abs(b))
            A = rnd(np.maximum(Z, 0.0))
            acts.append(A)
        else:
            A = Z
    logits = A
    yy = np.asarray(y, dtype=np.int64)
    lsm = _log_softmax(logits)
    per_sample = -lsm[np.arange(M), yy]
    loss = per_sample.reshape(n, B).mean(axis=1)
    dZ = np.exp(lsm)
    dZ[np.arange(M), yy] -= 1.0
    dZ = rnd(dZ / B)
    layers, d = param_layout(widths)
    G = np.empty((n, d), dtype=np.float64)
    Gmag = np.empty((n, d), dtype=np.float64) if return_magnitude else None
    for l in range(L - 1, -1, -1):
        offW, fout, fin, offb = layers[l]
        Ain = acts[l].reshape(n, B, fin)
        dZi = dZ.reshape(n, B, fout)
        G[:, offW:offW + fout * fin] = np.einsum("nbo,nbi->noi", dZi, Ain).reshape(n, -1)
        G[:, offb:offb + fout] = dZi.sum(axis=1)
        if return_magnitude:
            Gmag[:, offW:offW + fout * fin] = np.einsum("nbo,nbi->noi", np.abs(dZi), np.abs(Ain)).reshape(n, -1)
            Gmag[:, offb:offb + fout] = np.abs(dZi).sum(axis=1)
        if l > 0:
            W = params[l][0]
            live = zs[l - 1] > 0.0
            if relu_flip is not None and relu_flip[l - 1] is not None:
                live = live ^ relu_flip[l - 1]
            dZ = rnd((dZ @ W) * live)
    out = (G, loss)
    if return_preact:
        out = out + (zs, scales)
    if return_magnitude:
        out = out + (Gmag,)
    return out


def single_worker_grad(widths, w, X, y, B, bf16=False, relu_flip=None):
    """Eq. (2) for one worker only (its B rows); used for sampled checks at scale."""
    G, loss = worker_grads(widths, w, X, y, 1, B, bf16, relu_flip)
    return G[0], loss[0]


# ======================================== Eq. (4): arrival order and selection
def select_fastest(times, b):
    """Arrival order of the n gradients and the set kept by the PS (Eq. (4)).

    Worker i arrives before j iff (T_i, i) < (T_j, j) lexicographically (R10).
    Returns (order [n] int32: worker of each arrival rank, mask [n] uint8: 1 for
    the k = n - b first arrivals, tsorted [n] fp64: the order statistics).
    """
    t = np.asarray(times, dtype=np.float64)
    n = t.shape[0]
    if not (0 <= b <= n - 1):
        raise ValueError("b must be in [0, n-1]")
    k = n - b
    idx = np.arange(n)
    before = (t[None, :] < t[:, None]) | ((t[None, :] == t[:, None]) & (idx[None, :] < idx[:, None]))
    rank = before.sum(axis=1)          # rank[i] = number of workers that arrive before i
    order = np.empty(n, dtype=np.int32)
    order[rank] = idx
    tsorted = np.empty(n, dtype=np.float64)
    tsorted[rank] = t
    mask = (rank < k).astype(np.uint8)
    return order, mask, tsorted


def aggregate(G, mask):
    """Eq. (4): g_t = (1/k) sum over the k received rows (b = 0 gives Eq. (3)'s mean)."""
    sel = np.flatnonzero(np.asarray(mask))
    return np.asarray(G, dtype=np.float64)[sel].sum(axis=0) / len(sel)


def sgd_update(w, gbar, lr):
    """Eq. (3): w_{t+1} = w_t - eta * g_t."""
    return np.asarray(w, dtype=np.float64) - lr * gbar


# ============================================ Sect. 3.1: gradient statistics
def row_sqnorms(G, mask, all_rows=False):
    """||g_j||^2 for the received rows j (NaN for rows not received).

    R12: the statistics of Eq. (10) use the k received rows only.  With
    ``all_rows`` the norm of every row is reported as well (the rows the PS did
    not receive included); none of them enters a statistic."""
    G = np.asarray(G, dtype=np.float64)
    r = np.full(G.shape[0], np.nan)
    rows = range(G.shape[0]) if all_rows else np.flatnonzero(np.asarray(mask))
    for j in rows:
        r[j] = float(np.dot(G[j], G[j]))
    return r


def deviation_sumsq(G, mask, gbar):
    """sum_l sum_{j received} ([g_j - g_t]_l)^2 (two passes: mean first, then deviations)."""
    G = np.asarray(G, dtype=np.float64)
    s = 0.0
    for j in np.flatnonzero(np.asarray(mask)):
        dev = G[j] - gbar
        s += float(np.dot(dev, dev))
    return s


def variance_plus(SS, k):
    """Eq. (10): V^+ = SS / (k - 1); NaN when k = 1 (R1)."""
    if k < 2:
        return math.nan
    return SS / float(k - 1)


def norm_plus(gbar_sq, V, k):
    """Eq. (11): max(||g_t||^2 - V^+/k, 0)."""
    x = gbar_sq - V / float(k)
    return x if x > 0.0 else 0.0


def loss_hat(loss, mask):
    """F^_t: mean over the received workers of their minibatch mean loss (R5).

    Summed in increasing worker index in fp64.
    """
    acc = 0.0
    k = 0
    for j in np.flatnonzero(np.asarray(mask)):
        acc = acc + float(loss[j])
        k += 1
    return acc / float(k)


def L_plus(lr, N_prev, V_prev, k_prev, F_prev, F_now):
    """Eq. (12), solved from Eq. (9) with the observed gain F^_{t-1} - F^_t (R9)."""
    num = 2.0 * ((lr * N_prev) - (F_prev - F_now))
    den = (lr * lr) * (N_prev + (V_prev / float(k_prev)))
    return num, den


# ======================================================== estimator state
@dataclass
class State:
    """Everything the PS carries from iteration to iteration.

    Rings hold the last DMAX recorded "+" estimates (count = total recorded);
    S[k-1] is the running sum of the k-th order statistic, c the number of
    observed time vectors.
    """
    n: int
    D: int
    t: int = 0
    k_last: int = 0
    c: int = 0
    cntV: int = 0
    cntN: int = 0
    cntL: int = 0
    flags: int = 0
    has_last: int = 0
    F_last: float = math.nan
    F_prev: float = math.nan
    N_last: float = math.nan
    V_last: float = math.nan
    vclock: float = 0.0
    ringV: list = field(default_factory=lambda: [0.0] * DMAX)
    ringN: list = field(default_factory=lambda: [0.0] * DMAX)
    ringL: list = field(default_factory=lambda: [0.0] * DMAX)
    S: list = None

    def __post_init__(self):
        if self.S is None:
            self.S = [0.0] * self.n
        if not (1 <= self.D <= DMAX):
            raise ValueError("D must be in [1, DMAX]")


def _push(ring, cnt, x):
    ring[cnt % DMAX] = x
    return cnt + 1


def window_mean(ring, cnt, D):
    """Eqs. (13)-(15): mean of the m = min(D, cnt) most recent values, newest first (R2)."""
    m = min(D, cnt)
    acc = 0.0
    for v in range(1, m + 1):
        acc = acc + ring[(cnt - v) % DMAX]
    return acc / float(m)


FLAG_K1 = 1 << 0          # k = 1: no variance this iteration (R1)
FLAG_L_SKIPPED = 1 << 1   # Eq. (12) value not recorded (R4)


def record_iteration(st: State, k, SS, gbar_sq, loss, mask, tsorted, lr):
    """End-of-iteration bookkeeping (Sect. 3.1, 3.2): returns a dict of the "+" estimates.

    SS = sum of squared deviations (Eq. (10)'s double sum), gbar_sq = ||g_t||^2.
    """
    V = variance_plus(SS, k)
    N = norm_plus(gbar_sq, V, k) if k >= 2 else math.nan
    F = loss_hat(loss, mask)
    L = math.nan
    flags = 0
    if k < 2:
        flags |= FLAG_K1
    if st.t >= 1 and st.has_last:
        num, den = L_plus(lr, st.N_last, st.V_last, st.k_last, st.F_last, F)
        if den > 0.0:
            L = num / den
        if not (den > 0.0 and math.isfinite(L)):
            L = math.nan
            flags |= FLAG_L_SKIPPED
        else:
            st.cntL = _push(st.ringL, st.cntL, L)
    if k >= 2:
        st.cntV = _push(st.ringV, st.cntV, V)
        st.cntN = _push(st.ringN, st.cntN, N)
        st.N_last, st.V_last, st.has_last = N, V, 1
    else:
        st.N_last, st.V_last, st.has_last = math.nan, math.nan, 0
    # Sect. 3.2: all n arrivals are observed (late workers still notify).
    for i in range(st.n):
        st.S[i] = st.S[i] + float(tsorted[i])
    st.c += 1
    st.vclock = st.vclock + float(tsorted[k - 1])
    st.F_prev, st.F_last = st.F_last, F
    st.k_last = k
    st.t += 1
    st.flags |= flags
    return {"k": k, "SS": SS, "gbar_sq": gbar_sq, "V": V, "N": N, "F": F, "L": L,
            "flags": flags, "vclock": st.vclock}


def gain_estimates(st: State, lr):
    """Eq. (16) for k = 1..n with the window means of Eqs. (13)-(15); None before R3 holds."""
    if st.cntV == 0 or st.cntN == 0 or st.cntL == 0 or st.c == 0:
        return None
    Vh = window_mean(st.ringV, st.cntV, st.D)
    Nh = window_mean(st.ringN, st.cntN, st.D)
    Lh = window_mean(st.ringL, st.cntL, st.D)
    q = ((Lh * lr) * lr) / 2.0
    gains = []
    for k in range(1, st.n + 1):
        gains.append(((lr - q) * Nh) - (q * (Vh / float(k))))
    return gains


def time_estimates(st: State):
    """T^_k = S_k / c: the per-k mean order statistic (Eq. (17) under R11)."""
    return [st.S[k - 1] / float(st.c) for k in range(1, st.n + 1)]


def _ieee_div(a, b):
    """a / b with IEEE 754 semantics (x/0 = +-inf, 0/0 = NaN) instead of a Python error."""
    with np.errstate(divide="ignore", invalid="ignore"):
        return float(np.float64(a) / np.float64(b))


def choose_k(st: State, lr, beta, blind=False, T=None):
    """Eqs. (18)-(19): k_t for the iteration about to start; returns (k_t, ratio list).

    ``blind`` is the paper's B-DBW variant (Sect. 4): the gain is k itself.
    ``T`` replaces the push-and-interrupt time estimates S_k / c by given T^_k
    (the push-and-wait estimator of Eq. (17)); NaN estimates mean "none yet".
    """
    n = st.n
    ratio = [math.nan] * n
    kstar = n
    have_T = (st.c > 0) if T is None else (not math.isnan(T[0]))
    if T is None and st.c > 0:
        T = time_estimates(st)
    if blind:
        if have_T:
            best = -math.inf
            for k in range(1, n + 1):
                ratio[k - 1] = _ieee_div(float(k), T[k - 1])
                if ratio[k - 1] >= best:
                    best, kstar = ratio[k - 1], k
    else:
        gains = gain_estimates(st, lr)
        if gains is not None and have_T:
            best = -math.inf
            found = False
            for k in range(1, n + 1):
                ratio[k - 1] = _ieee_div(gains[k - 1], T[k - 1])
                if gains[k - 1] > 0.0 and ratio[k - 1] >= best:
                    best, kstar, found = ratio[k - 1], k, True
            if not found:
                kstar = n
    if st.t >= 2 and st.F_last > beta * st.F_prev and st.k_last < n:
        kstar = max(kstar, st.k_last + 1)
    return min(kstar, n), ratio


# ========================================================== one iteration
def step(st: State, widths, w, X, y, times, B, lr, beta, bf16=False, b=None, blind=False):
    """One DBW iteration: choose b (unless given), gradients, selection, update, statistics."""
    n = st.n
    if b is None:
        k, ratio = choose_k(st, lr, beta, blind)
        b = n - k
    else:
        ratio = None
    G, loss = worker_grads(widths, w, X, y, n, B, bf16)
    order, mask, tsorted = select_fastest(times, b)
    k = n - b
    gbar = aggregate(G, mask)
    w_new = sgd_update(w, gbar, lr)
    SS = deviation_sumsq(G, mask, gbar)
    gsq = float(np.dot(gbar, gbar))
    rec = record_iteration(st, k, SS, gsq, loss, mask, tsorted, lr)
    return {"b": b, "ratio": ratio, "G": G, "loss": loss, "order": order, "mask": mask,
            "tsorted": tsorted, "gbar": gbar, "w": w_new, "row_sqnorm": row_sqnorms(G, mask),
            **rec}
