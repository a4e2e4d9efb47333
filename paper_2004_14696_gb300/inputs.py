"""Seeded synthetic inputs for the DBW parameter-server iteration.

This module only draws random numbers and lays them out; it holds none of the
method's arithmetic (no gradients, no selection, no statistics).  Both the CUDA
path and the fp64 CPU oracle receive the arrays produced here, so the two sides
always see bit-identical inputs.

Every draw comes from numpy's PCG64 generator seeded with a ``SeedSequence``
keyed by ``(seed, stream, *counters)``, so the inputs of iteration ``t`` can be
produced without replaying iterations ``0..t-1``.

The time models are the round-trip-time families the paper's experiments use
(Sect. 4: shifted exponential ``1 - alpha + alpha * Exp(1)``, Pareto, slow
workers); the datasets are stand-ins with the shapes of MNIST (784 features,
10 classes) and CIFAR10 (3072 features), which are not available here.
"""
from __future__ import annotations

import numpy as np

# Streams: one independent generator family per kind of input.
STREAM_DATA = 1
STREAM_LABELS = 2
STREAM_INIT = 3
STREAM_INDEX = 4
STREAM_TIMES = 5
STREAM_GRADS = 6
STREAM_PICK = 7
STREAM_GRAD_COLS = 8
GRAD_COL_CHUNK = 1 << 16

BASE_SEED = 2004146960


def rng(seed: int, stream: int, *counters: int) -> np.random.Generator:
    """Generator for ``(seed, stream, counters...)``; independent across keys."""
    key = [int(seed) & 0xFFFFFFFF, int(stream)] + [int(c) for c in counters]
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence(key)))


def uniform01_open_left(g: np.random.Generator, size) -> np.ndarray:
    """U in (0, 1]: ``1 - U[0,1)``; never 0, so ``log U`` and ``U**-a`` are finite."""
    return 1.0 - g.random(size, dtype=np.float64)


# --------------------------------------------------------------------- datasets
def feature_pool(seed: int, S: int, dim: int, dist: str = "normal",
                 chunk_rows: int = 4096) -> np.ndarray:
    """Synthetic dataset features ``[S, dim]`` fp32, ``N(0,1)`` or ``U(0,1)``.

    Drawn in row chunks (each chunk keyed by its index) to bound peak memory.
    """
    out = np.empty((S, dim), dtype=np.float32)
    for c0 in range(0, S, chunk_rows):
        c1 = min(S, c0 + chunk_rows)
        g = rng(seed, STREAM_DATA, c0 // chunk_rows)
        if dist == "normal":
            out[c0:c1] = g.standard_normal((c1 - c0, dim), dtype=np.float32)
        elif dist == "uniform":
            out[c0:c1] = g.random((c1 - c0, dim), dtype=np.float32)
        else:
            raise ValueError(f"unknown feature distribution {dist!r}")
    return out


def label_pool(seed: int, S: int, classes: int) -> np.ndarray:
    """Uniform class labels ``[S]`` int32 in ``[0, classes)``."""
    return rng(seed, STREAM_LABELS).integers(0, classes, size=S, dtype=np.int32)


def teacher_labels(seed: int, X: np.ndarray, classes: int, chunk_rows: int = 8192) -> np.ndarray:
    """Learnable labels [S] int32: argmax over classes of X @ T, with T ~ N(0,1) [dim, classes]
    a fixed seeded "teacher" map (a task a classifier can actually fit, so that
    training losses fall steadily instead of fluctuating around log(classes))."""
    T = rng(seed, STREAM_LABELS, 1).standard_normal((X.shape[1], classes)).astype(np.float32)
    out = np.empty(X.shape[0], dtype=np.int32)
    for c0 in range(0, X.shape[0], chunk_rows):
        out[c0:c0 + chunk_rows] = np.argmax(X[c0:c0 + chunk_rows] @ T, axis=1)
    return out


# --------------------------------------------------------------------- model init
def param_count(widths) -> int:
    """Number of parameters of a fully connected net with these layer widths."""
    return sum(int(widths[l + 1]) * (int(widths[l]) + 1) for l in range(len(widths) - 1))


def kaiming_uniform_params(seed: int, widths) -> np.ndarray:
    """Flat fp32 parameter vector: per layer ``W [out, in]`` row-major then ``b [out]``.

    Weights ~ U(-sqrt(6/in), sqrt(6/in)) (He/Kaiming uniform for ReLU), biases 0.
    """
    d = param_count(widths)
    w = np.zeros(d, dtype=np.float32)
    off = 0
    for l in range(len(widths) - 1):
        fan_in, fan_out = int(widths[l]), int(widths[l + 1])
        bound = np.float32(np.sqrt(6.0 / fan_in))
        g = rng(seed, STREAM_INIT, l)
        W = g.random((fan_out, fan_in), dtype=np.float32)
        w[off:off + fan_out * fan_in] = ((W * 2.0 - 1.0) * bound).ravel()
        off += fan_out * fan_in + fan_out
    return w


# --------------------------------------------------------------------- per iteration
def minibatch_indices(seed: int, t: int, n: int, B: int, S: int) -> np.ndarray:
    """Indices ``[n*B]`` int32 of the samples of iteration t, drawn with replacement.

    Worker ``i`` owns entries ``i*B .. i*B+B-1``.  ``floor(U * S)`` with U in [0,1).
    """
    u = rng(seed, STREAM_INDEX, t).random(n * B, dtype=np.float64)
    return np.minimum((u * S).astype(np.int64), S - 1).astype(np.int32)


def completion_times(seed: int, t: int, n: int, model: str, **p) -> np.ndarray:
    """Per-worker round-trip times ``[n]`` fp64 of iteration t (fresh every iteration).

    Models (all strictly positive):
      ``shifted_exp``  shift + Exp(rate)              (p: shift, rate)
      ``lognormal``    exp(mu + sigma * N(0,1))        (p: mu, sigma)
      ``exp_slow``     Exp(rate), a fixed seeded set of ``floor(frac*n)`` workers
                       multiplied by ``factor``       (p: rate, frac, factor)
      ``pareto``       x_m * U**(-1/alpha)            (p: alpha, xm)
      ``constant``     all equal to ``value``          (p: value)
      ``slowdown``     ``value`` for everybody, workers ``0..n/2-1`` multiplied
                       by ``factor`` once ``t >= t_switch``
    """
    g = rng(seed, STREAM_TIMES, t)
    if model == "shifted_exp":
        u = uniform01_open_left(g, n)
        return p.get("shift", 1.0) - np.log(u) / p.get("rate", 1.0)
    if model == "lognormal":
        z = g.standard_normal(n)
        return np.exp(p.get("mu", 0.0) + p.get("sigma", 0.5) * z)
    if model == "exp_slow":
        u = uniform01_open_left(g, n)
        x = -np.log(u) / p.get("rate", 1.0)
        nslow = int(np.floor(p.get("frac", 0.05) * n))
        slow = rng(seed, STREAM_PICK).permutation(n)[:nslow]
        x[slow] *= p.get("factor", 10.0)
        return x
    if model == "pareto":
        u = uniform01_open_left(g, n)
        return p.get("xm", 1.0) * u ** (-1.0 / p.get("alpha", 2.0))
    if model == "constant":
        return np.full(n, float(p.get("value", 1.0)))
    if model == "slowdown":
        x = np.full(n, float(p.get("value", 1.0)))
        if t >= int(p.get("t_switch", 0)):
            x[: n // 2] *= p.get("factor", 5.0)
        return x
    raise ValueError(f"unknown time model {model!r}")


def gradient_matrix(seed: int, n: int, d: int, ld: int, mean: float = 0.0,
                    std: float = 1.0) -> np.ndarray:
    """Synthetic per-worker gradient matrix ``[n, ld]`` fp32, entries ``mean + std*N(0,1)``.

    Columns ``d .. ld-1`` (row padding) are filled with NaN so that a consumer
    reading past ``d`` shows up in every statistic.
    """
    G = np.empty((n, ld), dtype=np.float32)
    for i in range(n):
        g = rng(seed, STREAM_GRADS, i)
        G[i, :d] = mean + std * g.standard_normal(d, dtype=np.float32)
    G[:, d:] = np.nan
    return G


def gradient_columns(seed: int, rows, c0: int, c1: int, threads: int = 1) -> np.ndarray:
    """Columns ``[c0, c1)`` of the given rows of a synthetic gradient matrix, entries
    N(0,1) drawn in fp32 and returned as fp64 ``[len(rows), c1 - c0]``.  Column chunk q
    (``GRAD_COL_CHUNK`` columns) of row i comes from its own generator
    ``(seed, STREAM_GRAD_COLS, i, q)``, so any column range of any row can be drawn on
    its own, in any order, with the same values.  ``threads`` > 1 draws rows in
    parallel (numpy releases the GIL while it fills an array)."""
    rows = [int(i) for i in rows]
    q0, q1 = c0 // GRAD_COL_CHUNK, (c1 + GRAD_COL_CHUNK - 1) // GRAD_COL_CHUNK
    out = np.empty((len(rows), c1 - c0), dtype=np.float64)

    def fill(r):
        i = rows[r]
        for q in range(q0, q1):
            a, b = max(c0, q * GRAD_COL_CHUNK), min(c1, (q + 1) * GRAD_COL_CHUNK)
            block = rng(seed, STREAM_GRAD_COLS, i, q).standard_normal(GRAD_COL_CHUNK, dtype=np.float32)
            out[r, a - c0:b - c0] = block[a - q * GRAD_COL_CHUNK:b - q * GRAD_COL_CHUNK]

    if threads > 1:
        from concurrent.futures import ThreadPoolExecutor
        with ThreadPoolExecutor(threads) as ex:
            list(ex.map(fill, range(len(rows))))
    else:
        for r in range(len(rows)):
            fill(r)
    return out


def round_up(x: int, m: int) -> int:
    return (int(x) + m - 1) // m * m
