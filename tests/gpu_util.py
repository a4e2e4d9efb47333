"""Helpers shared by the GPU parity tests (no method arithmetic here)."""
import math

import numpy as np

RTOL_FP32 = 1e-5    # fp32 GEMM / fp32 accumulation paths
RTOL_BF16 = 2e-2    # bf16 GEMM operands with fp32 accumulation


def param_blocks(widths):
    """[start, end) of every parameter tensor (W_l, then b_l) in a row of G / in w."""
    blocks, off = [], 0
    for l in range(len(widths) - 1):
        fin, fout = int(widths[l]), int(widths[l + 1])
        blocks.append((off, off + fout * fin))
        blocks.append((off + fout * fin, off + fout * fin + fout))
        off += fout * fin + fout
    return blocks


def assert_close_rows(x, ref, rtol, what="", blocks=None):
    """|x - r| <= rtol * (|r| + rms(r))  elementwise.

    rms is taken over each row of r, or, when ``blocks`` ([start, end) column
    ranges, e.g. one per parameter tensor) is given, over each block of each row.
    The rms term keeps entries that cancel to ~0 in the reference (a mean of
    signed gradients, a weight gradient summed over samples of both signs) from
    demanding a relative accuracy no fp32 computation can give; taking it per
    parameter tensor keeps one tensor's scale from setting another's.
    """
    x = np.asarray(x, dtype=np.float64)
    r = np.asarray(ref, dtype=np.float64)
    assert x.shape == r.shape, (what, x.shape, r.shape)
    r2 = r.reshape(-1, r.shape[-1]) if r.ndim > 1 else r.reshape(1, -1)
    x2 = x.reshape(r2.shape)
    if blocks is None:
        blocks = [(0, r2.shape[1])]
    scale = np.empty_like(r2)
    for (a, b) in blocks:
        seg = r2[:, a:b]
        scale[:, a:b] = np.sqrt(np.mean(seg * seg, axis=1, keepdims=True))
    err = np.abs(x2 - r2)
    lim = rtol * (np.abs(r2) + scale)
    bad = ~(err <= lim)
    if bad.any():
        i = np.argwhere(bad)[0]
        worst = float(np.nanmax(err / np.where(lim > 0, lim, np.inf)))
        raise AssertionError(f"{what}: {bad.sum()} of {bad.size} entries off (worst {worst:.3g}x the limit); "
                             f"first at {tuple(i)}: got {x2[tuple(i)]!r} want {r2[tuple(i)]!r} "
                             f"(limit {lim[tuple(i)]:.3g})")


def assert_close_scalar(x, ref, rtol, what=""):
    assert math.isclose(float(x), float(ref), rel_tol=rtol, abs_tol=0.0), f"{what}: got {x!r} want {ref!r}"


def _rows_close(x, r, rtol, blocks):
    try:
        assert_close_rows(x, r, rtol, "", blocks)
        return None
    except AssertionError as e:
        return str(e)


def assert_worker_grads_match(G_gpu, loss_gpu, widths, w, X, y, B, bf16, workers, rtol,
                              amb=None, max_candidates=6, max_flips=3):
    """Each sampled worker's GPU gradient row matches the oracle's Eq. (2) row.

    A ReLU derivative whose pre-activation lies within rounding of 0 is a
    decision either value of which is correct at the kernel's precision (R13).
    When a row does not match, the oracle's own hidden pre-activations are ranked
    by |Z| / scale (scale = sum of |terms| of that dot product), the few most
    ambiguous ones (|Z| / scale <= amb) are flipped in every combination of up to
    ``max_flips`` of them, and the row must match one of those oracle results.
    Nothing of the GPU's enters the oracle; the GPU row is only compared.
    Returns {worker: (oracle row it matched, oracle loss)}: the valid reference a
    later check (the aggregation of these rows) must use.
    """
    import itertools

    from oracle import dbw_oracle as O

    if amb is None:
        amb = 2e-3 if bf16 else 1e-4
    blocks = param_blocks(widths)
    matched = {}
    for i in workers:
        Xi, yi = X[i * B:(i + 1) * B], y[i * B:(i + 1) * B]
        g, l, zs, scales = O.worker_grads(widths, w, Xi, yi, 1, B, bf16, return_preact=True)
        assert_close_scalar(loss_gpu[i], l[0], rtol, f"loss of worker {i}")
        msg = _rows_close(G_gpu[i], g[0], rtol, blocks)
        if msg is None:
            matched[i] = (g[0], float(l[0]))
            continue
        cand = []
        for h, (Z, S) in enumerate(zip(zs, scales)):
            rel = np.abs(Z) / np.where(S > 0, S, 1.0)
            for (r, u) in zip(*np.nonzero(rel <= amb)):
                cand.append((float(rel[r, u]), h, int(r), int(u)))
        cand = sorted(cand)[:max_candidates]
        ok = False
        for m in range(1, min(max_flips, len(cand)) + 1):
            for sub in itertools.combinations(cand, m):
                flips = [np.zeros(Z.shape, dtype=bool) for Z in zs]
                for (_, h, r, u) in sub:
                    flips[h][r, u] = True
                g2, _ = O.worker_grads(widths, w, Xi, yi, 1, B, bf16, relu_flip=flips)
                if _rows_close(G_gpu[i], g2[0], rtol, blocks) is None:
                    ok = True
                    matched[i] = (g2[0], float(l[0]))
                    break
            if ok:
                break
        assert ok, f"worker {i}: {msg} (no ReLU decision within rounding of 0 explains it; " \
                   f"{len(cand)} candidates)"
    return matched
