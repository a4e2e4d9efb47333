"""Helpers shared by the GPU parity tests (no method arithmetic here)."""
import math

import numpy as np

RTOL_FP32 = 1e-5    # fp32 GEMM / fp32 accumulation paths
RTOL_BF16 = 2e-2    # bf16 GEMM operands with fp32 accumulation


def assert_close_rows(x, ref, rtol, what=""):
    """|x - r| <= rtol * (|r| + rms(r)) elementwise, rms over each row of r.

    The rms term keeps entries that cancel to ~0 in the reference (a mean of
    signed gradients, a weight gradient of a dead unit) from demanding a
    relative accuracy no fp32 computation can give.
    """
    x = np.asarray(x, dtype=np.float64)
    r = np.asarray(ref, dtype=np.float64)
    assert x.shape == r.shape, (what, x.shape, r.shape)
    r2 = r.reshape(-1, r.shape[-1]) if r.ndim > 1 else r.reshape(1, -1)
    x2 = x.reshape(r2.shape)
    rms = np.sqrt(np.mean(r2 * r2, axis=1, keepdims=True))
    err = np.abs(x2 - r2)
    lim = rtol * (np.abs(r2) + rms)
    bad = ~(err <= lim)
    if bad.any():
        i = np.argwhere(bad)[0]
        raise AssertionError(f"{what}: {bad.sum()} of {bad.size} entries off; first at {tuple(i)}: "
                             f"got {x2[tuple(i)]!r} want {r2[tuple(i)]!r} (limit {lim[tuple(i)]:.3g})")


def assert_close_scalar(x, ref, rtol, what=""):
    assert math.isclose(float(x), float(ref), rel_tol=rtol, abs_tol=0.0), f"{what}: got {x!r} want {ref!r}"
