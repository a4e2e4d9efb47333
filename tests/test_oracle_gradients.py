"""Pins of the oracle's per-worker gradients (Eq. (2)): the textbook closed form of
softmax regression, fp64 central finite differences of the forward loss on tiny
MLPs, and bf16 rounding against torch's conversion."""
import numpy as np
import pytest
import torch

from oracle import dbw_oracle as O
from paper_2004_14696_gb300 import inputs


def _problem(widths, n, B, seed=0, S=50):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((n * B, widths[0])).astype(np.float32)
    y = rng.integers(0, widths[-1], size=n * B).astype(np.int32)
    w = inputs.kaiming_uniform_params(seed, widths)
    w[:] += (0.05 * rng.standard_normal(w.shape[0])).astype(np.float32)   # nonzero biases too
    return w, X, y


def test_softmax_regression_closed_form():
    """One layer: g_i = (1/B) sum_x (p(x) - e_y) x^T for W and (1/B) sum_x (p - e_y) for b."""
    widths, n, B = (7, 4), 3, 5
    w, X, y = _problem(widths, n, B, 1)
    G, loss = O.worker_grads(widths, w, X, y, n, B)
    W = w[:28].reshape(4, 7).astype(np.float64)
    b = w[28:].astype(np.float64)
    for i in range(n):
        Xi = X[i * B:(i + 1) * B].astype(np.float64)
        logits = Xi @ W.T + b
        p = np.exp(logits - logits.max(1, keepdims=True))
        p /= p.sum(1, keepdims=True)
        Y = np.eye(4)[y[i * B:(i + 1) * B]]
        gW = (p - Y).T @ Xi / B
        gb = (p - Y).sum(0) / B
        np.testing.assert_allclose(G[i, :28], gW.ravel(), rtol=1e-12, atol=1e-14)
        np.testing.assert_allclose(G[i, 28:], gb, rtol=1e-12, atol=1e-14)
        ce = -np.log(p[np.arange(B), y[i * B:(i + 1) * B]]).mean()
        assert abs(loss[i] - ce) < 1e-12


@pytest.mark.parametrize("widths", [(5, 4, 3), (6, 5, 4, 3), (3, 8, 2)])
def test_mlp_gradient_matches_central_differences(widths):
    n, B = 2, 4
    w, X, y = _problem(widths, n, B, 2)
    G, loss = O.worker_grads(widths, w, X, y, n, B)
    w64 = w.astype(np.float64)
    h = 1e-6
    for i in range(n):
        Xi, yi = X[i * B:(i + 1) * B], y[i * B:(i + 1) * B]
        f = lambda v: O.sample_losses(widths, v, Xi, yi).mean()
        assert abs(f(w64) - loss[i]) < 1e-12
        fd = np.empty_like(w64)
        for p in range(w64.shape[0]):
            e = np.zeros_like(w64)
            e[p] = h
            fd[p] = (f(w64 + e) - f(w64 - e)) / (2 * h)
        np.testing.assert_allclose(G[i], fd, rtol=1e-5, atol=1e-8)


def test_param_layout_matches_parameter_count():
    for widths in [(784, 10), (784, 256, 10), (3072, 1024, 1024, 10), (4096, 4096, 4096, 4096, 1000)]:
        _, d = O.param_layout(widths)
        assert d == inputs.param_count(widths)
    assert inputs.param_count((784, 256, 10)) == 203530
    assert inputs.param_count((3072, 1024, 1024, 10)) == 4206602
    assert inputs.param_count((4096, 4096, 4096, 4096, 1000)) == 54440936


def test_bf16_round_matches_torch_conversion():
    rng = np.random.default_rng(3)
    x = np.concatenate([rng.standard_normal(10000).astype(np.float32),
                        (rng.standard_normal(1000) * 1e-30).astype(np.float32),
                        np.float32([0.0, -0.0, 1.0, 1.00390625, 1.01171875, 3.0e38, -1.5])])
    # ties to even: 1 + 2^-8 is halfway between bf16 1 and 1 + 2^-7
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(O.bf16_round(x), ref)
    assert O.bf16_round(np.float32([1.00390625]))[0] == 1.0
    assert O.bf16_round(np.float32([1.01171875]))[0] == 1.015625


def test_bf16_mode_rounds_every_gemm_operand():
    """bf16 mode stays within bf16 precision of the fp64 gradient, differs from the
    fp64 computation on merely pre-rounded X and W (so the hidden operands really
    are rounded), and on a one-layer model equals the closed form on rounded X, W, dZ."""
    widths, n, B = (16, 12, 5), 3, 8
    w, X, y = _problem(widths, n, B, 4)
    G16, l16 = O.worker_grads(widths, w, X, y, n, B, bf16=True)
    G64, l64 = O.worker_grads(widths, w, X, y, n, B)
    # no ReLU (softmax regression): bf16 rounding only perturbs, by about 2^-8 relative
    ws, Xs, ys = _problem((64, 10), n, B, 7)
    Gs16, _ = O.worker_grads((64, 10), ws, Xs, ys, n, B, bf16=True)
    Gs64, _ = O.worker_grads((64, 10), ws, Xs, ys, n, B)
    assert np.linalg.norm(Gs16 - Gs64) <= 0.02 * np.linalg.norm(Gs64)
    assert np.all(np.abs(l16 - l64) <= 0.02 * np.abs(l64))
    layers, _ = O.param_layout(widths)
    wr = w.astype(np.float64).copy()
    for (offW, fout, fin, offb) in layers:
        wr[offW:offW + fout * fin] = O.bf16_round(w[offW:offW + fout * fin])
    Gpre, _ = O.worker_grads(widths, wr, O.bf16_round(X), y, n, B)
    assert not np.array_equal(G16, Gpre)
    # one layer: g_W = dZ^T X with dZ = bf16((p - e_y) / B), X and W rounded
    widths1 = (16, 5)
    w1, X1, y1 = _problem(widths1, 1, B, 5)
    G1, _ = O.worker_grads(widths1, w1, X1, y1, 1, B, bf16=True)
    Wr = O.bf16_round(w1[:80]).reshape(5, 16)
    Xr = O.bf16_round(X1)
    z = Xr @ Wr.T + w1[80:].astype(np.float64)
    p = np.exp(z - z.max(1, keepdims=True))
    p /= p.sum(1, keepdims=True)
    dZ = O.bf16_round(((p - np.eye(5)[y1]) / B).astype(np.float32))
    np.testing.assert_allclose(G1[0, :80], (dZ.T @ Xr).ravel(), rtol=1e-13, atol=1e-16)
    np.testing.assert_allclose(G1[0, 80:], dZ.sum(0), rtol=1e-13, atol=1e-16)


def test_relu_flip_changes_only_the_flipped_unit_and_below():
    widths, n, B = (6, 5, 4), 1, 3
    w, X, y = _problem(widths, n, B, 6)
    G, _, zs, scales = O.worker_grads(widths, w, X, y, n, B, return_preact=True)
    assert zs[0].shape == (3, 5) and np.all(scales[0] >= np.abs(zs[0]))
    flip = np.zeros((3, 5), dtype=bool)
    flip[1, 2] = True
    Gf, _ = O.worker_grads(widths, w, X, y, n, B, relu_flip=[flip])
    layers, _ = O.param_layout(widths)
    offW, fout, fin, offb = layers[0]
    changed = np.flatnonzero(G[0] != Gf[0])
    rows = set((c - offW) // fin for c in changed if c < offb)
    assert rows <= {2}                                   # only unit 2's weight row (and its bias)
    assert all(c < layers[1][0] for c in changed)        # the output layer is untouched


def test_single_worker_grad_equals_row_of_batch():
    widths, n, B = (5, 6, 3), 4, 3
    w, X, y = _problem(widths, n, B, 5)
    G, loss = O.worker_grads(widths, w, X, y, n, B)
    for i in range(n):
        g, l = O.single_worker_grad(widths, w, X[i * B:(i + 1) * B], y[i * B:(i + 1) * B], B)
        np.testing.assert_allclose(g, G[i], rtol=1e-13, atol=1e-16)
        assert abs(l - loss[i]) < 1e-13


def test_planted_dropped_term_is_caught(monkeypatch):
    """Losing the first layer's bias gradient must fail the finite-difference pin."""
    real = O.worker_grads

    def dropped_term(widths, w, X, y, n, B, bf16=False):
        G, loss = real(widths, w, X, y, n, B, bf16)
        layers, _ = O.param_layout(widths)
        offW, fout, fin, offb = layers[0]
        G[:, offb:offb + fout] = 0.0
        return G, loss

    monkeypatch.setattr(O, "worker_grads", dropped_term)
    with pytest.raises(AssertionError):
        test_mlp_gradient_matches_central_differences((5, 4, 3))


def test_gradient_magnitude_bounds_and_single_term_case():
    """The magnitude of an entry (sum of |products|) bounds |entry|, and equals it
    when the entry is a single product (one sample, one layer)."""
    widths = (6, 5, 4)
    w, X, y = _problem(widths, 2, 3, 8)
    G, _, Gm = O.worker_grads(widths, w, X, y, 2, 3, return_magnitude=True)
    assert np.all(Gm >= np.abs(G) - 1e-15)
    w1, X1, y1 = _problem((6, 4), 1, 1, 9)
    G1, _, Gm1 = O.worker_grads((6, 4), w1, X1, y1, 1, 1, return_magnitude=True)
    np.testing.assert_allclose(Gm1, np.abs(G1), rtol=1e-15, atol=0)
