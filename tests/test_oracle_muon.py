"""Pins of the Gefen-Muon oracle (oracle/muon.py) against what does not depend
on it: the Newton-Schulz iteration acts on each singular value separately, so
it must equal U f(S) V^T from an SVD with f the iterated quintic; the update
of a rank-one gradient has a closed form; and the codes are the nearest levels
by brute force."""
import numpy as np
import pytest

import oracle
from oracle import muon


def _f(sig, steps, coeffs):
    a, b, c = coeffs
    for _ in range(steps):
        sig = a * sig + b * sig ** 3 + c * sig ** 5
    return sig


@pytest.mark.parametrize("shape", [(5, 8), (8, 5), (16, 16), (3, 40)])
def test_newton_schulz_equals_the_singular_value_map(shape):
    rng = np.random.default_rng(sum(shape))
    Y = rng.normal(size=shape)
    U, S, Vt = np.linalg.svd(Y, full_matrices=False)
    ref = U @ np.diag(_f(S / np.linalg.norm(S), 5, muon.NS_COEFFICIENTS)) @ Vt
    np.testing.assert_allclose(muon.newton_schulz(Y), ref, rtol=1e-9, atol=1e-12)


def test_newton_schulz_pushes_singular_values_towards_one():
    rng = np.random.default_rng(7)
    Y = rng.normal(size=(32, 64))
    s = np.linalg.svd(muon.newton_schulz(Y, steps=5), compute_uv=False)
    assert s.min() > 0.6 and s.max() < 1.25  # the quintic's known band around 1


def _bf16(x):
    return (np.asarray(x, np.float32).view(np.uint32) >> 16).astype(np.uint16)


def test_rank_one_step_closed_form():
    # g = a b^T with bf16-exact entries, mu = 0: U = g, X = f(1) g / (|a| |b|)
    rows, cols = 4, 6
    a = np.array([1.0, -2.0, 0.5, 4.0])
    b = np.array([0.25, 1.0, -1.0, 2.0, 0.5, -0.125])
    g = np.outer(a, b)
    bits = _bf16(g.reshape(-1))
    theta = np.linspace(-1, 1, rows * cols).astype(np.float32)
    th0 = theta.astype(np.float64).copy()
    cb = np.linspace(-1, 1, 16).astype(np.float32)
    codes = np.full(rows * cols, 7, np.uint8)
    s = np.zeros(rows * cols // 6, np.float32)
    lr, wd = 0.02, 0.1
    muon.muon_step(theta, bits, codes, s, cb, cb, rows=rows, cols=cols, period=6, lr=lr, momentum=0.0,
                   weight_decay=wd, nesterov=True)
    f1 = _f(np.array(1.0), 5, muon.NS_COEFFICIENTS)
    X = f1 * g / (np.linalg.norm(a) * np.linalg.norm(b))
    want = th0 * (1 - lr * wd) - lr * X.reshape(-1)  # rows < cols: no lr adjustment
    np.testing.assert_allclose(theta, want.astype(np.float32), rtol=1e-6, atol=1e-7)
    # the buffer is g: its per-row absmax and nearest levels (brute force)
    np.testing.assert_allclose(s, np.abs(g).max(axis=1), rtol=0)
    for i, x in enumerate((g / np.abs(g).max(axis=1, keepdims=True)).reshape(-1)):
        assert codes[i] == oracle.nearest_level(float(x), cb)


def test_tall_matrix_learning_rate_adjustment():
    # rows > cols scales the step by sqrt(rows / cols)
    rng = np.random.default_rng(3)
    rows, cols = 12, 3
    g = rng.normal(size=(rows, cols)).astype(np.float32)
    bits = _bf16(g.reshape(-1))
    gb = (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64).reshape(rows, cols)
    cb = np.linspace(-1, 1, 16).astype(np.float32)
    theta = np.zeros(rows * cols, np.float32)
    codes = np.full(rows * cols, 7, np.uint8)
    s = np.zeros(rows, np.float32)
    muon.muon_step(theta, bits, codes, s, cb, cb, rows=rows, cols=cols, period=3, lr=0.01, momentum=0.0,
                   weight_decay=0.0)
    X = muon.newton_schulz(gb)
    np.testing.assert_allclose(theta, (-0.01 * 2.0 * X).reshape(-1).astype(np.float32), rtol=1e-6, atol=1e-9)


def test_momentum_and_nesterov_mix():
    # decoded buffer and gradient chosen so m and U are exact
    rows, cols = 2, 8
    cb = np.array([-1.0, -0.5, 0.0, 0.5, 1.0], np.float32)
    codes = np.array([4, 0, 3, 1, 2, 4, 0, 3] * 2, np.uint8)
    s = np.array([2.0, 4.0], np.float32)  # blocks are rows
    g = np.array([1.0, -1.0, 0.5, 0.25, 0.0, 2.0, -2.0, 1.0] * 2, np.float32)
    bits = _bf16(g)
    theta = np.zeros(16, np.float32)
    mu = 0.5
    X = muon.muon_step(theta, bits, codes.copy(), s.copy(), cb, cb, rows=rows, cols=cols, period=8, lr=1e-3,
                       momentum=mu, weight_decay=0.0, nesterov=True)
    buf = cb[codes].astype(np.float64) * np.repeat(s, 8)
    m = mu * buf + (1 - mu) * g
    U = g + mu * (m - g)
    ref = muon.newton_schulz(U.reshape(rows, cols))
    np.testing.assert_allclose(X, ref, rtol=1e-12)
    # without Nesterov the buffer itself is orthogonalised
    X2 = muon.muon_step(np.zeros(16, np.float32), bits, codes.copy(), s.copy(), cb, cb, rows=rows, cols=cols,
                        period=8, lr=1e-3, momentum=mu, weight_decay=0.0, nesterov=False)
    np.testing.assert_allclose(X2, muon.newton_schulz(m.reshape(rows, cols)), rtol=1e-12)


def test_nearest_codes_ties_go_to_the_lower_level():
    cb = np.array([-1.0, 0.0, 0.5, 1.0], np.float32)
    x = np.array([-0.5, 0.25, 0.75, -1.0, 1.0, 0.3])  # the first three sit on midpoints
    np.testing.assert_array_equal(muon.nearest_codes(x, cb), [0, 1, 2, 0, 3, 2])
    for xi in x:
        assert muon.nearest_codes(np.array([xi]), cb)[0] == oracle.nearest_level(float(xi), cb)
