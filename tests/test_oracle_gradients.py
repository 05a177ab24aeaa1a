"""Pins of the oracle's loss and per-partition gradient (§III ERM objective).

Independent references: closed forms (values at beta = 0, the least-squares
normal-equation form), central finite differences of the loss, a
scalar pure-Python loop over samples, and the K = 2 softmax / logistic
equivalence.
"""

import math

import numpy as np
import pytest

from oracle import pgc_oracle as O


def _data(loss, m=7, d=4, K=3, seed=0):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((m, d))
    if loss == O.LOGISTIC:
        y = (rng.random(m) < 0.5).astype(float)
        beta = rng.standard_normal(d)
    elif loss == O.LSQ:
        y = rng.standard_normal(m)
        beta = rng.standard_normal(d)
    else:
        y = rng.integers(0, K, m)
        beta = rng.standard_normal((K, d))
    return X, y, beta


def test_loss_at_zero_closed_forms():
    X, y, _ = _data(O.LOGISTIC)
    assert np.mean(O.sample_losses(O.LOGISTIC, X, y, np.zeros(4))) == pytest.approx(math.log(2), abs=1e-15)
    X, y, _ = _data(O.LSQ)
    assert np.mean(O.sample_losses(O.LSQ, X, y, np.zeros(4))) == pytest.approx(0.5 * np.mean(y ** 2), rel=1e-15)
    X, y, _ = _data(O.SOFTMAX, K=5)
    assert np.mean(O.sample_losses(O.SOFTMAX, X, y, np.zeros((5, 4)))) == pytest.approx(math.log(5), abs=1e-14)


@pytest.mark.parametrize("loss", [O.LOGISTIC, O.LSQ, O.SOFTMAX])
def test_gradient_matches_finite_differences(loss):
    X, y, beta = _data(loss)
    g = O.partition_gradient(loss, X, y, beta)
    assert g.shape == beta.shape
    h = 1e-6
    fd = np.zeros_like(beta)
    flat = beta.reshape(-1)
    for idx in range(flat.size):
        bp = flat.copy(); bp[idx] += h
        bm = flat.copy(); bm[idx] -= h
        fp = np.mean(O.sample_losses(loss, X, y, bp.reshape(beta.shape)))
        fm = np.mean(O.sample_losses(loss, X, y, bm.reshape(beta.shape)))
        fd.reshape(-1)[idx] = (fp - fm) / (2 * h)
    np.testing.assert_allclose(g, fd, rtol=1e-6, atol=1e-8)


def test_lsq_gradient_normal_equation_form():
    X, y, beta = _data(O.LSQ, m=11, d=5)
    g = O.partition_gradient(O.LSQ, X, y, beta)
    ref = (X.T @ X @ beta - X.T @ y) / X.shape[0]
    np.testing.assert_allclose(g, ref, rtol=1e-12, atol=1e-13)


def test_logistic_scalar_loop():
    X, y, beta = _data(O.LOGISTIC, m=5, d=3)
    g_ref = [0.0] * 3
    l_ref = 0.0
    for r in range(5):
        z = sum(X[r, j] * beta[j] for j in range(3))
        p = 1.0 / (1.0 + math.exp(-z))
        l_ref += math.log(1.0 + math.exp(z)) - y[r] * z
        for j in range(3):
            g_ref[j] += (p - y[r]) * X[r, j] / 5
    np.testing.assert_allclose(O.partition_gradient(O.LOGISTIC, X, y, beta), g_ref, rtol=1e-13)
    assert np.mean(O.sample_losses(O.LOGISTIC, X, y, beta)) == pytest.approx(l_ref / 5, rel=1e-13)


def test_softmax_scalar_loop():
    K, d, m = 4, 3, 6
    X, y, W = _data(O.SOFTMAX, m=m, d=d, K=K, seed=3)
    G_ref = [[0.0] * d for _ in range(K)]
    l_ref = 0.0
    for r in range(m):
        z = [sum(W[k, j] * X[r, j] for j in range(d)) for k in range(K)]
        e = [math.exp(v) for v in z]
        tot = sum(e)
        l_ref += math.log(tot) - z[int(y[r])]
        for k in range(K):
            rk = e[k] / tot - (1.0 if k == int(y[r]) else 0.0)
            for j in range(d):
                G_ref[k][j] += rk * X[r, j] / m
    np.testing.assert_allclose(O.partition_gradient(O.SOFTMAX, X, y, W), G_ref, rtol=1e-12, atol=1e-15)
    assert np.mean(O.sample_losses(O.SOFTMAX, X, y, W)) == pytest.approx(l_ref / m, rel=1e-13)


def test_softmax_rows_sum_to_zero():
    X, y, W = _data(O.SOFTMAX, m=9, d=5, K=6)
    G = O.partition_gradient(O.SOFTMAX, X, y, W)
    np.testing.assert_allclose(G.sum(axis=0), 0.0, atol=1e-14)


def test_softmax_two_classes_is_logistic():
    X, y, beta = _data(O.LOGISTIC, m=8, d=4)
    W = np.stack([np.zeros(4), beta])
    yc = y.astype(np.int64)
    np.testing.assert_allclose(O.sample_losses(O.SOFTMAX, X, yc, W),
                               O.sample_losses(O.LOGISTIC, X, y, beta), rtol=1e-13)
    G = O.partition_gradient(O.SOFTMAX, X, yc, W)
    g = O.partition_gradient(O.LOGISTIC, X, y, beta)
    np.testing.assert_allclose(G[1], g, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(G[0], -g, rtol=1e-12, atol=1e-15)


def test_full_loss_is_sample_mean_over_all_partitions():
    rng = np.random.default_rng(5)
    Xs = [rng.standard_normal((m, 3)) for m in (2, 5, 4)]
    ys = [rng.standard_normal(X.shape[0]) for X in Xs]
    beta = rng.standard_normal(3)
    Xall = np.concatenate(Xs)
    yall = np.concatenate(ys)
    ref = 0.5 * np.mean((Xall @ beta - yall) ** 2)
    assert O.full_loss(O.LSQ, Xs, ys, beta) == pytest.approx(ref, rel=1e-14)
