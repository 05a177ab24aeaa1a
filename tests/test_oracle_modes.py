"""Pins of the oracle's baselines (§VI-A) to facts that do not come from the
oracle itself: IS-SGD's average over all straggler sets is the full
gradient (each partition is received in C(n-1, s) of the C(n, s) sets, with
weight 1/(n-s)); with s = 0 both baselines are DGD (§III); GC-FR recovers the
full gradient exactly for every straggler set (§IV-A with current
gradients); and planted mistakes fail those pins."""

import numpy as np
import pytest

from oracle import pgc_oracle as O
from paper_2607_20739_gb300 import workloads as W


def _data(n, d=6, m=5, seed=0, K=1, loss=O.LOGISTIC):
    rng = np.random.default_rng(seed)
    Xs = [rng.standard_normal((m + k % 3, d)) for k in range(n)]
    if loss == O.SOFTMAX:
        ys = [rng.integers(0, K, size=len(X)).astype(np.int32) for X in Xs]
    else:
        ys = [(rng.random(len(X)) < 0.5).astype(np.float32) for X in Xs]
    return Xs, ys


def _full_gradient(loss, Xs, ys, beta):
    return sum(O.partition_gradient(loss, X, y, beta) for X, y in zip(Xs, ys)) / len(Xs)


@pytest.mark.parametrize("n,s", [(4, 1), (6, 2), (5, 3)])
def test_is_sgd_is_unbiased_over_all_masks(n, s):
    Xs, ys = _data(n)
    beta = np.linspace(-0.3, 0.4, 6)
    acc = np.zeros(6)
    cnt = 0
    for mask in O.all_masks(n, s):
        o = O.ISSGDOracle(n, s, O.LOGISTIC, Xs, ys, lr=0.0, beta0=beta)
        acc += o.step(mask)["grad"]
        cnt += 1
    assert cnt == O.binom(n, s)
    np.testing.assert_allclose(acc / cnt, _full_gradient(O.LOGISTIC, Xs, ys, beta), rtol=1e-12, atol=1e-14)


def test_is_sgd_coefficients():
    o = O.ISSGDOracle(5, 2, O.LSQ, *_data(5, loss=O.LSQ), lr=0.1)
    rec = o.step([0, 1, 0, 1, 0])
    np.testing.assert_array_equal(rec["coeff"], [1 / 3, 0, 1 / 3, 0, 1 / 3])


@pytest.mark.parametrize("n,s", [(4, 1), (6, 2), (6, 1)])
def test_gc_fr_recovers_the_full_gradient_for_every_mask(n, s):
    Xs, ys = _data(n, K=3, loss=O.SOFTMAX)
    beta = np.random.default_rng(3).standard_normal((3, 6)) * 0.1
    for mask in O.all_masks(n, s):
        o = O.GCFROracle(n, s, O.SOFTMAX, Xs, ys, lr=0.0, beta0=beta, K=3)
        np.testing.assert_allclose(o.step(mask)["grad"], _full_gradient(O.SOFTMAX, Xs, ys, beta),
                                   rtol=1e-12, atol=1e-14)


def test_gc_fr_trajectory_is_dgd_and_costs_c_evaluations_per_worker():
    n, s, T = 6, 2, 5
    Xs, ys = _data(n)
    w = W.WORKLOADS["cr_n8_logistic_d1024"].replace(n=n, s=s)
    masks = W.make_masks(w, T, 9)
    gc = O.run_mode("gc", O.FR, n, s, O.LOGISTIC, Xs, ys, 0.2, masks)
    dgd = O.run(O.CR, n, 0, O.LOGISTIC, Xs, ys, 0.2, [[0] * n] * T)
    for a, b in zip(gc, dgd):
        np.testing.assert_allclose(a["beta"], b["beta"], rtol=1e-12, atol=1e-14)
    o = O.GCFROracle(n, s, O.LOGISTIC, Xs, ys, 0.2)
    o.step(masks[0])
    assert o.inner.grad_evals == n * (s + 1)


def test_is_sgd_with_no_stragglers_is_dgd():
    n, T = 5, 4
    Xs, ys = _data(n, loss=O.LSQ)
    a = O.run_mode("is_sgd", O.CR, n, 0, O.LSQ, Xs, ys, 0.05, [[0] * n] * T)
    b = O.run(O.CR, n, 0, O.LSQ, Xs, ys, 0.05, [[0] * n] * T)
    for x, y in zip(a, b):
        np.testing.assert_allclose(x["beta"], y["beta"], rtol=1e-12, atol=1e-14)


def test_planted_mistake_fails_the_unbiasedness_pin(monkeypatch):
    # weight 1/n instead of 1/(n - s): the average over masks is then biased
    n, s = 5, 2
    Xs, ys = _data(n)
    beta = np.linspace(-0.2, 0.2, 6)
    orig = O.ISSGDOracle.step

    def wrong(self, mask):
        rec = orig(self, mask)
        rec["grad"] = rec["grad"] * (self.n - self.s) / self.n
        return rec

    monkeypatch.setattr(O.ISSGDOracle, "step", wrong)
    acc = sum(O.ISSGDOracle(n, s, O.LOGISTIC, Xs, ys, 0.0, beta0=beta).step(m)["grad"] for m in O.all_masks(n, s))
    assert not np.allclose(acc / O.binom(n, s), _full_gradient(O.LOGISTIC, Xs, ys, beta), rtol=1e-6)
