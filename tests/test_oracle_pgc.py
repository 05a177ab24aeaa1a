"""Pins of the oracle's PGC loop: encode, decode, the stale-gradient
bookkeeping and the update.

What each pin checks, and the passage that fixes it:

* ``pin_dgd_lsq_closed_form`` — §VI-A: DGD is PGC with c = 1, s = 0.  For
  least squares plain gradient descent is a linear recurrence whose T-th
  iterate has a closed form, solved here with numpy.linalg.
* ``pin_dgd_logistic_scalar`` — the same special case for logistic loss,
  against a scalar pure-Python gradient-descent loop.
* ``pin_fr_frozen_is_gc`` — §IV-A: with beta frozen (eta = 0) every PGC-FR
  coded gradient equals the GC-FR coded gradient sum_l g_{jc+l}, and the
  decode recovers (1/n) sum_k g_k for EVERY straggler set.
* ``pin_cr_fullsum`` — eq. cr-fullsum (§V-B): sum_j ghat_j equals
  sum_i sum_j g_i^{s(t,i,j)} at every step, with s(t,i,j) taken from the
  schedule's closed form and each g recomputed at the recorded beta.
* ``pin_cr_unbiased`` — eq. cr-unbiased (§V-B): the mean of the decoded
  gradient over all C(n, s) masks equals (1/(nc)) sum_{i,j} g_i^{s(t,i,j)}.

* ``test_lsq_converges_to_the_normal_equations`` — least squares with equal
  partitions: DGD and PGC-FR (stale copies, §IV-A) converge to the full-data
  least-squares solution, solved directly with numpy.linalg.lstsq.

``test_planted_*`` plant a mistake in the oracle (monkeypatched, on the CPU)
and check that at least one pin catches it.
"""

import math

import numpy as np
import pytest

from oracle import pgc_oracle as O


def _parts(n, m, d, loss=O.LSQ, K=3, seed=0, rows=None):
    rng = np.random.default_rng(seed)
    rows = rows or [m] * n
    Xs = [rng.standard_normal((r, d)) for r in rows]
    if loss == O.LSQ:
        ys = [rng.standard_normal(r) for r in rows]
    elif loss == O.LOGISTIC:
        ys = [(rng.random(r) < 0.5).astype(float) for r in rows]
    else:
        ys = [rng.integers(0, K, r) for r in rows]
    return Xs, ys


def _random_masks(n, s, T, seed=1):
    rng = np.random.default_rng(seed)
    out = []
    for _ in range(T):
        m = np.zeros(n, dtype=np.uint8)
        m[rng.choice(n, s, replace=False)] = 1
        out.append(list(m))
    return out


# ----------------------------------------------------------------------------
# pins
# ----------------------------------------------------------------------------

def pin_dgd_lsq_closed_form(scheme, rows=None):
    n, d, eta, T = 3, 5, 0.05, 30
    Xs, ys = _parts(n, 7, d, O.LSQ, rows=rows)
    # g(beta) = (1/n) sum_k (1/m_k) X_k^T (X_k beta - y_k) = A beta - b
    A = sum(X.T @ X / X.shape[0] for X in Xs) / n
    b = sum(X.T @ y / X.shape[0] for X, y in zip(Xs, ys)) / n
    I = np.eye(d)
    recs = O.run(scheme, n, 0, O.LSQ, Xs, ys, eta, [[0] * n] * T, record_loss=False)
    for t in (1, 2, 10, T):
        # beta^t = (I - (I - eta A)^t) A^{-1} b, from beta^0 = 0
        ref = (I - np.linalg.matrix_power(I - eta * A, t)) @ np.linalg.solve(A, b)
        np.testing.assert_allclose(recs[t - 1]["beta"], ref, rtol=1e-10, atol=1e-12)


def pin_dgd_logistic_scalar(scheme):
    n, d, m, eta, T = 2, 2, 3, 0.5, 5
    Xs, ys = _parts(n, m, d, O.LOGISTIC, seed=4)
    beta = [0.0] * d
    traj = []
    for _ in range(T):
        g = [0.0] * d
        for X, y in zip(Xs, ys):
            for r in range(m):
                z = sum(X[r, j] * beta[j] for j in range(d))
                p = 1.0 / (1.0 + math.exp(-z))
                for j in range(d):
                    g[j] += (p - y[r]) * X[r, j] / m / n
        beta = [beta[j] - eta * g[j] for j in range(d)]
        traj.append(list(beta))
    recs = O.run(scheme, n, 0, O.LOGISTIC, Xs, ys, eta, [[0] * n] * T, record_loss=False)
    for t in range(T):
        np.testing.assert_allclose(recs[t]["beta"], traj[t], rtol=1e-12, atol=1e-14)


def pin_fr_frozen_is_gc(n, s, loss=O.LOGISTIC):
    c = s + 1
    Xs, ys = _parts(n, 6, 3, loss)
    rng = np.random.default_rng(9)
    beta0 = rng.standard_normal((3, 3) if loss == O.SOFTMAX else 3)
    o = O.PGCOracle(O.FR, n, s, loss, Xs, ys, 0.0, beta0=beta0, K=3)
    gk = [O.partition_gradient(loss, Xs[k], ys[k], beta0) for k in range(n)]
    full = sum(gk) / n
    masks = list(O.all_masks(n, s))
    for t in range(2 * c + 1):
        o.step(masks[t % len(masks)])
        for i in range(n):
            j = i // c
            gc_coded = sum(gk[j * c + l] for l in range(c))
            np.testing.assert_allclose(o.coded(i), gc_coded, rtol=1e-12, atol=1e-14)
        for mask in masks:
            np.testing.assert_allclose(o.decode(mask), full, rtol=1e-12, atol=1e-14)


def staleness_closed_form(t, c, l):
    """Step at which slot l of a worker was last evaluated by step t:
    the largest tau in [1, t] with (tau - 1) mod c = l, else 0 (warm-up)."""
    best = 0
    for tau in range(1, t + 1):
        if (tau - 1) % c == l:
            best = tau
    return best


def pin_cr_fullsum(n, s, loss=O.LOGISTIC, eta=0.3, T=None):
    c = s + 1
    T = T or 3 * c + 2
    Xs, ys = _parts(n, 4, 3, loss, seed=2)
    o = O.PGCOracle(O.CR, n, s, loss, Xs, ys, eta, K=3)
    betas = [o.beta.copy()]
    for t, mask in enumerate(_random_masks(n, s, T)):
        o.step(mask)
        betas.append(o.beta.copy())
        lhs = sum(o.coded(j) for j in range(n))
        rhs = 0.0
        for i in range(n):
            for l in range(c):
                holder = (i - l) % n          # the worker holding D_i in its slot l
                sig = staleness_closed_form(t, c, l)
                assert max(0, t - c + 1) <= sig <= t
                assert o.ring_step[holder][l] == sig
                g = O.partition_gradient(loss, Xs[i], ys[i], betas[sig])
                # the holder's slot l stores exactly this copy of D_i's gradient
                np.testing.assert_allclose(o.ring[holder][l], g, rtol=1e-12, atol=1e-14)
                rhs = rhs + g
        np.testing.assert_allclose(lhs, rhs, rtol=1e-11, atol=1e-13)
    return o, betas


def pin_cr_unbiased(n, s, loss=O.LSQ, eta=0.2, T=None):
    c = s + 1
    T = T or 2 * c + 1
    Xs, ys = _parts(n, 5, 3, loss, seed=6)
    o = O.PGCOracle(O.CR, n, s, loss, Xs, ys, eta, K=3)
    betas = [o.beta.copy()]
    masks = list(O.all_masks(n, s))
    for t, mask in enumerate(_random_masks(n, s, T, seed=7)):
        o.step(mask)
        betas.append(o.beta.copy())
        mean = sum(o.decode(mk) for mk in masks) / len(masks)
        gbar = 0.0
        for i in range(n):
            for l in range(c):
                sig = staleness_closed_form(t, c, l)
                gbar = gbar + O.partition_gradient(loss, Xs[i], ys[i], betas[sig])
        gbar = gbar / (n * c)
        np.testing.assert_allclose(mean, gbar, rtol=1e-11, atol=1e-13)


# ----------------------------------------------------------------------------
# tests
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("scheme", [O.FR, O.CR])
def test_dgd_lsq_closed_form(scheme):
    pin_dgd_lsq_closed_form(scheme)


@pytest.mark.parametrize("scheme", [O.FR, O.CR])
def test_dgd_lsq_closed_form_unequal_partitions(scheme):
    pin_dgd_lsq_closed_form(scheme, rows=[3, 9, 6])


@pytest.mark.parametrize("scheme", [O.FR, O.CR])
def test_dgd_logistic_scalar(scheme):
    pin_dgd_logistic_scalar(scheme)


@pytest.mark.parametrize("n,s", [(4, 1), (6, 1), (6, 2), (8, 3), (4, 3)])
def test_fr_frozen_is_gc(n, s):
    pin_fr_frozen_is_gc(n, s)


def test_fr_frozen_is_gc_softmax():
    pin_fr_frozen_is_gc(4, 1, O.SOFTMAX)


@pytest.mark.parametrize("n,s", [(4, 1), (5, 2), (6, 3), (7, 6), (3, 0)])
def test_cr_fullsum(n, s):
    pin_cr_fullsum(n, s)


def test_cr_fullsum_softmax():
    pin_cr_fullsum(5, 2, O.SOFTMAX, eta=0.5)


@pytest.mark.parametrize("n,s", [(4, 1), (5, 2), (6, 2), (6, 4)])
def test_cr_unbiased(n, s):
    pin_cr_unbiased(n, s)


def test_fr_decode_ignores_which_group_member_straggles():
    n, s = 6, 2
    Xs, ys = _parts(n, 5, 3, O.LOGISTIC)
    o = O.PGCOracle(O.FR, n, s, O.LOGISTIC, Xs, ys, 0.4)
    masks = list(O.all_masks(n, s))
    for t in range(7):
        o.step(masks[(5 * t) % len(masks)])
        ref = o.decode(masks[0])
        for mk in masks:
            np.testing.assert_allclose(o.decode(mk), ref, rtol=1e-13, atol=1e-15)


def test_step_records_indices():
    n, s = 6, 2
    Xs, ys = _parts(n, 3, 2, O.LSQ)
    o = O.PGCOracle(O.FR, n, s, O.LSQ, Xs, ys, 0.1)
    r0 = o.step([0, 1, 1, 0, 0, 0])
    assert r0["slot"] == -1 and r0["eval_partition"] == [-1] * n
    assert r0["fr_rep"] == [0, 3]
    r1 = o.step([1, 1, 0, 0, 0, 0])
    assert r1["slot"] == 0 and r1["eval_partition"] == [0, 0, 0, 3, 3, 3]
    assert r1["fr_rep"] == [2, 3]
    r2 = o.step([0, 0, 0, 1, 1, 0])
    assert r2["slot"] == 1 and r2["fr_rep"] == [0, 5]
    assert r2["received"] == 4


def test_stragglers_still_advance_their_store():
    """§V-B / §VI-A: a straggler still evaluates and stores its gradient."""
    n, s = 4, 1
    Xs, ys = _parts(n, 3, 2, O.LSQ)
    o = O.PGCOracle(O.CR, n, s, O.LSQ, Xs, ys, 0.1)
    o.step([1, 0, 0, 0])
    o.step([1, 0, 0, 0])
    assert o.ring_step[0] == [1, 0]
    o.step([1, 0, 0, 0])
    assert o.ring_step[0] == [1, 2]


# ----------------------------------------------------------------------------
# planted mistakes: each must make at least one pin fail
# ----------------------------------------------------------------------------

def test_planted_schedule_off_by_one(monkeypatch):
    monkeypatch.setattr(O, "evaluated_slot", lambda t, c: None if t == 0 else t % c)
    with pytest.raises(AssertionError):
        pin_cr_fullsum(5, 2)


def test_planted_cr_placement_reversed(monkeypatch):
    orig = O.holdings

    def bad(scheme, n, c):
        if scheme == O.CR:
            return [[(i - l) % n for l in range(c)] for i in range(n)]
        return orig(scheme, n, c)

    monkeypatch.setattr(O, "holdings", bad)
    with pytest.raises(AssertionError):
        pin_cr_fullsum(5, 2)


def test_planted_cr_scale(monkeypatch):
    orig = O.decode_coefficients

    def bad(scheme, n, s, mask):
        a = orig(scheme, n, s, mask)
        return a * (s + 1) if scheme == O.CR else a     # 1/(n - s) instead of 1/((n - s) c)

    monkeypatch.setattr(O, "decode_coefficients", bad)
    with pytest.raises(AssertionError):
        pin_cr_unbiased(5, 2)


def test_planted_missing_mean(monkeypatch):
    orig = O.partition_gradient

    def bad(loss, X, y, beta):
        return orig(loss, X, y, beta) * np.asarray(X).shape[0]    # a sum, not a mean

    monkeypatch.setattr(O, "partition_gradient", bad)
    with pytest.raises(AssertionError):
        pin_dgd_lsq_closed_form(O.CR)


def test_planted_fr_uses_stale_slot_twice(monkeypatch):
    orig = O.PGCOracle.coded

    def bad(self, i):
        return orig(self, i) + self.ring[i][0] - self.ring[i][self.c - 1]

    monkeypatch.setattr(O.PGCOracle, "coded", bad)
    with pytest.raises(AssertionError):
        pin_fr_frozen_is_gc(4, 1)


def test_planted_straggler_skips_evaluation(monkeypatch):
    """A store that does not advance for stragglers breaks eq. cr-fullsum."""
    def bad_step(self, mask):
        O.check_mask(mask, self.n, self.s)
        t = self.t
        if t == 0:
            self.evaluate()
        else:
            l = O.evaluated_slot(t, self.c)
            for i in range(self.n):
                if int(mask[i]) == 0:
                    self.ring[i][l] = self.partition_grad(self.hold[i][l])
                    self.ring_step[i][l] = t
        g = self.decode(mask)
        self.beta = self.beta - self.lr * g
        self.t = t + 1
        return {"grad": g}

    monkeypatch.setattr(O.PGCOracle, "step", bad_step)
    with pytest.raises(AssertionError):
        pin_cr_fullsum(5, 2)


# ---------------------------------------------------------------------------
# Long-run sanity against a direct solve: least squares with equal partition
# sizes has the full-data least-squares solution as its only stationary point
# (sum_k X_k^T (X_k beta - y_k) = 0).  DGD (c = 1) converges to it; so does
# PGC-FR, whose stale copies all equal the current gradient at a fixed point,
# where the decode is (1/n) sum_k g_k = 0 (§IV-A; the theorem's geometric
# convergence for a small enough eta).
# ---------------------------------------------------------------------------

def _normal_equations_solution(Xs, ys):
    X = np.concatenate(Xs)
    y = np.concatenate(ys)
    return np.linalg.lstsq(X, y, rcond=None)[0]


@pytest.mark.parametrize("scheme,s,lr,T", [(O.CR, 0, 0.2, 1500), (O.FR, 0, 0.2, 1500), (O.FR, 1, 0.1, 3000),
                                           (O.FR, 3, 0.05, 6000)])
def test_lsq_converges_to_the_normal_equations(scheme, s, lr, T):
    n, m, d = 4, 6, 5
    Xs, ys = _parts(n, m, d, loss=O.LSQ, seed=11)
    o = O.PGCOracle(scheme, n, s, O.LSQ, Xs, ys, lr)
    masks = [[1 if (i - t) % n < s else 0 for i in range(n)] for t in range(T)]
    for mask in masks:
        o.step(mask)
    ref = _normal_equations_solution(Xs, ys)
    np.testing.assert_allclose(o.beta, ref, rtol=0, atol=1e-9 * (1 + np.abs(ref).max()))
