"""Pins of the GC-CR encoding and of the naive PGC-CR construction (§V-A) to
facts that do not come from the oracle itself: the published n = 3, s = 1
gradient-coding example; the paper's n = 4, c = 2 naive example (partition
D_1 decoded as -g_1^(t-1) + 2 g_1^(t)); exact recovery (sum_m alpha_{m,k} = 1
for every partition and every straggler set, and GC-CR with current
gradients equal to DGD); the null-space property the construction rests on;
s = 0 reducing to DGD; and the size of the coefficients at n = 12, c = 6
against PGC-CR's bound (1/mu)|N_k| < 2 (§V-B).  Planted mistakes fail them."""

import os

import numpy as np
import pytest

from oracle import pgc_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _read(name):
    out = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                k, v = line.rsplit(":", 1)
                out[k.strip()] = [float(x) for x in v.split()]
    return out


def _data(n, d=5, m=4, seed=0):
    rng = np.random.default_rng(seed)
    Xs = [rng.standard_normal((m + k % 2, d)) for k in range(n)]
    ys = [(rng.random(len(X)) < 0.5).astype(np.float32) for X in Xs]
    return Xs, ys


def test_encoding_reproduces_published_n3_example():
    g = _read("gc_cr_n3_s1.txt")
    Bpub = np.array([g[f"B {j}"] for j in range(3)])
    # the construction normalises B[j][j] = 1; the draws are those that make
    # its null-space matrix H = (-2, 1, 1), the one the published B satisfies
    assert np.allclose(np.array([-2.0, 1.0, 1.0]) @ Bpub.T, 0.0)
    B = O.gc_cr_encoding(3, 1, [-2.0, 1.0])
    scale = np.diag(Bpub)          # B[j] = Bpub[j] / scale[j], so the weights are d_pub = d / scale
    np.testing.assert_allclose(B, Bpub / scale[:, None], rtol=0, atol=1e-15)
    for i in range(3):
        mask = [0, 0, 0]
        mask[i] = 1
        d = O.gc_decode_weights(B, mask)
        np.testing.assert_allclose(d / scale, g[f"straggler {i}"], rtol=0, atol=1e-14)


def test_naive_example_n4_c2_coefficients_and_staleness():
    g = _read("naive_cr_n4_c2.txt")
    n, s = 4, 1
    mask = [0] * n
    mask[int(g["straggler"][0])] = 1
    B = O.gc_cr_encoding(n, s, g["draws"])
    d = O.gc_decode_weights(B, mask)
    alpha = O.decoding_alpha(B, d, mask, 2)
    assert alpha[(0, 1)] == pytest.approx(g["alpha D1 current (W0 slot 1)"][0], abs=1e-14)
    assert alpha[(1, 1)] == pytest.approx(g["alpha D1 stale (W1 slot 0)"][0], abs=1e-14)
    # run the naive construction: step 2 refreshes slot (2 - 1) mod 2 = 1, so
    # W_0's copy of D_1 is from step 2 and W_1's from step 1
    Xs, ys = _data(n)
    o = O.NaiveCROracle(n, s, O.LOGISTIC, Xs, ys, lr=0.5, draws=g["draws"], beta0=np.full(5, 0.1))
    betas = []
    for t in range(3):
        betas.append(o.beta.copy())
        rec = o.step(mask)
    assert rec["slot"] == 1
    # n * ghat = sum over received (j, l) of alpha * g_k at the step its copy was taken
    G = lambda k, t: O.partition_gradient(O.LOGISTIC, Xs[k], ys[k], betas[t])
    expect = np.zeros(5)
    for j in O.received_set(mask):
        for l in range(2):
            k = (j + l) % n
            expect += alpha[(j, k)] * G(k, 2 if l == 1 else 1)
    np.testing.assert_allclose(n * rec["grad"], expect, rtol=1e-12, atol=1e-14)
    # and D_1's part of it is exactly 2 g_1^(2) - g_1^(1)
    d1 = alpha[(0, 1)] * G(1, 2) + alpha[(1, 1)] * G(1, 1)
    np.testing.assert_allclose(d1, 2 * G(1, 2) - G(1, 1), rtol=1e-13, atol=1e-15)


@pytest.mark.parametrize("n,s,seed", [(7, 2, 1), (6, 3, 2), (5, 1, 3)])
def test_encoding_structure_and_exact_recovery_for_every_mask(n, s, seed):
    draws = np.random.default_rng(seed).standard_normal((s, n - 1))
    B = O.gc_cr_encoding(n, s, draws)
    c = s + 1
    H = np.concatenate([draws, -draws.sum(axis=1, keepdims=True)], axis=1)
    assert np.abs(H @ B.T).max() < 1e-9                      # rows in the null space of H
    for j in range(n):
        support = {(j + l) % n for l in range(c)}
        assert B[j, j] == 1.0
        assert all(B[j, k] == 0.0 for k in range(n) if k not in support)
    for mask in O.all_masks(n, s):
        d = O.gc_decode_weights(B, mask)
        assert all(d[i] == 0.0 for i in range(n) if mask[i])
        alpha = O.decoding_alpha(B, d, mask, c)
        per_k = np.zeros(n)
        for (j, k), a in alpha.items():
            per_k[k] += a
        np.testing.assert_allclose(per_k, 1.0, rtol=0, atol=1e-9)   # sum_m alpha_{m,k} = 1


@pytest.mark.parametrize("n,s", [(6, 2), (5, 4)])
def test_gc_cr_with_current_gradients_is_dgd(n, s):
    Xs, ys = _data(n, seed=4)
    draws = np.random.default_rng(5).standard_normal((s, n - 1))
    beta = np.linspace(-0.2, 0.3, 5)
    full = sum(O.partition_gradient(O.LOGISTIC, X, y, beta) for X, y in zip(Xs, ys)) / n
    for mask in list(O.all_masks(n, s))[:6]:
        o = O.NaiveCROracle(n, s, O.LOGISTIC, Xs, ys, lr=0.0, draws=draws, beta0=beta, pipelined=False)
        for _ in range(2):
            rec = o.step(mask)
            np.testing.assert_allclose(rec["grad"], full, rtol=1e-9, atol=1e-12)
    # the pipelined construction with lr = 0 keeps every copy at the same beta: exact too
    o = O.NaiveCROracle(n, s, O.LOGISTIC, Xs, ys, lr=0.0, draws=draws, beta0=beta)
    for t, mask in enumerate(list(O.all_masks(n, s))[:2 * (s + 1)]):
        np.testing.assert_allclose(o.step(mask)["grad"], full, rtol=1e-9, atol=1e-12)


def test_s0_is_dgd():
    n = 4
    Xs, ys = _data(n, seed=6)
    beta0 = np.linspace(0.1, -0.1, 5)
    ref = O.PGCOracle(O.CR, n, 0, O.LOGISTIC, Xs, ys, lr=0.3, beta0=beta0)
    o = O.NaiveCROracle(n, 0, O.LOGISTIC, Xs, ys, lr=0.3, beta0=beta0)
    for _ in range(3):
        a, b = ref.step([0] * n), o.step([0] * n)
        np.testing.assert_allclose(b["grad"], a["grad"], rtol=1e-13, atol=1e-15)
        assert b["alpha_max"] == b["alpha_min"] == 1.0


def test_coefficients_grow_large_at_n12_c6_while_pgc_cr_stays_below_two():
    n, s = 12, 5
    c = s + 1
    B = O.gc_cr_encoding(n, s, np.random.default_rng(7).standard_normal((s, n - 1)))
    amax = 0.0
    mu = (n - s) * c / n
    for mask in O.all_masks(n, s):
        d = O.gc_decode_weights(B, mask)
        amax = max(amax, max(abs(a) for a in O.decoding_alpha(B, d, mask, c).values()))
        assert O.appearance_counts(O.CR, n, s, mask).max() / mu < 2.0
    assert amax > 1000.0          # §V-A: they reach the thousands at n = 12, c = 6


def test_planted_mistakes_fail_the_pins():
    # a transposed encoding (coefficients read down columns) or a dropped
    # decode weight breaks exact recovery
    n, s = 6, 2
    B = O.gc_cr_encoding(n, s, np.random.default_rng(8).standard_normal((s, n - 1)))
    mask = [1, 0, 0, 1, 0, 0]
    d = O.gc_decode_weights(B, mask)
    assert np.abs(d @ B - 1.0).max() < 1e-9
    assert np.abs(d @ B.T - 1.0).max() > 1e-3
    d_bad = d.copy()
    d_bad[1] = 0.0
    assert np.abs(d_bad @ B - 1.0).max() > 1e-3
    with pytest.raises(ValueError):
        O.gc_decode_weights(np.eye(n), mask)      # the identity cannot tolerate stragglers
