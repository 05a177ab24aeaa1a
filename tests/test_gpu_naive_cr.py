"""GPU parity of the GC-CR modes (§V-A) through the C ABI: the naive
pipelined construction on cyclic repetition (PGC_MODE_NAIVE_CR) and GC-CR
itself (PGC_MODE_GC with PGC_CR), against the oracle's literal versions.

The device builds the encoding from the draws, solves for the decode weights
d(J) every step (fp64), reports the range of alpha_{m,k} = d_m c_{j_m,l} and
decodes (1/n) sum_j d_j sum_l c_{j,l} store[j][l] in fp32.  Because alpha
reaches the thousands, the oracle is teacher-forced: before each step it is
given the GPU's beta^(t), so both evaluate at the same parameters and the
comparison measures one step's arithmetic.  Bounds: encoding and decode
weights 1e-9 relative (fp64 on both sides, different elimination orders);
the alpha range 1e-9 relative; the decoded gradient within GRAD_TOL times
the decode's own scale (1/n) sum |alpha| max|store|, since each store
carries its fp32 (or bf16-input) error into the weighted sum."""

import numpy as np
import pytest

from oracle import pgc_oracle as O
from paper_2607_20739_gb300 import workloads as W

from parity import GRAD_TOL, LOSS, LOSS_TOL, generate, oracle_inputs

pytestmark = pytest.mark.gpu

WL = W.WORKLOADS


def _draws(w, seed):
    return np.random.default_rng(seed).standard_normal((w.s, w.n - 1))


def run_and_compare(libpgc, w, T, mode="naive_cr", seed=1, draws_seed=11):
    Xs, ys, masks = generate(w, T, seed)
    draws = _draws(w, draws_seed)
    g = libpgc.PGC(w.scheme, w.n, w.s, w.loss, w.dtype, w.d, K=w.K, rows=w.rows(), lr=w.lr, mode=mode)
    g.load(Xs, ys)
    g.set_gc_encoding(draws)
    o = O.NaiveCROracle(w.n, w.s, LOSS[w.loss], oracle_inputs(w, Xs), ys, w.lr, draws=draws, K=w.K,
                        pipelined=mode == "naive_cr")
    np.testing.assert_allclose(g.gc_encoding(), o.C, rtol=1e-9, atol=1e-12)
    P = w.K * w.d
    beta = np.zeros(P, dtype=np.float32)
    tol = GRAD_TOL[w.dtype]
    worst = 0.0
    amax_seen = 0.0
    for t, mask in enumerate(masks):
        o.beta = beta.astype(np.float64).reshape(o.beta.shape)          # teacher forcing
        lv_o = o.loss_value()
        lv_g = g.loss()
        assert abs(lv_g - lv_o) <= LOSS_TOL * abs(lv_o), (t, lv_g, lv_o)
        grad = np.zeros(P, dtype=np.float32)
        info = g.step(mask, grad, beta)
        d, (amax, amin) = g.gc_decode()
        rec = o.step(mask)
        assert info["t"] == rec["t"] == t
        assert info["slot"] == rec["slot"], (t, info["slot"], rec["slot"])
        assert list(info["eval_partition"]) == list(rec["eval_partition"]), t
        dscale = np.abs(rec["d"]).max()
        np.testing.assert_allclose(d, rec["d"], rtol=0, atol=1e-9 * dscale)
        assert ((d != 0) == (rec["d"] != 0)).all(), t
        ascale = max(abs(rec["alpha_max"]), abs(rec["alpha_min"]))
        assert abs(amax - rec["alpha_max"]) <= 1e-9 * ascale, (t, amax, rec["alpha_max"])
        assert abs(amin - rec["alpha_min"]) <= 1e-9 * ascale, (t, amin, rec["alpha_min"])
        np.testing.assert_allclose(g.decode_coefficients(), rec["coeff"], rtol=1e-6, atol=1e-7 * dscale / w.n)
        # the decode's scale: (1/n) sum over received (j, l) of |alpha| * max|store[j][l]|
        scale = sum(abs(a) * np.abs(o.ring[j][(k - j) % w.n]).max() for (j, k), a in rec["alpha"].items()) / w.n
        err = np.abs(grad.reshape(rec["grad"].shape) - rec["grad"]).max()
        worst = max(worst, err / scale)
        assert err <= tol * scale, f"step {t}: |ghat error| {err:.3g} > {tol} x {scale:.3g}"
        amax_seen = max(amax_seen, ascale)
    g.close()
    return worst, amax_seen


CASES = {
    "naive_cr_logistic_n6_s2": ("naive_cr", WL["cr_n8_logistic_d1024"].replace(n=6, s=2, m=300, d=200, lr=0.05), 7),
    "naive_cr_lsq_n12_c6_ragged": ("naive_cr", WL["cr_n64_lsq_d16384"].replace(n=12, s=5, m=64, d=257, lr=0.01), 8),
    "naive_cr_bf16_logistic": ("naive_cr", WL["cr_n8_logistic_d1024"].replace(n=5, s=1, m=90, d=1000, dtype="bf16",
                                                                               lr=0.05), 5),
    "naive_cr_softmax_few_class": ("naive_cr", WL["fr_n32_softmax_k10"].replace(scheme="CR", n=6, s=2, m=150, d=512), 5),
    "naive_cr_softmax_tc": ("naive_cr", WL["cr_n128_softmax_k1000"].replace(n=5, s=2, K=300, d=320, m=130), 4),
    "gc_cr_logistic_n6_s2": ("gc", WL["cr_n8_logistic_d1024"].replace(n=6, s=2, m=200, d=300, lr=0.05), 4),
    "gc_cr_softmax_cuda_cores": ("gc", WL["cr_n128_softmax_k1000"].replace(n=4, s=1, K=20, d=100, m=60,
                                                                           dtype="f32"), 3),
}


@pytest.mark.parametrize("name", list(CASES))
def test_gc_cr_mode_parity(libpgc, cuda, name):
    mode, w, T = CASES[name]
    run_and_compare(libpgc, w, T, mode=mode)


def test_paper_example_n4_c2_through_the_abi(libpgc, cuda):
    # §V-A's n = 4, c = 2 example: with draws giving c_{0,1} = 2 and W_3
    # straggling, D_1 is decoded with coefficients 2 (W_0) and -1 (W_1)
    w = WL["cr_n8_logistic_d1024"].replace(n=4, s=1, m=40, d=64)
    Xs, ys, _ = generate(w, 1)
    g = libpgc.PGC(w.scheme, w.n, w.s, w.loss, w.dtype, w.d, rows=w.rows(), lr=w.lr, mode="naive_cr")
    g.load(Xs, ys)
    g.set_gc_encoding(np.array([[2.0, -1.0, 1.0]]))
    np.testing.assert_allclose(g.gc_encoding(), [[1, 2], [1, 1], [1, 0.5], [1, 1]], rtol=0, atol=1e-15)
    g.step(np.array([0, 0, 0, 1], dtype=np.uint8))
    d, (amax, amin) = g.gc_decode()
    np.testing.assert_allclose(d, [1.0, -1.0, 2.0, 0.0], rtol=0, atol=1e-14)
    assert amax == pytest.approx(2.0, abs=1e-14) and amin == pytest.approx(-1.0, abs=1e-14)
    g.close()


def test_rows_kernel_without_fused_tail_matches_oracle(libpgc, cuda, monkeypatch):
    # the few-class kernel followed by the standalone commit and decode (the
    # GC-CR modes always run it this way)
    from parity import compare_runs, run_gpu, run_oracle
    monkeypatch.setenv("PGC_NO_ROWS_TAIL", "1")
    w = WL["fr_n32_softmax_k10"].replace(n=8, s=1, m=150, d=700)
    Xs, ys, masks = generate(w, 5)
    g, grecs = run_gpu(libpgc, w, Xs, ys, masks)
    assert g.gradient_path == "softmax_rows"
    compare_runs(w, grecs, run_oracle(w, Xs, ys, masks))
    g.close()


def test_gc_cr_errors(libpgc, cuda):
    w = WL["cr_n8_logistic_d1024"].replace(n=4, s=1, m=20, d=32)
    Xs, ys, _ = generate(w, 1)
    mk = lambda **kw: libpgc.PGC(kw.get("scheme", "CR"), kw.get("n", w.n), w.s, w.loss, w.dtype, w.d,
                                 rows=[w.m] * kw.get("n", w.n), lr=w.lr, mode=kw.get("mode", "naive_cr"))
    with pytest.raises(libpgc.PGCError) as ei:
        mk(scheme="FR")
    assert ei.value.code == libpgc.EINVAL
    with pytest.raises(libpgc.PGCError) as ei:
        mk(n=65)
    assert ei.value.code == libpgc.ENOTSUP
    p = mk(mode="pgc")
    with pytest.raises(libpgc.PGCError) as ei:
        p.set_gc_encoding(np.ones((1, 3)))
    assert ei.value.code == libpgc.EINVAL
    p.close()
    g = mk()
    g.load(Xs, ys)
    mask = np.array([0, 1, 0, 0], dtype=np.uint8)
    with pytest.raises(libpgc.PGCError) as ei:
        g.step(mask)                               # no encoding yet
    assert ei.value.code == libpgc.ESTATE
    with pytest.raises(libpgc.PGCError) as ei:
        g.set_gc_encoding(np.array([[1.0, 0.0, 1.0]]))   # H = (1, 0, 1, -2): W_0's system is 0 x = -1
    assert ei.value.code == libpgc.ESINGULAR
    with pytest.raises(libpgc.PGCError) as ei:
        g.set_gc_encoding(np.array([[1.0, np.nan, 1.0]]))
    assert ei.value.code == libpgc.EINVAL
    g.set_gc_encoding(np.array([[0.5, -1.5, 2.0]]))      # the context stayed usable
    grad = np.zeros(w.d, dtype=np.float32)
    g.step(mask, grad, None)
    assert np.isfinite(grad).all()
    g.close()


EDGE = {
    # the largest n the GC-CR modes take (one-warp fp64 solves over 64 rows)
    "naive_cr_n64_max": ("naive_cr", WL["cr_n8_logistic_d1024"].replace(n=64, s=3, m=9, d=40, lr=0.05), 5),
    # s = 0: B is the identity, every decode weight 1, the step is DGD
    "naive_cr_s0": ("naive_cr", WL["cr_n8_logistic_d1024"].replace(n=5, s=0, m=30, d=48, lr=0.05), 3),
    # c = n: every worker holds every partition, one coded gradient decodes
    "naive_cr_c_equals_n": ("naive_cr", WL["cr_n8_logistic_d1024"].replace(n=4, s=3, m=25, d=36, lr=0.05), 6),
    "gc_cr_c_equals_n": ("gc", WL["cr_n8_logistic_d1024"].replace(n=3, s=2, m=25, d=36, lr=0.05), 3),
    # one row per partition and d = 1
    "naive_cr_one_row_d1": ("naive_cr", WL["cr_n64_lsq_d16384"].replace(n=6, s=2, m=1, d=1, lr=0.05), 4),
}


@pytest.mark.parametrize("name", list(EDGE))
def test_gc_cr_edge_cases(libpgc, cuda, name):
    mode, w, T = EDGE[name]
    run_and_compare(libpgc, w, T, mode=mode)
