"""Checkpoint and resume (pgc_checkpoint_save / _load): a run stopped after
T0 steps and resumed in a fresh context from its checkpoint follows the fp64
oracle's uninterrupted run on the same masks (schedule and decode support
bit-exact, decoded gradient and parameters within the parity tolerances,
loss F(beta^(t)) within 1e-3 at every resumed step), and it reproduces the
GPU's own uninterrupted run (bit-exact where the step is deterministic; the
tensor-core path sums the slot total with reduce-adds in completion order,
so there to fp32 rounding).  A checkpoint of another configuration is
refused."""

import numpy as np
import pytest

from paper_2607_20739_gb300 import workloads as W

from parity import GRAD_TOL, compare_step, generate, make_gpu, rel_err, run_oracle

pytestmark = pytest.mark.gpu

WL = W.WORKLOADS

CASES = {
    "cr_logistic": ("pgc", WL["cr_n8_logistic_d1024"].replace(m=300, d=200), 7, 3, True),
    "fr_softmax_smallk": ("pgc", WL["fr_n32_softmax_k10"].replace(n=8, m=150), 6, 2, True),
    "cr_softmax_tensor_core": ("pgc", WL["cr_n128_softmax_k1000"].replace(n=5, s=2, K=300, d=320, m=130), 6, 4, False),
    # P = K d >= 2^20: the one-thread-per-column decode
    "cr_softmax_wide_decode": ("pgc", WL["cr_n128_softmax_k1000"].replace(n=5, s=2, K=256, d=4096, m=64), 7, 3, False),
    "is_sgd_lsq": ("is_sgd", WL["cr_n64_lsq_d16384"].replace(n=6, s=2, d=700, m=40), 5, 2, True),
}


def _steps(g, w, masks, ts):
    shape = (w.K, w.d) if w.loss == "softmax" else (w.d,)
    out = []
    for t in ts:
        lv = g.loss()
        grad = np.zeros(w.K * w.d, np.float32)
        beta = np.zeros(w.K * w.d, np.float32)
        rec = dict(g.step(masks[t], grad, beta))
        rec.update(grad=grad.reshape(shape), beta=beta.reshape(shape), coeff=g.decode_coefficients(), loss=lv)
        out.append(rec)
    return out


@pytest.mark.parametrize("name", list(CASES))
def test_resume_follows_the_oracle(libpgc, cuda, headroom, name):
    mode, w, T, T0, exact = CASES[name]
    Xs, ys, masks = generate(w, T)
    a = make_gpu(libpgc, w, Xs, ys, mode=mode)
    ref = _steps(a, w, masks, range(T))
    a.close()
    b = make_gpu(libpgc, w, Xs, ys, mode=mode)
    _steps(b, w, masks, range(T0))
    ck = b.checkpoint()
    b.close()
    c = make_gpu(libpgc, w, Xs, ys, mode=mode)
    c.restore(ck)
    assert c.t == T0
    got = _steps(c, w, masks, range(T0, T))
    c.close()
    # against the fp64 oracle's uninterrupted run
    orecs = run_oracle(w, Xs, ys, masks, mode=mode)
    worst = 0.0
    for t, (r, o) in enumerate(zip(got, orecs[T0:]), start=T0):
        e, _ = compare_step(w, t, r, o)
        worst = max(worst, e)
        assert rel_err(r["beta"], o["beta"]) <= GRAD_TOL[w.dtype], t
    headroom.append(f"resume {name} (steps {T0}..{T - 1}): decoded gradient {worst:.2e} / {GRAD_TOL[w.dtype]:g}")
    # against the GPU's own uninterrupted run
    for r1, r2 in zip(got, ref[T0:]):
        if exact:
            np.testing.assert_array_equal(r1["grad"], r2["grad"])
            np.testing.assert_array_equal(r1["beta"], r2["beta"])
        else:
            # the slot total's reduce-adds land in completion order; a few
            # free-running steps carry that rounding through the bf16 copy of beta
            assert rel_err(r1["grad"], r2["grad"]) < 1e-5 and rel_err(r1["beta"], r2["beta"]) < 1e-5


def test_checkpoint_of_another_configuration_is_refused(libpgc, cuda):
    w = WL["cr_n8_logistic_d1024"].replace(m=50, d=64)
    Xs, ys, masks = generate(w, 2)
    a = make_gpu(libpgc, w, Xs, ys)
    a.step(masks[0])
    ck = a.checkpoint()
    a.close()
    for other in (w.replace(s=1), w.replace(d=65)):
        Xo, yo, _ = generate(other, 1)
        g = make_gpu(libpgc, other, Xo, yo)
        with pytest.raises(libpgc.PGCError) as ei:
            g.restore(ck)
        assert ei.value.code == libpgc.EINVAL
        g.close()
    g = make_gpu(libpgc, w, Xs, ys)
    with pytest.raises(libpgc.PGCError):
        g.restore(ck[:-4])
    g.close()
