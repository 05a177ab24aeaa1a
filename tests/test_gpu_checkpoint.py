"""Checkpoint and resume (pgc_checkpoint_save / _load): a run stopped after
T0 steps and resumed in a fresh context from its checkpoint produces the same
decoded gradients and parameters as the uninterrupted run (bit-exact where
the step is deterministic; the tensor-core path sums the slot total with
reduce-adds in completion order, so there to fp32 rounding), and a
checkpoint of another configuration is refused."""

import numpy as np
import pytest

from paper_2607_20739_gb300 import workloads as W

from parity import generate, make_gpu, rel_err

pytestmark = pytest.mark.gpu

WL = W.WORKLOADS

CASES = {
    "cr_logistic": ("pgc", WL["cr_n8_logistic_d1024"].replace(m=300, d=200), 7, 3, True),
    "fr_softmax_smallk": ("pgc", WL["fr_n32_softmax_k10"].replace(n=8, m=150), 6, 2, True),
    "cr_softmax_tensor_core": ("pgc", WL["cr_n128_softmax_k1000"].replace(n=5, s=2, K=300, d=320, m=130), 6, 4, False),
    "is_sgd_lsq": ("is_sgd", WL["cr_n64_lsq_d16384"].replace(n=6, s=2, d=700, m=40), 5, 2, True),
}


def _steps(g, masks, ts, P):
    out = []
    for t in ts:
        grad = np.zeros(P, np.float32)
        beta = np.zeros(P, np.float32)
        g.step(masks[t], grad, beta)
        out.append((grad, beta))
    return out


@pytest.mark.parametrize("name", list(CASES))
def test_resume_reproduces_the_run(libpgc, cuda, name):
    mode, w, T, T0, exact = CASES[name]
    Xs, ys, masks = generate(w, T)
    P = w.K * w.d
    a = make_gpu(libpgc, w, Xs, ys, mode=mode)
    ref = _steps(a, masks, range(T), P)
    a.close()
    b = make_gpu(libpgc, w, Xs, ys, mode=mode)
    _steps(b, masks, range(T0), P)
    ck = b.checkpoint()
    b.close()
    c = make_gpu(libpgc, w, Xs, ys, mode=mode)
    c.restore(ck)
    assert c.t == T0
    got = _steps(c, masks, range(T0, T), P)
    for (g1, b1), (g2, b2) in zip(got, ref[T0:]):
        if exact:
            np.testing.assert_array_equal(g1, g2)
            np.testing.assert_array_equal(b1, b2)
        else:
            assert rel_err(g1, g2) < 1e-5 and rel_err(b1, b2) < 1e-6
    c.close()


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
