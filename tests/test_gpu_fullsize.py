"""Parity at the five measured workloads' full sizes, in the launch
configuration bench.py times (the library's stream, device outputs), on
outputs the fp64 oracle can compute one by one:

* every step: the schedule (evaluated partitions, slot, FR representatives)
  and the device-derived decode coefficients, bit-exact / exact;
* sampled workers: the gradient just written to their store slot against the
  oracle's partition gradient at the GPU's own beta of that step (the
  comparison point is the GPU state, so there is no drift to absorb);
* sampled columns of every store: the decoded gradient against the oracle's
  literal decode (sum over received workers of a_i times the c-slot coded
  gradient) of those same stored values, and the SGD update of beta.
"""

import numpy as np
import pytest

from oracle import pgc_oracle as O
from paper_2607_20739_gb300 import workloads as W

from parity import GRAD_TOL, LOSS, SCHEME, rel_err

pytestmark = pytest.mark.gpu

FULL = ["fr_n4_logistic_d64", "cr_n8_logistic_d1024", "fr_n32_softmax_k10", "cr_n64_lsq_d16384",
        "cr_n128_softmax_k1000"]

# decode of fp32 stores in fp32 (up to (n - s) c terms) against fp64
DECODE_TOL = 2e-5


def _col_blocks(P: int, rng, nblocks: int = 4, width: int = 64):
    if P <= nblocks * width:
        return [(0, P)]
    starts = np.sort(rng.choice(P - width, size=nblocks, replace=False))
    return [(int(s0), width) for s0 in starts]


@pytest.mark.parametrize("name", FULL)
def test_full_size_sampled(libpgc, cuda, name):
    torch = cuda
    w = W.WORKLOADS[name]
    T = w.c + 2                                   # every slot refreshed, then stale slots in the decode
    Xs, ys = W.make_partitions(w, 1)
    masks = W.make_masks(w, T, 1001)
    stream = torch.cuda.Stream()
    g = libpgc.PGC(w.scheme, w.n, w.s, w.loss, w.dtype, w.d, K=w.K, rows=w.rows(), lr=w.lr, stream=stream)
    g.load(Xs, ys)
    P = w.K * w.d
    gout = torch.empty(P, device="cuda")
    wout = torch.empty(P, device="cuda")
    scheme, loss = SCHEME[w.scheme], LOSS[w.loss]
    hold = O.holdings(scheme, w.n, w.c)
    rng = np.random.default_rng(7)
    blocks = _col_blocks(P, rng)
    shape = (w.K, w.d) if w.loss == "softmax" else (w.d,)
    for t in range(T):
        beta_t = np.asarray(g.weights()).reshape(-1)
        info = g.step(masks[t], gout, wout)
        g.sync()
        mask = masks[t]
        # schedule and coefficients
        o_t = O.evaluated_slot(t, w.c)
        assert info["slot"] == (-1 if o_t is None else o_t)
        exp_eval = [-1 if t == 0 else O.evaluated_partition(scheme, w.n, w.c, i, t) for i in range(w.n)]
        assert list(info["eval_partition"]) == exp_eval
        if w.scheme == "FR":
            assert list(info["fr_rep"]) == O.fr_representatives(mask, w.n, w.c)
        coeff = g.decode_coefficients()
        np.testing.assert_allclose(coeff, O.decode_coefficients(scheme, w.n, w.s, mask), rtol=2e-7, atol=0)
        # sampled workers: the gradient stored this step
        workers = rng.choice(w.n, size=2, replace=False)
        for i in workers:
            slot = int(rng.integers(w.c)) if t == 0 else o_t
            k = hold[i][slot]
            ref = O.partition_gradient(loss, W.features_as_float(Xs[k], w.dtype), ys[k], beta_t.reshape(shape))
            got = g.store(int(i), slot).reshape(shape)
            assert rel_err(got, ref) <= GRAD_TOL[w.dtype], (t, int(i), slot, k)
        # sampled columns: decode and SGD against the literal decode of the same stores
        ghat = gout.cpu().numpy().astype(np.float64)
        wnew = wout.cpu().numpy().astype(np.float64)
        for c0, nc in blocks:
            ref = np.zeros(nc)
            for i in range(w.n):
                if coeff[i] == 0.0:
                    continue
                coded = sum(g.store_cols(i, l, c0, nc).astype(np.float64) for l in range(w.c))
                ref += float(coeff[i]) * coded
            got = ghat[c0:c0 + nc]
            assert rel_err(got, ref) <= DECODE_TOL, (t, c0)
            exp_w = beta_t[c0:c0 + nc].astype(np.float64) - np.float64(np.float32(w.lr)) * got
            np.testing.assert_allclose(wnew[c0:c0 + nc], exp_w, rtol=1e-6, atol=1e-7)
    g.close()
