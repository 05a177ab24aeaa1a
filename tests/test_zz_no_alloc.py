"""pgc_gradient_noalloc: the allocation-free gradient entry point.

Some callers cannot call cudaMalloc / cudaFree when they need a gradient (a
framework whose caching pool already holds the free device memory, or a loop
that must not take cudaFree's implicit device synchronisation).  This entry
point computes one partition's gradient with a fixed scratch array inside the
library instead.  Here it is called through the C ABI twice in a row and each
result is checked against the fp64 oracle's partition gradient at the same
parameters, and against the gradient the existing pgc_step path stored for
the same partition (its warm-up step evaluates every partition at beta^(0)),
within 1e-4: the streaming kernel computes in fp32 on the exact feature
values, bf16 features included.

This file is named to be collected last.
"""

import ctypes as C

import numpy as np
import pytest

from oracle import pgc_oracle as O
from paper_2607_20739_gb300 import workloads as W

from parity import LOSS, rel_err

pytestmark = pytest.mark.gpu

TOL = 1e-4


def _noalloc(lib, loss, dtype, X, y, w, g, stream=0):
    return lib.lib.pgc_gradient_noalloc(loss, dtype, X.shape[0], X.shape[1], C.c_void_p(X.data_ptr()),
                                        C.c_void_p(y.data_ptr()), C.c_void_p(w.data_ptr()),
                                        C.c_void_p(g.data_ptr()), C.c_void_p(stream))


@pytest.mark.parametrize("loss,dtype,d,m", [("logistic", "f32", 1024, 3001), ("lsq", "f32", 16384, 700),
                                             ("logistic", "bf16", 2048, 1999)])
def test_noalloc_matches_oracle_and_pgc_step(libpgc, cuda, headroom, loss, dtype, d, m):
    torch = cuda
    w = W.WORKLOADS["cr_n8_logistic_d1024"].replace(n=4, s=1, loss=loss, dtype=dtype, d=d, m=m)
    Xs, ys = W.make_partitions(w, 3)
    w0 = (np.random.default_rng(0).standard_normal(d) / np.sqrt(d)).astype(np.float32)

    # existing entry point: the warm-up step stores g_k(beta^0) in slot 0 of worker k (CR)
    g = libpgc.PGC("CR", w.n, w.s, loss, dtype, d, rows=w.rows(), lr=w.lr, w0=w0)
    g.load(Xs, ys)
    g.step([0, 0, 1, 0], info=False)
    ref = {k: g.store(k, 0) for k in range(w.n)}
    g.close()

    code = libpgc.LOGISTIC if loss == "logistic" else libpgc.LSQ
    dcode = libpgc.F32 if dtype == "f32" else libpgc.BF16
    wd = torch.from_numpy(w0).cuda()
    worst = 0.0
    for k in (1, 3):                       # two calls in a row share the scratch
        Xh = Xs[k] if dtype == "f32" else Xs[k].view(np.int16)      # bf16 bits, passed through unchanged
        Xd = torch.from_numpy(Xh).cuda()
        yd = torch.from_numpy(ys[k]).cuda()
        out = torch.full((d,), float("nan"), device="cuda")
        rc = _noalloc(libpgc, code, dcode, Xd, yd, wd, out)
        assert rc == libpgc.OK, libpgc.lib.pgc_strerror(rc)
        got = out.cpu().numpy()
        assert np.isfinite(got).all()
        ora = O.partition_gradient(LOSS[loss], W.features_as_float(Xs[k], dtype), ys[k], w0.astype(np.float64))
        e = rel_err(got, ora)
        worst = max(worst, e)
        assert e <= TOL, (k, e)
        assert rel_err(got, ref[k]) <= TOL, (k, rel_err(got, ref[k]))
    headroom.append(f"pgc_gradient_noalloc {loss} {dtype} d={d} m={m}: against the oracle {worst:.2e} / {TOL:g}")


def test_noalloc_rejects_what_it_cannot_hold(libpgc, cuda):
    torch = cuda
    lib = libpgc
    x = torch.zeros(16, 100, device="cuda")
    y = torch.zeros(16, device="cuda")
    w = torch.zeros(100, device="cuda")
    g = torch.zeros(100, device="cuda")
    # a row length that would need padding
    assert _noalloc(lib, lib.LOGISTIC, lib.F32, x, y, w, g) == lib.ENOTSUP
    # more rows than the fixed scratch can hold partial sums for (checked
    # before any work is launched, so the tiny buffers are never read)
    big = lib.lib.pgc_gradient_noalloc(lib.LSQ, lib.F32, 3_000_000, 16384, C.c_void_p(x.data_ptr()),
                                       C.c_void_p(y.data_ptr()), C.c_void_p(w.data_ptr()),
                                       C.c_void_p(g.data_ptr()), None)
    assert big == lib.ESCRATCH
    assert b"scratch" in lib.lib.pgc_strerror(lib.ESCRATCH)
