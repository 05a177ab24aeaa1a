"""pgc_gradient_noalloc: the allocation-free gradient entry point.

Some callers cannot call cudaMalloc / cudaFree when they need a gradient (a
framework whose caching pool already holds the free device memory, or a loop
that must not take cudaFree's implicit device synchronisation).  This entry
point computes one partition's gradient with a fixed scratch array inside the
library instead.  Here it is called through the C ABI twice in a row and each
result is checked against the gradient the existing pgc_step path stored for
the same partition at the same parameters (its warm-up step evaluates every
partition at beta^(0)), within the fp32 tolerance of the parity tests.

This file is named to be collected last.
"""

import ctypes as C

import numpy as np
import pytest

from paper_2607_20739_gb300 import workloads as W

from parity import rel_err

pytestmark = pytest.mark.gpu

TOL = 1e-4


def _noalloc(lib, loss, dtype, X, y, w, g, stream=0):
    return lib.lib.pgc_gradient_noalloc(loss, dtype, X.shape[0], X.shape[1], C.c_void_p(X.data_ptr()),
                                        C.c_void_p(y.data_ptr()), C.c_void_p(w.data_ptr()),
                                        C.c_void_p(g.data_ptr()), C.c_void_p(stream))


@pytest.mark.parametrize("loss,d,m", [("logistic", 1024, 3001), ("lsq", 16384, 700)])
def test_noalloc_matches_pgc_step(libpgc, cuda, loss, d, m):
    torch = cuda
    w = W.WORKLOADS["cr_n8_logistic_d1024"].replace(n=4, s=1, loss=loss, d=d, m=m)
    Xs, ys = W.make_partitions(w, 3)
    w0 = (np.random.default_rng(0).standard_normal(d) / np.sqrt(d)).astype(np.float32)

    # existing entry point: the warm-up step stores g_k(beta^0) in slot 0 of worker k (CR)
    g = libpgc.PGC("CR", w.n, w.s, loss, "f32", d, rows=w.rows(), lr=w.lr, w0=w0)
    g.load(Xs, ys)
    g.step([0, 0, 1, 0], info=False)
    ref = {k: g.store(k, 0) for k in range(w.n)}
    g.close()

    code = libpgc.LOGISTIC if loss == "logistic" else libpgc.LSQ
    wd = torch.from_numpy(w0).cuda()
    for k in (1, 3):                       # two calls in a row share the scratch
        Xd = torch.from_numpy(Xs[k]).cuda()
        yd = torch.from_numpy(ys[k]).cuda()
        out = torch.full((d,), float("nan"), device="cuda")
        rc = _noalloc(libpgc, code, libpgc.F32, Xd, yd, wd, out)
        assert rc == libpgc.OK, libpgc.lib.pgc_strerror(rc)
        got = out.cpu().numpy()
        assert np.isfinite(got).all()
        assert rel_err(got, ref[k]) <= TOL, (k, rel_err(got, ref[k]))


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
