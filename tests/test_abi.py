"""The C ABI without a GPU: the library loads, exports every entry point the
header declares, its host-only index helpers agree bit for bit with the
oracle's placement and schedule (§III, §IV-A, §V-B), and bad arguments are
rejected before any CUDA call."""

import ctypes as C
import os
import re

import numpy as np
import pytest

from oracle import pgc_oracle as O


def _declared(root):
    src = open(os.path.join(root, "include", "pgc.h")).read()
    return sorted(set(re.findall(r"^\s*(?:int|int64_t|const char \*)\s*(pgc_\w+)\s*\(", src, re.M)))


def test_every_declared_symbol_is_exported(libpgc, root_dir):
    names = _declared(root_dir)
    assert len(names) >= 14
    for name in names:
        assert hasattr(libpgc.lib, name), name
    assert set(names) == set(libpgc.EXPORTED)


def test_strerror_covers_codes(libpgc):
    for code in range(0, -10, -1):
        assert libpgc.lib.pgc_strerror(code)
    assert b"GC-CR" in libpgc.lib.pgc_strerror(libpgc.ESINGULAR)
    assert b"unknown" in libpgc.lib.pgc_strerror(-99)


@pytest.mark.parametrize("scheme", [O.FR, O.CR])
@pytest.mark.parametrize("n,s", [(1, 0), (4, 1), (6, 2), (8, 3), (12, 5), (5, 4), (9, 2), (128, 7), (64, 3)])
def test_placement_matches_oracle(libpgc, scheme, n, s):
    if scheme == O.FR and n % (s + 1):
        assert libpgc.lib.pgc_placement(scheme, n, s, (C.c_int32 * (n * (s + 1)))()) == libpgc.EINVAL
        return
    got = libpgc.placement(scheme, n, s)
    assert got.tolist() == O.holdings(scheme, n, s + 1)


@pytest.mark.parametrize("scheme", [O.FR, O.CR])
@pytest.mark.parametrize("n,s", [(4, 1), (6, 2), (8, 3), (12, 5), (9, 8), (128, 7)])
def test_schedule_matches_oracle(libpgc, scheme, n, s):
    c = s + 1
    if scheme == O.FR and n % c:
        pytest.skip("FR needs c | n")
    for t in list(range(0, 3 * c + 2)) + [1000, 10 ** 12 + 7]:
        ev, slot = libpgc.schedule(scheme, n, s, t)
        ref_slot = O.evaluated_slot(t, c)
        assert slot == (-1 if ref_slot is None else ref_slot)
        ref = [O.evaluated_partition(scheme, n, c, i, t) for i in range(n)]
        assert ev.tolist() == [-1 if r is None else r for r in ref]


def _create(lib, n=4, s=1, scheme=0, loss=0, dtype=0, d=8, K=1, rows=None, lr=0.1, null_rows=False):
    h = C.c_void_p()
    r = (C.c_int64 * n)(*(rows if rows is not None else [3] * n)) if n > 0 else (C.c_int64 * 1)(3)
    rc = lib.lib.pgc_create(C.byref(h), n, s, scheme, loss, dtype, d, K, None if null_rows else r, C.c_float(lr),
                            None, None)
    assert not h.value
    return rc


@pytest.mark.parametrize("kw", [
    dict(n=0), dict(s=-1), dict(n=3, s=3), dict(n=6, s=3, scheme=0), dict(scheme=2), dict(loss=3),
    dict(dtype=2), dict(d=0), dict(K=2), dict(loss=2, K=1), dict(loss=2, K=5000), dict(rows=[3, 0, 3, 3]),
    dict(null_rows=True), dict(n=1025, s=0, rows=[1] * 1025), dict(lr=float("nan")),
])
def test_create_rejects_bad_arguments(libpgc, kw):
    assert _create(libpgc, **kw) == libpgc.EINVAL


def test_null_context_calls(libpgc):
    L = libpgc.lib
    assert L.pgc_destroy(None) == libpgc.OK
    assert L.pgc_step(None, None, None, None, 0, None) == libpgc.EINVAL
    assert L.pgc_loss(None, None) == libpgc.EINVAL
    assert L.pgc_sync(None) == libpgc.EINVAL
    assert L.pgc_step_count(None) == -1
    assert L.pgc_schedule(0, 4, 1, -1, None, None) == libpgc.EINVAL


def _create_mode(lib, mode, n=4, s=1, scheme=1, loss=0, dtype=0, d=8, K=1):
    h = C.c_void_p()
    r = (C.c_int64 * n)(*([3] * n))
    rc = lib.lib.pgc_create_mode(C.byref(h), mode, n, s, scheme, loss, dtype, d, K, r, C.c_float(0.1), None, None)
    assert not h.value
    return rc


@pytest.mark.parametrize("mode,scheme,n,s,code", [
    (7, 1, 4, 1, "EINVAL"),          # unknown mode
    (1, 0, 4, 1, "EINVAL"),          # IS-SGD needs CR
    (3, 0, 4, 1, "EINVAL"),          # naive PGC-CR needs CR
    (3, 1, 65, 2, "ENOTSUP"),        # the GC-CR modes stop at n = 64
    (2, 1, 65, 2, "ENOTSUP"),        # GC on CR placement uses the same decode weights
])
def test_create_mode_rejects_before_any_cuda_call(libpgc, mode, scheme, n, s, code):
    assert _create_mode(libpgc, mode, n=n, s=s, scheme=scheme) == getattr(libpgc, code)


def test_gc_cr_calls_on_a_null_context(libpgc):
    L = libpgc.lib
    assert L.pgc_set_gc_encoding(None, None) == libpgc.EINVAL
    assert L.pgc_get_gc_encoding(None, None) == libpgc.EINVAL
    assert L.pgc_get_gc_decode(None, None, None) == libpgc.EINVAL
