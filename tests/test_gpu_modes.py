"""GPU parity of the paper's baselines (§VI-A) run on the same kernels
(`pgc_create_mode`): IS-SGD (CR, one slot per worker, mean of the n - s
received gradients) and GC with FR placement (every slot refreshed every
step), against the oracle's literal per-worker versions; and the argument
checks of the mode/scheme pairs."""

import pytest

from paper_2607_20739_gb300 import workloads as W

from parity import compare_runs, generate, run_gpu, run_oracle

pytestmark = pytest.mark.gpu

WL = W.WORKLOADS

CASES = {
    "is_sgd_cr_logistic": ("is_sgd", WL["cr_n8_logistic_d1024"].replace(m=300, d=200), 6),
    "is_sgd_cr_lsq_long_rows": ("is_sgd", WL["cr_n64_lsq_d16384"].replace(n=6, s=2, d=5000, m=40), 5),
    "is_sgd_cr_softmax_tc": ("is_sgd", WL["cr_n128_softmax_k1000"].replace(n=5, s=2, K=300, d=320, m=130), 4),
    "gc_fr_logistic": ("gc", WL["fr_n4_logistic_d64"].replace(n=6, s=2, m=50), 5),
    "gc_fr_softmax_smallk": ("gc", WL["fr_n32_softmax_k10"].replace(n=8, s=1, m=150), 4),
    "gc_fr_bf16_lsq": ("gc", WL["cr_n64_lsq_d16384"].replace(scheme="FR", n=4, s=1, dtype="bf16", d=3000, m=33), 4),
}


@pytest.mark.parametrize("name", list(CASES))
def test_mode_parity_with_oracle(libpgc, cuda, name):
    mode, w, T = CASES[name]
    Xs, ys, masks = generate(w, T)
    g, grecs = run_gpu(libpgc, w, Xs, ys, masks, mode=mode)
    orecs = run_oracle(w, Xs, ys, masks, mode=mode)
    compare_runs(w, grecs, orecs)
    g.close()


def test_mode_scheme_pairs_are_checked(libpgc, cuda):
    w = WL["fr_n4_logistic_d64"]
    for mode, scheme in (("is_sgd", "FR"), ("naive_cr", "FR"), (7, "CR")):
        with pytest.raises(libpgc.PGCError) as ei:
            libpgc.PGC(scheme, w.n, w.s, w.loss, w.dtype, w.d, rows=w.rows(), lr=w.lr, mode=mode)
        assert ei.value.code == libpgc.EINVAL
