"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle on
the same seeded inputs, at sizes the oracle finishes in seconds that still
span several work items, stages and a ragged tail.  Every workload shape
(row length, dtype, loss, scheme) of the five measured workloads is
covered, plus edge cases: unequal partitions, n = 1, c = n, d = 1, ragged d,
s = 0 (plain distributed gradient descent)."""

import numpy as np
import pytest

from paper_2607_20739_gb300 import workloads as W

from parity import compare_runs, generate, rel_err, run_gpu, run_oracle

pytestmark = pytest.mark.gpu

WL = W.WORKLOADS

CASES = {
    # the five workloads, scaled so the oracle stays fast
    "fr_n4_logistic_d64": (WL["fr_n4_logistic_d64"], 20),
    "cr_n8_logistic_d1024_m1000": (WL["cr_n8_logistic_d1024"].replace(m=1000), 8),
    "fr_n8_softmax_k10_m333": (WL["fr_n32_softmax_k10"].replace(n=8, m=333), 6),
    "cr_n12_lsq_d16384_m45": (WL["cr_n64_lsq_d16384"].replace(n=12, m=45), 6),
    "cr_n10_softmax_k1000_m40": (WL["cr_n128_softmax_k1000"].replace(n=10, m=40), 3),
    # edge cases
    "fr_unequal_rows": (WL["fr_n4_logistic_d64"].replace(m=(1, 300, 17, 64)), 7),
    "cr_unequal_rows_lsq": (WL["cr_n64_lsq_d16384"].replace(n=5, s=2, d=3000, m=(7, 1, 40, 9, 33)), 6),
    "cr_n1_s0": (WL["cr_n8_logistic_d1024"].replace(n=1, s=0, m=77, d=33), 4),
    "fr_dgd_s0": (WL["fr_n4_logistic_d64"].replace(s=0, d=129, m=50), 4),
    "cr_c_equals_n": (WL["cr_n8_logistic_d1024"].replace(n=3, s=2, m=21, d=100), 7),
    "fr_c_equals_n": (WL["fr_n4_logistic_d64"].replace(n=3, s=2, m=21, d=1), 7),
    "cr_ragged_d_block_row": (WL["cr_n64_lsq_d16384"].replace(n=6, s=1, d=5000, m=37), 5),
    "fr_bf16_logistic": (WL["fr_n4_logistic_d64"].replace(dtype="bf16", d=700, m=90), 5),
    "cr_bf16_lsq_long_rows": (WL["cr_n64_lsq_d16384"].replace(n=4, s=1, dtype="bf16", d=9000, m=20), 5),
    "cr_f32_softmax_k3": (WL["cr_n128_softmax_k1000"].replace(n=4, s=1, dtype="f32", K=3, d=50, m=30), 6),
    "fr_bf16_softmax_k2": (WL["fr_n32_softmax_k10"].replace(n=4, s=1, K=2, d=70, m=65), 6),
    # tensor-core softmax: ragged class, feature and row tiles
    "cr_tc_k300_d320_m200": (WL["cr_n128_softmax_k1000"].replace(n=4, s=1, K=300, d=320, m=200), 5),
    "fr_tc_k256_unequal_rows": (WL["cr_n128_softmax_k1000"].replace(scheme="FR", n=4, s=1, K=256, d=600,
                                                                     m=(130, 1, 64, 257)), 5),
    "cr_tc_k128_c_equals_n": (WL["cr_n128_softmax_k1000"].replace(n=3, s=2, K=128, d=256, m=300), 5),
    # fused logits + residual with 8-CTA clusters (K > 1792), and K = 1500
    # (six 256-class tiles: the three-kernel path)
    "cr_tc_k2000_nt8": (WL["cr_n128_softmax_k1000"].replace(n=3, s=1, K=2000, d=300, m=150), 4),
    "fr_tc_k1500_unfused": (WL["cr_n128_softmax_k1000"].replace(scheme="FR", n=4, s=1, K=1500, d=256, m=(90, 200, 3, 128)), 4),
    # few-class softmax (whole-row kernel on CTA pairs): ragged tiles, partition
    # boundaries inside a cluster's run, empty feature slices, K = 16
    "fr_smallk_k10_unequal_rows": (WL["fr_n32_softmax_k10"].replace(n=4, s=1, d=3072, m=(300, 1, 129, 700)), 5),
    "cr_smallk_k16_d1000": (WL["fr_n32_softmax_k10"].replace(scheme="CR", n=6, s=2, K=16, d=1000, m=257), 5),
    "cr_smallk_k5_d64": (WL["fr_n32_softmax_k10"].replace(scheme="CR", n=5, s=1, K=5, d=64, m=(1, 2, 128, 129, 40)), 5),
    # more slots per store (c = 6) than the fused tail's short route takes:
    # its decode reads the stores and slot totals back from L2; ten steps
    # cover every slot after the warm-up
    "cr_smallk_c6_k10_d256": (WL["fr_n32_softmax_k10"].replace(scheme="CR", n=8, s=5, K=10, d=256, m=(40, 97, 1, 64, 33, 120, 8, 71)), 10),
    # P = K d >= 2^20: the one-thread-per-column decode
    "cr_tc_wide_decode": (WL["cr_n128_softmax_k1000"].replace(n=5, s=2, K=256, d=4096, m=64), 5),
    "fr_tc_wide_decode": (WL["cr_n128_softmax_k1000"].replace(scheme="FR", n=4, s=1, K=300, d=4000, m=(70, 129, 1, 64)), 5),
}


@pytest.mark.parametrize("name", list(CASES))
def test_parity_with_oracle(libpgc, cuda, name):
    w, T = CASES[name]
    Xs, ys, masks = generate(w, T)
    g, grecs = run_gpu(libpgc, w, Xs, ys, masks)
    orecs = run_oracle(w, Xs, ys, masks)
    compare_runs(w, grecs, orecs)
    g.close()


CLUSTER_CASES = {
    "fr_smallk_k10_d2048_unequal_rows": (WL["fr_n32_softmax_k10"].replace(n=4, s=1, d=2048, m=(300, 1, 129, 700)), 5),
    "cr_smallk_k16_d1000": CASES["cr_smallk_k16_d1000"],
}


@pytest.mark.parametrize("name", list(CLUSTER_CASES))
def test_parity_cluster_few_class_kernel(libpgc, cuda, monkeypatch, name):
    """Few-class cases with the 8-CTA cluster kernel (the fall-back taken when
    the whole-row kernel does not apply; its shared memory holds rows of up
    to 2048 features)."""
    monkeypatch.setenv("PGC_NO_ROWS", "1")
    w, T = CLUSTER_CASES[name]
    Xs, ys, masks = generate(w, T)
    g, grecs = run_gpu(libpgc, w, Xs, ys, masks)
    assert g.gradient_path == "softmax_cluster"
    orecs = run_oracle(w, Xs, ys, masks)
    compare_runs(w, grecs, orecs)
    g.close()


@pytest.mark.parametrize("run", ["1", "3", "8"])
def test_parity_gradient_runs(libpgc, cuda, monkeypatch, run):
    """The tensor-core gradient contraction with runs of 1, 3 and 8 partitions
    per output tile (5 evaluated partitions: a shorter last run, or one run
    holding them all); each run's sum goes into the slot total once."""
    monkeypatch.setenv("PGC_GRAD_RUN", run)
    w, T = WL["cr_n128_softmax_k1000"].replace(n=5, s=2, K=260, d=300, m=(70, 129, 1, 64, 200)), 5
    Xs, ys, masks = generate(w, T)
    g, grecs = run_gpu(libpgc, w, Xs, ys, masks)
    assert g.gradient_path == "tc_fused"
    orecs = run_oracle(w, Xs, ys, masks)
    compare_runs(w, grecs, orecs)
    g.close()


@pytest.mark.parametrize("name", ["cr_tc_wide_decode", "fr_tc_wide_decode"])
def test_parity_early_decode_terms(libpgc, cuda, monkeypatch, name):
    """The decode split around the tensor-core GEMMs, forced on for cases too
    small for it to pay (the full-size cr_n128_softmax_k1000 runs take it by
    default): the logits kernel sums the terms of the slots other than o_t,
    the decode after the contraction adds the slot o_t terms."""
    monkeypatch.setenv("PGC_PRE_DECODE", "1")
    w, T = CASES[name]
    Xs, ys, masks = generate(w, T)
    g, grecs = run_gpu(libpgc, w, Xs, ys, masks)
    assert g.gradient_path == "tc_fused"
    orecs = run_oracle(w, Xs, ys, masks)
    compare_runs(w, grecs, orecs)
    g.close()


def test_parity_unfused_tensor_core_path(libpgc, cuda, monkeypatch):
    """A class count the fused kernel covers, forced through the three-kernel
    fall-back (logits GEMM, residual kernel, gradient contraction)."""
    monkeypatch.setenv("PGC_NO_FUSED", "1")
    w, T = CASES["cr_tc_k300_d320_m200"]
    Xs, ys, masks = generate(w, T)
    g, grecs = run_gpu(libpgc, w, Xs, ys, masks)
    assert g.gradient_path == "tc"
    orecs = run_oracle(w, Xs, ys, masks)
    compare_runs(w, grecs, orecs)
    g.close()


def test_stores_hold_the_scheduled_gradients(libpgc, cuda):
    """After each step every worker's store slot l holds the gradient of its
    slot-l partition at the step it was last evaluated (s(t,i,j), §V-B)."""
    from oracle import pgc_oracle as O
    from parity import oracle_inputs, make_gpu, rel_err, SCHEME, LOSS
    for base in (WL["cr_n8_logistic_d1024"].replace(n=5, s=2, m=40, d=96),
                 WL["fr_n4_logistic_d64"].replace(n=6, s=2, m=30)):
        Xs, ys, masks = generate(base, 7)
        g = make_gpu(libpgc, base, Xs, ys)
        o = O.PGCOracle(SCHEME[base.scheme], base.n, base.s, LOSS[base.loss], oracle_inputs(base, Xs), ys, base.lr)
        for t in range(7):
            g.step(masks[t], info=False)
            o.step(masks[t])
            for i in range(base.n):
                for l in range(base.c):
                    assert rel_err(g.store(i, l), o.ring[i][l]) < 1e-5, (t, i, l)
        g.close()


def test_mask_errors_leave_state_unchanged(libpgc, cuda):
    w = WL["cr_n8_logistic_d1024"].replace(m=50, d=64)
    Xs, ys, masks = generate(w, 3)
    g = make_ctx = None
    from parity import make_gpu
    g = make_gpu(libpgc, w, Xs, ys)
    g.step(masks[0], info=False)
    w_before = g.weights().copy()
    bad = [np.zeros(w.n, np.uint8), np.ones(w.n, np.uint8), np.array([2] + [0] * (w.n - 1), np.uint8)]
    for m in bad:
        with pytest.raises(libpgc.PGCError) as ei:
            g.step(m)
        assert ei.value.code == libpgc.EMASK
    assert g.t == 1
    np.testing.assert_array_equal(g.weights(), w_before)
    g.step(masks[1], info=False)
    assert g.t == 2
    g.close()


def test_step_before_load_is_a_state_error(libpgc, cuda):
    w = WL["fr_n4_logistic_d64"]
    g = libpgc.PGC(w.scheme, w.n, w.s, w.loss, w.dtype, w.d, rows=w.rows(), lr=w.lr)
    with pytest.raises(libpgc.PGCError) as ei:
        g.step([0, 1, 0, 0])
    assert ei.value.code == libpgc.ESTATE
    g.close()


def test_device_outputs_match_host_outputs(libpgc, cuda):
    torch = cuda
    w = WL["cr_n8_logistic_d1024"].replace(m=300)
    Xs, ys, masks = generate(w, 4)
    from parity import make_gpu
    a = make_gpu(libpgc, w, Xs, ys)
    b = make_gpu(libpgc, w, [torch.from_numpy(X).cuda() for X in Xs], [torch.from_numpy(y).cuda() for y in ys])
    for t in range(4):
        gh = np.zeros(w.d, np.float32)
        wh = np.zeros(w.d, np.float32)
        a.step(masks[t], gh, wh)
        gd = torch.zeros(w.d, device="cuda")
        wd = torch.zeros(w.d, device="cuda")
        b.step(masks[t], gd, wd)
        b.sync()
        np.testing.assert_array_equal(gd.cpu().numpy(), gh)
        np.testing.assert_array_equal(wd.cpu().numpy(), wh)
    a.close()
    b.close()


@pytest.mark.parametrize("name", ["cr_n8_logistic_d1024_m1000", "cr_tc_wide_decode", "fr_n8_softmax_k10_m333"])
def test_pinned_host_outputs_match_device_outputs(libpgc, cuda, name):
    """Pinned host outputs are written by the decode itself (no copy after
    it); they match the device outputs of an identical run bit for bit."""
    torch = cuda
    from parity import make_gpu
    w, _ = CASES[name]
    T = 4
    Xs, ys, masks = generate(w, T)
    a = make_gpu(libpgc, w, Xs, ys)
    b = make_gpu(libpgc, w, Xs, ys)
    P = w.K * w.d
    gh = torch.zeros(P).pin_memory()
    wh = torch.zeros(P).pin_memory()
    gd = torch.zeros(P, device="cuda")
    wd = torch.zeros(P, device="cuda")
    for t in range(T):
        a.step(masks[t], gh, wh)
        b.step(masks[t], gd, wd)
        b.sync()
        if w.loss == "softmax" and w.K >= 128:
            # the tensor-core slot total is summed in completion order
            assert rel_err(gh.numpy(), gd.cpu().numpy()) < 1e-5
            assert rel_err(wh.numpy(), wd.cpu().numpy()) < 1e-5
        else:
            np.testing.assert_array_equal(gh.numpy(), gd.cpu().numpy())
            np.testing.assert_array_equal(wh.numpy(), wd.cpu().numpy())
    a.close()
    b.close()


def test_teacher_forced_gradient(libpgc, cuda):
    """Set beta on the device from the oracle each step; the decoded gradient
    must then match the oracle's at that same beta (no drift)."""
    from oracle import pgc_oracle as O
    from parity import make_gpu, oracle_inputs, rel_err, SCHEME, LOSS
    w = WL["fr_n32_softmax_k10"].replace(n=8, m=200)
    Xs, ys, masks = generate(w, 6)
    g = make_gpu(libpgc, w, Xs, ys)
    o = O.PGCOracle(SCHEME[w.scheme], w.n, w.s, LOSS[w.loss], oracle_inputs(w, Xs), ys, w.lr, K=w.K)
    for t in range(6):
        g.set_weights(o.beta.astype(np.float32))
        grad = np.zeros(w.K * w.d, np.float32)
        g.step(masks[t], grad)
        rec = o.step(masks[t])
        assert rel_err(grad.reshape(w.K, w.d), rec["grad"]) < 2e-2
    g.close()


EXPECTED_PATHS = {
    "fr_n4_logistic_d64": "grad_rows",
    "cr_f32_softmax_k3": "softmax_cc",
    "fr_bf16_softmax_k2": "softmax_rows",
    "fr_smallk_k10_unequal_rows": "softmax_rows",
    "cr_smallk_k16_d1000": "softmax_rows",
    "cr_smallk_c6_k10_d256": "softmax_rows",
    "cr_tc_k300_d320_m200": "tc_fused",
    "cr_tc_k2000_nt8": "tc_fused",
    "fr_tc_k1500_unfused": "tc",
}


@pytest.mark.parametrize("name", list(EXPECTED_PATHS))
def test_gradient_path_chosen(libpgc, cuda, name):
    """Each workload shape runs on the kernel path meant for it (a silent
    fallback to a slower path would still pass parity)."""
    w, _ = CASES[name]
    g = libpgc.PGC(w.scheme, w.n, w.s, w.loss, w.dtype, w.d, K=w.K, rows=w.rows(), lr=w.lr)
    assert g.gradient_path == EXPECTED_PATHS[name]
    g.close()


def test_gradient_path_overrides(libpgc, cuda, monkeypatch):
    monkeypatch.setenv("PGC_NO_ROWS", "1")
    w, _ = CLUSTER_CASES["fr_smallk_k10_d2048_unequal_rows"]
    g = libpgc.PGC(w.scheme, w.n, w.s, w.loss, w.dtype, w.d, K=w.K, rows=w.rows(), lr=w.lr)
    assert g.gradient_path == "softmax_cluster"
    g.close()
    # rows longer than the cluster kernel's shared memory holds: CUDA cores
    w, _ = CASES["fr_smallk_k10_unequal_rows"]
    g = libpgc.PGC(w.scheme, w.n, w.s, w.loss, w.dtype, w.d, K=w.K, rows=w.rows(), lr=w.lr)
    assert g.gradient_path == "softmax_cc"
    g.close()
    w, _ = CASES["cr_tc_k300_d320_m200"]
    monkeypatch.setenv("PGC_NO_FUSED", "1")
    g = libpgc.PGC(w.scheme, w.n, w.s, w.loss, w.dtype, w.d, K=w.K, rows=w.rows(), lr=w.lr)
    assert g.gradient_path == "tc"
    g.close()
