"""Shared helpers of the parity tests: run one seeded workload through the
CUDA library (via its C ABI) and through the fp64 oracle, and compare.

Tolerances (decoded gradient, normwise max|gpu - oracle| / max|oracle|):
1e-4 for fp32 features, 2e-2 for bf16 features; loss trajectory 1e-3
relative per step.  Index outputs (schedule, slot, FR representatives,
the support of the device-derived decode coefficients) are bit-exact.
"""

from __future__ import annotations

import numpy as np

from oracle import pgc_oracle as O
from paper_2607_20739_gb300 import workloads as W

SCHEME = {"FR": O.FR, "CR": O.CR}
LOSS = {"logistic": O.LOGISTIC, "lsq": O.LSQ, "softmax": O.SOFTMAX}

GRAD_TOL = {"f32": 1e-4, "bf16": 2e-2}
LOSS_TOL = 1e-3


def rel_err(a, b) -> float:
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    den = np.max(np.abs(b))
    if den == 0.0:
        return float(np.max(np.abs(a)))
    return float(np.max(np.abs(a - b)) / den)


def generate(w: W.Workload, steps: int, seed: int = 1):
    Xs, ys = W.make_partitions(w, seed)
    masks = W.make_masks(w, steps, seed + 1000)
    return Xs, ys, masks


def oracle_inputs(w: W.Workload, Xs):
    return [W.features_as_float(X, w.dtype) for X in Xs]


def run_oracle(w: W.Workload, Xs, ys, masks, record_loss=True, mode="pgc"):
    return O.run_mode(mode, SCHEME[w.scheme], w.n, w.s, LOSS[w.loss], oracle_inputs(w, Xs), ys, w.lr, list(masks),
                      K=w.K, record_loss=record_loss)


def make_gpu(binding, w: W.Workload, Xs, ys, stream=None, mode="pgc"):
    g = binding.PGC(w.scheme, w.n, w.s, w.loss, w.dtype, w.d, K=w.K, rows=w.rows(), lr=w.lr, stream=stream,
                    mode=mode)
    g.load(Xs, ys)
    return g


def run_gpu(binding, w: W.Workload, Xs, ys, masks, record_loss=True, mode="pgc"):
    g = make_gpu(binding, w, Xs, ys, mode=mode)
    P = w.K * w.d
    out = []
    for mask in masks:
        lv = g.loss() if record_loss else None
        grad = np.zeros(P, dtype=np.float32)
        beta = np.zeros(P, dtype=np.float32)
        info = g.step(mask, grad, beta)
        rec = dict(info)
        rec["grad"] = grad.reshape(w.K, w.d) if w.loss == "softmax" else grad
        rec["beta"] = beta.reshape(w.K, w.d) if w.loss == "softmax" else beta
        rec["coeff"] = g.decode_coefficients()
        rec["loss"] = lv
        out.append(rec)
    return g, out


def compare_step(w: W.Workload, t: int, a: dict, b: dict, check_loss=True):
    """One step of a GPU record `a` against the oracle's `b`: schedule, slot,
    FR representatives and the decode support bit-exact, the coefficients to
    fp32 rounding, the decoded gradient within GRAD_TOL and (check_loss) the
    loss F(beta^(t)) within LOSS_TOL.  Returns (gradient error, loss error)."""
    tol = GRAD_TOL[w.dtype]
    assert a["t"] == b["t"] == t
    assert a["slot"] == b["slot"], (t, a["slot"], b["slot"])
    assert list(a["eval_partition"]) == list(b["eval_partition"]), t
    if w.scheme == "FR":
        assert list(a["fr_rep"]) == list(b["fr_rep"]), t
    assert a["received"] == b["received"]
    # device-derived coefficients: same support, same values (fp32)
    ca = np.asarray(a["coeff"], dtype=np.float64)
    cb = np.asarray(b["coeff"], dtype=np.float64)
    assert ((ca != 0) == (cb != 0)).all(), (t, ca, cb)
    np.testing.assert_allclose(ca, cb, rtol=2e-7, atol=0)
    e = rel_err(a["grad"], b["grad"])
    assert e <= tol, f"step {t}: decoded-gradient error {e:.3g} > {tol}"
    le = 0.0
    if check_loss and a["loss"] is not None:
        le = abs(a["loss"] - b["loss"]) / abs(b["loss"])
        assert le <= LOSS_TOL, f"step {t}: loss {a['loss']} vs {b['loss']} ({le:.3g})"
    return e, le


def compare_runs(w: W.Workload, gpu_recs, ora_recs, check_loss=True):
    worst = 0.0
    for t, (a, b) in enumerate(zip(gpu_recs, ora_recs)):
        e, _ = compare_step(w, t, a, b, check_loss)
        worst = max(worst, e)
    return worst
