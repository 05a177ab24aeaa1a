"""Free-running training trajectories at the five workloads' full sizes.

The CUDA path (through the C ABI, on its own stream with device outputs, the
launch configuration bench.py times) and the fp64 oracle each run the same
seeded workload from beta^(0) = 0 with the same straggler masks, neither
seeing the other's state.  Every step is compared: the schedule, slot, FR
representatives and decode support bit-exact, the decoded gradient within
1e-4 (fp32 features) or 2e-2 (bf16 features) normwise, and the full-data loss
F(beta^(t)) within 1e-3 relative (the iterations of §IV-A and §V-B).

Steps per workload: the whole run where the oracle finishes it within a
minute or two (fr_n4_logistic_d64: 20, cr_n8_logistic_d1024: 200,
fr_n32_softmax_k10: 500, cr_n64_lsq_d16384: 300); for cr_n128_softmax_k1000
a prefix of 9 of its 200 steps, which refreshes every store slot once after
the warm-up step (c = 8) and then decodes with stale slots: its literal
oracle evaluates 1024 partition gradients in its warm-up step, about 17
GFLOP each, and keeps 33.5 GB of fp64 stores.  The worst error of each run is
reported in the headroom summary.
"""

import gc

import numpy as np
import pytest

from oracle import pgc_oracle as O
from paper_2607_20739_gb300 import workloads as W

from parity import GRAD_TOL, LOSS, LOSS_TOL, SCHEME, compare_step

pytestmark = pytest.mark.gpu

STEPS = {
    "fr_n4_logistic_d64": 20,
    "cr_n8_logistic_d1024": 200,
    "fr_n32_softmax_k10": 500,
    "cr_n64_lsq_d16384": 300,
    "cr_n128_softmax_k1000": 9,
}


@pytest.mark.parametrize("name", list(STEPS))
def test_free_running_trajectory(libpgc, cuda, headroom, name):
    torch = cuda
    w = W.WORKLOADS[name]
    T = STEPS[name]
    assert T == w.T or T >= 2 * w.c or T == w.c + 1
    Xs, ys = W.make_partitions(w, 1)
    masks = W.make_masks(w, T, 1001)
    stream = torch.cuda.Stream()
    g = libpgc.PGC(w.scheme, w.n, w.s, w.loss, w.dtype, w.d, K=w.K, rows=w.rows(), lr=w.lr, stream=stream)
    g.load(Xs, ys)
    # the oracle reads the exact feature values in fp64 (converted once here,
    # so that its per-step arithmetic is not dominated by conversions)
    X64 = []
    for k in range(w.n):
        X64.append(W.features_as_float(Xs[k], w.dtype).astype(np.float64))
        Xs[k] = None
    o = O.PGCOracle(SCHEME[w.scheme], w.n, w.s, LOSS[w.loss], X64, ys, w.lr, K=w.K)

    P = w.K * w.d
    gout = torch.empty(P, device="cuda")
    wout = torch.empty(P, device="cuda")
    shape = (w.K, w.d) if w.loss == "softmax" else (w.d,)
    worst_g, worst_l, worst_w = 0.0, 0.0, 0.0
    try:
        for t in range(T):
            gl = g.loss()
            info = g.step(masks[t], gout, wout)
            g.sync()
            a = dict(info)
            a["grad"] = gout.cpu().numpy().reshape(shape)
            a["coeff"] = g.decode_coefficients()
            a["loss"] = gl
            ol = o.loss_value()
            b = o.step(masks[t])
            b["loss"] = ol
            eg, el = compare_step(w, t, a, b)
            worst_g, worst_l = max(worst_g, eg), max(worst_l, el)
            beta = wout.cpu().numpy().reshape(shape).astype(np.float64)
            worst_w = max(worst_w, float(np.max(np.abs(beta - o.beta)) / max(np.max(np.abs(o.beta)), 1e-30)))
    finally:
        g.close()
    headroom.append(f"trajectory {name} ({T} of {w.T} steps, free-running): decoded gradient "
                    f"{worst_g:.2e} / {GRAD_TOL[w.dtype]:g}, loss {worst_l:.2e} / {LOSS_TOL:g}, "
                    f"beta (normwise) {worst_w:.2e}")
    del o, X64
    gc.collect()
