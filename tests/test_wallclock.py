"""The simulated step clock (§VI "time per step"): a hand-computed case, the
orderings the model implies for any delays, and agreement with the seeded
straggler masks."""

import numpy as np
import pytest

from paper_2607_20739_gb300 import wallclock as WC
from paper_2607_20739_gb300 import workloads as W


def test_hand_computed_case():
    # n = 4, s = 1 (c = 2), compute 1, delay unit 1, decode 0.25
    t = WC.step_times([[0.1, 0.5, 0.3, 0.9]], n=4, s=1, compute_s=1.0, delay_unit_s=1.0, decode_s=0.25)
    assert t["pgc"][0] == pytest.approx(1.5 + 0.25)      # 3rd fastest of 1.1 1.5 1.3 1.9
    assert t["is_sgd"][0] == pytest.approx(1.5 + 0.25)
    assert t["gc"][0] == pytest.approx(2.5 + 0.25)       # 3rd fastest of 2.1 2.5 2.3 2.9
    assert t["dgd"][0] == pytest.approx(1.9 + 0.25)      # slowest of all four


@pytest.mark.parametrize("name", list(W.WORKLOADS))
def test_orderings_for_seeded_delays(name):
    w = W.WORKLOADS[name]
    D = W.draw_delays(w, 200, 7)
    t = WC.step_times(D, w.n, w.s, compute_s=2.0, delay_unit_s=1.0)
    assert np.all(t["pgc"] <= t["dgd"])                  # never waits for the s slowest
    np.testing.assert_array_equal(t["pgc"], t["is_sgd"])  # same work, same wait
    assert np.all(t["gc"] >= t["pgc"])                   # c partitions per worker
    if w.s > 0:
        assert np.all(t["gc"] - t["pgc"] >= (w.c - 1) * 2.0 - 1e-12)


def test_no_stragglers_reduces_to_dgd():
    w = W.WORKLOADS["cr_n8_logistic_d1024"].replace(s=0)
    D = W.draw_delays(w, 50, 3)
    t = WC.step_times(D, w.n, 0, compute_s=1.0, delay_unit_s=0.5)
    np.testing.assert_array_equal(t["pgc"], t["dgd"])
    np.testing.assert_array_equal(t["gc"], t["dgd"])


@pytest.mark.parametrize("name", list(W.WORKLOADS))
def test_waited_for_workers_are_the_non_stragglers(name):
    # equal compute: the n - s fastest finishers are the workers the mask keeps,
    # so the step ends with the slowest non-straggler
    w = W.WORKLOADS[name]
    D = W.draw_delays(w, 100, 11)
    M = W.make_masks(w, 100, 11)
    t = WC.step_times(D, w.n, w.s, compute_s=1.0, delay_unit_s=1.0)
    for k in range(100):
        assert t["pgc"][k] == pytest.approx(1.0 + D[k][M[k] == 0].max())


def test_summary_normalises_by_dgd():
    w = W.WORKLOADS["cr_n128_softmax_k1000"]
    sm = WC.summary(W.draw_delays(w, 100, 5), w.n, w.s, 1e-3, 1e-3, 2e-4)
    assert sm["normalized_to_dgd"]["dgd"] == pytest.approx(1.0)
    assert 0 < sm["normalized_to_dgd"]["pgc"] < 1 < sm["normalized_to_dgd"]["gc"]
