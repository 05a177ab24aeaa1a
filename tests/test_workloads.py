"""The seeded input generators: determinism, shapes, bf16 rounding, masks."""

import numpy as np
import pytest

from paper_2607_20739_gb300 import workloads as W


def test_bf16_rounding_ties_to_even():
    vals = np.array([1.0, 1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, -2.5, 0.0, 1.0 + 2.0 ** -7], dtype=np.float32)
    bits = W.f32_to_bf16_bits(vals)
    assert list(bits) == [0x3F80, 0x3F80, 0x3F82, 0xC020, 0x0000, 0x3F81]
    np.testing.assert_array_equal(W.bf16_bits_to_f32(bits)[[0, 3, 4]], [1.0, -2.5, 0.0])


def test_bf16_rounding_error_bound():
    x = np.random.default_rng(0).standard_normal(10000).astype(np.float32)
    r = W.bf16_bits_to_f32(W.f32_to_bf16_bits(x))
    assert np.all(np.abs(r - x) <= np.abs(x) * 2.0 ** -8)


@pytest.mark.parametrize("name", W.WORKLOAD_ORDER)
def test_partitions_are_deterministic(name):
    w = W.WORKLOADS[name].replace(m=5, n=min(W.WORKLOADS[name].n, 8))
    a = W.make_partition(w, 3, 1)
    b = W.make_partition(w, 3, 1)
    c = W.make_partition(w, 4, 1)
    np.testing.assert_array_equal(a[0], b[0])
    np.testing.assert_array_equal(a[1], b[1])
    assert not np.array_equal(a[0], c[0])
    assert a[0].shape == (5, w.d)
    assert a[0].dtype == (np.uint16 if w.dtype == "bf16" else np.float32)
    if w.loss == "softmax":
        assert a[1].dtype == np.int32 and a[1].min() >= 0 and a[1].max() < w.K
    if w.loss == "logistic":
        assert set(np.unique(a[1])) <= {0.0, 1.0}


def test_threaded_generation_matches_serial():
    w = W.WORKLOADS["cr_n8_logistic_d1024"].replace(m=33)
    Xa, ya = W.make_partitions(w, 7, threads=1)
    Xb, yb = W.make_partitions(w, 7, threads=4)
    for k in range(w.n):
        np.testing.assert_array_equal(Xa[k], Xb[k])
        np.testing.assert_array_equal(ya[k], yb[k])


@pytest.mark.parametrize("name", W.WORKLOAD_ORDER)
def test_masks_mark_the_s_slowest(name):
    w = W.WORKLOADS[name]
    masks = W.make_masks(w, 25, 11)
    D = W.draw_delays(w, 25, 11)
    assert masks.shape == (25, w.n) and masks.dtype == np.uint8
    assert (masks.sum(axis=1) == w.s).all()
    for t in range(25):
        slow = D[t][masks[t] == 1]
        fast = D[t][masks[t] == 0]
        assert slow.min() >= fast.max()
    np.testing.assert_array_equal(masks, W.make_masks(w, 25, 11))


def test_unequal_rows():
    w = W.WORKLOADS["fr_n4_logistic_d64"].replace(m=(3, 1, 7, 2))
    Xs, ys = W.make_partitions(w, 1)
    assert [X.shape[0] for X in Xs] == [3, 1, 7, 2]
    assert [len(y) for y in ys] == [3, 1, 7, 2]
