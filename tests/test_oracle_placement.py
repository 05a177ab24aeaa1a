"""Pins of the oracle's placement, schedule and decode-weight rules.

Sources: §III (FR and CR placement, the n = 4, c = 2 FR example), §IV-A
(PGC-FR schedule), §V-B (PGC-CR schedule, |N_k|, mu and the bound
0 <= |N_k| / mu < 2).
"""

import os

import numpy as np
import pytest

from oracle import pgc_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _read_table(name):
    rows = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            w, parts = line.split(":")
            rows[int(w)] = [int(p) for p in parts.split()]
    return [rows[i] for i in range(len(rows))]


def test_fr_placement_matches_paper_example():
    assert O.holdings(O.FR, 4, 2) == _read_table("fr_placement_n4_c2.txt")


def test_fr_rejects_c_not_dividing_n():
    with pytest.raises(ValueError):
        O.holdings(O.FR, 6, 4)
    with pytest.raises(ValueError):
        O.holdings(O.CR, 3, 4)


@pytest.mark.parametrize("scheme", [O.FR, O.CR])
@pytest.mark.parametrize("n,c", [(1, 1), (4, 1), (4, 2), (6, 3), (8, 4), (9, 3), (12, 6), (5, 5)])
def test_every_partition_has_c_holders_and_workers_hold_distinct(scheme, n, c):
    if scheme == O.FR and n % c:
        pytest.skip("FR needs c | n")
    hold = O.holdings(scheme, n, c)
    assert len(hold) == n
    count = np.zeros(n, dtype=int)
    for i in range(n):
        assert len(set(hold[i])) == c
        for k in hold[i]:
            assert 0 <= k < n
            count[k] += 1
    assert (count == c).all()


@pytest.mark.parametrize("n,c", [(4, 2), (6, 3), (8, 4), (12, 6)])
def test_fr_groups_are_disjoint_and_share_placement(n, c):
    hold = O.holdings(O.FR, n, c)
    for i in range(n):
        # every member of a group holds the same c partitions
        assert hold[i] == hold[(i // c) * c]
    groups = [set(hold[j * c]) for j in range(n // c)]
    for a in range(len(groups)):
        for b in range(a + 1, len(groups)):
            assert not groups[a] & groups[b]


@pytest.mark.parametrize("n,c", [(4, 2), (5, 3), (7, 7), (9, 4)])
def test_cr_is_cyclic(n, c):
    hold = O.holdings(O.CR, n, c)
    # worker i + 1 holds worker i's list shifted by one partition, mod n
    for i in range(n):
        assert hold[(i + 1) % n] == [(k + 1) % n for k in hold[i]]
    assert hold[0] == list(range(c))


@pytest.mark.parametrize("scheme", [O.FR, O.CR])
@pytest.mark.parametrize("n,c", [(4, 2), (6, 3), (8, 4), (6, 1)])
def test_schedule_rotates_through_every_slot(scheme, n, c):
    hold = O.holdings(scheme, n, c)
    assert O.evaluated_slot(0, c) is None
    for t0 in range(1, 2 * c + 1):
        for i in range(n):
            seen = [O.evaluated_partition(scheme, n, c, i, t) for t in range(t0, t0 + c)]
            assert sorted(seen) == sorted(hold[i])
    for t in range(1, 3 * c):
        ev = [O.evaluated_partition(scheme, n, c, i, t) for i in range(n)]
        if scheme == O.CR:
            # CR: the n workers evaluate n distinct partitions at every step
            assert sorted(ev) == list(range(n))
        else:
            # FR: all c members of a group evaluate the same partition
            o = (t - 1) % c
            assert ev == [(i // c) * c + o for i in range(n)]


def test_schedule_first_steps_by_hand():
    # FR n=4 c=2: step 1 evaluates slot 0 (D0 for group 0, D2 for group 1),
    # step 2 slot 1 (D1, D3), step 3 slot 0 again.
    assert [O.evaluated_partition(O.FR, 4, 2, i, 1) for i in range(4)] == [0, 0, 2, 2]
    assert [O.evaluated_partition(O.FR, 4, 2, i, 2) for i in range(4)] == [1, 1, 3, 3]
    assert [O.evaluated_partition(O.FR, 4, 2, i, 3) for i in range(4)] == [0, 0, 2, 2]
    # CR n=4 c=2: step 1: W_j evaluates D_j; step 2: D_{j+1 mod 4}
    assert [O.evaluated_partition(O.CR, 4, 2, i, 1) for i in range(4)] == [0, 1, 2, 3]
    assert [O.evaluated_partition(O.CR, 4, 2, i, 2) for i in range(4)] == [1, 2, 3, 0]


@pytest.mark.parametrize("n", range(2, 10))
def test_cr_appearance_counts_and_weight_bound(n):
    """§V-B: sum_k |N_k| = (n - s) c and 0 <= |N_k| / mu < 2 for every mask."""
    for s in range(0, n):
        c = s + 1
        mu = (n - s) * c / n
        for mask in O.all_masks(n, s):
            N = O.appearance_counts(O.CR, n, s, mask)
            assert N.sum() == (n - s) * c
            assert (N >= 0).all()
            assert (N / mu < 2.0).all()
            assert N.max() <= min(c, n - s)


@pytest.mark.parametrize("n,s", [(4, 1), (6, 2), (8, 3), (6, 5)])
def test_cr_mean_weight_is_one(n, s):
    """§V-B: E[|N_k| / mu] = 1 when every worker is equally likely to straggle."""
    c = s + 1
    mu = (n - s) * c / n
    tot = np.zeros(n)
    cnt = 0
    for mask in O.all_masks(n, s):
        tot += O.appearance_counts(O.CR, n, s, mask) / mu
        cnt += 1
    np.testing.assert_allclose(tot / cnt, np.ones(n), rtol=0, atol=1e-12)


def test_decode_coefficients_by_hand():
    # FR n=4 c=2, W1 straggles: groups {0,1} -> W0, {2,3} -> W2; a = 1/4 each.
    a = O.decode_coefficients(O.FR, 4, 1, [0, 1, 0, 0])
    assert list(a) == [0.25, 0.0, 0.25, 0.0]
    a = O.decode_coefficients(O.FR, 4, 1, [1, 0, 0, 0])
    assert list(a) == [0.0, 0.25, 0.25, 0.0]
    # CR n=4 s=1: 1/(n mu) = 1/((n - s) c) = 1/6 for the three received.
    a = O.decode_coefficients(O.CR, 4, 1, [0, 0, 1, 0])
    assert list(a) == [1 / 6, 1 / 6, 0.0, 1 / 6]


def test_mask_validation():
    with pytest.raises(ValueError):
        O.check_mask([1, 1, 0, 0], 4, 1)
    with pytest.raises(ValueError):
        O.check_mask([2, 0, 0, 0], 4, 1)
    with pytest.raises(ValueError):
        O.check_mask([0, 0, 0], 4, 1)
    O.check_mask([0, 0, 1, 0], 4, 1)
