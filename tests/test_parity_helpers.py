"""The decision-margin helpers of the parity harness (tests/parity.py), on hand-made cases:
the relative gap at a top-k boundary, the best-versus-runner-up gap of bucket routing, and
the near-tie rule of the top-k comparison (a swap is accepted only inside DELTA)."""
import math

import numpy as np
import pytest

import parity as P


def test_boundary_gap():
    v = np.array([1.0, 4.0, 2.0, 2.0, 3.0])
    assert P.boundary_gap(v, 1) == pytest.approx((4.0 - 3.0) / 4.0)
    assert P.boundary_gap(v, 3) == 0.0            # 2.0 taken, 2.0 left out: an exact tie
    assert P.boundary_gap(v, 4) == pytest.approx((2.0 - 1.0) / 2.0)
    assert math.isinf(P.boundary_gap(v, 5)) and math.isinf(P.boundary_gap(v, 0))


def test_route_gap():
    # bucket 4: positions 0-3 and 4-7; kept 0, 1, 5; bucket 0 evicts 2, 3 and keeps two
    kept = np.zeros(8, dtype=bool)
    kept[[0, 1, 5]] = True
    a = np.array([0.5, 0.4, 0.1, 0.1, 0.9, 0.3, 0.2, 0.2])
    assert P.route_gap(a, kept, 4) == pytest.approx((0.5 - 0.4) / 0.5)
    # bucket 1 keeps only one token: it has no runner-up and does not count
    kept[0] = False
    assert math.isinf(P.route_gap(a, kept, 4))


def test_topk_choice_near_tie_rule():
    v = np.array([3.0, 2.0, 2.0 * (1 - 0.5 * P.DELTA), 1.0])
    own = np.array([True, True, False, False])
    assert P.check_topk_choice(own, v, 2, "exact") == 0
    swapped = np.array([True, False, True, False])   # within DELTA of the threshold: accepted
    assert P.check_topk_choice(swapped, v, 2, "near tie") == 2
    wrong = np.array([True, False, False, True])     # 1.0 is far below the threshold
    with pytest.raises(AssertionError):
        P.check_topk_choice(wrong, v, 2, "wrong")


def test_stats_merge_low_and_counts():
    st = P.Stats()
    st.low("topk_min_gap", 0.3)
    st.low("topk_min_gap", 0.1)
    st.add("topk_near_ties", 0)
    st.add("route_near_ties", 2)
    assert st["topk_min_gap"] == 0.1 and st.near_ties() == 2
