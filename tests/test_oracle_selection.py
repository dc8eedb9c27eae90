"""Pins for oracle.selection: the paper's bin table and worked example (tests/golden/),
closed forms of the scores, and hand-computed cases."""
import json
import math
import os

import numpy as np
import pytest

from oracle import selection as sel

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def test_bin_table_matches_the_paper():
    g = _golden("speedup_bins.json")
    assert list(sel.UPPER_EDGES) == g["upper_edges"]
    assert [g["interior_representatives"][str(b)] for b in range(2, 8)] == list(sel.INTERIOR_REPRESENTATIVES)
    # interior representatives are the geometric centres of their bins (caption of the table)
    for b in range(2, 8):
        lo, hi = sel.LOWER_EDGES[b - 1], sel.UPPER_EDGES[b - 1]
        assert abs(math.sqrt(lo * hi) - sel.INTERIOR_REPRESENTATIVES[b - 2]) < 0.01


@pytest.mark.parametrize("S,b", [(0.1, 1), (0.25, 1), (0.2501, 2), (0.5, 2), (0.7, 3), (0.71, 3), (0.8, 4),
                                 (1.0, 4), (1.2, 5), (1.41, 5), (1.71, 6), (2.0, 6), (3.9, 7), (4.0, 7), (4.01, 8),
                                 (100.0, 8)])
def test_speedup_bin_edges(S, b):
    assert sel.speedup_bin(S) == b


def test_expected_speedup_and_ranking():
    m = sel.representatives(0.1, 6.0)
    p = np.zeros((3, 8))
    p[0, 6] = 1.0                        # all mass on bin 7 -> 2.83
    p[1, :] = 1.0 / 8                    # uniform -> mean of m
    p[2, 4], p[2, 5] = 0.5, 0.5          # -> (1.19 + 1.68) / 2
    s = sel.expected_speedup(p, m)
    np.testing.assert_allclose(s, [2.83, m.mean(), 1.435], atol=1e-12)
    assert list(sel.ranking([1.0, 2.0, 2.0, 0.5])) == [1, 2, 0, 3]   # ties: lower index first


def test_recovered_perfect_and_worst_rankings():
    S = np.array([0.5, 3.0, 1.0, 2.0])
    assert sel.recovered(S, S) == pytest.approx(100.0)
    # ranking the fastest last with n = 4: budgets 1, 5, 10, 25 % take the single slowest (0.5),
    # the 50 % budget takes the two slowest (best 1.0): 100/5 * (4 * 0.5/3 + 1.0/3)
    assert sel.recovered(-S, S) == pytest.approx(100.0 / 5 * (4 * 0.5 / 3 + 1.0 / 3))


def test_brier_and_crps_closed_forms():
    one_hot = np.eye(8)[3]
    assert sel.brier(one_hot, 4) == 0.0 and sel.crps(one_hot, 4) == 0.0
    uni = np.full(8, 1.0 / 8)
    assert sel.brier(uni, 5) == pytest.approx(0.5 * (7 / 64 + 49 / 64))
    assert sel.crps(uni, 1) == pytest.approx((49 + 36 + 25 + 16 + 9 + 4 + 1) / 64 / 7)
    # mass one bin away costs less CRPS than mass seven bins away; Brier treats them alike
    near, far = np.eye(8)[1], np.eye(8)[7]
    assert sel.crps(near, 1) < sel.crps(far, 1)
    assert sel.brier(near, 1) == sel.brier(far, 1) == 1.0


def test_ece_extremes():
    assert sel.ece([0.7] * 10, [1] * 7 + [0] * 3) == pytest.approx(0.0)
    assert sel.ece([1.0] * 4, [0] * 4) == pytest.approx(1.0)
    assert sel.ece([0.25, 0.95], [1, 1]) == pytest.approx(0.5 * 0.75 + 0.5 * 0.05)


def test_forecast_error_hand_value():
    m = sel.representatives(0.2, 5.0)
    assert sel.forecast_error(np.array([7, 2]), np.array([3.0, 0.4]), m) == pytest.approx((0.17 + 0.05) / 2)


def test_discovery_worked_example():
    g = _golden("discovery_example.json")
    assert sel.speedup_bin(g["g"]) == 7 and g["g"] >= g["cutoff_x"]
    p = np.zeros(8)
    p[6], p[7], p[4] = 0.5, 0.2, 0.3     # 0.7 of the mass on g >= 2 (bins 7 and 8)
    s = sel.discovery_score(p, g["cutoff_x"])
    assert s == pytest.approx(g["score_s"])
    tau_max = g["predicted_positive_for_tau_at_most"]
    assert sel.discovery_predict(s, tau_max) == 1
    assert sel.discovery_predict(s, tau_max + 1e-9) == 0


def test_discovery_cutoffs_use_bins_at_or_above_x():
    p = np.arange(1, 9, dtype=np.float64) / 36.0
    assert sel.discovery_score(p, 1.25) == pytest.approx((6 + 7 + 8) / 36)   # bins 6, 7, 8
    assert sel.discovery_score(p, 1.5) == pytest.approx((7 + 8) / 36)
    assert sel.discovery_score(p, 2.0) == pytest.approx((7 + 8) / 36)
    assert sel.discovery_score(p, 0.0) == pytest.approx(1.0)


def test_poorly_grounded_trace_example():
    # Sec. A (failure cases): 0.65 of the mass on bins 6-8 with the arg max at bin 8 (0.25) and 0.15 on
    # bin 5; the remaining 0.20 is placed on bins 1-4 here
    p = np.array([0.05, 0.05, 0.05, 0.05, 0.15, 0.2, 0.2, 0.25])
    assert p.sum() == pytest.approx(1.0) and p[5:].sum() == pytest.approx(0.65)
    assert int(np.argmax(p)) + 1 == 8 and p.max() == 0.25
