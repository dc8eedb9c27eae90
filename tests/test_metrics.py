"""Host evaluation of 8-bin forecasts in the library (gf_speedup_bin, gf_score_forecasts) against the
oracle's restatement of the paper's scores (oracle/selection.py, pinned in test_oracle_selection.py):
speedup recovered, ECE and forecast error (Sec. 3.1), Brier and CRPS (Sec. 2.2).  No GPU needed."""
import numpy as np
import pytest

from oracle import selection as sel


@pytest.fixture(scope="module")
def gf():
    from paper_2605_31464_gb300 import _build
    _build.build()
    import paper_2605_31464_gb300 as g
    return g


@pytest.mark.parametrize("S", [0.1, 0.25, 0.2501, 0.5, 0.71, 0.8, 1.0, 1.2, 1.41, 1.71, 2.0, 3.9, 4.0, 4.01, 100.0])
def test_speedup_bin(gf, S):
    assert gf.gf_speedup_bin(S) == sel.speedup_bin(S)


def _case(n, seed, peaked=False):
    rng = np.random.default_rng(seed)
    logits = rng.standard_normal((n, 8)) * (4.0 if peaked else 1.0)
    p = np.exp(logits)
    p /= p.sum(axis=1, keepdims=True)
    S = np.exp(rng.normal(0.0, 1.0, n))
    return p, S


@pytest.mark.parametrize("n,seed,peaked", [(1, 1, False), (7, 2, False), (64, 3, True), (480, 4, False),
                                           (1000, 5, True)])
def test_scores_match_the_oracle(gf, n, seed, peaked):
    p, S = _case(n, seed, peaked)
    m = sel.representatives(0.12, 6.5)
    got = gf.score_forecasts(p, S, m)
    pred = np.argmax(p, axis=1) + 1
    y = np.array([sel.speedup_bin(s) for s in S])
    np.testing.assert_allclose(got["recovered"], sel.recovered(sel.expected_speedup(p, m), S), rtol=1e-12)
    np.testing.assert_allclose(got["ece"], sel.ece(p.max(axis=1), pred == y), rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(got["forecast_error"], sel.forecast_error(pred, S, m), rtol=1e-12)
    np.testing.assert_allclose(got["brier"], np.mean([sel.brier(p[i], y[i]) for i in range(n)]), rtol=1e-12)
    np.testing.assert_allclose(got["crps"], np.mean([sel.crps(p[i], y[i]) for i in range(n)]), rtol=1e-12)


def test_ties_and_one_hot(gf):
    m = sel.representatives(0.12, 6.5)
    # one-hot forecasts on the measured bins: Brier 0, CRPS 0, ECE 0, recovered 100
    S = np.array([0.2, 1.1, 3.0])
    p = np.zeros((3, 8))
    for i, s in enumerate(S):
        p[i, sel.speedup_bin(s) - 1] = 1.0
    got = gf.score_forecasts(p, S, m)
    assert got["brier"] == 0.0 and got["crps"] == 0.0 and got["ece"] == 0.0
    assert got["recovered"] == pytest.approx(100.0)
    # a uniform forecast predicts the lowest bin (ties) and ranks by index
    u = np.full((2, 8), 1.0 / 8)
    got = gf.score_forecasts(u, np.array([0.3, 5.0]), m)
    assert got["forecast_error"] == pytest.approx(np.mean([abs(m[0] - 0.3), abs(m[0] - 5.0)]))


def test_bad_arguments_are_refused(gf):
    m = sel.representatives(0.12, 6.5)
    with pytest.raises(gf.GfError):
        gf.score_forecasts(np.full((2, 8), 0.125), np.array([1.0, -1.0]), m)
    with pytest.raises(gf.GfError):
        gf.score_forecasts(np.full((1, 8), np.nan), np.array([1.0]), m)
    with pytest.raises(ValueError):
        gf.score_forecasts(np.full((2, 7), 0.125), np.array([1.0, 1.0]), m)
