"""Pins for oracle.sampling (temperature sampling with repeats, Sec. 3.1 setup).

* The generator: the oracle's Philox4x64-10 blocks (numpy's bit generator)
  equal the published Random123 known answer and the separately pinned C
  implementation in ``synth`` at the counters the draw uses.
* The Gumbel-max draw: empirical token frequencies match softmax(l / T) for
  three temperatures (a wrong sign, a T multiplied instead of divided, or a
  single log instead of two all fail); a vanishing temperature gives the
  greedy token.
* Repeat statistics: hand-computed mean and population standard deviation.
* The sampled forecast: vanishing temperature reproduces the greedy forecast,
  the same (seed, row) reproduces itself, other rows or seeds draw otherwise.
"""
import dataclasses
import math

import numpy as np
import pytest

import oracle
from oracle import sampling as smp
import synth


@pytest.mark.parametrize("seed,t,r,V", [(0, 0, 0, 3), (7, 0, 5, 9), (123456789, 4, 13, 5), (2 ** 63 + 5, 1, 0, 2),
                                        (3, 255, 97, 4)])
def test_words_equal_the_pinned_c_philox_at_the_draw_counters(seed, t, r, V):
    got = smp.philox_words(seed, t, r, V)
    for v in range(V):
        ref = synth.philox4x64_10([v, t, r // 4, 0], [seed, 0])
        assert int(got[v]) == int(ref[r % 4])


def test_random123_known_answer_gives_the_first_uniform():
    # Random123 philox4x64_10 at counter 0, key 0: first word 0x16554D9ECA36314C
    assert int(smp.philox_words(0, 0, 0, 1)[0]) == 0x16554D9ECA36314C
    u = smp.uniforms(0, 0, 0, 1)[0]
    assert u == (0x16554D9ECA36314C // 2 ** 41 + 0.5) / 2 ** 23
    assert u == (731814 + 0.5) / 8388608


def test_uniforms_stay_inside_the_open_interval():
    u = smp.uniforms(11, 3, 6, 20000)
    assert u.min() > 0.0 and u.max() < 1.0
    # 23 bits + 1/2: every value is an odd multiple of 2^-24, exact in float32
    assert np.all(np.float64(np.float32(u)) == u)
    assert np.all(np.mod(u * 2 ** 24, 2) == 1)
    # roughly uniform: mean 1/2, variance 1/12
    assert abs(u.mean() - 0.5) < 0.01 and abs(u.var() - 1 / 12) < 0.005


def test_gumbel_of_known_uniforms():
    assert smp.gumbel(np.exp(-1.0)) == pytest.approx(0.0, abs=1e-15)
    assert smp.gumbel(np.exp(-np.exp(-2.0))) == pytest.approx(2.0, abs=1e-12)


@pytest.mark.parametrize("T", [1.0, 0.5, 2.0])
def test_gumbel_max_draws_follow_the_tempered_softmax(T):
    logits = np.log(np.array([1.0, 2.0, 3.0, 4.0]))
    target = np.array([1.0, 2.0, 3.0, 4.0]) ** (1.0 / T)
    target /= target.sum()
    n = 12000
    counts = np.zeros(4)
    for r in range(n):
        counts[smp.sample(logits, T, smp.uniforms(2024, 0, r, 4))] += 1
    freq = counts / n
    sd = np.sqrt(target * (1 - target) / n)
    assert np.all(np.abs(freq - target) < 5 * sd), (freq, target)


def test_draws_over_tokens_and_rows_are_distinct_streams():
    a = smp.uniforms(5, 0, 0, 64)
    b = smp.uniforms(5, 1, 0, 64)
    c = smp.uniforms(5, 0, 1, 64)
    d = smp.uniforms(6, 0, 0, 64)
    for x, y in [(a, b), (a, c), (a, d), (b, c)]:
        assert not np.any(x == y)


def test_vanishing_temperature_is_greedy():
    rng = np.random.default_rng(3)
    for r in range(20):
        l = rng.normal(size=300)
        assert smp.sample(l, 1e-9, smp.uniforms(1, 0, r, 300)) == int(np.argmax(l))


def test_repeat_stats_by_hand():
    mean, std = smp.repeat_stats(np.array([0.2, 0.4, 0.9]))
    assert mean == pytest.approx(0.5, abs=1e-15)
    assert std == pytest.approx(math.sqrt((0.09 + 0.01 + 0.16) / 3), abs=1e-15)
    m2, s2 = smp.repeat_stats(np.array([[0.3, 0.7], [0.3, 0.7], [0.3, 0.7]]))
    np.testing.assert_allclose(m2, [0.3, 0.7], atol=1e-15)
    np.testing.assert_allclose(s2, [0.0, 0.0], atol=1e-15)


TINY2 = dataclasses.replace(synth.SHAPE_TINY, vocab=512)


def test_sampled_forecast_at_vanishing_temperature_is_the_greedy_forecast():
    W = oracle.Weights(TINY2)
    ids = synth.uniform_int(1, 60, 20, 0, TINY2.vocab - 1)
    g = oracle.forecast_one(W, ids, 5, (10, 11), 0.8)
    s = smp.forecast_sampled_one(W, ids, 5, (10, 11), 0.8, seed=9, row=2, temperature=1e-9)
    np.testing.assert_array_equal(g["tokens"], s["tokens"])
    np.testing.assert_array_equal(g["step_logits"], s["step_logits"])


def test_sampled_forecast_rows_and_seeds():
    W = oracle.Weights(TINY2)
    ids = synth.uniform_int(1, 61, 20, 0, TINY2.vocab - 1)
    a = smp.forecast_sampled_one(W, ids, 6, (10, 11), 0.8, seed=9, row=0, temperature=1.0)
    a2 = smp.forecast_sampled_one(W, ids, 6, (10, 11), 0.8, seed=9, row=0, temperature=1.0)
    b = smp.forecast_sampled_one(W, ids, 6, (10, 11), 0.8, seed=9, row=1, temperature=1.0)
    c = smp.forecast_sampled_one(W, ids, 6, (10, 11), 0.8, seed=10, row=0, temperature=1.0)
    np.testing.assert_array_equal(a["tokens"], a2["tokens"])
    assert not np.array_equal(a["tokens"], b["tokens"])
    assert not np.array_equal(a["tokens"], c["tokens"])
    # the prompt's logits do not depend on the draw
    np.testing.assert_array_equal(a["step_logits"][0], b["step_logits"][0])
    # teacher forcing with the row's own tokens reproduces it
    f = smp.forecast_sampled_one(W, ids, 6, (10, 11), 0.8, seed=0, row=7, temperature=1.0, forced_tokens=a["tokens"])
    np.testing.assert_array_equal(f["step_logits"], a["step_logits"])


def _frequency_pin_holds():
    try:
        for T in (1.0, 0.5, 2.0):
            test_gumbel_max_draws_follow_the_tempered_softmax(T)
    except AssertionError:
        return False
    return True


@pytest.mark.parametrize("name,bad", [
    ("gumbel", lambda u: np.log(-np.log(np.asarray(u, dtype=np.float64)))),         # sign flipped
    ("gumbel", lambda u: -np.log(np.asarray(u, dtype=np.float64))),                 # one log only
    ("sample", lambda l, T, u: int(np.argmax(np.asarray(l) * T + smp.gumbel(u)))),  # T multiplies
    ("sample", lambda l, T, u: int(np.argmax(np.asarray(l) + smp.gumbel(u)))),      # T dropped
])
def test_planted_sampling_mistakes_are_caught(monkeypatch, name, bad):
    assert _frequency_pin_holds()
    monkeypatch.setattr(smp, name, bad)
    assert not _frequency_pin_holds()
