"""Algebraic properties of the oracle's steps, on seeded random inputs.

Each property holds exactly in real arithmetic, so the float64 oracle must
satisfy it to rounding; each one fails for a plausible slip in a step
(a missing max-shift, a scale-dependent norm, a rotation that does not
compose, a mask that depends on key order, a restricted softmax that is not
renormalised).
"""
import numpy as np
import pytest

import oracle
from oracle import model as om

SEEDS = range(6)


def rng(seed):
    return np.random.default_rng(1000 + seed)


@pytest.mark.parametrize("seed", SEEDS)
def test_softmax_is_shift_invariant_and_normalised(seed):
    r = rng(seed)
    s = r.normal(0, 5, size=(7, 33))
    c = r.normal(0, 100, size=(7, 1))
    p = oracle.softmax(s)
    np.testing.assert_allclose(oracle.softmax(s + c), p, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(p.sum(-1), 1.0, rtol=0, atol=1e-12)
    # large logits do not overflow (max-shifted)
    assert np.isfinite(oracle.softmax(s * 1e3)).all()


@pytest.mark.parametrize("seed", SEEDS)
def test_rms_norm_is_scale_invariant(seed):
    r = rng(seed)
    x = r.normal(0, 1, size=(5, 64))
    g = r.normal(1, 0.1, size=64)
    c = np.exp(r.normal(0, 2))
    np.testing.assert_allclose(oracle.rms_norm(c * x, g, 0.0), oracle.rms_norm(x, g, 0.0), rtol=1e-12, atol=1e-12)
    # with the gain divided out, every row has mean square 1
    y = oracle.rms_norm(x, np.ones(64), 0.0)
    np.testing.assert_allclose((y * y).mean(-1), 1.0, rtol=1e-12)


@pytest.mark.parametrize("seed", SEEDS)
@pytest.mark.parametrize("hd,theta", [(64, 1e4), (128, 1e6)])
def test_rope_rotations_compose_and_invert(seed, hd, theta):
    r = rng(seed)
    x = r.normal(0, 1, size=(4, 3, hd))
    m = r.integers(0, 20000, size=4)
    n = r.integers(0, 20000, size=4)
    mn = oracle.rope(oracle.rope(x, m, theta), n, theta)
    np.testing.assert_allclose(mn, oracle.rope(x, m + n, theta), rtol=1e-9, atol=1e-9)
    back = oracle.rope(oracle.rope(x, m, theta), -m, theta)
    np.testing.assert_allclose(back, x, rtol=1e-9, atol=1e-9)


@pytest.mark.parametrize("seed", SEEDS)
def test_attention_of_the_last_query_ignores_key_order(seed):
    r = rng(seed)
    T, nq, nkv, hd = 9, 4, 2, 16
    q = r.normal(0, 1, size=(1, nq, hd))
    k = r.normal(0, 1, size=(T, nkv, hd))
    v = r.normal(0, 1, size=(T, nkv, hd))
    pos = np.arange(T)
    out = oracle.attention(q, k, v, np.array([T - 1]), pos)
    perm = r.permutation(T)
    out_p = oracle.attention(q, k[perm], v[perm], np.array([T - 1]), pos[perm])
    np.testing.assert_allclose(out_p, out, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("seed", SEEDS)
def test_attention_is_a_convex_combination_of_visible_values(seed):
    r = rng(seed)
    T, hd = 11, 8
    q = r.normal(0, 3, size=(T, 1, hd))
    k = r.normal(0, 3, size=(T, 1, hd))
    v = r.normal(0, 1, size=(T, 1, hd))
    pos = np.arange(T)
    out = oracle.attention(q, k, v, pos, pos)
    for t in range(T):
        lo = v[:t + 1, 0].min(axis=0) - 1e-12
        hi = v[:t + 1, 0].max(axis=0) + 1e-12
        assert ((out[t, 0] >= lo) & (out[t, 0] <= hi)).all(), t


@pytest.mark.parametrize("seed", SEEDS)
def test_feed_forward_is_linear_in_the_down_projection(seed):
    r = rng(seed)
    h = r.normal(0, 1, size=(3, 32))
    wg, wu = r.normal(0, 0.2, size=(48, 32)), r.normal(0, 0.2, size=(48, 32))
    wd1, wd2 = r.normal(0, 0.2, size=(32, 48)), r.normal(0, 0.2, size=(32, 48))
    a = oracle.swiglu_ffn(h, wg, wu, wd1 + 2.0 * wd2)
    b = oracle.swiglu_ffn(h, wg, wu, wd1) + 2.0 * oracle.swiglu_ffn(h, wg, wu, wd2)
    np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-12)
    # silu(z) = z * sigmoid(z) and silu(-z) = silu(z) - z
    z = r.normal(0, 4, size=50)
    np.testing.assert_allclose(oracle.silu(-z), oracle.silu(z) - z, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("seed", SEEDS)
def test_verdict_depends_only_on_the_verdict_logits_up_to_a_shift(seed):
    r = rng(seed)
    V = 64
    logits = r.normal(0, 2, size=(5, V))
    ids = [10, 11, 40, 3]
    p, conf, arg, defer = oracle.verdict(logits, ids, 0.6)
    # a common shift, and any change to the other tokens, leave the verdict unchanged
    other = logits + 7.5
    mask = np.ones(V, bool)
    mask[ids] = False
    other[:, mask] = r.normal(0, 50, size=(5, int(mask.sum())))
    p2, conf2, arg2, defer2 = oracle.verdict(other, ids, 0.6)
    np.testing.assert_allclose(p2, p, rtol=1e-12, atol=1e-15)
    assert (arg2 == arg).all() and (defer2 == defer).all()
    # permuting the verdict ids permutes p
    order = [2, 0, 3, 1]
    p3, _, _, _ = oracle.verdict(logits, [ids[i] for i in order], 0.6)
    np.testing.assert_allclose(p3, p[:, order], rtol=1e-12, atol=1e-15)
    # p is the full softmax renormalised on the verdict ids
    full = oracle.softmax(logits)[:, ids]
    np.testing.assert_allclose(p, full / full.sum(-1, keepdims=True), rtol=1e-12)
