"""Pins for the oracle: brute force on tiny inputs, invariants, closed forms.

Each check ties the oracle to something other than itself: an independent
pure-Python loop computation on tiny inputs, an invariant the mathematics
fixes (causality, cache equivalence, permutation, rotation), or a closed form
of the verdict (Sec. 2.1).  ``test_planted_mistakes_are_caught`` plants
plausible mistakes into the oracle and checks that some pin fails for each.
"""
import dataclasses
import math
import struct

import numpy as np
import pytest

import oracle
import oracle.model as om
import synth

MICRO = synth.ModelShape(layers=2, d_model=8, n_q=4, n_kv=2, head_dim=4, ffn=6, vocab=16, rope_theta=10.0,
                         rms_eps=1e-6, sigma=0.3, head_sigma=0.3)


# ----------------------------------------------------------------------------
# an independent, loop-only transformer for tiny shapes
# ----------------------------------------------------------------------------

def _bf16(bits):
    return struct.unpack("<f", struct.pack("<I", int(bits) << 16))[0]


def _mat(bits2d):
    return [[_bf16(b) for b in row] for row in np.asarray(bits2d)]


def _matvec(w, x):  # w: rows of output features
    return [sum(w[o][i] * x[i] for i in range(len(x))) for o in range(len(w))]


def brute_force_logits(shape, seed, ids):
    """Logits of every position, computed with Python loops and the math module."""
    d, hd, nq, nkv = shape.d_model, shape.head_dim, shape.n_q, shape.n_kv
    emb = _mat(synth.embed_bf16(shape, seed))
    head = _mat(synth.head_bf16(shape, seed))
    xs = [list(emb[t]) for t in ids]
    T = len(ids)

    def norm(v):
        r = 1.0 / math.sqrt(sum(a * a for a in v) / len(v) + shape.rms_eps)
        return [a * r for a in v]

    def rot(vec, p):
        out = list(vec)
        half = hd // 2
        for i in range(half):
            ang = p * shape.rope_theta ** (-2.0 * i / hd)
            a, b = vec[i], vec[i + half]
            out[i] = a * math.cos(ang) - b * math.sin(ang)
            out[i + half] = b * math.cos(ang) + a * math.sin(ang)
        return out

    for l in range(shape.layers):
        lw = {k: _mat(v) for k, v in synth.layer_weights_bf16(shape, l, seed).items()}
        hs = [norm(x) for x in xs]
        qs = [_matvec(lw["wq"], h) for h in hs]
        ks = [_matvec(lw["wk"], h) for h in hs]
        vs = [_matvec(lw["wv"], h) for h in hs]
        new = []
        for t in range(T):
            att = []
            for h in range(nq):
                g = h * nkv // nq
                qh = rot(qs[t][h * hd:(h + 1) * hd], t)
                scores = []
                for u in range(t + 1):
                    kh = rot(ks[u][g * hd:(g + 1) * hd], u)
                    scores.append(sum(qh[i] * kh[i] for i in range(hd)) / math.sqrt(hd))
                mx = max(scores)
                e = [math.exp(s - mx) for s in scores]
                z = sum(e)
                for i in range(hd):
                    att.append(sum(e[u] / z * vs[u][g * hd + i] for u in range(t + 1)))
            o = _matvec(lw["wo"], att)
            x1 = [xs[t][i] + o[i] for i in range(d)]
            h2 = norm(x1)
            gt = _matvec(lw["w_gate"], h2)
            up = _matvec(lw["w_up"], h2)
            act = [gt[j] / (1.0 + math.exp(-gt[j])) * up[j] for j in range(len(gt))]
            dn = _matvec(lw["w_down"], act)
            new.append([x1[i] + dn[i] for i in range(d)])
        xs = new
    return np.array([_matvec(head, norm(x)) for x in xs])


def _micro_ids(n=6, seed=4):
    return synth.uniform_int(seed, 0, n, 0, MICRO.vocab - 1)


def test_whole_model_matches_brute_force():
    ids = _micro_ids()
    W = oracle.Weights(MICRO, seed=5)
    got, _ = oracle.prefill(W, ids, all_logits=True)
    ref = brute_force_logits(MICRO, 5, ids)
    np.testing.assert_allclose(got, ref, rtol=0, atol=1e-11)


# ----------------------------------------------------------------------------
# attention
# ----------------------------------------------------------------------------

def _rand(shape, seed):
    return synth.normal_f32(seed, 1, int(np.prod(shape)), 1.0).astype(np.float64).reshape(shape)


def test_attention_brute_force_tiny():
    T, nq, nkv, hd = 7, 2, 1, 4
    q, k, v = _rand((T, nq, hd), 1), _rand((T, nkv, hd), 2), _rand((T, nkv, hd), 3)
    got = oracle.attention(q, k, v, np.arange(T), np.arange(T))
    for t in range(T):
        for h in range(nq):
            s = [sum(q[t, h, i] * k[u, 0, i] for i in range(hd)) / 2.0 for u in range(t + 1)]
            e = [math.exp(x) for x in s]
            for i in range(hd):
                ref = sum(e[u] * v[u, 0, i] for u in range(t + 1)) / sum(e)
                assert abs(got[t, h, i] - ref) < 1e-12


def test_attention_single_key_returns_its_value():
    q, k, v = _rand((1, 3, 8), 4), _rand((1, 3, 8), 5), _rand((1, 3, 8), 6)
    np.testing.assert_array_equal(oracle.attention(q, k, v, np.array([0]), np.array([0])), v)


def test_attention_uniform_scores_give_prefix_mean():
    T = 6
    q = np.zeros((T, 2, 4))
    k, v = _rand((T, 1, 4), 7), _rand((T, 1, 4), 8)
    got = oracle.attention(q, k, v, np.arange(T), np.arange(T))
    for t in range(T):
        np.testing.assert_allclose(got[t, 0], v[:t + 1, 0].mean(axis=0), atol=1e-14)


def test_gqa_equals_mha_with_duplicated_kv_heads():
    T, nq, nkv, hd = 5, 6, 2, 4
    q, k, v = _rand((T, nq, hd), 9), _rand((T, nkv, hd), 10), _rand((T, nkv, hd), 11)
    grp = nq // nkv
    k_rep = np.repeat(k, grp, axis=1)
    v_rep = np.repeat(v, grp, axis=1)
    a = oracle.attention(q, k, v, np.arange(T), np.arange(T))
    b = oracle.attention(q, k_rep, v_rep, np.arange(T), np.arange(T))
    np.testing.assert_allclose(a, b, atol=1e-15)


# ----------------------------------------------------------------------------
# RMSNorm, RoPE, SwiGLU, softmax
# ----------------------------------------------------------------------------

def test_rmsnorm_constant_vector_and_unit_mean_square():
    g = np.ones(16)
    for c in (3.0, -0.5):
        out = oracle.rms_norm(np.full(16, c), g, 0.0)
        np.testing.assert_allclose(out, np.sign(c), atol=1e-15)
    x = _rand((4, 64), 12)
    y = oracle.rms_norm(x, np.ones(64), 0.0)
    np.testing.assert_allclose(np.mean(y * y, axis=-1), 1.0, atol=1e-14)
    gains = _rand((64,), 13)
    np.testing.assert_allclose(oracle.rms_norm(x, gains, 0.0), y * gains, atol=1e-14)


def test_rope_identity_at_zero_norm_preserving_and_relative():
    hd, theta = 16, 1e4
    x = _rand((1, 1, hd), 14)
    np.testing.assert_array_equal(oracle.rope(x, np.array([0]), theta), x)
    y = oracle.rope(x, np.array([37]), theta)
    half = hd // 2
    for i in range(half):
        n0 = x[0, 0, i] ** 2 + x[0, 0, i + half] ** 2
        n1 = y[0, 0, i] ** 2 + y[0, 0, i + half] ** 2
        assert abs(n0 - n1) < 1e-13
    q, k = _rand((1, 1, hd), 15), _rand((1, 1, hd), 16)
    dots = []
    for m, n in [(5, 2), (103, 100), (3, 0), (1003, 1000)]:
        a = oracle.rope(q, np.array([m]), theta)[0, 0]
        b = oracle.rope(k, np.array([n]), theta)[0, 0]
        dots.append(float(a @ b))
    np.testing.assert_allclose(dots, dots[0], atol=1e-11)


def test_rope_first_pair_turns_by_position_radians():
    # pair 0 has inverse frequency theta^0 = 1, so position p turns it by p radians
    x = np.zeros((1, 1, 4))
    x[0, 0, 0] = 1.0
    y = oracle.rope(x, np.array([1]), 1e4)[0, 0]
    assert abs(y[0] - math.cos(1.0)) < 1e-15 and abs(y[2] - math.sin(1.0)) < 1e-15


def test_swiglu_zero_gate_and_silu_values():
    assert oracle.silu(np.array([0.0]))[0] == 0.0
    assert abs(oracle.silu(np.array([40.0]))[0] - 40.0) < 1e-12
    h = _rand((3, 8), 17)
    out = oracle.swiglu_ffn(h, np.zeros((5, 8)), _rand((5, 8), 18), _rand((8, 5), 19))
    np.testing.assert_array_equal(out, 0.0)


def test_softmax_rows_sum_to_one():
    s = _rand((50, 33), 20) * 30
    np.testing.assert_allclose(oracle.softmax(s).sum(axis=-1), 1.0, atol=1e-12)


# ----------------------------------------------------------------------------
# verdict (Sec. 2.1): closed forms
# ----------------------------------------------------------------------------

def test_verdict_equal_logits():
    logits = np.zeros((3, 20))
    for k in (2, 8):
        p, conf, arg, defer = oracle.verdict(logits, list(range(k)), 0.5 + 1e-9 if k == 2 else 0.2)
        np.testing.assert_allclose(p, 1.0 / k, atol=1e-15)
        np.testing.assert_allclose(conf, 1.0 / k, atol=1e-15)
        assert np.all(arg == 0)  # ties resolve to the lowest index
        assert np.all(defer == 1)
    # a confidence exactly at the threshold is accepted: defer only when q < tau
    assert oracle.verdict(np.zeros((1, 4)), [0, 1], 0.5)[3][0] == 0


def test_verdict_ln4_gap_gives_confidence_point_eight():
    logits = np.zeros((1, 16))
    logits[0, 11] = math.log(4.0)
    p, conf, arg, defer = oracle.verdict(logits, [10, 11], 0.8)
    np.testing.assert_allclose(p[0], [0.2, 0.8], atol=1e-15)
    assert arg[0] == 1
    assert oracle.verdict(logits, [10, 11], 0.8 + 1e-9)[3][0] == 1
    assert oracle.verdict(logits, [10, 11], 0.8 - 1e-9)[3][0] == 0
    np.testing.assert_allclose(p.sum(), 1.0, atol=1e-15)


def test_greedy_lowest_id_on_ties():
    x = np.array([[0.0, 2.0, 1.0, 2.0]])
    assert oracle.greedy(x)[0] == 1


# ----------------------------------------------------------------------------
# whole-model invariants
# ----------------------------------------------------------------------------

TINY2 = dataclasses.replace(synth.SHAPE_TINY, vocab=512)


def test_causal_prefix_invariance_bit_identical():
    W = oracle.Weights(TINY2)
    ids = synth.uniform_int(1, 50, 40, 0, TINY2.vocab - 1)
    full, _ = oracle.prefill(W, ids, all_logits=True)
    part, _ = oracle.prefill(W, ids[:23], all_logits=True)
    np.testing.assert_allclose(full[:23], part, rtol=0, atol=1e-12)


def test_kv_cache_decode_equals_full_recompute():
    W = oracle.Weights(TINY2)
    ids = synth.uniform_int(1, 51, 30, 0, TINY2.vocab - 1)
    logits, st = oracle.prefill(W, ids[:20])
    for t in range(20, 30):
        logits = oracle.decode_step(W, st, int(ids[t]))
        ref = oracle.full_recompute_logits(W, ids[:t + 1])
        np.testing.assert_allclose(logits, ref, rtol=0, atol=1e-10)


def test_batch_permutation_invariance():
    W = oracle.Weights(TINY2)
    w = synth.workload("tiny", model=TINY2, batch=3, prompt_len=24, inc_len=8, n_decode=3)
    ids, off = synth.packed_prompts(w)
    a = oracle.forecast_batch(W, ids, off, 3, (10, 11), 0.8)
    perm = [2, 0, 1]
    ids_p = np.concatenate([ids[off[i]:off[i + 1]] for i in perm])
    off_p = np.concatenate([[0], np.cumsum([off[i + 1] - off[i] for i in perm])])
    b = oracle.forecast_batch(W, ids_p, off_p, 3, (10, 11), 0.8)
    for j, i in enumerate(perm):
        np.testing.assert_array_equal(a[i]["step_logits"], b[j]["step_logits"])
        assert a[i]["defer"] == b[j]["defer"]


def test_layer_rows_equals_layer_forward_rows():
    W = oracle.Weights(TINY2)
    x = _rand((33, TINY2.d_model), 21)
    full, _, _ = oracle.layer_forward(x, W.layer(1), TINY2, np.arange(33))
    rows = [0, 7, 20, 32]
    np.testing.assert_allclose(oracle.layer_rows(x, W.layer(1), TINY2, rows), full[rows], atol=1e-12)


def test_teacher_forcing_replays_own_tokens():
    W = oracle.Weights(TINY2)
    ids = synth.uniform_int(1, 52, 16, 0, TINY2.vocab - 1)
    a = oracle.forecast_one(W, ids, 4, (10, 11), 0.8)
    b = oracle.forecast_one(W, ids, 4, (10, 11), 0.8, forced_tokens=a["tokens"])
    np.testing.assert_array_equal(a["step_logits"], b["step_logits"])


# ----------------------------------------------------------------------------
# planted mistakes: each must make at least one pin fail
# ----------------------------------------------------------------------------

def _pins():
    return [test_whole_model_matches_brute_force, test_attention_brute_force_tiny,
            test_attention_single_key_returns_its_value, test_attention_uniform_scores_give_prefix_mean,
            test_gqa_equals_mha_with_duplicated_kv_heads, test_rmsnorm_constant_vector_and_unit_mean_square,
            test_rope_identity_at_zero_norm_preserving_and_relative, test_rope_first_pair_turns_by_position_radians,
            test_swiglu_zero_gate_and_silu_values, test_verdict_equal_logits,
            test_verdict_ln4_gap_gives_confidence_point_eight, test_causal_prefix_invariance_bit_identical,
            test_kv_cache_decode_equals_full_recompute]


def _bad_rope_sign(x, positions, theta):
    hd = x.shape[-1]
    half = hd // 2
    inv = theta ** (-(2.0 * np.arange(half)) / hd)
    ang = np.asarray(positions, dtype=np.float64)[:, None] * inv[None, :]
    c, s = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c + x2 * s, x2 * c - x1 * s], axis=-1)


def _bad_attention_mask(q, k, v, q_pos, k_pos):  # strict inequality: drops the diagonal
    return _orig_attention(q, k, v, np.asarray(q_pos) - 1, k_pos) if len(k_pos) > 1 else v * 0


def _bad_gqa(q, k, v, q_pos, k_pos):  # kv-head chosen as h % n_kv
    tq, n_q, hd = q.shape
    n_kv = k.shape[1]
    order = [h % n_kv for h in range(n_q)]
    k2 = k[:, order, :]
    v2 = v[:, order, :]
    return _orig_attention(q, k2, v2, q_pos, k_pos)


def _bad_norm(x, g, eps):  # mean instead of mean square
    return x / np.sqrt(np.abs(np.mean(x, axis=-1, keepdims=True)) + eps) * g


def _bad_ffn(h, wg, wu, wd):  # gate and up swapped
    return (oracle.silu(h @ wu.T) * (h @ wg.T)) @ wd.T


def _bad_post(x, a, lw, shape):  # residual dropped around the feed-forward block
    t = x.shape[0]
    x = x + a.reshape(t, shape.n_q * shape.head_dim) @ lw["wo"].T
    h = om.rms_norm(x, lw["ffn_norm"], shape.rms_eps)
    return om.swiglu_ffn(h, lw["w_gate"], lw["w_up"], lw["w_down"])


def _bad_verdict(logits, ids, tau):
    p, conf, arg, defer = _orig_verdict(logits, ids, tau)
    return p, conf, arg, (conf <= tau).astype(np.uint8)


_orig_attention = om.attention
_orig_verdict = om.verdict


@pytest.mark.parametrize("target,bad", [
    ("rope", _bad_rope_sign), ("attention", _bad_attention_mask), ("attention", _bad_gqa),
    ("rms_norm", _bad_norm), ("swiglu_ffn", _bad_ffn), ("attn_out_and_ffn", _bad_post),
    ("verdict", _bad_verdict),
])
def test_planted_mistakes_are_caught(monkeypatch, target, bad):
    monkeypatch.setattr(om, target, bad)
    monkeypatch.setattr(oracle, target, bad)
    failed = 0
    for pin in _pins():
        try:
            with np.errstate(invalid="ignore"):  # a planted mask can leave a row with no key (NaN)
                pin()
        except (AssertionError, FloatingPointError, ValueError, IndexError):
            failed += 1
    assert failed >= 1, f"no pin caught the planted mistake in {target}"
