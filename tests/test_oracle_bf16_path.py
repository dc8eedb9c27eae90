"""Pins of oracle/bf16_path.py, the precision model the full-depth parity tests are held to.

- Its rounding equals torch's float32 -> bfloat16 conversion (round to nearest even), ties included.
- With the rounding switched off it computes the float64 oracle's prompt logits (the folded RMS scale
  equals the normalised product in exact arithmetic), so its layer order, RoPE, attention and SwiGLU
  are the oracle's.
- Each rounding point it names does move the result, and the whole stays within a few percent of the
  oracle on a small model.
"""
import numpy as np
import pytest

import oracle
import synth
from oracle import bf16_path

torch = pytest.importorskip("torch")

SMALL = synth.ModelShape(layers=2, d_model=64, n_q=4, n_kv=2, head_dim=64, ffn=96, vocab=256, rope_theta=1e4)


def test_rounding_matches_torch_bfloat16():
    rng = np.random.default_rng(3)
    x = np.concatenate([rng.standard_normal(20000) * 10.0 ** rng.integers(-6, 6, 20000),
                        [0.0, -0.0, 1.0, 1.00390625, 1.01171875, -1.01171875, 3.0e38]])
    # values exactly half-way between two bf16 numbers (ties to even)
    ties = (np.arange(1, 200, dtype=np.uint32) << 16 | 0x8000).view(np.float32).astype(np.float64)
    x = np.concatenate([x, ties, -ties])
    want = torch.from_numpy(x.astype(np.float32)).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(bf16_path.bf16_round(x), want)


def test_without_rounding_it_is_the_oracle():
    W = oracle.Weights(SMALL)
    ids = synth.uniform_int(7, 1, 40, 0, SMALL.vocab - 1)
    ref = oracle.prefill(W, ids)[0]
    got = bf16_path.prompt_logits_bf16(W, ids, rnd=bf16_path.identity_rounding())
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-12)


def test_rounding_moves_the_logits_by_a_bf16_sized_amount():
    W = oracle.Weights(SMALL)
    ids = synth.uniform_int(7, 2, 40, 0, SMALL.vocab - 1)
    ref = oracle.prefill(W, ids)[0]
    got = bf16_path.prompt_logits_bf16(W, ids)
    rel = np.sqrt(np.mean((got - ref) ** 2)) / np.sqrt(np.mean(ref ** 2))
    assert 1e-4 < rel < 3e-2
