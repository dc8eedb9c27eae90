"""The forward pass with every tensor a bf16 data path stores rounded to bf16: a precision model.

TEST INFRASTRUCTURE ONLY (imported by ``tests/`` and by the script that writes
``tests/golden/bf16_drift.json``).  It shares no code with the CUDA path.

The float64 oracle (``model.py``) is the definition of what the surrogate
computes.  A bf16 implementation cannot match it exactly: its matmul operands
must be bf16 like the weights, and its KV cache holds bf16.  This module
computes the same prompt forward pass in float64 but rounds to bf16 (round to
nearest even) at those points, so that the distance between the two tells how
far an implementation that rounds there, and nowhere else, drifts from the
definition after many layers:

* the input of every matmul with a weight matrix: the residual times the norm
  gain before the QKV and gate/up products (the RMS scale 1/sqrt(mean(x^2)+eps)
  is applied to the product's rows, which is the same number in exact
  arithmetic), the attention output before the output projection, the SwiGLU
  product before the down projection, and the final normalised hidden state
  before the LM head;
* the rotated queries and keys and the values (what the KV cache holds);
* the softmax numerators exp(s - max) that multiply the values; their sum
  stays unrounded.

The layer order, RoPE, attention, SwiGLU and the readings of the paper are
those of ``model.py`` (Sec. 2.1 and the workload shapes); this module reuses
its step functions.
"""
from __future__ import annotations

import math

import numpy as np

from .model import Weights, rope, silu


def bf16_round(x: np.ndarray) -> np.ndarray:
    """Round to the nearest bf16 value (ties to even), returned as float64.

    x is first rounded to float32 (as any fp32 accumulator holding it would be), then its 32-bit
    pattern is rounded to the upper 16 bits.
    """
    x32 = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    u = x32.view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16) << 16
    return r.astype(np.uint32).view(np.float32).astype(np.float64)


def _identity(x):
    return np.asarray(x, dtype=np.float64)


def layer_forward_bf16(x: np.ndarray, lw: dict, shape, positions: np.ndarray, rnd=bf16_round) -> np.ndarray:
    """One layer over the prompt tokens x ([T, d]) with the rounding points above (rnd: the rounding)."""
    t = x.shape[0]
    hd = shape.head_dim
    rs = 1.0 / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + shape.rms_eps)
    xn = rnd(x * lw["attn_norm"])
    q = rnd(rope(((xn @ lw["wq"].T) * rs).reshape(t, shape.n_q, hd), positions, shape.rope_theta))
    k = rnd(rope(((xn @ lw["wk"].T) * rs).reshape(t, shape.n_kv, hd), positions, shape.rope_theta))
    v = rnd(((xn @ lw["wv"].T) * rs).reshape(t, shape.n_kv, hd))
    group = shape.n_q // shape.n_kv
    allowed = positions[None, :] <= positions[:, None]
    a = np.empty((t, shape.n_q, hd))
    for h in range(shape.n_q):
        s = (q[:, h, :] @ k[:, h // group, :].T) / math.sqrt(hd)
        s = np.where(allowed, s, -np.inf)
        p = np.exp(s - np.max(s, axis=-1, keepdims=True))
        a[:, h, :] = (rnd(p) @ v[:, h // group, :]) / np.sum(p, axis=-1, keepdims=True)
    x = x + rnd(a.reshape(t, shape.n_q * hd)) @ lw["wo"].T
    rs = 1.0 / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + shape.rms_eps)
    xn = rnd(x * lw["ffn_norm"])
    act = rnd(silu((xn @ lw["w_gate"].T) * rs) * ((xn @ lw["w_up"].T) * rs))
    return x + act @ lw["w_down"].T


def prompt_logits_bf16(weights: Weights, ids: np.ndarray, rnd=bf16_round) -> np.ndarray:
    """Logits of the last prompt position ([V]) with the rounding points above."""
    m = weights.shape
    ids = np.asarray(ids, dtype=np.int64)
    x = weights.embed_rows(ids)
    pos = np.arange(len(ids))
    for l in range(m.layers):
        x = layer_forward_bf16(x, weights.layer(l), m, pos, rnd)
    last = x[-1:]
    h = rnd(last / np.sqrt(np.mean(last * last, axis=-1, keepdims=True) + m.rms_eps) * weights.final_norm())
    return (h @ weights.head().T)[0]


def identity_rounding():
    """The rounding hook that rounds nothing (this module then computes the float64 oracle's numbers)."""
    return _identity
