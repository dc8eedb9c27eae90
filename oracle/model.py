"""CPU oracle for the surrogate forecaster's forward pass and selective deferral.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s CPU-baseline / reference arm may import this module.  It shares
no code with the CUDA path; its only shared dependency is the seeded input
generator ``synth`` (which draws numbers and holds none of the method).

Everything is plain numpy in float64.  Weights are the bf16 values drawn by
``synth``, widened exactly to float64.  A library matmul is the only
primitive used for contractions; there is no blocking, fusion or reordering.

What is computed (the surrogate of Sec. 2.1: a language model reads
x_i = (r, k_i, h) as tokens, reasons for a few tokens, then emits a
distribution p_i over verdicts; q_i = max_b p_{i,b} is its confidence and a
forecast is accepted only when q_i clears a threshold):

* the language model is a pre-norm decoder-only transformer (the paper uses an
  off-the-shelf LLM and does not describe its layers, Sec. 2.2 / App. C; the
  layer structure below is the standard one its workload shapes name):
  token embedding; per layer RMSNorm -> q,k,v projections -> rotary position
  embedding on q and k -> causal grouped-query attention -> output projection
  added to the residual -> RMSNorm -> SwiGLU feed-forward added to the
  residual; final RMSNorm -> LM head.
* greedy decoding: the next token is the arg max of the logits (lowest id on
  ties), fed back for ``n_decode`` steps ("generate a brief chain of
  reasoning", Sec. 2.1).
* verdict (Sec. 2.1, the unnumbered display defining p_i, y_hat_i and q_i):
  p = softmax of the final logits restricted to the K verdict token ids,
  y_hat = arg max p (lowest index on ties), q = max p, and the candidate is
  deferred to real GPU measurement when q < tau (forecasts are accepted with
  q "above a confidence threshold", Sec. 2.1, Selective Use).

Readings where the paper is silent:
* the verdict is read from the logits produced by the last decode step (the
  logits that would choose decode token n_decode+1); with n_decode = 0 from
  the last prompt position;
* RoPE is the rotate-half form, pairs (i, i + hd/2), inverse frequency
  theta^(-2i/hd), positions from 0;
* attention scale 1/sqrt(hd); q-head h reads kv-head h // (n_q / n_kv);
* no biases, untied LM head, RMSNorm gains from the weights (1 here).
"""
from __future__ import annotations

import math

import numpy as np

import synth


# ----------------------------------------------------------------------------
# weights
# ----------------------------------------------------------------------------

def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float64."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


class Weights:
    """The model's weights in float64, drawn layer by layer from ``synth``.

    ``cache_layers`` keeps every layer resident (small models); otherwise a
    layer is regenerated when asked for, so 7B/14B shapes fit in host memory.
    """

    def __init__(self, shape: synth.ModelShape, seed: int = 0, cache_layers: bool = True):
        self.shape = shape
        self.seed = seed
        self.cache_layers = cache_layers
        self._layers = {}
        self._embed = None
        self._head = None

    def layer(self, l: int) -> dict:
        if l in self._layers:
            return self._layers[l]
        m = self.shape
        raw = synth.layer_weights_bf16(m, l, self.seed)
        lw = {k: bf16_bits_to_f64(v) for k, v in raw.items()}
        lw["attn_norm"] = bf16_bits_to_f64(synth.ones_bf16(m.d_model))
        lw["ffn_norm"] = bf16_bits_to_f64(synth.ones_bf16(m.d_model))
        if self.cache_layers:
            self._layers[l] = lw
        return lw

    def embed_rows(self, ids: np.ndarray) -> np.ndarray:
        if self._embed is None:
            self._embed = synth.embed_bf16(self.shape, self.seed)  # bf16 bits, widened per row
        return bf16_bits_to_f64(self._embed[np.asarray(ids, dtype=np.int64)])

    def head(self) -> np.ndarray:
        if self._head is None:
            self._head = bf16_bits_to_f64(synth.head_bf16(self.shape, self.seed))
        return self._head

    def final_norm(self) -> np.ndarray:
        return bf16_bits_to_f64(synth.ones_bf16(self.shape.d_model))


# ----------------------------------------------------------------------------
# the layer's steps, one function each
# ----------------------------------------------------------------------------

def rms_norm(x: np.ndarray, g: np.ndarray, eps: float) -> np.ndarray:
    """RMSNorm over the last axis: x / sqrt(mean(x^2) + eps) * g."""
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * g


def rope(x: np.ndarray, positions: np.ndarray, theta: float) -> np.ndarray:
    """Rotary position embedding, rotate-half form.

    x: [T, H, hd]; element pairs (i, i + hd/2) of the token at position p are
    rotated by the angle p * theta^(-2i/hd).
    """
    hd = x.shape[-1]
    half = hd // 2
    inv_freq = theta ** (-(2.0 * np.arange(half, dtype=np.float64)) / hd)
    ang = np.asarray(positions, dtype=np.float64)[:, None] * inv_freq[None, :]  # [T, half]
    cos = np.cos(ang)[:, None, :]
    sin = np.sin(ang)[:, None, :]
    x1 = x[..., :half]
    x2 = x[..., half:]
    return np.concatenate([x1 * cos - x2 * sin, x2 * cos + x1 * sin], axis=-1)


def softmax(s: np.ndarray, axis: int = -1) -> np.ndarray:
    """Max-subtracted softmax."""
    m = np.max(s, axis=axis, keepdims=True)
    e = np.exp(s - m)
    return e / np.sum(e, axis=axis, keepdims=True)


def attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, q_pos: np.ndarray, k_pos: np.ndarray) -> np.ndarray:
    """Causal grouped-query attention with an explicit score matrix.

    q: [Tq, n_q, hd]; k, v: [Tk, n_kv, hd].  Query at position p sees keys at
    positions <= p.  q-head h uses kv-head h // (n_q // n_kv).
    Returns [Tq, n_q, hd].
    """
    tq, n_q, hd = q.shape
    n_kv = k.shape[1]
    group = n_q // n_kv
    out = np.empty_like(q)
    allowed = np.asarray(k_pos)[None, :] <= np.asarray(q_pos)[:, None]  # [Tq, Tk]
    scale = 1.0 / math.sqrt(hd)
    for h in range(n_q):
        g = h // group
        s = (q[:, h, :] @ k[:, g, :].T) * scale
        s = np.where(allowed, s, -np.inf)
        out[:, h, :] = softmax(s, axis=-1) @ v[:, g, :]
    return out


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


def swiglu_ffn(h: np.ndarray, w_gate: np.ndarray, w_up: np.ndarray, w_down: np.ndarray) -> np.ndarray:
    """(silu(h W_gate^T) * (h W_up^T)) W_down^T."""
    return (silu(h @ w_gate.T) * (h @ w_up.T)) @ w_down.T


def q_proj(x: np.ndarray, lw: dict, shape: synth.ModelShape, positions: np.ndarray) -> np.ndarray:
    """Queries of the tokens x at `positions`: RMSNorm, W_q, RoPE.  [T, n_q, hd]"""
    h = rms_norm(x, lw["attn_norm"], shape.rms_eps)
    q = (h @ lw["wq"].T).reshape(x.shape[0], shape.n_q, shape.head_dim)
    return rope(q, positions, shape.rope_theta)


def kv_proj(x: np.ndarray, lw: dict, shape: synth.ModelShape, positions: np.ndarray):
    """Keys (rotated) and values of the tokens x at `positions`.  [T, n_kv, hd] each."""
    h = rms_norm(x, lw["attn_norm"], shape.rms_eps)
    k = (h @ lw["wk"].T).reshape(x.shape[0], shape.n_kv, shape.head_dim)
    v = (h @ lw["wv"].T).reshape(x.shape[0], shape.n_kv, shape.head_dim)
    return rope(k, positions, shape.rope_theta), v


def qkv(x: np.ndarray, lw: dict, shape: synth.ModelShape, positions: np.ndarray):
    """Pre-attention half of a layer for the tokens x: norm, projections, RoPE."""
    k, v = kv_proj(x, lw, shape, positions)
    return q_proj(x, lw, shape, positions), k, v


def attn_out_and_ffn(x: np.ndarray, a: np.ndarray, lw: dict, shape: synth.ModelShape) -> np.ndarray:
    """Post-attention half: output projection + residual, then the SwiGLU block + residual."""
    t = x.shape[0]
    x = x + a.reshape(t, shape.n_q * shape.head_dim) @ lw["wo"].T
    h = rms_norm(x, lw["ffn_norm"], shape.rms_eps)
    return x + swiglu_ffn(h, lw["w_gate"], lw["w_up"], lw["w_down"])


def layer_forward(x: np.ndarray, lw: dict, shape: synth.ModelShape, positions: np.ndarray,
                  cache_k: np.ndarray | None = None, cache_v: np.ndarray | None = None):
    """One transformer layer for the new tokens x ([T, d]) of one sequence.

    cache_k / cache_v hold the keys and values of the earlier positions
    0..P-1 ([P, n_kv, hd]); the new tokens sit at ``positions``.
    Returns (x_out, k_all, v_all) with the caches extended by the new tokens.
    """
    q, k, v = qkv(x, lw, shape, positions)
    if cache_k is not None and cache_k.shape[0]:
        k_all = np.concatenate([cache_k, k], axis=0)
        v_all = np.concatenate([cache_v, v], axis=0)
    else:
        k_all, v_all = k, v
    k_pos = np.arange(k_all.shape[0])
    a = attention(q, k_all, v_all, np.asarray(positions), k_pos)
    return attn_out_and_ffn(x, a, lw, shape), k_all, v_all


def layer_rows(x_all: np.ndarray, lw: dict, shape: synth.ModelShape, rows) -> np.ndarray:
    """One layer's output at selected positions of a single sequence.

    x_all: the layer's input for positions 0..T-1 ([T, d]).  Keys and values
    are formed for positions <= max(rows); queries and the feed-forward block
    are evaluated at ``rows`` alone.  Equal, row for row, to
    layer_forward(x_all, ...)[0][rows].
    """
    rows = np.asarray(rows, dtype=np.int64)
    hi = int(rows.max()) + 1
    k, v = kv_proj(x_all[:hi], lw, shape, np.arange(hi))
    q = q_proj(x_all[rows], lw, shape, rows)
    a = attention(q, k, v, rows, np.arange(hi))
    return attn_out_and_ffn(x_all[rows], a, lw, shape)


def lm_head(x: np.ndarray, weights: Weights) -> np.ndarray:
    """Final RMSNorm and the LM head: logits [T, V]."""
    h = rms_norm(x, weights.final_norm(), weights.shape.rms_eps)
    return h @ weights.head().T


def greedy(logits: np.ndarray) -> np.ndarray:
    """Arg max over the vocabulary, lowest id on ties (np.argmax takes the first)."""
    return np.argmax(logits, axis=-1).astype(np.int32)


# ----------------------------------------------------------------------------
# verdict and deferral (Sec. 2.1)
# ----------------------------------------------------------------------------

def verdict(logits: np.ndarray, verdict_ids, tau: float):
    """Restricted softmax over the verdict ids, confidence, predicted verdict, defer bit.

    logits: [B, V].  p[b] = softmax(logits[b, verdict_ids]); q = max p;
    y_hat = arg max p (lowest index on ties); defer = q < tau.
    """
    z = np.asarray(logits, dtype=np.float64)[:, list(verdict_ids)]
    p = softmax(z, axis=-1)
    conf = p.max(axis=-1)
    arg = np.argmax(p, axis=-1).astype(np.int32)
    defer = (conf < tau).astype(np.uint8)
    return p, conf, arg, defer


# ----------------------------------------------------------------------------
# whole-sequence drivers
# ----------------------------------------------------------------------------

class SequenceState:
    """KV cache (dense, per layer) and position of one sequence."""

    def __init__(self, layers: int):
        self.k = [None] * layers
        self.v = [None] * layers
        self.length = 0


def prefill(weights: Weights, ids: np.ndarray, all_logits: bool = False):
    """Run the prompt ``ids`` of one sequence; return (logits, state).

    logits are those of the last prompt position ([V]), or of every position
    ([T, V]) when all_logits is set.
    """
    m = weights.shape
    ids = np.asarray(ids, dtype=np.int64)
    st = SequenceState(m.layers)
    x = weights.embed_rows(ids)
    pos = np.arange(len(ids))
    for l in range(m.layers):
        x, st.k[l], st.v[l] = layer_forward(x, weights.layer(l), m, pos)
    st.length = len(ids)
    if all_logits:
        return lm_head(x, weights), st
    return lm_head(x[-1:], weights)[0], st


def decode_step(weights: Weights, st: SequenceState, token: int) -> np.ndarray:
    """Feed one token at position st.length using the KV cache; return its logits [V]."""
    m = weights.shape
    x = weights.embed_rows(np.array([token]))
    pos = np.array([st.length])
    for l in range(m.layers):
        x, st.k[l], st.v[l] = layer_forward(x, weights.layer(l), m, pos, st.k[l], st.v[l])
    st.length += 1
    return lm_head(x, weights)[0]


def full_recompute_logits(weights: Weights, ids: np.ndarray) -> np.ndarray:
    """Logits of the last position by running every token from scratch (no cache)."""
    logits, _ = prefill(weights, ids)
    return logits


def forecast_one(weights: Weights, prompt: np.ndarray, n_decode: int, verdict_ids, tau: float,
                 forced_tokens=None):
    """One candidate: prefill, n_decode greedy steps, verdict on the final logits.

    forced_tokens (optional, length n_decode) replays given decode inputs
    instead of the oracle's own greedy choices (teacher forcing), so that the
    logits of every step can be compared with another implementation's even
    where near-tied arg maxes would send the two trajectories apart.
    Returns dict(step_logits [n_decode+1, V], tokens [n_decode], p, conf, arg, defer).
    """
    logits, st = prefill(weights, prompt)
    step_logits = [logits]
    tokens = []
    for s in range(n_decode):
        tok = int(greedy(logits[None, :])[0]) if forced_tokens is None else int(forced_tokens[s])
        tokens.append(tok)
        logits = decode_step(weights, st, tok)
        step_logits.append(logits)
    p, conf, arg, defer = verdict(logits[None, :], verdict_ids, tau)
    return dict(step_logits=np.stack(step_logits), tokens=np.array(tokens, dtype=np.int32),
                p=p[0], conf=float(conf[0]), arg=int(arg[0]), defer=int(defer[0]))


def forecast_batch(weights: Weights, ids: np.ndarray, offsets: np.ndarray, n_decode: int, verdict_ids, tau: float,
                   forced_tokens=None):
    """forecast_one for every prompt ids[offsets[i]:offsets[i+1]] (items are independent)."""
    out = []
    for i in range(len(offsets) - 1):
        f = None if forced_tokens is None else forced_tokens[i]
        out.append(forecast_one(weights, ids[offsets[i]:offsets[i + 1]], n_decode, verdict_ids, tau, f))
    return out
