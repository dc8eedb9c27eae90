"""CPU oracle for temperature sampling with repeats.

TEST INFRASTRUCTURE ONLY (like ``oracle.model``): imported by the tests,
``__graft_entry__.smoke()`` and the benchmark's CPU baseline, never by the
library.  Plain numpy, float64.

What the paper fixes (Sec. 3.1, setup): every row is sampled three times from
the surrogate at temperature 1.0, and tables give the mean and the population
standard deviation over the three repeats.

Readings where the paper is silent (each repeated where it is used):
* A token is drawn by the Gumbel-max identity: argmax_v (l_v / T + G_v) with
  G_v = -ln(-ln U_v) and U_v uniform on (0, 1) is an exact draw from
  softmax(l / T).  The lowest id wins an exact tie.
* U_v comes from a counter-based generator so that another implementation can
  reproduce the draw: Philox4x64-10 (Salmon et al., SC 2011) under key
  (seed, 0) at counter (v, t, r // 4, 0); the draw for row r is output word
  r mod 4, w, and U = (floor(w / 2^41) + 1/2) / 2^23.  Here r numbers the
  sampled rows of one call (item i, repeat j -> r = i * R + j) and t the
  generated token (t = 0 from the prompt's logits, t = s + 1 from decode
  step s).  numpy's Philox bit generator supplies the blocks.
* The verdict reads the final logits exactly as in greedy decoding: the
  readout is a probability, not a sampled token.
* Repeats of an item run the same prompt; only their draws differ.
* Population statistics divide by R (not R - 1).
"""
from __future__ import annotations

import numpy as np

from .model import Weights, decode_step, prefill, verdict

_MASK64 = (1 << 64) - 1


def _counter_minus_one(c):
    """256-bit counter (4 little-endian words) minus one, with borrow."""
    value = sum(int(w) << (64 * i) for i, w in enumerate(c))
    value = (value - 1) % (1 << 256)
    return np.array([(value >> (64 * i)) & _MASK64 for i in range(4)], dtype=np.uint64)


def philox_words(seed: int, t: int, r: int, V: int) -> np.ndarray:
    """Output word r mod 4 of the Philox4x64-10 blocks at counters (v, t, r // 4, 0), v = 0..V-1."""
    # numpy's Philox advances its counter before producing a block, so start one below block 0
    start = _counter_minus_one([0, t, r // 4, 0])
    g = np.random.Philox(counter=start, key=np.array([seed & _MASK64, 0], dtype=np.uint64))
    return g.random_raw(4 * V).reshape(V, 4)[:, r % 4]


def uniforms(seed: int, t: int, r: int, V: int) -> np.ndarray:
    """U_v = (floor(w_v / 2^41) + 1/2) / 2^23, strictly inside (0, 1)."""
    w = philox_words(seed, t, r, V)
    return ((w >> np.uint64(41)).astype(np.float64) + 0.5) / float(1 << 23)


def gumbel(u: np.ndarray) -> np.ndarray:
    """G = -ln(-ln U)."""
    return -np.log(-np.log(np.asarray(u, dtype=np.float64)))


def sample(logits: np.ndarray, temperature: float, u: np.ndarray) -> int:
    """argmax_v (l_v / T + G_v), lowest v among equals."""
    z = np.asarray(logits, dtype=np.float64) / float(temperature) + gumbel(u)
    return int(np.argmax(z))


def sample_scores(logits: np.ndarray, temperature: float, u: np.ndarray) -> np.ndarray:
    """The perturbed scores l_v / T + G_v whose arg max is the sampled token."""
    return np.asarray(logits, dtype=np.float64) / float(temperature) + gumbel(u)


def forecast_sampled_one(weights: Weights, prompt: np.ndarray, n_decode: int, verdict_ids, tau: float, seed: int,
                         row: int, temperature: float, forced_tokens=None):
    """One sampled row: prefill, n_decode sampled steps, verdict on the final logits.

    Token t (the input of decode step t) is drawn from the logits before it
    with the uniforms of (seed, t, row).  forced_tokens replays another
    implementation's tokens (teacher forcing) so that every step's logits can
    be compared even where a near tie sends two trajectories apart.
    Returns dict(step_logits [n_decode+1, V], tokens [n_decode], p, conf, arg, defer).
    """
    logits, st = prefill(weights, prompt)
    V = logits.shape[-1]
    step_logits = [logits]
    tokens = []
    for t in range(n_decode):
        if forced_tokens is None:
            tok = sample(logits, temperature, uniforms(seed, t, row, V))
        else:
            tok = int(forced_tokens[t])
        tokens.append(tok)
        logits = decode_step(weights, st, tok)
        step_logits.append(logits)
    p, conf, arg, defer = verdict(logits[None, :], verdict_ids, tau)
    return dict(step_logits=np.stack(step_logits), tokens=np.array(tokens, dtype=np.int32),
                p=p[0], conf=float(conf[0]), arg=int(arg[0]), defer=int(defer[0]))


def repeat_stats(x: np.ndarray):
    """Mean and population standard deviation over the repeats (axis 0)."""
    x = np.asarray(x, dtype=np.float64)
    mean = x.sum(axis=0) / x.shape[0]
    return mean, np.sqrt(((x - mean) ** 2).sum(axis=0) / x.shape[0])
