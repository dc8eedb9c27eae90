"""Seeded synthetic workloads: model shapes, weights and prompt token ids.

This module is shared by the oracle (``oracle/``) and by the CUDA path's
tests and benchmark.  It holds no arithmetic of the forecasting method: it
names the workload shapes, draws weights and token ids from a counter-based
generator (Philox4x64-10, implemented in ``synth.c``) and returns them as
plain numpy arrays.  Weights are returned as bf16 bit patterns (uint16); each
consumer converts them to its own working type.

Workload recipe (the five model/prompt configurations the surrogate is run
on, standing in for the paper's tokenised kernel-source prompts, whose
tokenizer, model and data are not available):

* weights: Irwin-Hall(8) draws with mean 0 and standard deviation 0.02,
  rounded once to bf16; RMSNorm gains are 1.
* prompts: prompt i = incumbent ids (one draw shared by the whole batch, the
  reference kernel r of x_i = (r, k_i, h), Sec. 2.1) followed by candidate i's
  ids.  Ids are uniform for ``tiny`` and Zipf(1.1) for the others.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "synth.c")
_LIB_PATH = os.path.join(_HERE, "_build", "libsynth.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile synth.c into a shared library (plain gcc, OpenMP)."""
    os.makedirs(os.path.dirname(_LIB_PATH), exist_ok=True)
    stale = (not os.path.exists(_LIB_PATH)) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC)
    if force or stale:
        tmp = _LIB_PATH + f".{os.getpid()}.tmp"
        subprocess.check_call(["gcc", "-O2", "-fopenmp", "-shared", "-fPIC", "-std=c11", _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            u64, u32, i64, f32, f64, p = (ctypes.c_uint64, ctypes.c_uint32, ctypes.c_int64, ctypes.c_float,
                                          ctypes.c_double, ctypes.c_void_p)
            lib.synth_philox4x64_10.argtypes = [p, p, p]
            lib.synth_philox4x64_10.restype = None
            lib.synth_normal_bf16.argtypes = [u64, u64, u64, u64, f32, p]
            lib.synth_normal_bf16.restype = None
            lib.synth_normal_f32.argtypes = [u64, u64, u64, u64, f32, p]
            lib.synth_normal_f32.restype = None
            lib.synth_uniform_int.argtypes = [u64, u64, u64, i64, i64, p]
            lib.synth_uniform_int.restype = None
            lib.synth_uniform_f64.argtypes = [u64, u64, u64, p]
            lib.synth_uniform_f64.restype = None
            lib.synth_zipf_ids.argtypes = [u64, u64, u64, u32, f64, p]
            lib.synth_zipf_ids.restype = ctypes.c_int
            lib.synth_irwin_hall_scale.argtypes = [f32]
            lib.synth_irwin_hall_scale.restype = f32
            _lib = lib
    return _lib


# ----------------------------------------------------------------------------
# raw generators
# ----------------------------------------------------------------------------

def philox4x64_10(counter, key) -> np.ndarray:
    """One Philox4x64-10 block: four 64-bit words for a 256-bit counter and 128-bit key."""
    c = np.ascontiguousarray(np.asarray(counter, dtype=np.uint64).reshape(4))
    k = np.ascontiguousarray(np.asarray(key, dtype=np.uint64).reshape(2))
    out = np.zeros(4, dtype=np.uint64)
    _load().synth_philox4x64_10(c.ctypes.data, k.ctypes.data, out.ctypes.data)
    return out


def normal_bf16(seed: int, stream: int, n: int, sigma: float, start: int = 0) -> np.ndarray:
    """n bf16 bit patterns of Irwin-Hall(8) draws with mean 0 and std sigma."""
    out = np.empty(int(n), dtype=np.uint16)
    if n:
        _load().synth_normal_bf16(seed, stream, start, n, sigma, out.ctypes.data)
    return out


def normal_f32(seed: int, stream: int, n: int, sigma: float, start: int = 0) -> np.ndarray:
    """The same draws as normal_bf16 before the bf16 rounding."""
    out = np.empty(int(n), dtype=np.float32)
    if n:
        _load().synth_normal_f32(seed, stream, start, n, sigma, out.ctypes.data)
    return out


def uniform_int(seed: int, stream: int, n: int, lo: int, hi: int) -> np.ndarray:
    out = np.empty(int(n), dtype=np.int32)
    if n:
        _load().synth_uniform_int(seed, stream, n, lo, hi, out.ctypes.data)
    return out


def uniform_f64(seed: int, stream: int, n: int) -> np.ndarray:
    out = np.empty(int(n), dtype=np.float64)
    if n:
        _load().synth_uniform_f64(seed, stream, n, out.ctypes.data)
    return out


def zipf_ids(seed: int, stream: int, n: int, vocab: int, s: float = 1.1) -> np.ndarray:
    out = np.empty(int(n), dtype=np.int32)
    if n:
        rc = _load().synth_zipf_ids(seed, stream, n, vocab, s, out.ctypes.data)
        if rc != 0:
            raise MemoryError("synth_zipf_ids: out of memory")
    return out


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Reinterpret bf16 bit patterns as float32 (exact)."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


# ----------------------------------------------------------------------------
# workload configurations
# ----------------------------------------------------------------------------

@dataclasses.dataclass(frozen=True)
class ModelShape:
    layers: int
    d_model: int
    n_q: int
    n_kv: int
    head_dim: int
    ffn: int
    vocab: int
    rope_theta: float
    rms_eps: float = 1e-6
    sigma: float = 0.02
    head_sigma: float = 0.02  # std of the LM-head weights (a separate knob for defer tests)


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    model: ModelShape
    batch: int
    prompt_len: int          # maximum prompt length
    inc_len: int             # shared incumbent prefix length
    id_dist: str             # "uniform" or "zipf"
    n_decode: int
    tau: float
    verdict_ids: tuple = (10, 11)
    ragged: tuple | None = None  # (lo, hi) inclusive prompt-length range, else all prompt_len
    weight_seed: int = 0
    id_seed: int = 1
    len_seed: int = 2


SHAPE_TINY = ModelShape(layers=2, d_model=256, n_q=4, n_kv=4, head_dim=64, ffn=688, vocab=4096, rope_theta=1e4)
SHAPE_1P5B = ModelShape(layers=28, d_model=1536, n_q=12, n_kv=2, head_dim=128, ffn=8960, vocab=151936,
                        rope_theta=1e6)
SHAPE_7B = ModelShape(layers=28, d_model=3584, n_q=28, n_kv=4, head_dim=128, ffn=18944, vocab=152064,
                      rope_theta=1e6)
SHAPE_14B = ModelShape(layers=48, d_model=5120, n_q=40, n_kv=8, head_dim=128, ffn=13824, vocab=152064,
                       rope_theta=1e6)

WORKLOADS = {
    "tiny": Workload("tiny", SHAPE_TINY, batch=4, prompt_len=256, inc_len=128, id_dist="uniform", n_decode=8,
                     tau=0.8),
    "1p5b": Workload("1p5b", SHAPE_1P5B, batch=16, prompt_len=4096, inc_len=2048, id_dist="zipf", n_decode=64,
                     tau=0.8),
    "7b_prefill": Workload("7b_prefill", SHAPE_7B, batch=32, prompt_len=6144, inc_len=3072, id_dist="zipf",
                           n_decode=256, tau=0.8),
    "7b_decode": Workload("7b_decode", SHAPE_7B, batch=128, prompt_len=2048, inc_len=512, id_dist="zipf",
                          n_decode=2048, tau=0.8, ragged=(1024, 2048)),
    "14b_long": Workload("14b_long", SHAPE_14B, batch=8, prompt_len=16384, inc_len=8192, id_dist="zipf",
                         n_decode=128, tau=0.9),
}


def workload(name: str, **overrides) -> Workload:
    w = WORKLOADS[name]
    return dataclasses.replace(w, **overrides) if overrides else w


# Per-tensor streams of the weight generator.
KIND = {"wq": 0, "wk": 1, "wv": 2, "wo": 3, "w_gate": 4, "w_up": 5, "w_down": 6}
STREAM_EMBED = 1
STREAM_HEAD = 2


def layer_tensor_shapes(m: ModelShape) -> dict:
    """Canonical per-layer weight shapes, rows = output features (row-major)."""
    return {
        "wq": (m.n_q * m.head_dim, m.d_model),
        "wk": (m.n_kv * m.head_dim, m.d_model),
        "wv": (m.n_kv * m.head_dim, m.d_model),
        "wo": (m.d_model, m.n_q * m.head_dim),
        "w_gate": (m.ffn, m.d_model),
        "w_up": (m.ffn, m.d_model),
        "w_down": (m.d_model, m.ffn),
    }


def layer_weights_bf16(m: ModelShape, layer: int, seed: int = 0) -> dict:
    """Weights of one layer as bf16 bit patterns (uint16), canonical shapes."""
    out = {}
    for name, shape in layer_tensor_shapes(m).items():
        stream = (layer + 1) * 16 + KIND[name]
        out[name] = normal_bf16(seed, stream, shape[0] * shape[1], m.sigma).reshape(shape)
    return out


def embed_bf16(m: ModelShape, seed: int = 0) -> np.ndarray:
    return normal_bf16(seed, STREAM_EMBED, m.vocab * m.d_model, m.sigma).reshape(m.vocab, m.d_model)


def head_bf16(m: ModelShape, seed: int = 0) -> np.ndarray:
    return normal_bf16(seed, STREAM_HEAD, m.vocab * m.d_model, m.head_sigma).reshape(m.vocab, m.d_model)


def ones_bf16(n: int) -> np.ndarray:
    return np.full(n, 0x3F80, dtype=np.uint16)  # bf16(1.0)


def prompt_lengths(w: Workload) -> np.ndarray:
    if w.ragged is None:
        return np.full(w.batch, w.prompt_len, dtype=np.int32)
    lo, hi = w.ragged
    return uniform_int(w.len_seed, 3000, w.batch, lo, hi)


def _ids(w: Workload, stream: int, n: int) -> np.ndarray:
    if w.id_dist == "uniform":
        return uniform_int(w.id_seed, stream, n, 0, w.model.vocab - 1)
    return zipf_ids(w.id_seed, stream, n, w.model.vocab, 1.1)


def prompts(w: Workload, items=None):
    """Token ids of the batch (or of the listed items).

    Returns (inc_ids, inc_offsets, cand_ids, cand_offsets): packed int32 arrays
    with B+1 offsets each; prompt i = inc_ids[inc_offsets[i]:inc_offsets[i+1]]
    followed by cand_ids[cand_offsets[i]:cand_offsets[i+1]].
    """
    items = list(range(w.batch)) if items is None else list(items)
    lens = prompt_lengths(w)
    inc = _ids(w, 1000, w.inc_len)
    inc_parts, cand_parts = [], []
    for i in items:
        inc_parts.append(inc)
        cand_parts.append(_ids(w, 2000 + i, int(lens[i]) - w.inc_len))
    inc_off = np.concatenate([[0], np.cumsum([len(x) for x in inc_parts])]).astype(np.int32)
    cand_off = np.concatenate([[0], np.cumsum([len(x) for x in cand_parts])]).astype(np.int32)
    return (np.concatenate(inc_parts).astype(np.int32), inc_off,
            np.concatenate(cand_parts).astype(np.int32), cand_off)


def packed_prompts(w: Workload, items=None):
    """Whole prompts packed: (ids, offsets) with prompt i = ids[offsets[i]:offsets[i+1]]."""
    inc, inc_off, cand, cand_off = prompts(w, items)
    parts = []
    for i in range(len(inc_off) - 1):
        parts.append(inc[inc_off[i]:inc_off[i + 1]])
        parts.append(cand[cand_off[i]:cand_off[i + 1]])
    ids = np.concatenate(parts).astype(np.int32)
    lens = (np.diff(inc_off) + np.diff(cand_off)).astype(np.int64)
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    return ids, off
