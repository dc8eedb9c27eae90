"""GB300 surrogate forecaster: thin Python binding of the C ABI in include/gf.h.

Every step of the forward pass, the greedy decode and the verdict/defer step
runs in the CUDA library ``_build/libgf.so`` (hand-written sm_103a kernels).
This module only marshals arguments: functions named like the C entry points
take raw pointers and sizes; ``Model`` wraps them for torch tensors, which
serve only as device memory and streams.  There is no fallback path: if the
library is missing, every call raises.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libgf.so")

GF_OK, GF_EINVAL, GF_ECAPACITY, GF_ENOMEM, GF_ECUDA, GF_ENOTIMPL, GF_ETIMEOUT = range(7)

_c_i32, _c_i64, _c_f32, _p = ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_void_p


class GfError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"gf error {code}: {msg}")
        self.code = code


class gf_config(ctypes.Structure):
    _fields_ = [("layers", _c_i32), ("d_model", _c_i32), ("n_q", _c_i32), ("n_kv", _c_i32), ("head_dim", _c_i32),
                ("ffn", _c_i32), ("vocab", _c_i32), ("rope_theta", _c_f32), ("rms_eps", _c_f32),
                ("max_batch", _c_i32), ("max_seq", _c_i32), ("max_prefill_tokens", _c_i64), ("kv_pages", _c_i64)]


_PP = ctypes.POINTER(_p)


class gf_weights(ctypes.Structure):
    _fields_ = [("embed", _p), ("lm_head", _p), ("final_norm", _p), ("attn_norm", _PP), ("wq", _PP), ("wk", _PP),
                ("wv", _PP), ("wo", _PP), ("ffn_norm", _PP), ("w_gate", _PP), ("w_up", _PP), ("w_down", _PP)]


EXPORTS = ["gf_create", "gf_destroy", "gf_prefill", "gf_decode_step", "gf_release", "gf_forecast_batch",
           "gf_forecast_batch_host", "gf_verdict", "gf_debug_capture", "gf_debug_read_kv", "gf_device_status",
           "gf_launch_count", "gf_last_error", "gf_gemm_bf16", "gf_gemm_status", "gf_profile_enable",
           "gf_profile_read", "gf_decode_attention", "gf_decode_attention_workspace",
           "gf_decode_attention_static", "gf_decode_attention_static_status", "gf_selftest_timeout_static",
           "gf_forecast_batch_shared", "gf_speedup_bin", "gf_score_forecasts", "gf_free_pages", "gf_selftest_timeout", "gf_select",
           "gf_forecast_batch_sampled", "gf_sample_tokens", "gf_plan_gemm", "gf_plan_decode_chunk"]

GF_GEMM_STORE_F32, GF_GEMM_ADD_F32, GF_GEMM_ATOMIC_F32, GF_GEMM_STORE_BF16, GF_GEMM_SWIGLU = range(5)
GF_PROF_PREFILL_GEMM, GF_PROF_DECODE_GEMM, GF_PROF_PREFILL_ATTN, GF_PROF_DECODE_ATTN, GF_PROF_DECODE_STEPS = range(5)

_lib = None


def load(path: str = LIB_PATH):
    """Load libgf.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"CUDA library {path} is missing: build it with paper_2605_31464_gb300._build.build()")
    lib = ctypes.CDLL(path)
    sig = {
        "gf_create": ([ctypes.POINTER(gf_config), ctypes.POINTER(gf_weights), _p, ctypes.POINTER(_p)], ctypes.c_int),
        "gf_destroy": ([_p], None),
        "gf_prefill": ([_p, _c_i32, _p, _p, _p, _p, _p, _p], ctypes.c_int),
        "gf_decode_step": ([_p, _c_i32, _p, _p, _p, _p, _p], ctypes.c_int),
        "gf_release": ([_p, _c_i32, _p], ctypes.c_int),
        "gf_forecast_batch": ([_p, _c_i32, _p, _p, _p, _p, _c_i32, _p, _c_i32, _c_f32, _p, _p, _p, _p, _p, _p, _p],
                              ctypes.c_int),
        "gf_forecast_batch_host": ([_p, _c_i32, _p, _p, _p, _p, _c_i32, _p, _c_i32, _c_f32, _p, _p, _p, _p, _p, _p],
                                   ctypes.c_int),
        "gf_forecast_batch_shared": ([_p, _c_i32, _p, _c_i32, _p, _p, _c_i32, _p, _c_i32, _c_f32, _p, _p, _p, _p, _p,
                                      _p, _p], ctypes.c_int),
        "gf_forecast_batch_sampled": ([_p, _c_i32, _p, _p, _p, _p, _c_i32, _c_i32, _c_f32, ctypes.c_uint64, _p, _c_i32,
                                       _c_f32, _p, _p, _p, _p, _p, _p, _p, _p, _p, _p, _p], ctypes.c_int),
        "gf_sample_tokens": ([_c_i32, _p, _c_i64, _c_i32, ctypes.c_uint64, _c_i32, _c_f32, _p, _p], ctypes.c_int),
        "gf_free_pages": ([_p], _c_i64),
        "gf_selftest_timeout": ([ctypes.c_uint32, _p], ctypes.c_int),
        "gf_selftest_timeout_static": ([ctypes.c_uint32, _p], ctypes.c_int),
        "gf_speedup_bin": ([ctypes.c_double], ctypes.c_int),
        "gf_score_forecasts": ([_c_i32, _p, _p, _p, _p], ctypes.c_int),
        "gf_decode_attention_static_status": ([_p], ctypes.c_int),
        "gf_select": ([_c_i32, _p, _p, _c_f32, _c_f32, _p, _p, _p, _p, _p], ctypes.c_int),
        "gf_verdict": ([_c_i32, _p, _c_i64, _p, _c_i32, _c_f32, _p, _p, _p, _p, _p], ctypes.c_int),
        "gf_debug_capture": ([_p, _c_i32, _c_i32, _p, _c_i64], ctypes.c_int),
        "gf_debug_read_kv": ([_p, _c_i32, _c_i32, _c_i32, _c_i32, _p, _p, _p], ctypes.c_int),
        "gf_device_status": ([_p, _p], ctypes.c_int),
        "gf_launch_count": ([_p], _c_i64),
        "gf_last_error": ([], ctypes.c_char_p),
        "gf_gemm_bf16": ([_p, _p, _c_i32, _c_i32, _c_i32, _p, _c_i64, _c_i32, _c_i32, _c_i32, _c_i32, _p],
                         ctypes.c_int),
        "gf_gemm_status": ([_p], ctypes.c_int),
        "gf_plan_gemm": ([_c_i32, _c_i32, _c_i32, _c_i32, _c_i32, ctypes.POINTER(_c_i32), ctypes.POINTER(_c_i32),
                          ctypes.POINTER(_c_i32)], ctypes.c_int),
        "gf_plan_decode_chunk": ([_c_i32, _c_i32, _c_i32, _c_i32], _c_i32),
        "gf_decode_attention_workspace": ([_c_i32, _c_i32, _c_i32, _c_i32], ctypes.c_size_t),
        "gf_decode_attention_static": ([_p, _p, _p, _c_i64, _p, _c_i32, _p, _c_i32, _c_i32, _c_i32, _c_i32, _c_i32,
                                        _p, _p], ctypes.c_int),
        "gf_decode_attention": ([_p, _p, _p, _c_i64, _p, _c_i32, _p, _c_i32, _c_i32, _c_i32, _c_i32, _c_i32, _p, _p,
                                 ctypes.c_size_t, _p], ctypes.c_int),
        "gf_profile_enable": ([_p, ctypes.c_uint32], ctypes.c_int),
        "gf_profile_read": ([_p, _c_i32, ctypes.POINTER(_c_i64), ctypes.POINTER(ctypes.c_double),
                             ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double)], ctypes.c_int),
    }
    for name, (args, res) in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    _lib = lib
    return lib


def _check(rc: int):
    if rc != GF_OK:
        raise GfError(rc, load().gf_last_error().decode())


# ---------------------------------------------------------------- raw entry points (pointers and sizes)

def gf_create(cfg: gf_config, weights: gf_weights, stream: int) -> int:
    out = _p()
    _check(load().gf_create(ctypes.byref(cfg), ctypes.byref(weights), stream, ctypes.byref(out)))
    return out.value


def gf_destroy(model: int) -> None:
    load().gf_destroy(model)


def gf_prefill(model, B, ids, offsets, seq_handles, last_logits, next_ids, stream):
    _check(load().gf_prefill(model, B, ids, offsets, seq_handles, last_logits, next_ids, stream))


def gf_decode_step(model, B, seq_handles, ids, logits, next_ids, stream):
    _check(load().gf_decode_step(model, B, seq_handles, ids, logits, next_ids, stream))


def gf_release(model, B, seq_handles):
    _check(load().gf_release(model, B, seq_handles))


def gf_forecast_batch(model, B, inc_ids, inc_offsets, cand_ids, cand_offsets, n_decode, verdict_ids, K, tau, p,
                      conf, verdict_arg, defer, tokens, final_logits, stream):
    _check(load().gf_forecast_batch(model, B, inc_ids, inc_offsets, cand_ids, cand_offsets, n_decode, verdict_ids,
                                    K, tau, p, conf, verdict_arg, defer, tokens, final_logits, stream))


def gf_forecast_batch_host(model, B, inc_ids, inc_offsets, cand_ids, cand_offsets, n_decode, verdict_ids, K, tau, p,
                           conf, verdict_arg, defer, tokens, stream):
    _check(load().gf_forecast_batch_host(model, B, inc_ids, inc_offsets, cand_ids, cand_offsets, n_decode,
                                         verdict_ids, K, tau, p, conf, verdict_arg, defer, tokens, stream))


def gf_forecast_batch_shared(model, B, prefix_ids, prefix_len, cand_ids, cand_offsets, n_decode, verdict_ids, K, tau,
                             p, conf, verdict_arg, defer, tokens, final_logits, stream):
    _check(load().gf_forecast_batch_shared(model, B, prefix_ids, prefix_len, cand_ids, cand_offsets, n_decode,
                                           verdict_ids, K, tau, p, conf, verdict_arg, defer, tokens, final_logits,
                                           stream))


def gf_forecast_batch_sampled(model, B, inc_ids, inc_offsets, cand_ids, cand_offsets, n_decode, repeats, temperature,
                              seed, verdict_ids, K, tau, p, conf, verdict_arg, defer, p_mean, p_std, conf_mean,
                              conf_std, tokens, final_logits, stream):
    _check(load().gf_forecast_batch_sampled(model, B, inc_ids, inc_offsets, cand_ids, cand_offsets, n_decode, repeats,
                                            temperature, seed, verdict_ids, K, tau, p, conf, verdict_arg, defer,
                                            p_mean, p_std, conf_mean, conf_std, tokens, final_logits, stream))


def gf_sample_tokens(B, logits, ld, V, seed, token_index, temperature, out_ids, stream):
    _check(load().gf_sample_tokens(B, logits, ld, V, seed, token_index, temperature, out_ids, stream))


def sample_tokens(logits, seed, token_index, temperature, stream=None):
    """Temperature draw (Gumbel-max, counter-based) for each row of a [B, V] float32 CUDA tensor."""
    import torch
    _check_tensor(logits, "logits", dtype=torch.float32, rows_strided=True)
    s = stream if stream is not None else torch.cuda.current_stream()
    out = torch.empty(logits.shape[0], dtype=torch.int32, device=logits.device)
    gf_sample_tokens(logits.shape[0], logits.data_ptr(), logits.stride(0), logits.shape[1], int(seed),
                     int(token_index), float(temperature), out.data_ptr(), s.cuda_stream)
    return out


def gf_select(B, p, m_bins, x_cut, tau_disc, s_hat, order, disc, disc_pred, stream):
    _check(load().gf_select(B, p, m_bins, x_cut, tau_disc, s_hat, order, disc, disc_pred, stream))


def select(p, m_bins, x_cut, tau_disc, stream=None):
    """Expected speedup, ranking and discovery score of a [B, 8] CUDA tensor of bin probabilities."""
    import torch
    _check_tensor(p, "p", (p.shape[0], 8), torch.float32)
    s = stream if stream is not None else torch.cuda.current_stream()
    B = p.shape[0]
    m = np.ascontiguousarray(np.asarray(m_bins, dtype=np.float32))
    s_hat = torch.empty(B, dtype=torch.float32, device=p.device)
    order = torch.empty(B, dtype=torch.int32, device=p.device)
    disc = torch.empty(B, dtype=torch.float32, device=p.device)
    pred = torch.empty(B, dtype=torch.uint8, device=p.device)
    gf_select(B, p.data_ptr(), m.ctypes.data_as(_p), float(x_cut), float(tau_disc), s_hat.data_ptr(),
              order.data_ptr(), disc.data_ptr(), pred.data_ptr(), s.cuda_stream)
    return s_hat, order, disc, pred


def gf_selftest_timeout(limit_ms, stream):
    """Returns the status code (GF_ETIMEOUT expected) instead of raising."""
    return int(load().gf_selftest_timeout(limit_ms, stream))


def gf_speedup_bin(S) -> int:
    """Bin 1..8 of a measured speedup (host arithmetic only; needs no GPU)."""
    return int(load().gf_speedup_bin(float(S)))


def score_forecasts(p, S, m_bins) -> dict:
    """Speedup recovered, ECE, forecast error, mean Brier and CRPS of 8-bin forecasts p [n, 8] against
    measured speedups S [n] (host arithmetic only; needs no GPU)."""
    p = np.ascontiguousarray(np.asarray(p, dtype=np.float64))
    S = np.ascontiguousarray(np.asarray(S, dtype=np.float64))
    m = np.ascontiguousarray(np.asarray(m_bins, dtype=np.float64))
    if p.ndim != 2 or p.shape[1] != 8 or S.shape != (p.shape[0],) or m.shape != (8,):
        raise ValueError("p must be [n, 8], S [n] and m_bins [8]")
    out = np.zeros(5, dtype=np.float64)
    _check(load().gf_score_forecasts(p.shape[0], _ptr(p), _ptr(S), _ptr(m), _ptr(out)))
    return dict(recovered=out[0], ece=out[1], forecast_error=out[2], brier=out[3], crps=out[4])


def gf_free_pages(model) -> int:
    return int(load().gf_free_pages(model))


def gf_verdict(B, logits, ld, verdict_ids, K, tau, p, conf, verdict_arg, defer, stream):
    _check(load().gf_verdict(B, logits, ld, verdict_ids, K, tau, p, conf, verdict_arg, defer, stream))


def gf_debug_capture(model, layer, item, dst, cap_rows):
    _check(load().gf_debug_capture(model, layer, item, dst, cap_rows))


def gf_debug_read_kv(model, layer, handle, start, n, k_dst, v_dst, stream):
    _check(load().gf_debug_read_kv(model, layer, handle, start, n, k_dst, v_dst, stream))


def gf_device_status(model, stream):
    _check(load().gf_device_status(model, stream))


def gf_launch_count(model) -> int:
    return int(load().gf_launch_count(model))


def gf_last_error() -> str:
    return load().gf_last_error().decode()


def gf_gemm_bf16(A, W, M, N, K, out, ldo, mode, bn, splits, group_m, stream):
    _check(load().gf_gemm_bf16(A, W, M, N, K, out, ldo, mode, bn, splits, group_m, stream))


def gf_gemm_status(stream):
    _check(load().gf_gemm_status(stream))


def gf_plan_gemm(sms, M, N, K, mode) -> dict:
    """The GEMM tiling the library chooses (host arithmetic only; needs no GPU)."""
    bn, splits, swap = _c_i32(), _c_i32(), _c_i32()
    _check(load().gf_plan_gemm(sms, M, N, K, mode, ctypes.byref(bn), ctypes.byref(splits), ctypes.byref(swap)))
    return dict(bn=bn.value, splits=splits.value, swap=bool(swap.value))


def gf_plan_decode_chunk(B, n_kv, max_ctx, sms) -> int:
    """Keys per decode-attention CTA (host arithmetic only; needs no GPU)."""
    rc = int(load().gf_plan_decode_chunk(B, n_kv, max_ctx, sms))
    if rc not in (256, 512, 1024):
        raise GfError(rc, load().gf_last_error().decode())
    return rc


def gf_decode_attention_workspace(B, n_kv, head_dim, max_ctx) -> int:
    return int(load().gf_decode_attention_workspace(B, n_kv, head_dim, max_ctx))


def gf_decode_attention(q, k_cache, v_cache, num_pages, block_table, max_pages, ctx_len, max_ctx, B, n_q, n_kv,
                        head_dim, out, workspace, workspace_bytes, stream):
    _check(load().gf_decode_attention(q, k_cache, v_cache, num_pages, block_table, max_pages, ctx_len, max_ctx, B,
                                      n_q, n_kv, head_dim, out, workspace, workspace_bytes, stream))


def gf_decode_attention_static(q, k_cache, v_cache, num_pages, block_table, max_pages, ctx_len, max_ctx, B, n_q,
                               n_kv, head_dim, out, stream):
    """gf_decode_attention with its scratch in the library's fixed device array (no allocation)."""
    _check(load().gf_decode_attention_static(q, k_cache, v_cache, num_pages, block_table, max_pages, ctx_len, max_ctx,
                                             B, n_q, n_kv, head_dim, out, stream))


def gf_decode_attention_static_status(stream):
    """Returns the status code (GF_OK, or GF_ETIMEOUT once after a timed-out wait) instead of raising."""
    return int(load().gf_decode_attention_static_status(stream))


def gf_selftest_timeout_static(limit_ms, stream):
    """Returns the status code (GF_ETIMEOUT expected) instead of raising."""
    return int(load().gf_selftest_timeout_static(limit_ms, stream))


def decode_attention(q, k_cache, v_cache, block_table, ctx_len, max_ctx, n_q, n_kv, stream=None):
    """Paged decode attention on torch tensors; allocates the workspace with torch."""
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    B = q.shape[0]
    hd = k_cache.shape[-1]
    _check_tensor(q, "q", (B, n_q * hd), torch.bfloat16)
    _check_tensor(k_cache, "k_cache", (k_cache.shape[0], n_kv, 64, hd), torch.bfloat16)
    _check_tensor(v_cache, "v_cache", (k_cache.shape[0], n_kv, hd, 64), torch.bfloat16)
    _check_tensor(block_table, "block_table", (B, block_table.shape[1]), torch.int32)
    _check_ids(ctx_len, "ctx_len", B)
    ws_bytes = gf_decode_attention_workspace(B, n_kv, hd, max_ctx)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=q.device)
    out = torch.empty_like(q)
    gf_decode_attention(q.data_ptr(), k_cache.data_ptr(), v_cache.data_ptr(), k_cache.shape[0],
                        block_table.data_ptr(), block_table.shape[1], ctx_len.data_ptr(), max_ctx, B, n_q, n_kv, hd,
                        out.data_ptr(), ws.data_ptr(), ws_bytes, s.cuda_stream)
    return out


def gf_profile_enable(model, mask):
    _check(load().gf_profile_enable(model, mask))


def gf_profile_read(model, kind):
    n, ms, fl, by = _c_i64(), ctypes.c_double(), ctypes.c_double(), ctypes.c_double()
    _check(load().gf_profile_read(model, kind, ctypes.byref(n), ctypes.byref(ms), ctypes.byref(fl), ctypes.byref(by)))
    return dict(launches=n.value, ms=ms.value, flops=fl.value, bytes=by.value)


def gemm(A, W, out, mode=GF_GEMM_STORE_F32, bn=0, splits=0, stream=None, group_m=0):
    """out (op)= A . W^T on the tensor cores (A [M,K], W [N,K] bf16 CUDA tensors)."""
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    M, K = A.shape
    N = W.shape[0]
    _check_tensor(A, "A", (M, K), torch.bfloat16)
    _check_tensor(W, "W", (N, K), torch.bfloat16)
    bf16_out = mode in (GF_GEMM_STORE_BF16, GF_GEMM_SWIGLU)
    _check_tensor(out, "out", dtype=torch.bfloat16 if bf16_out else torch.float32, rows_strided=True)
    if out.shape[0] < M or out.shape[1] < (N // 2 if mode == GF_GEMM_SWIGLU else N):
        raise ValueError(f"out: shape {tuple(out.shape)} too small for {M} x {N}")
    gf_gemm_bf16(A.data_ptr(), W.data_ptr(), M, N, K, out.data_ptr(), out.stride(0), mode, bn, splits, group_m,
                 s.cuda_stream)


# ---------------------------------------------------------------- torch-facing wrapper

def _i32_host(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(_p)


def _check_tensor(t, name, shape=None, dtype=None, rows_strided=False):
    """Refuse what the C ABI cannot see through a pointer: a wrong shape or dtype, a tensor
    in host memory, or a layout other than row-major (rows_strided: any row stride)."""
    import torch
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name}: expected a torch tensor, got {type(t).__name__}")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name}: shape {tuple(t.shape)}, expected {tuple(shape)}")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name}: dtype {t.dtype}, expected {dtype}")
    dense = (t.dim() == 2 and t.stride(1) == 1 and t.stride(0) >= t.shape[1]) if rows_strided else t.is_contiguous()
    if not dense:
        raise ValueError(f"{name}: layout not supported (strides {tuple(t.stride())})")
    if not t.is_cuda:
        raise ValueError(f"{name}: must be a CUDA tensor")


def _check_ids(t, name, n):
    """A 1-D int32 CUDA tensor holding at least the n ids the call reads."""
    import torch
    _check_tensor(t, name, dtype=torch.int32)
    if t.dim() != 1 or t.numel() < n:
        raise ValueError(f"{name}: shape {tuple(t.shape)}, expected 1-D with at least {n} ids")


def _check_weights(shape, weights: dict):
    """Shapes and dtypes gf_create reads (it copies bytes by those shapes)."""
    import torch
    d, hd, L = shape.d_model, shape.head_dim, shape.layers
    bf16 = torch.bfloat16
    for name, shp in (("embed", (shape.vocab, d)), ("lm_head", (shape.vocab, d)), ("final_norm", (d,))):
        _check_tensor(weights[name], name, shp, bf16)
    per_layer = {"attn_norm": (d,), "ffn_norm": (d,), "wq": (shape.n_q * hd, d), "wk": (shape.n_kv * hd, d),
                 "wv": (shape.n_kv * hd, d), "wo": (d, shape.n_q * hd), "w_gate": (shape.ffn, d),
                 "w_up": (shape.ffn, d), "w_down": (d, shape.ffn)}
    for name, shp in per_layer.items():
        if len(weights[name]) != L:
            raise ValueError(f"{name}: {len(weights[name])} tensors for {L} layers")
        for l, t in enumerate(weights[name]):
            _check_tensor(t, f"{name}[{l}]", shp, bf16)


class Model:
    """A model on the current CUDA device.

    ``shape`` has the fields of gf_config's model part (layers, d_model, n_q,
    n_kv, head_dim, ffn, vocab, rope_theta, rms_eps).  ``weights`` maps
    names to bf16 CUDA tensors: embed, lm_head, final_norm and per layer
    lists attn_norm, wq, wk, wv, wo, ffn_norm, w_gate, w_up, w_down.
    """

    def __init__(self, shape, weights: dict, max_batch: int, max_seq: int, max_prefill_tokens: int,
                 kv_pages: int = 0, stream=None):
        import torch
        _check_weights(shape, weights)
        self.torch = torch
        self.shape = shape
        self.stream = stream if stream is not None else torch.cuda.current_stream()
        cfg = gf_config(layers=shape.layers, d_model=shape.d_model, n_q=shape.n_q, n_kv=shape.n_kv,
                        head_dim=shape.head_dim, ffn=shape.ffn, vocab=shape.vocab, rope_theta=shape.rope_theta,
                        rms_eps=shape.rms_eps, max_batch=max_batch, max_seq=max_seq,
                        max_prefill_tokens=max_prefill_tokens, kv_pages=kv_pages)
        L = shape.layers

        def arr(name):
            a = (_p * L)(*[t.data_ptr() for t in weights[name]])
            return ctypes.cast(a, _PP), a

        keep = {}
        fields = {}
        for name in ("attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "w_gate", "w_up", "w_down"):
            fields[name], keep[name] = arr(name)
        w = gf_weights(embed=weights["embed"].data_ptr(), lm_head=weights["lm_head"].data_ptr(),
                       final_norm=weights["final_norm"].data_ptr(), **fields)
        self.cfg = cfg
        self.max_batch, self.max_seq = max_batch, max_seq
        self.handle = gf_create(cfg, w, self.stream.cuda_stream)

    @property
    def s(self) -> int:
        return self.stream.cuda_stream

    def close(self):
        if getattr(self, "handle", None):
            gf_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- calls
    def prefill(self, ids, offsets, want_logits: bool = True):
        torch = self.torch
        off = _i32_host(offsets)
        B = len(off) - 1
        _check_ids(ids, "ids", int(off[-1]))
        handles = np.zeros(B, dtype=np.int32)
        logits = torch.empty(B, self.shape.vocab, dtype=torch.float32, device="cuda") if want_logits else None
        nxt = torch.empty(B, dtype=torch.int32, device="cuda")
        gf_prefill(self.handle, B, ids.data_ptr(), _ptr(off), _ptr(handles),
                   logits.data_ptr() if logits is not None else None, nxt.data_ptr(), self.s)
        return handles, logits, nxt

    def decode_step(self, handles, ids, want_logits: bool = True):
        torch = self.torch
        h = _i32_host(handles)
        B = len(h)
        _check_ids(ids, "ids", B)
        logits = torch.empty(B, self.shape.vocab, dtype=torch.float32, device="cuda") if want_logits else None
        nxt = torch.empty(B, dtype=torch.int32, device="cuda")
        gf_decode_step(self.handle, B, _ptr(h), ids.data_ptr(), logits.data_ptr() if logits is not None else None,
                       nxt.data_ptr(), self.s)
        return logits, nxt

    def release(self, handles):
        h = _i32_host(handles)
        gf_release(self.handle, len(h), _ptr(h))

    def forecast_batch(self, inc_ids, inc_offsets, cand_ids, cand_offsets, n_decode, verdict_ids, tau,
                       want_tokens=True, want_logits=False):
        torch = self.torch
        io, co, vid = _i32_host(inc_offsets), _i32_host(cand_offsets), _i32_host(verdict_ids)
        B, K = len(io) - 1, len(vid)
        _check_ids(inc_ids, "inc_ids", int(io[-1]))
        _check_ids(cand_ids, "cand_ids", int(co[-1]))
        p = torch.empty(B, K, dtype=torch.float32, device="cuda")
        conf = torch.empty(B, dtype=torch.float32, device="cuda")
        arg = torch.empty(B, dtype=torch.int32, device="cuda")
        defer = torch.empty(B, dtype=torch.uint8, device="cuda")
        toks = torch.empty(B, max(n_decode, 1), dtype=torch.int32, device="cuda") if want_tokens else None
        lg = torch.empty(B, self.shape.vocab, dtype=torch.float32, device="cuda") if want_logits else None
        gf_forecast_batch(self.handle, B, inc_ids.data_ptr(), _ptr(io), cand_ids.data_ptr(), _ptr(co), n_decode,
                          _ptr(vid), K, float(tau), p.data_ptr(), conf.data_ptr(), arg.data_ptr(), defer.data_ptr(),
                          toks.data_ptr() if toks is not None and n_decode > 0 else None,
                          lg.data_ptr() if lg is not None else None, self.s)
        return dict(p=p, conf=conf, arg=arg, defer=defer, tokens=toks, logits=lg)

    def forecast_batch_shared(self, prefix_ids, cand_ids, cand_offsets, n_decode, verdict_ids, tau, want_tokens=True,
                              want_logits=False):
        """Forecasts for candidates that all share one incumbent prefix (prefilled once)."""
        torch = self.torch
        co, vid = _i32_host(cand_offsets), _i32_host(verdict_ids)
        B, K = len(co) - 1, len(vid)
        _check_ids(prefix_ids, "prefix_ids", prefix_ids.numel())
        _check_ids(cand_ids, "cand_ids", int(co[-1]))
        p = torch.empty(B, K, dtype=torch.float32, device="cuda")
        conf = torch.empty(B, dtype=torch.float32, device="cuda")
        arg = torch.empty(B, dtype=torch.int32, device="cuda")
        defer = torch.empty(B, dtype=torch.uint8, device="cuda")
        toks = torch.empty(B, max(n_decode, 1), dtype=torch.int32, device="cuda") if want_tokens else None
        lg = torch.empty(B, self.shape.vocab, dtype=torch.float32, device="cuda") if want_logits else None
        gf_forecast_batch_shared(self.handle, B, prefix_ids.data_ptr() if prefix_ids.numel() else None,
                                 int(prefix_ids.numel()), cand_ids.data_ptr() if cand_ids.numel() else None, _ptr(co),
                                 n_decode, _ptr(vid), K, float(tau), p.data_ptr(), conf.data_ptr(), arg.data_ptr(),
                                 defer.data_ptr(), toks.data_ptr() if toks is not None and n_decode > 0 else None,
                                 lg.data_ptr() if lg is not None else None, self.s)
        return dict(p=p, conf=conf, arg=arg, defer=defer, tokens=toks, logits=lg)

    def forecast_batch_sampled(self, inc_ids, inc_offsets, cand_ids, cand_offsets, n_decode, verdict_ids, tau,
                               repeats=3, temperature=1.0, seed=0, want_tokens=True, want_logits=False):
        """Forecasts by temperature sampling, `repeats` rows per item (row = item * repeats + repeat),
        with the mean and population standard deviation of p and conf over each item's repeats."""
        torch = self.torch
        io, co, vid = _i32_host(inc_offsets), _i32_host(cand_offsets), _i32_host(verdict_ids)
        B, K = len(io) - 1, len(vid)
        _check_ids(inc_ids, "inc_ids", int(io[-1]))
        _check_ids(cand_ids, "cand_ids", int(co[-1]))
        BR = B * repeats
        f32 = dict(dtype=torch.float32, device="cuda")
        p, conf = torch.empty(BR, K, **f32), torch.empty(BR, **f32)
        arg = torch.empty(BR, dtype=torch.int32, device="cuda")
        defer = torch.empty(BR, dtype=torch.uint8, device="cuda")
        p_mean, p_std = torch.empty(B, K, **f32), torch.empty(B, K, **f32)
        conf_mean, conf_std = torch.empty(B, **f32), torch.empty(B, **f32)
        toks = torch.empty(BR, max(n_decode, 1), dtype=torch.int32, device="cuda") if want_tokens else None
        lg = torch.empty(BR, self.shape.vocab, **f32) if want_logits else None
        gf_forecast_batch_sampled(self.handle, B, inc_ids.data_ptr(), _ptr(io), cand_ids.data_ptr(), _ptr(co),
                                  n_decode, repeats, float(temperature), int(seed), _ptr(vid), K, float(tau),
                                  p.data_ptr(), conf.data_ptr(), arg.data_ptr(), defer.data_ptr(), p_mean.data_ptr(),
                                  p_std.data_ptr(), conf_mean.data_ptr(), conf_std.data_ptr(),
                                  toks.data_ptr() if toks is not None and n_decode > 0 else None,
                                  lg.data_ptr() if lg is not None else None, self.s)
        return dict(p=p, conf=conf, arg=arg, defer=defer, p_mean=p_mean, p_std=p_std, conf_mean=conf_mean,
                    conf_std=conf_std, tokens=toks, logits=lg)

    def free_pages(self) -> int:
        return gf_free_pages(self.handle)

    def forecast_batch_host(self, inc_ids, inc_offsets, cand_ids, cand_offsets, n_decode, verdict_ids, tau,
                            want_tokens=True):
        inc, cand = _i32_host(inc_ids), _i32_host(cand_ids)
        io, co, vid = _i32_host(inc_offsets), _i32_host(cand_offsets), _i32_host(verdict_ids)
        B, K = len(io) - 1, len(vid)
        p = np.zeros((B, K), dtype=np.float32)
        conf = np.zeros(B, dtype=np.float32)
        arg = np.zeros(B, dtype=np.int32)
        defer = np.zeros(B, dtype=np.uint8)
        toks = np.zeros((B, max(n_decode, 1)), dtype=np.int32) if want_tokens else None
        gf_forecast_batch_host(self.handle, B, _ptr(inc), _ptr(io), _ptr(cand), _ptr(co), n_decode, _ptr(vid), K,
                               float(tau), _ptr(p), _ptr(conf), _ptr(arg), _ptr(defer),
                               _ptr(toks) if toks is not None and n_decode > 0 else None, self.s)
        return dict(p=p, conf=conf, arg=arg, defer=defer, tokens=toks)

    def capture(self, layer: int, item: int, rows: int):
        """Arm a copy of the residual stream entering `layer` for batch item `item` (next call)."""
        buf = self.torch.zeros(rows, self.shape.d_model, dtype=self.torch.float32, device="cuda")
        gf_debug_capture(self.handle, layer, item, buf.data_ptr(), rows)
        return buf

    def read_kv(self, layer: int, handle: int, start: int, n: int):
        torch = self.torch
        k = torch.empty(n, self.shape.n_kv, self.shape.head_dim, dtype=torch.bfloat16, device="cuda")
        v = torch.empty_like(k)
        gf_debug_read_kv(self.handle, layer, handle, start, n, k.data_ptr(), v.data_ptr(), self.s)
        return k, v

    def status(self):
        gf_device_status(self.handle, self.s)

    def launch_count(self) -> int:
        return gf_launch_count(self.handle)

    def profile(self, mask: int):
        gf_profile_enable(self.handle, mask)

    def profile_read(self, kind: int) -> dict:
        return gf_profile_read(self.handle, kind)


def verdict(logits, verdict_ids, tau, stream=None):
    """Stand-alone verdict step on a [B, V] float32 CUDA tensor."""
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    vid = _i32_host(verdict_ids)
    _check_tensor(logits, "logits", dtype=torch.float32, rows_strided=True)
    B, K = logits.shape[0], len(vid)
    p = torch.empty(B, K, dtype=torch.float32, device=logits.device)
    conf = torch.empty(B, dtype=torch.float32, device=logits.device)
    arg = torch.empty(B, dtype=torch.int32, device=logits.device)
    defer = torch.empty(B, dtype=torch.uint8, device=logits.device)
    gf_verdict(B, logits.data_ptr(), logits.stride(0), _ptr(vid), K, float(tau), p.data_ptr(), conf.data_ptr(),
               arg.data_ptr(), defer.data_ptr(), s.cuda_stream)
    return p, conf, arg, defer
