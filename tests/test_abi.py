"""The C-ABI library: it builds, loads without a GPU, exports every declared
symbol, and rejects bad arguments before touching the device."""
import ctypes
import os
import re

import numpy as np
import pytest

import paper_2605_31464_gb300 as gf
from paper_2605_31464_gb300 import _build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    _build.build()
    return gf.load()


def declared_symbols():
    text = open(os.path.join(ROOT, "include", "gf.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(gf_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_boundary():
    syms = declared_symbols()
    for name in ("gf_prefill", "gf_decode_step", "gf_forecast_batch", "gf_forecast_batch_host", "gf_create",
                 "gf_destroy", "gf_release", "gf_verdict", "gf_last_error"):
        assert name in syms


def test_every_declared_symbol_is_exported(lib):
    for name in declared_symbols():
        assert hasattr(lib, name), name
    assert sorted(gf.EXPORTS) == sorted(declared_symbols())


def test_config_struct_layout():
    # int32 x7, float x2, int32 x2, int64 x2 with natural alignment
    assert ctypes.sizeof(gf.gf_config) == 64
    assert gf.gf_config.max_prefill_tokens.offset == 48
    assert ctypes.sizeof(gf.gf_weights) == 12 * ctypes.sizeof(ctypes.c_void_p)


def test_verdict_argument_validation_needs_no_gpu(lib):
    ids = np.array([10, 11], dtype=np.int32)
    dummy = ctypes.c_void_p(16)
    for K, tau in [(0, 0.5), (9, 0.5), (2, -0.1), (2, 1.5)]:
        with pytest.raises(gf.GfError) as e:
            gf.gf_verdict(1, dummy, 4096, ids.ctypes.data_as(ctypes.c_void_p), K, tau, dummy, dummy, dummy, dummy,
                          None)
        assert e.value.code == gf.GF_EINVAL
    bad = np.array([10, 5000], dtype=np.int32)
    with pytest.raises(gf.GfError):
        gf.gf_verdict(1, dummy, 4096, bad.ctypes.data_as(ctypes.c_void_p), 2, 0.5, dummy, dummy, dummy, dummy, None)
    assert "outside" in gf.gf_last_error()


def test_create_rejects_bad_configs_before_any_device_call(lib):
    w = gf.gf_weights()
    for kw in [dict(head_dim=96), dict(n_q=6, n_kv=4), dict(d_model=100), dict(vocab=1000)]:
        base = dict(layers=1, d_model=128, n_q=2, n_kv=2, head_dim=64, ffn=64, vocab=1024, rope_theta=1e4,
                    rms_eps=1e-6, max_batch=2, max_seq=64, max_prefill_tokens=64, kv_pages=0)
        base.update(kw)
        cfg = gf.gf_config(**base)
        with pytest.raises(gf.GfError) as e:
            gf.gf_create(cfg, w, None)
        assert e.value.code in (gf.GF_EINVAL, gf.GF_ENOTIMPL)


def test_null_model_calls_fail_cleanly(lib):
    with pytest.raises(gf.GfError):
        gf.gf_release(None, 1, None)
    with pytest.raises(gf.GfError):
        gf.gf_device_status(None, None)
    assert gf.gf_launch_count(None) == 0


def test_sampling_argument_validation_needs_no_gpu(lib):
    dummy = ctypes.c_void_p(16)
    for T, t, V, ld in [(0.0, 0, 8, 8), (float("nan"), 0, 8, 8), (float("inf"), 0, 8, 8), (1.0, -1, 8, 8),
                        (1.0, 0, 8, 4), (1.0, 0, 0, 8)]:
        with pytest.raises(gf.GfError) as e:
            gf.gf_sample_tokens(2, dummy, ld, V, 0, t, T, dummy, None)
        assert e.value.code == gf.GF_EINVAL
    off = np.array([0, 1], dtype=np.int32)
    vid = np.array([10, 11], dtype=np.int32)
    with pytest.raises(gf.GfError) as e:
        gf.gf_forecast_batch_sampled(None, 1, dummy, off.ctypes.data_as(ctypes.c_void_p), dummy,
                                     off.ctypes.data_as(ctypes.c_void_p), 4, 3, 1.0, 0,
                                     vid.ctypes.data_as(ctypes.c_void_p), 2, 0.8, dummy, dummy, dummy, dummy, None,
                                     None, None, None, None, None, None)
    assert e.value.code == gf.GF_EINVAL


def test_decode_attention_argument_validation_needs_no_gpu(lib):
    d = ctypes.c_void_p(256)
    ws = gf.gf_decode_attention_workspace(4, 2, 128, 1000)
    ok = dict(q=d, k=d, v=d, num_pages=64, table=d, max_pages=16, ctx=d, max_ctx=1000, B=4, n_q=8, n_kv=2, hd=128,
              out=d, ws=d, ws_bytes=ws)

    def call(**kw):
        a = dict(ok, **kw)
        return (a["q"], a["k"], a["v"], a["num_pages"], a["table"], a["max_pages"], a["ctx"], a["max_ctx"], a["B"],
                a["n_q"], a["n_kv"], a["hd"], a["out"])

    cases = [(dict(q=None), gf.GF_EINVAL), (dict(B=0), gf.GF_EINVAL), (dict(n_q=6, n_kv=4), gf.GF_EINVAL),
             (dict(n_q=34, n_kv=2), gf.GF_EINVAL), (dict(hd=96), gf.GF_ENOTIMPL),
             (dict(max_ctx=16 * 64 + 1), gf.GF_EINVAL), (dict(num_pages=0), gf.GF_EINVAL),
             (dict(num_pages=1 << 26), gf.GF_EINVAL)]
    for kw, code in cases:
        for static in (False, True):
            with pytest.raises(gf.GfError) as e:
                if static:
                    gf.gf_decode_attention_static(*call(**kw), None)
                else:
                    gf.gf_decode_attention(*call(**kw), ok["ws"], ok["ws_bytes"], None)
            assert e.value.code == code, (kw, static)
    with pytest.raises(gf.GfError) as e:
        gf.gf_decode_attention(*call(), d, ws - 1, None)
    assert e.value.code == gf.GF_EINVAL
    # the fixed scratch of the allocation-free variant (16 MiB) bounds its problem size
    big = dict(B=512, n_kv=8, max_ctx=16384, max_pages=256, num_pages=4096)
    assert gf.gf_decode_attention_workspace(512, 8, 128, 16384) > 16 << 20
    with pytest.raises(gf.GfError) as e:
        gf.gf_decode_attention_static(*call(**big), None)
    assert e.value.code == gf.GF_ECAPACITY


def test_decode_attention_workspace_covers_every_chunking():
    # partial results: 16 query rows x (head_dim outputs + max + sum) floats per (sequence, kv head, chunk);
    # chunks are at least 256 keys, so the 256-key count bounds every plan
    for B, n_kv, hd, ctx in [(1, 1, 64, 1), (4, 2, 128, 1000), (32, 4, 128, 6400), (128, 4, 128, 4096)]:
        ws = gf.gf_decode_attention_workspace(B, n_kv, hd, ctx)
        for chunk in (256, 512, 1024):
            assert ws >= B * n_kv * -(-ctx // chunk) * 16 * (hd + 2) * 4
        assert gf.gf_decode_attention_workspace(2 * B, n_kv, hd, ctx) == 2 * ws
    assert gf.gf_decode_attention_workspace(0, 1, 128, 64) == 0


def test_gemm_argument_validation_needs_no_gpu(lib):
    d = ctypes.c_void_p(256)
    ok = dict(A=d, W=d, M=32, N=256, K=128, out=d, ldo=256, mode=gf.GF_GEMM_STORE_F32, bn=0, splits=0, group_m=0)
    cases = [dict(A=None), dict(out=None), dict(N=0), dict(K=32), dict(K=96), dict(N=48), dict(mode=5),
             dict(mode=-1), dict(bn=96), dict(bn=32), dict(splits=2), dict(ldo=255),
             dict(mode=gf.GF_GEMM_SWIGLU, ldo=127)]
    for kw in cases:
        a = dict(ok, **kw)
        with pytest.raises(gf.GfError) as e:
            gf.gf_gemm_bf16(a["A"], a["W"], a["M"], a["N"], a["K"], a["out"], a["ldo"], a["mode"], a["bn"],
                            a["splits"], a["group_m"], None)
        assert e.value.code == gf.GF_EINVAL, kw
    # an empty product is a no-op (no device work)
    gf.gf_gemm_bf16(d, d, 0, 256, 128, d, 256, gf.GF_GEMM_STORE_F32, 0, 0, 0, None)


def test_select_and_selftest_argument_validation_needs_no_gpu(lib):
    d = ctypes.c_void_p(256)
    for B, tau, p in [(0, 0.5, d), (1025, 0.5, d), (4, -0.1, d), (4, 1.5, d), (4, float("nan"), d), (4, 0.5, None)]:
        with pytest.raises(gf.GfError) as e:
            gf.gf_select(B, p, d, 1.5, tau, d, d, d, d, None)
        assert e.value.code == gf.GF_EINVAL, (B, tau)
    assert gf.gf_selftest_timeout(0, None) == gf.GF_EINVAL
    assert gf.gf_selftest_timeout(2001, None) == gf.GF_EINVAL
