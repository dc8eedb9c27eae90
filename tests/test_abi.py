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
