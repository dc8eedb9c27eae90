"""gf_decode_attention_static: decode attention that allocates nothing.

Some callers cannot allocate device memory where they run decode attention:
their memory is already reserved by another allocator, or they must not call
cudaMalloc/cudaFree (which can synchronise the whole device) once they are
running.  For them the library keeps the kernel's scratch in a fixed device
array.  This file checks, through the C ABI:
  - two calls in a row on the same case give identical results, equal to the
    float64 oracle's attention and to gf_decode_attention (which takes a
    caller workspace) within the attention tolerance;
  - a small call between two large ones is not disturbed by what the large
    call left in the shared array, nor disturbs the next large call;
  - a request larger than the fixed array is refused;
  - a bounded wait that runs out is reported by the entry point's own status
    query, which then clears it.
It is collected last so that a stop at the first failure has already run every
other test.
"""
import ctypes

import numpy as np
import pytest

import oracle
import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

ATOL = RTOL = 2e-2  # the decode-attention tolerance of the other GPU tests (bf16 P and output)


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2605_31464_gb300 import _build
    _build.build()
    assert torch.cuda.is_available()


def _paged_case(ctx, n_q, n_kv, hd, seed):
    """Random bf16 queries and K/V pages (a shuffled pool); also the dense float64 copies."""
    B = len(ctx)
    pages_per = [(c + 63) // 64 for c in ctx]
    max_pages = max(pages_per)
    n_pages = sum(pages_per) + 2
    perm = np.random.default_rng(seed).permutation(n_pages)
    table = np.zeros((B, max_pages), dtype=np.int32)
    k = 0
    for b in range(B):
        for j in range(pages_per[b]):
            table[b, j] = perm[k]
            k += 1
    kbits = synth.normal_bf16(seed, 1, n_pages * n_kv * 64 * hd, 1.0).reshape(n_pages, n_kv, 64, hd)
    vtbits = synth.normal_bf16(seed, 2, n_pages * n_kv * 64 * hd, 1.0).reshape(n_pages, n_kv, hd, 64)
    qbits = synth.normal_bf16(seed, 3, B * n_q * hd, 1.0).reshape(B, n_q, hd)
    dense = []
    for b in range(B):
        idx = table[b, :pages_per[b]]
        kd = oracle.bf16_bits_to_f64(kbits[idx]).transpose(0, 2, 1, 3).reshape(-1, n_kv, hd)[:ctx[b]]
        vd = oracle.bf16_bits_to_f64(vtbits[idx]).transpose(0, 3, 1, 2).reshape(-1, n_kv, hd)[:ctx[b]]
        dense.append((kd, vd))

    def dev(bits):
        return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()

    return dict(q=dev(qbits).reshape(B, n_q * hd), kc=dev(kbits), vc=dev(vtbits), table=torch.from_numpy(table).cuda(),
                ctx=torch.tensor(ctx, dtype=torch.int32, device="cuda"), ctx_list=list(ctx), max_ctx=max(ctx), B=B,
                n_q=n_q, n_kv=n_kv, hd=hd, n_pages=n_pages, max_pages=max_pages, q64=oracle.bf16_bits_to_f64(qbits),
                dense=dense)


def _stream():
    return torch.cuda.current_stream().cuda_stream


def _with_workspace(c):
    import paper_2605_31464_gb300 as gf
    out = gf.decode_attention(c["q"], c["kc"], c["vc"], c["table"], c["ctx"], c["max_ctx"], c["n_q"], c["n_kv"])
    gf.gf_gemm_status(_stream())
    return out.float().cpu().numpy()


def _without_allocation(c):
    import paper_2605_31464_gb300 as gf
    out = torch.full_like(c["q"], float("nan"))
    gf.gf_decode_attention_static(c["q"].data_ptr(), c["kc"].data_ptr(), c["vc"].data_ptr(), c["n_pages"],
                                  c["table"].data_ptr(), c["max_pages"], c["ctx"].data_ptr(), c["max_ctx"], c["B"],
                                  c["n_q"], c["n_kv"], c["hd"], out.data_ptr(), _stream())
    assert gf.gf_decode_attention_static_status(_stream()) == gf.GF_OK, gf.gf_last_error()
    got = out.float().cpu().numpy()
    assert np.isfinite(got).all()
    return got


def _check_oracle(got, c):
    g = got.reshape(c["B"], c["n_q"], c["hd"])
    for b, n in enumerate(c["ctx_list"]):
        k, v = c["dense"][b]
        ref = oracle.attention(c["q64"][b][None], k, v, np.array([n - 1]), np.arange(n))[0]
        np.testing.assert_allclose(g[b], ref, atol=ATOL, rtol=RTOL, err_msg=f"context {n}")


def _large():
    return _paged_case([1, 64, 65, 300, 1000, 2100], n_q=28, n_kv=4, hd=128, seed=21)


def _small():
    return _paged_case([700, 5, 128], n_q=4, n_kv=4, hd=64, seed=22)


@pytest.mark.parametrize("make", [_large, _small], ids=["gqa_hd128", "mha_hd64"])
def test_two_calls_in_a_row_match_the_oracle_and_the_workspace_entry_point(make):
    c = make()
    first = _without_allocation(c)
    second = _without_allocation(c)
    np.testing.assert_array_equal(first, second)
    _check_oracle(first, c)
    np.testing.assert_allclose(first, _with_workspace(c), atol=ATOL, rtol=RTOL)


def test_a_small_call_between_large_ones_is_unaffected_by_the_shared_array():
    big, small = _large(), _small()
    a = _without_allocation(big)
    b = _without_allocation(small)
    c = _without_allocation(big)
    np.testing.assert_allclose(a, _with_workspace(big), atol=ATOL, rtol=RTOL)
    np.testing.assert_allclose(b, _with_workspace(small), atol=ATOL, rtol=RTOL)
    _check_oracle(b, small)
    np.testing.assert_array_equal(a, c)


def test_oversized_request_is_refused():
    import paper_2605_31464_gb300 as gf
    assert gf.gf_decode_attention_workspace(512, 8, 128, 16384) > 16 << 20
    dummy = ctypes.c_void_p(256)
    with pytest.raises(gf.GfError) as e:
        gf.gf_decode_attention_static(dummy, dummy, dummy, 4096, dummy, 256, dummy, 16384, 512, 40, 8, 128, dummy,
                                      None)
    assert e.value.code == gf.GF_ECAPACITY
    assert "scratch" in gf.gf_last_error()


def test_a_timed_out_wait_is_reported_once_by_the_status_query():
    import paper_2605_31464_gb300 as gf
    s = _stream()
    # a kernel waits on a barrier that nothing completes; after 50 ms it records the timeout in the
    # entry point's word and returns
    assert gf.gf_selftest_timeout_static(50, s) == gf.GF_ETIMEOUT
    assert "timed out" in gf.gf_last_error()
    assert gf.gf_selftest_timeout_static(0, s) == gf.GF_EINVAL
    # the query cleared the word, and the entry point still computes correctly
    assert gf.gf_decode_attention_static_status(s) == gf.GF_OK
    c = _small()
    _check_oracle(_without_allocation(c), c)
