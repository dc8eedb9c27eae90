"""gf_decode_attention_static: decode attention that allocates nothing.

Some callers cannot allocate device memory where they run decode attention
(their memory is already reserved by another allocator, or they must not
call cudaMalloc/cudaFree, which can synchronise the device, after start-up).
For them the library keeps the kernel's scratch in a fixed device array.
This file checks, through the C ABI, that two calls in a row give the same
results as gf_decode_attention (which takes a caller workspace), and that a
request larger than the fixed array is refused.  It is collected last so
that a stop at the first failure has already run every other test.
"""
import ctypes

import numpy as np
import pytest

import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

ATOL = RTOL = 2e-2  # the attention tolerance the other GPU tests use


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2605_31464_gb300 import _build
    _build.build()
    assert torch.cuda.is_available()


def _paged_case(ctx, n_q, n_kv, hd, seed):
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

    def bf16(stream, n):
        bits = synth.normal_bf16(seed, stream, n, 1.0)
        return torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).cuda()

    kc = bf16(1, n_pages * n_kv * 64 * hd).reshape(n_pages, n_kv, 64, hd)
    vc = bf16(2, n_pages * n_kv * 64 * hd).reshape(n_pages, n_kv, hd, 64)  # pages stored transposed
    q = bf16(3, B * n_q * hd).reshape(B, n_q * hd)
    return dict(q=q, kc=kc, vc=vc, table=torch.from_numpy(table).cuda(),
                ctx=torch.tensor(ctx, dtype=torch.int32, device="cuda"), max_ctx=max(ctx), B=B, n_q=n_q, n_kv=n_kv,
                hd=hd, n_pages=n_pages, max_pages=max_pages)


def _with_workspace(c):
    import paper_2605_31464_gb300 as gf
    return gf.decode_attention(c["q"], c["kc"], c["vc"], c["table"], c["ctx"], c["max_ctx"], c["n_q"], c["n_kv"])


def _without_allocation(c):
    import paper_2605_31464_gb300 as gf
    out = torch.full_like(c["q"], float("nan"))
    gf.gf_decode_attention_static(c["q"].data_ptr(), c["kc"].data_ptr(), c["vc"].data_ptr(), c["n_pages"],
                                  c["table"].data_ptr(), c["max_pages"], c["ctx"].data_ptr(), c["max_ctx"], c["B"],
                                  c["n_q"], c["n_kv"], c["hd"], out.data_ptr(),
                                  torch.cuda.current_stream().cuda_stream)
    return out


def test_two_calls_in_a_row_match_the_workspace_entry_point():
    import paper_2605_31464_gb300 as gf
    cases = [_paged_case([1, 64, 65, 300, 1000, 2100], n_q=28, n_kv=4, hd=128, seed=21),
             _paged_case([700, 5, 128], n_q=4, n_kv=4, hd=64, seed=22)]
    for c in cases:
        got = _without_allocation(c)
        ref = _with_workspace(c)
        gf.gf_gemm_status(torch.cuda.current_stream().cuda_stream)
        torch.cuda.synchronize()
        g, r = got.float().cpu().numpy(), ref.float().cpu().numpy()
        assert np.isfinite(g).all()
        np.testing.assert_allclose(g, r, atol=ATOL, rtol=RTOL)


def test_oversized_request_is_refused():
    import paper_2605_31464_gb300 as gf
    assert gf.gf_decode_attention_workspace(512, 8, 128, 16384) > 16 << 20
    dummy = ctypes.c_void_p(256)
    with pytest.raises(gf.GfError) as e:
        gf.gf_decode_attention_static(dummy, dummy, dummy, 4096, dummy, 256, dummy, 16384, 512, 40, 8, 128, dummy,
                                      None)
    assert e.value.code == gf.GF_ECAPACITY
    assert "scratch" in gf.gf_last_error()
