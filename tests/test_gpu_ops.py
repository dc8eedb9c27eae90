"""Building blocks through the C ABI vs the oracle's definitions.

* gf_gemm_bf16: every epilogue, every tile width, split-K, ragged M and N
  tails and long K, against a float64 matmul of the same bf16 operands.
* gf_decode_attention: paged decode attention over a shuffled page pool with
  ragged context lengths (1 key, page-boundary lengths, several 256-key
  chunks), against the oracle's explicit-softmax attention.
"""
import numpy as np
import pytest

import oracle
import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2605_31464_gb300 import _build
    _build.build()
    assert torch.cuda.is_available()


def _bf16(shape, seed, scale=1.0):
    bits = synth.normal_bf16(seed, 77, int(np.prod(shape)), scale).reshape(shape)
    t = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).cuda()
    return t, oracle.bf16_bits_to_f64(bits)


def _gemm_ref(a64, w64):
    return a64 @ w64.T


@pytest.mark.parametrize("M,N,K", [(1, 256, 64), (7, 4608, 3584), (128, 256, 128), (129, 96, 192),
                                   (1000, 768, 256), (300, 1408, 1024)])
@pytest.mark.parametrize("bn", [64, 128, 256])
def test_gemm_store_f32(M, N, K, bn):
    import paper_2605_31464_gb300 as gf
    A, a64 = _bf16((M, K), 1)
    W, w64 = _bf16((N, K), 2, 0.05)
    out = torch.full((M, N), float("nan"), device="cuda")
    gf.gemm(A, W, out, gf.GF_GEMM_STORE_F32, bn=bn, splits=1)
    gf.gf_gemm_status(torch.cuda.current_stream().cuda_stream)
    ref = _gemm_ref(a64, w64)
    np.testing.assert_allclose(out.cpu().numpy(), ref, rtol=1e-4, atol=1e-4 * np.abs(ref).max())


@pytest.mark.parametrize("splits", [1, 3, 8])
def test_gemm_split_k_atomic_accumulates(splits):
    import paper_2605_31464_gb300 as gf
    M, N, K = 33, 512, 2048
    A, a64 = _bf16((M, K), 3)
    W, w64 = _bf16((N, K), 4, 0.05)
    base = torch.randn(M, N, device="cuda", dtype=torch.float64).float()
    out = base.clone()
    gf.gemm(A, W, out, gf.GF_GEMM_ATOMIC_F32, bn=64, splits=splits)
    gf.gf_gemm_status(torch.cuda.current_stream().cuda_stream)
    ref = base.cpu().double().numpy() + _gemm_ref(a64, w64)
    np.testing.assert_allclose(out.cpu().numpy(), ref, rtol=1e-4, atol=1e-4 * np.abs(ref).max())


def test_gemm_residual_add_and_bf16_store():
    import paper_2605_31464_gb300 as gf
    M, N, K = 700, 512, 576
    A, a64 = _bf16((M, K), 5)
    W, w64 = _bf16((N, K), 6, 0.05)
    base = torch.randn(M, N, device="cuda")
    out = base.clone()
    gf.gemm(A, W, out, gf.GF_GEMM_ADD_F32, bn=256)
    ref = base.cpu().double().numpy() + _gemm_ref(a64, w64)
    np.testing.assert_allclose(out.cpu().numpy(), ref, rtol=1e-4, atol=1e-4 * np.abs(ref).max())
    ob = torch.zeros(M, N, device="cuda", dtype=torch.bfloat16)
    gf.gemm(A, W, ob, gf.GF_GEMM_STORE_BF16, bn=128)
    r2 = _gemm_ref(a64, w64)
    np.testing.assert_allclose(ob.float().cpu().numpy(), r2, rtol=8e-3, atol=8e-3 * np.abs(r2).max())


@pytest.mark.parametrize("bn", [128, 256])
def test_gemm_swiglu_epilogue(bn):
    import paper_2605_31464_gb300 as gf
    M, F, K = 260, 208, 320  # F = 13 blocks of 16
    A, a64 = _bf16((M, K), 7)
    G, g64 = _bf16((F, K), 8, 0.05)
    U, u64 = _bf16((F, K), 9, 0.05)
    # interleave blocks of 16 rows: gate block c, then up block c
    Wi = torch.cat([torch.cat([G[16 * c:16 * c + 16], U[16 * c:16 * c + 16]]) for c in range(F // 16)])
    out = torch.zeros(M, F, device="cuda", dtype=torch.bfloat16)
    gf.gemm(A, Wi, out, gf.GF_GEMM_SWIGLU, bn=bn)
    g = a64 @ g64.T
    ref = oracle.silu(g) * (a64 @ u64.T)
    np.testing.assert_allclose(out.float().cpu().numpy(), ref, rtol=1e-2, atol=1e-2 * np.abs(ref).max())


@pytest.mark.parametrize("M", [1, 7, 32, 33, 100, 128])
@pytest.mark.parametrize("mode", ["f32", "atomic", "swiglu"])
def test_gemm_few_rows_swapped_operands(M, mode):
    # with few rows (decode) the library puts the weights in the 128-row MMA operand
    import paper_2605_31464_gb300 as gf
    N, K = (4608 if mode != "swiglu" else 1024), 1024
    A, a64 = _bf16((M, K), 11)
    W, w64 = _bf16((N, K), 12, 0.05)
    if mode == "swiglu":
        out = torch.zeros(M, N // 2, device="cuda", dtype=torch.bfloat16)
        gf.gemm(A, W, out, gf.GF_GEMM_SWIGLU)
        gu = a64 @ w64.T
        g = np.concatenate([gu[:, 32 * c:32 * c + 16] for c in range(N // 32)], axis=1)
        u = np.concatenate([gu[:, 32 * c + 16:32 * c + 32] for c in range(N // 32)], axis=1)
        ref = oracle.silu(g) * u
        got = out.float().cpu().numpy()
        np.testing.assert_allclose(got, ref, rtol=1e-2, atol=1e-2 * np.abs(ref).max())
        return
    base = torch.randn(M, N, device="cuda") if mode == "atomic" else torch.zeros(M, N, device="cuda")
    out = base.clone()
    gf.gemm(A, W, out, gf.GF_GEMM_ATOMIC_F32 if mode == "atomic" else gf.GF_GEMM_STORE_F32)
    gf.gf_gemm_status(torch.cuda.current_stream().cuda_stream)
    ref = base.cpu().double().numpy() + a64 @ w64.T
    np.testing.assert_allclose(out.cpu().numpy(), ref, rtol=1e-4, atol=1e-4 * np.abs(ref).max())


def test_gemm_rejects_bad_shapes():
    import paper_2605_31464_gb300 as gf
    A, _ = _bf16((4, 96), 1)
    W, _ = _bf16((64, 96), 2)
    out = torch.zeros(4, 64, device="cuda")
    with pytest.raises(gf.GfError):
        gf.gemm(A, W, out)  # K not a multiple of 64


# ----------------------------------------------------------------------------- decode attention

def make_paged(ctx, n_kv, hd, seed, page_order_seed=11):
    """Random K/V for each sequence, stored in a shuffled pool of 64-token pages."""
    B = len(ctx)
    pages_per = [(c + 63) // 64 for c in ctx]
    max_pages = max(pages_per)
    n_pages = sum(pages_per) + 3
    perm = np.random.default_rng(page_order_seed).permutation(n_pages)
    kbits = synth.normal_bf16(seed, 1, n_pages * n_kv * 64 * hd, 1.0).reshape(n_pages, n_kv, 64, hd)
    vbits = synth.normal_bf16(seed, 2, n_pages * n_kv * 64 * hd, 1.0).reshape(n_pages, n_kv, 64, hd)
    table = np.zeros((B, max_pages), dtype=np.int32)
    nxt = 0
    for b in range(B):
        for j in range(pages_per[b]):
            table[b, j] = perm[nxt]
            nxt += 1
    dense = []
    for b in range(B):
        idx = table[b, :pages_per[b]]
        k = oracle.bf16_bits_to_f64(kbits[idx]).transpose(0, 2, 1, 3).reshape(-1, n_kv, hd)[:ctx[b]]
        v = oracle.bf16_bits_to_f64(vbits[idx]).transpose(0, 2, 1, 3).reshape(-1, n_kv, hd)[:ctx[b]]
        dense.append((k, v))
    to = lambda x: torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).view(torch.bfloat16).cuda()
    # the value cache holds each page transposed: [page][kv head][hd][64 tokens]
    return to(kbits), to(vbits.transpose(0, 1, 3, 2)), torch.from_numpy(table).cuda(), dense, max_pages


@pytest.mark.parametrize("n_q,n_kv,hd", [(28, 4, 128), (12, 2, 128), (4, 4, 64), (40, 8, 128)])
def test_decode_attention_matches_oracle(n_q, n_kv, hd):
    import paper_2605_31464_gb300 as gf
    ctx = [1, 63, 64, 65, 256, 257, 700, 1500]
    kc, vc, table, dense, max_pages = make_paged(ctx, n_kv, hd, seed=5)
    qbits = synth.normal_bf16(6, 3, len(ctx) * n_q * hd, 1.0).reshape(len(ctx), n_q, hd)
    q = torch.from_numpy(qbits.view(np.int16)).view(torch.bfloat16).cuda().reshape(len(ctx), n_q * hd)
    ctx_d = torch.tensor(ctx, dtype=torch.int32, device="cuda")
    out = gf.decode_attention(q, kc, vc, table, ctx_d, max(ctx), n_q, n_kv)
    gf.gf_gemm_status(torch.cuda.current_stream().cuda_stream)
    got = out.float().cpu().numpy().reshape(len(ctx), n_q, hd)
    q64 = oracle.bf16_bits_to_f64(qbits)
    for b, c in enumerate(ctx):
        k, v = dense[b]
        ref = oracle.attention(q64[b][None], k, v, np.array([c - 1]), np.arange(c))[0]
        np.testing.assert_allclose(got[b], ref, atol=2e-2, rtol=2e-2, err_msg=f"ctx {c}")
