"""Shared-incumbent prefix reuse (gf_forecast_batch_shared) vs the plain path and the oracle.

Every candidate of a search step shares the reference kernel r of
x_i = (r, k_i, h) (Sec. 2.1).  The shared path prefills the prefix's full
64-token pages once and points every candidate's block table at them; its
forecasts must match the plain path (each prompt prefilled in full) and the
oracle, for prefix lengths that are, are not, and are less than a multiple of
the page size, and the page pool must get every page back.
"""
import numpy as np
import pytest

import oracle
import synth
from _helpers import check_logits, check_verdict, make_model

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

GQA = synth.ModelShape(layers=2, d_model=512, n_q=8, n_kv=2, head_dim=128, ffn=1000, vocab=2048, rope_theta=1e6)


@pytest.fixture(scope="module")
def model():
    from paper_2605_31464_gb300 import _build
    _build.build()
    m = make_model(GQA, max_batch=8, max_seq=1024, max_prefill_tokens=4096)
    yield m, oracle.Weights(GQA)
    m.close()


def _cuda(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.int32)).cuda()


@pytest.mark.parametrize("prefix_len", [192, 200, 30, 64])
def test_shared_prefix_matches_plain_path_and_oracle(model, prefix_len):
    m, W = model
    prefix = synth.zipf_ids(4, 1, prefix_len, GQA.vocab)
    cands = [synth.zipf_ids(4, 10 + i, n, GQA.vocab) for i, n in enumerate([50, 1, 130, 77])]
    B = len(cands)
    cand = np.concatenate(cands).astype(np.int32)
    co = np.concatenate([[0], np.cumsum([len(c) for c in cands])]).astype(np.int32)
    n_dec, vid, tau = 6, (10, 11, 12), 0.5
    free0 = m.free_pages()
    sh = m.forecast_batch_shared(_cuda(prefix), _cuda(cand), co, n_dec, vid, tau, want_tokens=True, want_logits=True)
    torch.cuda.synchronize()
    m.status()
    assert m.free_pages() == free0, "pages leaked by the shared path"
    inc = np.concatenate([prefix] * B).astype(np.int32)
    io = np.arange(B + 1, dtype=np.int32) * prefix_len
    pl = m.forecast_batch(_cuda(inc), io, _cuda(cand), co, n_dec, vid, tau, want_tokens=True, want_logits=True)
    torch.cuda.synchronize()
    toks = sh["tokens"].cpu().numpy()
    for i in range(B):
        prompt = np.concatenate([prefix, cands[i]])
        ref = oracle.forecast_one(W, prompt, n_dec, vid, tau, forced_tokens=toks[i])
        check_logits(sh["logits"][i].cpu().numpy(), ref["step_logits"][-1], f"shared item {i}")
        check_verdict(sh["p"][i].cpu().numpy(), sh["conf"][i].item(), sh["arg"][i].item(), sh["defer"][i].item(),
                      ref["p"], ref["conf"], ref["arg"], ref["defer"], tau)
        if np.array_equal(toks[i], pl["tokens"][i].cpu().numpy()):
            np.testing.assert_allclose(sh["logits"][i].cpu().numpy(), pl["logits"][i].cpu().numpy(), atol=2e-2,
                                       rtol=2e-2)


def test_shared_prefix_rejects_prompts_without_own_tokens(model):
    import paper_2605_31464_gb300 as gf
    m, _ = model
    prefix = synth.zipf_ids(4, 1, 128, GQA.vocab)
    with pytest.raises(gf.GfError):
        m.forecast_batch_shared(_cuda(prefix), _cuda(np.zeros(0, np.int32)), [0, 0], 2, (10, 11), 0.5)
