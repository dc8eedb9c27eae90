"""gf_select (8-bin expected speedup, ranking, discovery score) vs oracle.selection,
and an end-to-end 8-bin forecast: K = 8 verdict ids through gf_forecast_batch."""
import numpy as np
import pytest

import oracle
import synth
from oracle import selection as sel
from _helpers import check_verdict, make_model

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2605_31464_gb300 import _build
    _build.build()


@pytest.mark.parametrize("B", [1, 7, 300, 1024])
@pytest.mark.parametrize("x,tau", [(1.25, 0.3), (1.5, 0.5), (2.0, 0.7)])
def test_select_matches_oracle(B, x, tau):
    import paper_2605_31464_gb300 as gf
    rng = np.random.default_rng(B)
    z = rng.normal(size=(B, 8)) * 2
    p = np.exp(z - z.max(1, keepdims=True))
    p /= p.sum(1, keepdims=True)
    p = p.astype(np.float32)
    if B > 4:
        p[3] = p[1]  # a tie in the expected speedup
    m = sel.representatives(0.15, 6.0)
    s_hat, order, disc, pred = gf.select(torch.from_numpy(p).cuda(), m.astype(np.float32), x, tau)
    p64 = p.astype(np.float64)
    ref_s = sel.expected_speedup(p64, m)
    np.testing.assert_allclose(s_hat.cpu().numpy(), ref_s, rtol=1e-5, atol=1e-6)
    got_order = order.cpu().numpy()
    # the order is unique up to values within float rounding; check it sorts the GPU's own values
    g = s_hat.cpu().numpy()
    assert sorted(got_order.tolist()) == list(range(B))
    for a, b in zip(got_order[:-1], got_order[1:]):
        assert g[a] > g[b] or (g[a] == g[b] and a < b)
    # and agrees with the oracle's ranking wherever the oracle's values are not near-ties
    ref_order = sel.ranking(ref_s)
    gaps = np.abs(np.diff(ref_s[ref_order]))
    if B > 1 and gaps.min() > 1e-5:
        np.testing.assert_array_equal(got_order, ref_order)
    ref_d = sel.discovery_score(p64, x)
    np.testing.assert_allclose(disc.cpu().numpy(), ref_d, atol=1e-6)
    far = np.abs(ref_d - tau) > 1e-6
    np.testing.assert_array_equal(pred.cpu().numpy()[far], sel.discovery_predict(ref_d, tau)[far])


def test_eight_bin_forecast_end_to_end():
    import paper_2605_31464_gb300 as gf
    shape = synth.SHAPE_TINY
    w = synth.workload("tiny", n_decode=3)
    m = make_model(shape, max_batch=8, max_seq=300, max_prefill_tokens=4096)
    W = oracle.Weights(shape)
    vid = tuple(range(100, 108))   # one token id per speedup bin
    inc, io, cand, co = synth.prompts(w)
    out = m.forecast_batch(torch.from_numpy(inc).cuda(), io, torch.from_numpy(cand).cuda(), co, w.n_decode, vid,
                           0.3, want_tokens=True)
    reps = sel.representatives(0.15, 6.0)
    s_hat, order, disc, pred = gf.select(out["p"], reps.astype(np.float32), 2.0, 0.5)
    torch.cuda.synchronize()
    ids, off = synth.packed_prompts(w)
    toks = out["tokens"].cpu().numpy()
    for i in range(w.batch):
        ref = oracle.forecast_one(W, ids[off[i]:off[i + 1]], w.n_decode, vid, 0.3, forced_tokens=toks[i])
        check_verdict(out["p"][i].cpu().numpy(), out["conf"][i].item(), out["arg"][i].item(), out["defer"][i].item(),
                      ref["p"], ref["conf"], ref["arg"], ref["defer"], 0.3)
        assert abs(s_hat[i].item() - sel.expected_speedup(ref["p"][None], reps)[0]) < 1e-2 * reps.max()
        assert abs(disc[i].item() - sel.discovery_score(ref["p"][None], 2.0)[0]) < 2e-2
    m.close()
