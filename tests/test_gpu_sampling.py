"""Temperature sampling with repeats (Sec. 3.1 setup) through the C ABI vs the oracle.

* gf_sample_tokens: the device draw equals the oracle's Gumbel-max draw on
  the same float32 logits (counter-based uniforms, so both sides see the
  same noise); the two may part only where the perturbed scores of the top
  two ids lie within float32 rounding of each other.
* gf_forecast_batch_sampled, teacher-forced: the oracle replays each row's
  sampled tokens; final logits, every draw (up to the greedy tie band),
  the per-row verdict and the repeat statistics are compared.  Prompts are
  ragged so that forks copy partial KV pages, and whole pages are shared.
* Determinism in (seed, row), distinct repeats, page bookkeeping, argument
  checks, and the vanishing-temperature limit (the greedy first token).
"""
import numpy as np
import pytest

import oracle
from oracle import sampling as smp
import synth
from _helpers import ARGMAX_GAP, check_logits, check_verdict, make_model

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

GQA = synth.ModelShape(layers=2, d_model=512, n_q=8, n_kv=2, head_dim=128, ffn=1000, vocab=2048, rope_theta=1e6)
VIDS = (10, 11)
TAU = 0.8


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2605_31464_gb300 import _build
    _build.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"


def _cuda_i32(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.int32)).cuda()


def _draw_agrees(gpu_tok, scores, band):
    top = int(np.argmax(scores))
    return gpu_tok == top or scores[top] - scores[gpu_tok] < band


@pytest.mark.parametrize("T", [1.0, 0.7, 3.0])
@pytest.mark.parametrize("seed,t", [(0, 0), (2 ** 64 - 7, 5), (12345, 255)])
def test_sample_tokens_match_the_oracle_draw(T, seed, t):
    import paper_2605_31464_gb300 as gf
    B, V = 13, 5000  # a ragged group of four rows and a ragged last pass over the vocabulary
    logits = np.random.default_rng(seed % 1000 + t).normal(0.0, 2.0, size=(B, V)).astype(np.float32)
    got = gf.sample_tokens(torch.from_numpy(logits).cuda(), seed, t, T).cpu().numpy()
    exact = 0
    for r in range(B):
        sc = smp.sample_scores(logits[r].astype(np.float64), T, smp.uniforms(seed, t, r, V))
        assert _draw_agrees(int(got[r]), sc, 1e-4 * (1 + np.abs(sc).max())), f"row {r}"
        exact += int(got[r]) == int(np.argmax(sc))
    assert exact >= B - 1


def test_sample_tokens_spread_like_the_softmax():
    import paper_2605_31464_gb300 as gf
    V, rows = 4, 4096
    base = np.log(np.array([1.0, 2.0, 3.0, 4.0], dtype=np.float32))
    logits = torch.from_numpy(np.tile(base, (rows, 1))).cuda()
    got = gf.sample_tokens(logits, 77, 0, 1.0).cpu().numpy()
    freq = np.bincount(got, minlength=V) / rows
    target = np.array([0.1, 0.2, 0.3, 0.4])
    assert np.all(np.abs(freq - target) < 5 * np.sqrt(target * (1 - target) / rows)), freq


def test_sample_tokens_rejects_bad_arguments():
    import paper_2605_31464_gb300 as gf
    x = torch.zeros(2, 64, device="cuda")
    for T in (0.0, -1.0, float("nan"), float("inf")):
        with pytest.raises(gf.GfError):
            gf.sample_tokens(x, 0, 0, T)
    with pytest.raises(gf.GfError):
        gf.sample_tokens(x, 0, -1, 1.0)


@pytest.fixture(scope="module")
def tiny():
    w = synth.workload("tiny")
    m = make_model(w.model, max_batch=16, max_seq=512, max_prefill_tokens=4096)
    yield w.model, m, oracle.Weights(w.model)
    m.close()


@pytest.fixture(scope="module")
def gqa():
    m = make_model(GQA, max_batch=16, max_seq=1024, max_prefill_tokens=8192)
    yield GQA, m, oracle.Weights(GQA)
    m.close()


def _tiny_prompts():
    w = synth.workload("tiny")
    return synth.prompts(w)


def _ragged_prompts(vocab):
    inc_len, cand_len = [40, 64, 100, 1], [60, 0, 50, 0]  # totals 100, 64, 150, 1: partial and whole pages
    inc = [synth.uniform_int(3, 100 + i, n, 0, vocab - 1) for i, n in enumerate(inc_len)]
    cand = [synth.uniform_int(3, 200 + i, n, 0, vocab - 1) for i, n in enumerate(cand_len)]
    off = lambda parts: np.concatenate([[0], np.cumsum([len(p) for p in parts])]).astype(np.int32)
    return (np.concatenate(inc).astype(np.int32), off(inc), np.concatenate(cand).astype(np.int32), off(cand))


def _prompt(inc, io, cand, co, i):
    return np.concatenate([inc[io[i]:io[i + 1]], cand[co[i]:co[i + 1]]])


def _run_sampled(m, prompts, n_decode, R, T, seed):
    inc, io, cand, co = prompts
    return m.forecast_batch_sampled(_cuda_i32(inc), io, _cuda_i32(cand), co, n_decode, VIDS, TAU, repeats=R,
                                    temperature=T, seed=seed, want_tokens=True, want_logits=True)


@pytest.mark.parametrize("case", ["tiny", "gqa_ragged"])
def test_sampled_forecast_teacher_forced_parity(case, tiny, gqa):
    shape, m, W = tiny if case == "tiny" else gqa
    prompts = _tiny_prompts() if case == "tiny" else _ragged_prompts(shape.vocab)
    n_decode, R, T, seed = (8, 3, 1.0, 2024) if case == "tiny" else (6, 3, 1.0, 99)
    free0 = m.free_pages()
    out = _run_sampled(m, prompts, n_decode, R, T, seed)
    m.status()
    torch.cuda.synchronize()
    assert m.free_pages() == free0
    B = len(prompts[1]) - 1
    toks = out["tokens"].cpu().numpy()
    lg = out["logits"].cpu().numpy()
    p, conf = out["p"].cpu().numpy(), out["conf"].cpu().numpy()
    arg, defer = out["arg"].cpu().numpy(), out["defer"].cpu().numpy()
    ref_p = np.zeros((B * R, len(VIDS)))
    ref_conf = np.zeros(B * R)
    for r in range(B * R):
        i = r // R
        ref = smp.forecast_sampled_one(W, _prompt(*prompts, i), n_decode, VIDS, TAU, seed, r, T,
                                       forced_tokens=toks[r])
        check_logits(lg[r], ref["step_logits"][-1], f"row {r} final logits")
        for t in range(n_decode):
            sc = smp.sample_scores(ref["step_logits"][t], T, smp.uniforms(seed, t, r, shape.vocab))
            assert _draw_agrees(int(toks[r, t]), sc, ARGMAX_GAP / T), f"row {r} token {t}"
        check_verdict(p[r], conf[r], arg[r], defer[r], ref["p"], ref["conf"], ref["arg"], ref["defer"], TAU)
        ref_p[r], ref_conf[r] = ref["p"], ref["conf"]
    # repeat statistics: against the GPU's own rows (same inputs) and against the oracle's rows
    pm, ps = out["p_mean"].cpu().numpy(), out["p_std"].cpu().numpy()
    cm, cs = out["conf_mean"].cpu().numpy(), out["conf_std"].cpu().numpy()
    for i in range(B):
        rows = slice(i * R, (i + 1) * R)
        m_own, s_own = smp.repeat_stats(p[rows])
        np.testing.assert_allclose(pm[i], m_own, atol=1e-6)
        np.testing.assert_allclose(ps[i], s_own, atol=1e-5)
        mc_own, sc_own = smp.repeat_stats(conf[rows])
        assert abs(cm[i] - mc_own) < 1e-6 and abs(cs[i] - sc_own) < 1e-5
        m_ref, s_ref = smp.repeat_stats(ref_p[rows])
        np.testing.assert_allclose(pm[i], m_ref, atol=1e-2)
        np.testing.assert_allclose(ps[i], s_ref, atol=1e-2)
    # the repeats of an item are distinct draws
    for i in range(B):
        assert len({tuple(toks[i * R + j]) for j in range(R)}) > 1, f"item {i}: repeats drew the same tokens"


def test_same_seed_repeats_itself_and_other_seeds_differ(tiny):
    _, m, _ = tiny
    a = _run_sampled(m, _tiny_prompts(), 6, 2, 1.0, 5)["tokens"].cpu().numpy()
    b = _run_sampled(m, _tiny_prompts(), 6, 2, 1.0, 5)["tokens"].cpu().numpy()
    c = _run_sampled(m, _tiny_prompts(), 6, 2, 1.0, 6)["tokens"].cpu().numpy()
    np.testing.assert_array_equal(a, b)
    assert not np.array_equal(a, c)


def test_single_repeat_and_no_decode(tiny):
    shape, m, W = tiny
    prompts = _tiny_prompts()
    out = _run_sampled(m, prompts, 0, 1, 1.0, 3)
    torch.cuda.synchronize()
    lg = out["logits"].cpu().numpy()
    for i in range(len(prompts[1]) - 1):
        ref, _ = oracle.prefill(W, _prompt(*prompts, i))
        check_logits(lg[i], ref, f"item {i} prompt logits")
    assert np.all(out["p_std"].cpu().numpy() == 0) and np.all(out["conf_std"].cpu().numpy() == 0)


def test_vanishing_temperature_draws_the_greedy_first_token(tiny):
    _, m, _ = tiny
    inc, io, cand, co = _tiny_prompts()
    g = m.forecast_batch(_cuda_i32(inc), io, _cuda_i32(cand), co, 2, VIDS, TAU)["tokens"].cpu().numpy()
    s = _run_sampled(m, (inc, io, cand, co), 2, 3, 1e-6, 8)["tokens"].cpu().numpy()
    for r in range(s.shape[0]):
        assert s[r, 0] == g[r // 3, 0]


def test_sampled_forecast_rejects_bad_arguments(tiny):
    import paper_2605_31464_gb300 as gf
    _, m, _ = tiny
    prompts = _tiny_prompts()
    free0 = m.free_pages()
    for kw in [dict(R=0, T=1.0), dict(R=3, T=0.0), dict(R=3, T=float("nan")), dict(R=5, T=1.0)]:  # 4 x 5 > 16 rows
        with pytest.raises(gf.GfError) as e:
            _run_sampled(m, prompts, 2, kw["R"], kw["T"], 0)
        assert e.value.code == gf.GF_EINVAL
    assert m.free_pages() == free0


@pytest.fixture(scope="module")
def gqa_wide():
    m = make_model(GQA, max_batch=128, max_seq=512, max_prefill_tokens=4096)
    yield GQA, m, oracle.Weights(GQA)
    m.close()


def test_many_rows_use_the_wide_lm_head_tiles(gqa_wide):
    # 4 items x 25 repeats = 100 rows: the LM-head draw runs on 128-column tiles with several
    # 32-row chunks and a ragged last chunk; the oracle checks the prompt draw and one decode draw
    shape, m, W = gqa_wide
    prompts = _ragged_prompts(shape.vocab)
    R, T, seed = 25, 1.0, 31337
    out = _run_sampled(m, prompts, 2, R, T, seed)
    m.status()
    toks = out["tokens"].cpu().numpy()
    lg = out["logits"].cpu().numpy()
    prompt_logits = {}
    for r in range(4 * R):
        i = r // R
        if i not in prompt_logits:
            prompt_logits[i] = oracle.prefill(W, _prompt(*prompts, i))[0]
        sc = smp.sample_scores(prompt_logits[i], T, smp.uniforms(seed, 0, r, shape.vocab))
        assert _draw_agrees(int(toks[r, 0]), sc, ARGMAX_GAP), f"row {r} token 0"
    for r in (0, 1, 27, 50, 77, 99):
        ref = smp.forecast_sampled_one(W, _prompt(*prompts, r // R), 2, VIDS, TAU, seed, r, T, forced_tokens=toks[r])
        sc = smp.sample_scores(ref["step_logits"][1], T, smp.uniforms(seed, 1, r, shape.vocab))
        assert _draw_agrees(int(toks[r, 1]), sc, ARGMAX_GAP), f"row {r} token 1"
        check_logits(lg[r], ref["step_logits"][-1], f"row {r} final logits")
    # 25 draws from one prompt's distribution are not all the same token
    for i in range(4):
        assert len(set(toks[i * R:(i + 1) * R, 0].tolist())) > 1


@pytest.fixture(scope="module")
def tiny_wide():
    w = synth.workload("tiny")
    m = make_model(w.model, max_batch=160, max_seq=512, max_prefill_tokens=4096)
    yield w.model, m, oracle.Weights(w.model)
    m.close()


def test_more_than_128_rows_draw_outside_the_lm_head_gemm(tiny_wide):
    # 4 items x 40 repeats = 160 rows: beyond the widest fused LM-head tile the logits are written out
    # and a separate kernel draws every row, in the prompt step and inside the captured decode graph
    shape, m, W = tiny_wide
    prompts = _tiny_prompts()
    R, T, seed, n_decode = 40, 1.0, 4242, 3
    free0 = m.free_pages()
    out = _run_sampled(m, prompts, n_decode, R, T, seed)
    m.status()
    assert m.free_pages() == free0
    toks = out["tokens"].cpu().numpy()
    lg = out["logits"].cpu().numpy()
    for r in (0, 1, 39, 40, 77, 120, 159):
        ref = smp.forecast_sampled_one(W, _prompt(*prompts, r // R), n_decode, VIDS, TAU, seed, r, T,
                                       forced_tokens=toks[r])
        for t in range(n_decode):
            sc = smp.sample_scores(ref["step_logits"][t], T, smp.uniforms(seed, t, r, shape.vocab))
            assert _draw_agrees(int(toks[r, t]), sc, ARGMAX_GAP), f"row {r} token {t}"
        check_logits(lg[r], ref["step_logits"][-1], f"row {r} final logits")
    for i in range(4):
        assert len({tuple(toks[i * R + j]) for j in range(R)}) > 1
