"""GPU path vs the oracle, element by element, on seeded synthetic inputs.

Whole-model parity at sizes the oracle finishes in seconds but that span
several GEMM/attention tiles, KV pages and a ragged tail:
  * the tiny workload (2 layers, d 256, 4 MHA heads x 64, vocab 4096,
    4 prompts of 256 uniform ids, 8 greedy steps, verdict ids {10, 11}, tau 0.8);
  * a GQA shape with head_dim 128 (the head layout of the 1.5B/7B/14B shapes)
    and ragged prompts that straddle pages, q tiles and decode page boundaries.
Decode is teacher-forced: the oracle replays the tokens the GPU emitted, so
the logits of every step are compared even where near-tied arg maxes would
let the two trajectories drift apart; greedy agreement is checked separately.
"""
import dataclasses
import math

import numpy as np
import pytest

import oracle
import synth
from _helpers import (check_logits, check_verdict, greedy_agrees, make_model)

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

GQA = synth.ModelShape(layers=2, d_model=512, n_q=8, n_kv=2, head_dim=128, ffn=1000, vocab=2048, rope_theta=1e6)


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2605_31464_gb300 import _build
    _build.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"


def _cuda_i32(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.int32)).cuda()


def run_teacher_forced(model, W, ids, off, n_decode):
    """Prefill + n_decode steps through the step API; compare every step's logits."""
    B = len(off) - 1
    handles, logits, nxt = model.prefill(_cuda_i32(ids), off)
    torch.cuda.synchronize()
    states, max_err = [], 0.0
    g = logits.cpu().numpy()
    for i in range(B):
        ref, st = oracle.prefill(W, ids[off[i]:off[i + 1]])
        states.append(st)
        max_err = max(max_err, check_logits(g[i], ref, f"prefill item {i}"))
        assert greedy_agrees(int(nxt[i]), ref)
    toks = nxt
    for step in range(n_decode):
        lg, nxt2 = model.decode_step(handles, toks)
        torch.cuda.synchronize()
        g = lg.cpu().numpy()
        t_host = toks.cpu().numpy()
        for i in range(B):
            ref = oracle.decode_step(W, states[i], int(t_host[i]))
            max_err = max(max_err, check_logits(g[i], ref, f"decode step {step} item {i}"))
            assert greedy_agrees(int(nxt2[i]), ref), f"step {step} item {i}"
        toks = nxt2
    model.release(handles)
    model.status()
    return max_err


@pytest.fixture(scope="module")
def tiny():
    w = synth.workload("tiny")
    m = make_model(w.model, max_batch=8, max_seq=512, max_prefill_tokens=4096)
    yield w, m, oracle.Weights(w.model)
    m.close()


@pytest.fixture(scope="module")
def gqa():
    m = make_model(GQA, max_batch=8, max_seq=1024, max_prefill_tokens=8192)
    yield m, oracle.Weights(GQA)
    m.close()


def test_tiny_workload_teacher_forced(tiny):
    w, m, W = tiny
    ids, off = synth.packed_prompts(w)
    run_teacher_forced(m, W, ids, off, w.n_decode)


def test_tiny_forecast_batch_verdict_matches_oracle(tiny):
    w, m, W = tiny
    inc, io, cand, co = synth.prompts(w)
    out = m.forecast_batch(_cuda_i32(inc), io, _cuda_i32(cand), co, w.n_decode, w.verdict_ids, w.tau,
                           want_tokens=True, want_logits=True)
    torch.cuda.synchronize()
    m.status()
    ids, off = synth.packed_prompts(w)
    toks = out["tokens"].cpu().numpy()
    lg = out["logits"].cpu().numpy()
    for i in range(w.batch):
        ref = oracle.forecast_one(W, ids[off[i]:off[i + 1]], w.n_decode, w.verdict_ids, w.tau, forced_tokens=toks[i])
        check_logits(lg[i], ref["step_logits"][-1], f"final logits item {i}")
        check_verdict(out["p"][i].cpu().numpy(), out["conf"][i].item(), out["arg"][i].item(), out["defer"][i].item(),
                      ref["p"], ref["conf"], ref["arg"], ref["defer"], w.tau)
        # the tokens the GPU generated are the greedy choices of its own logits; check them against the oracle's
        free = oracle.forecast_one(W, ids[off[i]:off[i + 1]], 1, w.verdict_ids, w.tau)
        assert greedy_agrees(int(toks[i, 0]), free["step_logits"][0])


def test_host_buffer_variant_matches_oracle(tiny):
    w, m, W = tiny
    inc, io, cand, co = synth.prompts(w)
    host = m.forecast_batch_host(inc, io, cand, co, w.n_decode, w.verdict_ids, w.tau)
    ids, off = synth.packed_prompts(w)
    for i in range(w.batch):
        ref = oracle.forecast_one(W, ids[off[i]:off[i + 1]], w.n_decode, w.verdict_ids, w.tau,
                                  forced_tokens=host["tokens"][i])
        check_verdict(host["p"][i], host["conf"][i], host["arg"][i], host["defer"][i], ref["p"], ref["conf"],
                      ref["arg"], ref["defer"], w.tau)


def test_gqa_hd128_ragged_teacher_forced(gqa):
    m, W = gqa
    # lengths straddle 64-token pages and 128-row query tiles; 70 decode steps cross page boundaries
    lens = [1, 63, 64, 65, 130, 257, 300]
    ids = synth.uniform_int(7, 1, sum(lens), 0, GQA.vocab - 1)
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    run_teacher_forced(m, W, ids, off, 70)


def test_gqa_forecast_with_empty_incumbent_and_shared_prefix(gqa):
    m, W = gqa
    inc_ids = synth.zipf_ids(3, 1, 40, GQA.vocab)
    cands = [synth.zipf_ids(3, 10 + i, n, GQA.vocab) for i, n in enumerate([5, 77, 1])]
    inc = np.concatenate([inc_ids, inc_ids, np.zeros(0, np.int32)]).astype(np.int32)
    io = np.array([0, 40, 80, 80], dtype=np.int32)
    cand = np.concatenate(cands).astype(np.int32)
    co = np.concatenate([[0], np.cumsum([len(c) for c in cands])]).astype(np.int32)
    n_dec, vid, tau = 5, (3, 7, 11, 200), 0.3
    out = m.forecast_batch(_cuda_i32(inc), io, _cuda_i32(cand), co, n_dec, vid, tau, want_tokens=True,
                           want_logits=True)
    torch.cuda.synchronize()
    toks = out["tokens"].cpu().numpy()
    for i in range(3):
        prompt = np.concatenate([inc[io[i]:io[i + 1]], cand[co[i]:co[i + 1]]])
        ref = oracle.forecast_one(W, prompt, n_dec, vid, tau, forced_tokens=toks[i])
        check_logits(out["logits"][i].cpu().numpy(), ref["step_logits"][-1])
        check_verdict(out["p"][i].cpu().numpy(), out["conf"][i].item(), out["arg"][i].item(),
                      out["defer"][i].item(), ref["p"], ref["conf"], ref["arg"], ref["defer"], tau)


def test_zero_decode_steps_reads_last_prompt_position(gqa):
    m, W = gqa
    inc = synth.uniform_int(5, 1, 100, 0, GQA.vocab - 1)
    cand = synth.uniform_int(5, 2, 60, 0, GQA.vocab - 1)
    out = m.forecast_batch(_cuda_i32(inc), [0, 100], _cuda_i32(cand), [0, 60], 0, (10, 11), 0.8, want_tokens=False,
                           want_logits=True)
    ref, _ = oracle.prefill(W, np.concatenate([inc, cand]))
    check_logits(out["logits"][0].cpu().numpy(), ref)
    p, conf, arg, defer = oracle.verdict(ref[None, :], (10, 11), 0.8)
    check_verdict(out["p"][0].cpu().numpy(), out["conf"][0].item(), out["arg"][0].item(), out["defer"][0].item(),
                  p[0], conf[0], arg[0], defer[0], 0.8)


def test_defer_mask_takes_both_values():
    # a sharper LM head spreads the verdict confidence across tau so that both mask values occur
    shape = dataclasses.replace(synth.SHAPE_TINY, head_sigma=0.25)
    w = synth.workload("tiny", model=shape, batch=8, n_decode=2)
    m = make_model(shape, max_batch=8, max_seq=300, max_prefill_tokens=4096)
    W = oracle.Weights(shape)
    inc, io, cand, co = synth.prompts(w)
    ids, off = synth.packed_prompts(w)
    for tau in (0.6, 0.8, 0.95):
        out = m.forecast_batch(_cuda_i32(inc), io, _cuda_i32(cand), co, w.n_decode, w.verdict_ids, tau)
        torch.cuda.synchronize()
        toks = out["tokens"].cpu().numpy()
        refs = [oracle.forecast_one(W, ids[off[i]:off[i + 1]], w.n_decode, w.verdict_ids, tau,
                                    forced_tokens=toks[i]) for i in range(w.batch)]
        for i, ref in enumerate(refs):
            check_verdict(out["p"][i].cpu().numpy(), out["conf"][i].item(), out["arg"][i].item(),
                          out["defer"][i].item(), ref["p"], ref["conf"], ref["arg"], ref["defer"], tau)
        if tau == 0.8:
            assert len({r["defer"] for r in refs}) == 2, "the sharper head should give both defer values"
    m.close()


def test_verdict_kernel_closed_forms():
    import paper_2605_31464_gb300 as gf
    lg = torch.zeros(4, 64, dtype=torch.float32, device="cuda")
    lg[1, 11] = math.log(4.0)           # p = (0.2, 0.8)
    lg[2, 10] = 50.0                    # p ~ (1, 0)
    lg[3, 10], lg[3, 11] = -3.0, -3.0   # tie: lowest index wins
    p, conf, arg, defer = gf.verdict(lg, (10, 11), 0.79)
    p, conf, arg, defer = p.cpu().numpy(), conf.cpu().numpy(), arg.cpu().numpy(), defer.cpu().numpy()
    np.testing.assert_allclose(p[0], [0.5, 0.5], atol=1e-7)
    np.testing.assert_allclose(p[1], [0.2, 0.8], atol=1e-6)
    np.testing.assert_allclose(p.sum(axis=1), 1.0, atol=1e-6)
    assert list(arg) == [0, 1, 0, 0]
    assert list(defer) == [1, 0, 0, 1]
    np.testing.assert_allclose(conf, [0.5, 0.8, 1.0, 0.5], atol=1e-6)


def test_pool_exhaustion_and_bad_handles_are_reported():
    import paper_2605_31464_gb300 as gf
    shape = dataclasses.replace(synth.SHAPE_TINY, layers=1)
    m = make_model(shape, max_batch=2, max_seq=256, max_prefill_tokens=1024, kv_pages=3)
    ids = _cuda_i32(synth.uniform_int(1, 1, 300, 0, shape.vocab - 1))
    with pytest.raises(gf.GfError) as e:
        m.prefill(ids, [0, 150, 300])            # needs 6 pages, pool has 3
    assert e.value.code == gf.GF_ECAPACITY
    h, _, nxt = m.prefill(ids, [0, 128])         # 2 pages
    with pytest.raises(gf.GfError) as e:
        m.decode_step([h[0], h[0]], _cuda_i32([1, 2]))
    assert e.value.code == gf.GF_EINVAL
    with pytest.raises(gf.GfError) as e:
        m.decode_step([1], _cuda_i32([1]))       # slot 1 is not live
    assert e.value.code == gf.GF_EINVAL
    lg, nxt = m.decode_step(h, nxt)              # position 128 needs a third page: fits
    m.release(h)
    m.status()
    m.close()


def test_more_than_128_sequences_use_the_wide_decode_tiles():
    # 160 sequences: the decode GEMMs leave the few-rows (swapped) path, the greedy token comes from a
    # separate arg-max kernel, and decode attention runs 160 x n_kv groups
    m = make_model(GQA, max_batch=160, max_seq=256, max_prefill_tokens=160 * 48)
    W = oracle.Weights(GQA)
    try:
        lens = [17 + (i * 7) % 31 for i in range(160)]  # 17..47 tokens
        ids = synth.uniform_int(9, 3, sum(lens), 0, GQA.vocab - 1)
        off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
        io = np.zeros(161, dtype=np.int32)  # no incumbent: every prompt is its candidate part
        out = m.forecast_batch(_cuda_i32(np.zeros(1, dtype=np.int32)), io, _cuda_i32(ids), off, 4, (10, 11), 0.8,
                               want_tokens=True, want_logits=True)
        torch.cuda.synchronize()
        m.status()
        toks = out["tokens"].cpu().numpy()
        lg = out["logits"].cpu().numpy()
        for i in (0, 1, 63, 64, 127, 128, 129, 159):
            ref = oracle.forecast_one(W, ids[off[i]:off[i + 1]], 4, (10, 11), 0.8, forced_tokens=toks[i])
            check_logits(lg[i], ref["step_logits"][-1], f"final logits item {i}")
            for t in range(4):
                assert greedy_agrees(int(toks[i, t]), ref["step_logits"][t]), f"item {i} token {t}"
    finally:
        m.close()


@pytest.mark.parametrize("T", [1, 50, 128, 129])
def test_gqa_short_prefill_uses_row_major_tiles_for_the_folded_norm(gqa, T):
    # at most 128 prompt tokens would put the SwiGLU GEMM on the swapped (few-rows) tiles; the folded
    # RMSNorm keeps it on the row-major ones
    m, W = gqa
    ids = synth.uniform_int(6, T, T, 0, GQA.vocab - 1)
    out = m.forecast_batch(_cuda_i32(np.zeros(1, np.int32)), [0, 0], _cuda_i32(ids), [0, T], 3, (10, 11), 0.8,
                           want_tokens=True, want_logits=True)
    torch.cuda.synchronize()
    m.status()
    toks = out["tokens"].cpu().numpy()
    ref = oracle.forecast_one(W, ids, 3, (10, 11), 0.8, forced_tokens=toks[0])
    check_logits(out["logits"][0].cpu().numpy(), ref["step_logits"][-1], f"T={T}")
    assert greedy_agrees(int(toks[0, 0]), ref["step_logits"][0])
