"""Parity at the full workload sizes, in the launch configuration bench.py uses.

End to end from token ids (test_*_end_to_end): the whole batch goes through
gf_forecast_batch at its full size, and the oracle runs one item in float64
from its token ids:
  - 1p5b (16 x 4096, 64 decode steps): one item's prompt, every decode step
    teacher-forced with the GPU's own greedy tokens.  Checked: the final
    logits the verdict reads, the verdict and defer bit, every one of the 64
    greedy choices against the oracle's logits of that step, and the logits
    of every eighth step (and the last) from a second, eager pass of the same
    batch fed the same tokens; and the same item's prompt logits through the
    shared-incumbent forecast (gf_forecast_batch_shared) and the sampled
    forecast (gf_forecast_batch_sampled, one repeat) of the whole batch.
  - 7b_prefill (32 x 6144) items 17 and 3 and 7b_decode (128 ragged prompts)
    items 11 and 76, with n_decode = 0: the prompt logits and verdicts, against
    oracle logits stored by tests/golden/make_bf16_drift.py (a 7B prompt
    forward pass takes minutes of host time); and 8 decode steps of items 17
    and 11 fed the oracle's own greedy tokens.
  All 256 (2048) decode steps of a 7B model, and 14b_long end to end, are out
  of the oracle's reach; those keep the layer-level checks below.
  Logits at full depth are held to the distance that bf16 rounding alone puts
  between the float64 oracle and the same forward pass rounded at a bf16
  path's rounding points (tests/golden/bf16_drift.json; check_logits_deep):
  that rounding itself misses the per-element bound 3e-2 + 2e-2 |o| on a few
  logits.  The verdict probabilities follow from those logits: they are held
  to max(1e-2, three times the spread that logit drift implies) (verdict_tol_deep).

Layer level (test_full_size_workload): the oracle cannot run a whole 7B/14B
forward pass in seconds, so these tests compare outputs it can compute one by
one.  The whole batch is prefilled at
its full size through gf_prefill and decoded through gf_decode_step (the
kernels, tile plans and split factors gf_forecast_batch uses); the GPU's
residual stream is captured entering and leaving sampled layers, and the
oracle recomputes those layers from the captured input at sampled rows
(teacher-forced at layer level).  Also checked: the rotated keys and values
the GPU cached at sampled positions, the final logits of sampled items
(from the captured final hidden state), the last decode step of the full
n_decode run (layer outputs from the GPU's own cache), greedy agreement,
and the verdict/defer step on the whole batch's final logits.

Layer outputs must match within 2 % of the layer's largest update on that
row (the update o - x is what bf16 rounding inside the layer perturbs);
keys/values within bf16 rounding; logits and verdict within the standard
tolerances.
"""
import numpy as np
import pytest

import oracle
import synth
from _helpers import (bf16_drift, check_logits, check_logits_deep, check_verdict, greedy_agrees, make_model,
                      verdict_tol_deep)

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

LAYER_TOL = 2e-2


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2605_31464_gb300 import _build
    _build.build()
    assert torch.cuda.is_available()


def check_layer(got, ref, x_in, what):
    upd = np.abs(ref - x_in).max(axis=-1, keepdims=True)
    err = np.abs(np.asarray(got, dtype=np.float64) - ref)
    ratio = (err / (upd + 1e-30)).max()
    assert ratio <= LAYER_TOL, f"{what}: max error {err.max():.3g} = {ratio:.3g} of the layer update"
    return ratio


def check_kv(got_bf16, ref, what):
    g = got_bf16.float().cpu().numpy().astype(np.float64)
    err = np.abs(g - ref)
    bound = 1e-2 * np.abs(ref) + 2e-2 * np.abs(ref).max()
    assert (err <= bound).all(), f"{what}: max error {err.max():.3g} (scale {np.abs(ref).max():.3g})"


def sample_rows(n, seed):
    base = {0, 1, n // 2, n - 2, n - 1}
    rng = np.random.default_rng(seed)
    base |= set(rng.integers(0, n, 3).tolist())
    return sorted(r for r in base if 0 <= r < n)


@pytest.mark.parametrize("name", ["1p5b", "7b_prefill", "7b_decode", "14b_long"])
def test_full_size_workload(name):
    import paper_2605_31464_gb300 as gf
    w = synth.workload(name)
    m = w.model
    ids, off = synth.packed_prompts(w)
    lens = np.diff(off)
    B, L = w.batch, m.layers
    model = make_model(m, max_batch=B, max_seq=int(lens.max()) + w.n_decode,
                       max_prefill_tokens=int(off[-1]))
    Wo = oracle.Weights(m, cache_layers=False)
    a = int(np.argmax(lens))            # longest prompt
    b = int(np.argmin(lens)) if w.ragged else B - 1
    plan = [(a, 0), (a, L - 1), (b, L // 2)]
    caps = {}
    for item, l in plan:
        for ll in (l, l + 1):
            if (item, ll) not in caps:
                caps[(item, ll)] = model.capture(ll, item, int(lens[item]))
    handles, logits, nxt = model.prefill(torch.from_numpy(ids).cuda(), off)
    torch.cuda.synchronize()
    model.status()

    # ---- prefill: sampled layers, cached keys/values, final logits
    for item, l in plan:
        n = int(lens[item])
        x_in = caps[(item, l)].cpu().numpy().astype(np.float64)
        x_out = caps[(item, l + 1)].cpu().numpy()
        rows = sample_rows(n, seed=l)
        lw = Wo.layer(l)
        ref = oracle.layer_rows(x_in, lw, m, rows)
        check_layer(x_out[rows], ref, x_in[rows], f"{name} prefill layer {l} item {item}")
        k_ref, v_ref = oracle.kv_proj(x_in[rows], lw, m, np.array(rows))
        k_gpu, v_gpu = model.read_kv(l, int(handles[item]), 0, n)
        check_kv(k_gpu[rows], k_ref, f"{name} cached K layer {l}")
        check_kv(v_gpu[rows], v_ref, f"{name} cached V layer {l}")
    h_final = caps[(a, L)].cpu().numpy().astype(np.float64)
    ref_logits = oracle.lm_head(h_final[-1:], Wo)[0]
    lg0 = logits[a].cpu().numpy()
    check_logits(lg0, ref_logits, f"{name} prefill logits item {a}")
    assert greedy_agrees(int(nxt[a]), ref_logits)

    # ---- the full decode run; checks at its last step
    toks = nxt
    for _ in range(w.n_decode - 1):
        _, toks = model.decode_step(handles, toks, want_logits=False)
    dec_plan = [(a, 0), (a, L - 1)]
    dcaps = {}
    for item, l in dec_plan:
        for ll in (l, l + 1):
            dcaps[(item, ll)] = model.capture(ll, item, 1)
    lg, nx = model.decode_step(handles, toks)
    torch.cuda.synchronize()
    model.status()
    pos = int(lens[a]) + w.n_decode - 1
    for item, l in dec_plan:
        x_in = dcaps[(item, l)].cpu().numpy().astype(np.float64)
        k_prev, v_prev = model.read_kv(l, int(handles[item]), 0, pos)
        kp = k_prev.float().cpu().numpy().astype(np.float64)
        vp = v_prev.float().cpu().numpy().astype(np.float64)
        ref, _, _ = oracle.layer_forward(x_in, Wo.layer(l), m, np.array([pos]), kp, vp)
        check_layer(dcaps[(item, l + 1)].cpu().numpy(), ref, x_in, f"{name} decode layer {l} at position {pos}")
    ref_logits = oracle.lm_head(dcaps[(a, L)].cpu().numpy().astype(np.float64), Wo)[0]
    check_logits(lg[a].cpu().numpy(), ref_logits, f"{name} decode logits at position {pos}")
    assert greedy_agrees(int(nx[a]), ref_logits)

    # ---- verdict and defer on the whole batch's final logits
    p, conf, arg, defer = gf.verdict(lg, w.verdict_ids, w.tau)
    rp, rc, ra, rd = oracle.verdict(lg.cpu().numpy().astype(np.float64), w.verdict_ids, w.tau)
    p, conf, arg, defer = p.cpu().numpy(), conf.cpu().numpy(), arg.cpu().numpy(), defer.cpu().numpy()
    for i in range(B):
        check_verdict(p[i], conf[i], arg[i], defer[i], rp[i], rc[i], ra[i], rd[i], w.tau)
    model.release(handles)
    model.close()
    del model
    torch.cuda.empty_cache()


# ----------------------------------------------------------------------------- end to end from token ids

def _forecast_whole_batch(w, n_decode, want_tokens):
    """gf_forecast_batch on the workload's whole batch, sized as the benchmark sizes it."""
    m = w.model
    inc, io, cand, co = synth.prompts(w)
    lens = np.diff(io) + np.diff(co)
    model = make_model(m, max_batch=w.batch + 1, max_seq=int(lens.max()) + n_decode,
                       max_prefill_tokens=int(lens.sum()) + w.batch * n_decode + 64)
    out = model.forecast_batch(torch.from_numpy(inc).cuda(), io, torch.from_numpy(cand).cuda(), co, n_decode,
                               w.verdict_ids, w.tau, want_tokens=want_tokens, want_logits=True)
    torch.cuda.synchronize()
    model.status()
    return model, out


def _check_item_verdict(out, item, ref, tau, p_atol):
    check_verdict(out["p"][item].cpu().numpy(), float(out["conf"][item]), int(out["arg"][item]),
                  int(out["defer"][item]), ref["p"], ref["conf"], ref["arg"], ref["defer"], tau, p_atol=p_atol)


def _prompt_logits_other_paths(model, w, item):
    """Prompt logits of `item` (n_decode = 0) through the shared-incumbent forecast (the incumbent's
    pages prefilled once) and the sampled forecast (one repeat per item), on the same model."""
    inc, io, cand, co = synth.prompts(w)
    cand_d = torch.from_numpy(cand).cuda()
    sh = model.forecast_batch_shared(torch.from_numpy(inc[:w.inc_len]).cuda(), cand_d, co, 0, w.verdict_ids, w.tau,
                                     want_tokens=False, want_logits=True)
    sa = model.forecast_batch_sampled(torch.from_numpy(inc).cuda(), io, cand_d, co, 0, w.verdict_ids, w.tau,
                                      repeats=1, temperature=1.0, seed=3, want_tokens=False, want_logits=True)
    torch.cuda.synchronize()
    model.status()
    return {"shared-incumbent": sh["logits"][item].cpu().numpy(), "sampled": sa["logits"][item].cpu().numpy()}


def test_1p5b_forecast_end_to_end_from_token_ids():
    w = synth.workload("1p5b")
    m, n_dec = w.model, w.n_decode
    item = 5
    model, out = _forecast_whole_batch(w, n_dec, want_tokens=True)
    toks = out["tokens"].cpu().numpy()
    final = out["logits"][item].cpu().numpy()
    # a second pass over the whole batch, eager (no graph), fed the tokens the forecast generated
    ids, off = synth.packed_prompts(w)
    steps = sorted(set(range(0, n_dec, 8)) | {n_dec - 1})
    handles, lg0, _ = model.prefill(torch.from_numpy(ids).cuda(), off)
    step_logits = {-1: lg0[item].cpu().numpy()}
    tok_d = torch.from_numpy(np.ascontiguousarray(toks)).cuda()
    for s in range(n_dec):
        lg, _ = model.decode_step(handles, tok_d[:, s].contiguous(), want_logits=s in steps)
        if s in steps:
            step_logits[s] = lg[item].cpu().numpy()
    torch.cuda.synchronize()
    model.status()
    model.release(handles)
    others = _prompt_logits_other_paths(model, w, item)
    model.close()
    del model
    torch.cuda.empty_cache()

    Wo = oracle.Weights(m, cache_layers=True)
    ref = oracle.forecast_one(Wo, ids[off[item]:off[item + 1]], n_dec, w.verdict_ids, w.tau,
                              forced_tokens=toks[item])
    del Wo
    # product path: the logits the verdict reads, the verdict, and every greedy choice
    drift = bf16_drift("1p5b", item)
    print(check_logits_deep(final, ref["step_logits"][n_dec], drift, f"1p5b item {item}: final logits (step {n_dec})"))
    _check_item_verdict(out, item, ref, w.tau, verdict_tol_deep(drift, ref["p"]))
    for s in range(n_dec):
        assert greedy_agrees(int(toks[item, s]), ref["step_logits"][s]), f"greedy token of decode input {s}"
    # the eager pass: prompt logits and the logits of the sampled steps
    for s, lg in step_logits.items():
        print(check_logits_deep(lg, ref["step_logits"][s + 1], drift, f"1p5b item {item}: logits after decode input {s}"))
    # the shared-incumbent and sampled forecasts of the same batch: the prompt logits
    for path, lg in others.items():
        print(check_logits_deep(lg, ref["step_logits"][0], drift, f"1p5b item {item}: {path} prompt logits"))



@pytest.mark.parametrize("name,items", [("7b_prefill", (17, 3)), ("7b_decode", (11, 76))])
def test_7b_forecast_prompt_logits_end_to_end_from_token_ids(name, items):
    """7b_prefill (32 x 6144) and 7b_decode (128 ragged prompts of U[1024, 2048] ids; item 76 is the
    shortest, 1029 tokens) through gf_forecast_batch with n_decode = 0, whole batch: two items' prompt
    logits and verdicts against the float64 oracle's 28-layer pass from each item's token ids.  That pass
    takes minutes of host time, so tests/golden/make_bf16_drift.py (which calls only oracle/) stored its
    logits in tests/golden/prompt_logits_<workload>_<item>.npy."""
    import os
    w = synth.workload(name)
    model, out = _forecast_whole_batch(w, 0, want_tokens=False)
    finals = {item: out["logits"][item].cpu().numpy() for item in items}
    model.close()
    del model
    torch.cuda.empty_cache()
    for item in items:
        ref_logits = np.load(os.path.join(os.path.dirname(__file__), "golden",
                                          f"prompt_logits_{name}_{item}.npy")).astype(np.float64)
        assert ref_logits.shape == (w.model.vocab,)
        drift = bf16_drift(name, item)
        print(check_logits_deep(finals[item], ref_logits, drift, f"{name} item {item}: prompt logits"))
        rp, rc, ra, rd = oracle.verdict(ref_logits[None], w.verdict_ids, w.tau)
        tol = verdict_tol_deep(drift, rp[0])
        print(f"{name} item {item}: verdict p {out['p'][item].cpu().numpy()} vs oracle {rp[0]} (tolerance {tol:.4f})")
        _check_item_verdict(out, item, {"p": rp[0], "conf": float(rc[0]), "arg": int(ra[0]), "defer": int(rd[0])},
                            w.tau, tol)


@pytest.mark.parametrize("name,item", [("7b_prefill", 17), ("7b_decode", 11)])
def test_7b_decode_steps_fed_the_oracle_tokens(name, item):
    """7b_prefill (32 x 6144) and 7b_decode (128 ragged prompts): the whole batch prefilled and then decoded
    for 8 steps in the benchmark's launch configuration, every sequence fed the float64 oracle's own greedy
    tokens for one item; that item's logits after decode inputs 3 and 7 against the oracle's
    (tests/golden/decode_steps_<workload>_<item>.npz, written by tests/golden/make_decode_steps.py, which
    calls only oracle/)."""
    import os
    w = synth.workload(name)
    m = w.model
    g = np.load(os.path.join(os.path.dirname(__file__), "golden", f"decode_steps_{name}_{item}.npz"))
    toks = g["tokens"]
    ids, off = synth.packed_prompts(w)
    lens = np.diff(off)
    model = make_model(m, max_batch=w.batch, max_seq=int(lens.max()) + len(toks) + 1,
                       max_prefill_tokens=int(off[-1]))
    handles, _, _ = model.prefill(torch.from_numpy(ids).cuda(), off)
    got = {}
    for s in range(len(toks)):
        step_ids = torch.full((w.batch,), int(toks[s]), dtype=torch.int32, device="cuda")
        lg, _ = model.decode_step(handles, step_ids, want_logits=f"logits_{s + 1}" in g.files)
        if f"logits_{s + 1}" in g.files:
            got[s + 1] = lg[item].cpu().numpy()
    torch.cuda.synchronize()
    model.status()
    model.release(handles)
    model.close()
    del model
    torch.cuda.empty_cache()
    assert sorted(got) == [4, 8]
    drift = bf16_drift(name, item)
    for s, lg in got.items():
        print(check_logits_deep(lg, g[f"logits_{s}"].astype(np.float64), drift,
                                f"{name} item {item}: logits after decode input {s - 1}"))
