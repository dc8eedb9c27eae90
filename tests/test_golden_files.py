"""The stored oracle outputs the full-size GPU tests read agree with one another (CPU).

tests/golden/make_bf16_drift.py writes the float64 oracle's prompt logits of sampled 7B items and the
bf16-rounding drift records; tests/golden/make_decode_steps.py writes the oracle's own greedy decode of
one item per 7B workload.  Both call only oracle/.  Here: every stored file has the vocabulary's shape and
finite values, every logits file has a drift record, the first greedy token of a decode-step file is the
arg max of the same item's stored prompt logits, and the drift records are internally consistent.
"""
import json
import os

import numpy as np
import pytest

import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _drift_cases():
    with open(os.path.join(GOLDEN, "bf16_drift.json")) as f:
        return {(c["workload"], c["item"]): c for c in json.load(f)["cases"]}


def _files(prefix, suffix):
    out = []
    for f in sorted(os.listdir(GOLDEN)):
        if f.startswith(prefix) and f.endswith(suffix):
            name, item = f[len(prefix):-len(suffix)].rsplit("_", 1)
            out.append((name, int(item), os.path.join(GOLDEN, f)))
    return out


def test_drift_records_are_consistent():
    cases = _drift_cases()
    assert cases
    for (name, item), c in cases.items():
        w = synth.workload(name)
        assert 0 <= item < w.batch
        assert c["logits"] == w.model.vocab
        assert 0 < c["mean_err"] <= c["rms_err"] <= c["max_err"]
        assert 0 <= c["outside_elementwise_bound"] <= c["logits"]
        assert 0 <= c["verdict_p_err"] < 1
        ids, _ = synth.packed_prompts(w, items=[item])
        assert c["prompt_len"] == len(ids)


@pytest.mark.parametrize("name,item,path", _files("prompt_logits_", ".npy"))
def test_prompt_logits_files(name, item, path):
    lg = np.load(path)
    assert lg.dtype == np.float32 and lg.shape == (synth.workload(name).model.vocab,)
    assert np.isfinite(lg).all()
    assert (name, item) in _drift_cases(), "every stored logits file has its drift record"


@pytest.mark.parametrize("name,item,path", _files("decode_steps_", ".npz"))
def test_decode_step_files(name, item, path):
    g = np.load(path)
    V = synth.workload(name).model.vocab
    toks = g["tokens"]
    assert toks.dtype == np.int32 and toks.ndim == 1 and len(toks) >= 8
    assert ((toks >= 0) & (toks < V)).all()
    for key in ("logits_4", "logits_8"):
        assert g[key].shape == (V,) and np.isfinite(g[key]).all()
    # the first decode input is the oracle's greedy choice from the prompt's logits
    pl = os.path.join(GOLDEN, f"prompt_logits_{name}_{item}.npy")
    if os.path.exists(pl):
        lg = np.load(pl).astype(np.float64)
        top2 = np.sort(lg)[-2:]
        if top2[1] - top2[0] > 1e-5:
            assert int(np.argmax(lg)) == int(toks[0])
    # and the 5th input is the greedy choice from the stored logits after 4 inputs
    lg4 = g["logits_4"].astype(np.float64)
    top2 = np.sort(lg4)[-2:]
    if top2[1] - top2[0] > 1e-5:
        assert int(np.argmax(lg4)) == int(toks[4])
