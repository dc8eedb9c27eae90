"""Write bf16_drift.json: how far bf16 rounding alone moves the prompt logits of full-size items.

For each listed (workload, item), the float64 oracle's prompt logits (oracle.model) and those of the
same forward pass rounded to bf16 at a bf16 data path's rounding points (oracle.bf16_path) are
compared: root-mean-square and largest absolute difference of the logits, how many logits fall
outside |g - o| <= 3e-2 + 2e-2 |o|, and the largest difference of the verdict probabilities.  The
end-to-end parity tests hold the GPU's own difference from the oracle to a small multiple of these.
For the cases in SAVE_LOGITS the float64 oracle's prompt logits are also written, as float32, to
prompt_logits_<workload>_<item>.npy: a whole 7B prompt forward pass takes minutes of host time, so
the GPU test reads them instead of recomputing them.

Calls only oracle/ and the seeded input generator; runs for about two hours on eight host cores
(28-layer prompt forward passes of 4096, 2 x 6144, 2038 and 1029 tokens, twice each).

    python tests/golden/make_bf16_drift.py [workload:item ...]
"""
from __future__ import annotations

import json
import os
import sys
import time

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
import synth  # noqa: E402
from oracle import bf16_path  # noqa: E402

CASES = [("1p5b", 5), ("7b_prefill", 17), ("7b_prefill", 3), ("7b_decode", 11), ("7b_decode", 76)]
SAVE_LOGITS = {("7b_prefill", 17), ("7b_prefill", 3), ("7b_decode", 11), ("7b_decode", 76)}
OUT = os.path.join(HERE, "bf16_drift.json")


def drift(name: str, item: int) -> dict:
    w = synth.workload(name)
    m = w.model
    ids, off = synth.packed_prompts(w, items=[item])
    W = oracle.Weights(m, cache_layers=False)
    pos = np.arange(len(ids))
    x = W.embed_rows(ids)
    xb = x.copy()
    t0 = time.time()
    for l in range(m.layers):
        lw = W.layer(l)  # one draw of the layer's weights serves both passes
        x, _, _ = oracle.layer_forward(x, lw, m, pos)
        xb = bf16_path.layer_forward_bf16(xb, lw, m, pos)
        print(f"{name} item {item}: layer {l + 1}/{m.layers} ({time.time() - t0:.0f} s)", flush=True)
    ref = oracle.lm_head(x[-1:], W)[0]
    if (name, item) in SAVE_LOGITS:
        np.save(os.path.join(HERE, f"prompt_logits_{name}_{item}.npy"), ref.astype(np.float32))
    last = xb[-1:]
    h = bf16_path.bf16_round(last / np.sqrt(np.mean(last * last, axis=-1, keepdims=True) + m.rms_eps) *
                             W.final_norm())
    emu = (h @ W.head().T)[0]
    err = np.abs(emu - ref)
    p_ref = oracle.verdict(ref[None], w.verdict_ids, w.tau)[0][0]
    p_emu = oracle.verdict(emu[None], w.verdict_ids, w.tau)[0][0]
    return {"workload": name, "item": item, "prompt_len": int(len(ids)),
            "rms_err": float(np.sqrt(np.mean(err ** 2))), "max_err": float(err.max()),
            "mean_err": float(err.mean()),
            "outside_elementwise_bound": int((err > 3e-2 + 2e-2 * np.abs(ref)).sum()), "logits": int(err.size),
            "ref_rms": float(np.sqrt(np.mean(ref ** 2))), "verdict_p_err": float(np.abs(p_emu - p_ref).max())}


def main(argv):
    cases = [(a.split(":")[0], int(a.split(":")[1])) for a in argv] or CASES
    out = {"source": "tests/golden/make_bf16_drift.py (oracle.model vs oracle.bf16_path, prompt logits)",
           "cases": []}
    if os.path.exists(OUT):
        with open(OUT) as f:
            out = json.load(f)
    for name, item in cases:
        r = drift(name, item)
        out["cases"] = [c for c in out["cases"] if (c["workload"], c["item"]) != (name, item)] + [r]
        with open(OUT, "w") as f:
            json.dump(out, f, indent=1)
        print(json.dumps(r), flush=True)


if __name__ == "__main__":
    main(sys.argv[1:])
