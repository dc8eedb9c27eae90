"""Write decode_steps_<workload>_<item>.npz: the float64 oracle's own greedy decode of one 7B prompt.

The item's prompt is prefilled by oracle.forecast_one, which then takes 8 greedy decode steps with its KV
cache.  Stored: the 8 tokens it chose, and as float32 its logits after 4 and after 8 decode inputs.  The
GPU test feeds the GPU the same 8 tokens, so the two compare logits at the same positions even where a
near-tied arg max could send free-running trajectories apart.

Calls only oracle/ and the seeded input generator; 21 minutes on eight host cores for 7b_prefill item 17
(6144 prompt tokens), about 10 for 7b_decode item 11 (2038), weights regenerated layer by layer.

    python tests/golden/make_decode_steps.py [workload:item ...]
"""
from __future__ import annotations

import os
import sys
import time

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
import synth  # noqa: E402

CASES = [("7b_prefill", 17), ("7b_decode", 11)]
N_DECODE, KEEP = 8, (4, 8)


def run(name: str, item: int):
    out = os.path.join(HERE, f"decode_steps_{name}_{item}.npz")
    w = synth.workload(name)
    ids, _ = synth.packed_prompts(w, items=[item])
    W = oracle.Weights(w.model, cache_layers=False)
    t0 = time.time()
    ref = oracle.forecast_one(W, ids, N_DECODE, w.verdict_ids, w.tau)
    print(f"{name} item {item}: {len(ids)} prompt tokens + {N_DECODE} decode steps in {time.time() - t0:.0f} s; "
          f"tokens {ref['tokens'].tolist()}", flush=True)
    stored = os.path.join(HERE, f"prompt_logits_{name}_{item}.npy")
    if os.path.exists(stored):
        d = np.abs(np.load(stored).astype(np.float64) - ref["step_logits"][0]).max()
        print(f"prompt logits vs {os.path.basename(stored)}: largest difference {d:.3g}", flush=True)
    np.savez(out, tokens=ref["tokens"].astype(np.int32),
             **{f"logits_{s}": ref["step_logits"][s].astype(np.float32) for s in KEEP})
    print(f"wrote {out}", flush=True)


def main(argv):
    for name, item in [(a.split(":")[0], int(a.split(":")[1])) for a in argv] or CASES:
        run(name, item)


if __name__ == "__main__":
    main(sys.argv[1:])
