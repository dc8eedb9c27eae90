"""Write decode_steps_7b_prefill_17.npz: the float64 oracle's own greedy decode of one 7B prompt.

7b_prefill item 17 (6144 tokens) is prefilled by oracle.forecast_one, which then takes 8 greedy decode
steps with its KV cache.  Stored: the 8 tokens it chose, and as float32 its logits after 4 and after 8
decode inputs.  The GPU test feeds the GPU the same 8 tokens, so the two compare logits at the same
positions even where a near-tied arg max could send free-running trajectories apart.

Calls only oracle/ and the seeded input generator; about half an hour on eight host cores (one
28-layer prompt pass at 6144 tokens and 8 decode steps, weights regenerated layer by layer).

    python tests/golden/make_decode_steps.py
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

NAME, ITEM, N_DECODE, KEEP = "7b_prefill", 17, 8, (4, 8)
OUT = os.path.join(HERE, f"decode_steps_{NAME}_{ITEM}.npz")


def main():
    w = synth.workload(NAME)
    ids, _ = synth.packed_prompts(w, items=[ITEM])
    W = oracle.Weights(w.model, cache_layers=False)
    t0 = time.time()
    ref = oracle.forecast_one(W, ids, N_DECODE, w.verdict_ids, w.tau)
    print(f"{NAME} item {ITEM}: {len(ids)} prompt tokens + {N_DECODE} decode steps in {time.time() - t0:.0f} s; "
          f"tokens {ref['tokens'].tolist()}", flush=True)
    stored = os.path.join(HERE, f"prompt_logits_{NAME}_{ITEM}.npy")
    if os.path.exists(stored):
        d = np.abs(np.load(stored).astype(np.float64) - ref["step_logits"][0]).max()
        print(f"prompt logits vs {os.path.basename(stored)}: largest difference {d:.3g}", flush=True)
    np.savez(OUT, tokens=ref["tokens"].astype(np.int32),
             **{f"logits_{s}": ref["step_logits"][s].astype(np.float32) for s in KEEP})
    print(f"wrote {OUT}", flush=True)


if __name__ == "__main__":
    main()
