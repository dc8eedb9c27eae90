"""The oracle: a plain, slow, float64 CPU restatement of the surrogate's forward
pass, greedy decoding and verdict/deferral (Sec. 2.1).

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline / reference arm of ``bench.py``, never by the product
package.  It shares no code with the CUDA path.
"""
from .model import (Weights, attention, bf16_bits_to_f64, decode_step, forecast_batch, forecast_one,
                    full_recompute_logits, greedy, kv_proj, layer_forward, layer_rows, lm_head, prefill, q_proj, qkv, rms_norm,
                    rope, silu, softmax, swiglu_ffn, verdict, SequenceState, attn_out_and_ffn)
