"""Run one hot-path kernel at a chosen workload shape (for profilers).

    python profile_cases.py gemm --M 8192 --N 37888 --K 3584 --mode swiglu
    python profile_cases.py decode_attn --B 128 --ctx 3072 --n_q 28 --n_kv 4
    python profile_cases.py prefill --workload 7b_prefill --batch 2 --layers 2
    python profile_cases.py forecast --workload 7b_prefill --layers 4 --n_decode 16

Each case launches the kernel `--repeat` times on synthetic data through
the C ABI and prints the mean CUDA-event time and the algorithmic rate.
"""
from __future__ import annotations

import argparse
import os
import sys

import numpy as np


def _gemm(a):
    import torch
    import paper_2605_31464_gb300 as gf
    mode = {"f32": gf.GF_GEMM_STORE_F32, "add": gf.GF_GEMM_ADD_F32, "atomic": gf.GF_GEMM_ATOMIC_F32,
            "bf16": gf.GF_GEMM_STORE_BF16, "swiglu": gf.GF_GEMM_SWIGLU}[a.mode]
    A = (torch.randn(a.M, a.K, device="cuda") * 0.5).bfloat16()
    W = (torch.randn(a.N, a.K, device="cuda") * 0.02).bfloat16()
    cols = a.N // 2 if mode == gf.GF_GEMM_SWIGLU else a.N
    dt = torch.bfloat16 if mode in (gf.GF_GEMM_STORE_BF16, gf.GF_GEMM_SWIGLU) else torch.float32
    out = torch.zeros(a.M, cols, device="cuda", dtype=dt)
    s = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    gf.gemm(A, W, out, mode, bn=a.bn, splits=a.splits, group_m=a.group_m)
    e0.record(s)
    for _ in range(a.repeat):
        gf.gemm(A, W, out, mode, bn=a.bn, splits=a.splits, group_m=a.group_m)
    e1.record(s)
    torch.cuda.synchronize()
    gf.gf_gemm_status(s.cuda_stream)
    ms = e0.elapsed_time(e1) / a.repeat
    tf = 2.0 * a.M * a.N * a.K / (ms / 1e3) / 1e12
    gbs = (a.M * a.K * 2 + a.N * a.K * 2 + a.M * cols * out.element_size()) / (ms / 1e3) / 1e9
    print(f"gemm M{a.M} N{a.N} K{a.K} {a.mode} bn{a.bn} splits{a.splits} group_m{a.group_m}: {ms:.3f} ms, "
          f"{tf:.1f} TFLOP/s, "
          f"{gbs:.0f} GB/s")


def _decode_attn(a):
    import torch
    import paper_2605_31464_gb300 as gf
    hd = a.hd
    pages_per = (a.ctx + 63) // 64
    n_pages = a.B * pages_per
    rng = np.random.default_rng(0)
    table = torch.from_numpy(rng.permutation(n_pages).astype(np.int32).reshape(a.B, pages_per)).cuda()
    kc = torch.randn(n_pages, a.n_kv, 64, hd, device="cuda").bfloat16()
    vc = torch.randn(n_pages, a.n_kv, hd, 64, device="cuda").bfloat16()  # pages stored transposed
    q = torch.randn(a.B, a.n_q * hd, device="cuda").bfloat16()
    ctx = torch.full((a.B,), a.ctx, dtype=torch.int32, device="cuda")
    s = torch.cuda.current_stream()
    gf.decode_attention(q, kc, vc, table, ctx, a.ctx, a.n_q, a.n_kv)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(s)
    for _ in range(a.repeat):
        gf.decode_attention(q, kc, vc, table, ctx, a.ctx, a.n_q, a.n_kv)
    e1.record(s)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / a.repeat
    by = a.B * a.ctx * a.n_kv * hd * 2 * 2
    print(f"decode_attn B{a.B} ctx{a.ctx} {a.n_q}/{a.n_kv}x{hd}: {ms:.3f} ms, {by / (ms / 1e3) / 1e9:.0f} GB/s of KV")


def _prefill(a):
    import dataclasses
    import torch
    import synth
    import paper_2605_31464_gb300 as gf
    w = synth.workload(a.workload, batch=a.batch or 2)
    shape = dataclasses.replace(w.model, layers=a.layers) if a.layers else w.model
    ids, off = synth.packed_prompts(w)
    dev = lambda bits: torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()
    W = {"embed": dev(synth.embed_bf16(shape)), "lm_head": dev(synth.head_bf16(shape)),
         "final_norm": dev(synth.ones_bf16(shape.d_model))}
    for k in ("attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "w_gate", "w_up", "w_down"):
        W[k] = []
    for l in range(shape.layers):
        for k, v in synth.layer_weights_bf16(shape, l).items():
            W[k].append(dev(v))
        W["attn_norm"].append(dev(synth.ones_bf16(shape.d_model)))
        W["ffn_norm"].append(dev(synth.ones_bf16(shape.d_model)))
    m = gf.Model(shape, W, max_batch=w.batch, max_seq=int(np.diff(off).max()) + 8,
                 max_prefill_tokens=int(off[-1]))
    ids_d = torch.from_numpy(ids).cuda()
    s = torch.cuda.current_stream()
    for r in range(a.repeat + 1):
        if r == min(1, a.repeat):  # with --repeat 0 the single run is timed (no warm-up)
            e0 = torch.cuda.Event(enable_timing=True)
            e0.record(s)
        h, _, _ = m.prefill(ids_d, off, want_logits=False)
        m.release(h)
    e1 = torch.cuda.Event(enable_timing=True)
    e1.record(s)
    torch.cuda.synchronize()
    m.status()
    ms = e0.elapsed_time(e1) / max(a.repeat, 1)
    print(f"prefill {a.workload} batch {a.batch} layers {shape.layers}: {ms:.2f} ms, "
          f"{off[-1] / (ms / 1e3):.0f} tok/s")
    m.close()


def _forecast(a):
    """gf_forecast_batch on a workload with `--layers` layers (default all): prefill + decode + verdict."""
    import dataclasses
    import torch
    import synth
    import paper_2605_31464_gb300 as gf
    w = synth.workload(a.workload, batch=a.batch or synth.workload(a.workload).batch)
    shape = dataclasses.replace(w.model, layers=a.layers) if a.layers else w.model
    n_dec = a.n_decode or w.n_decode
    inc, io, cand, co = synth.prompts(w)
    lens = np.diff(io) + np.diff(co)
    dev = lambda bits: torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()
    W = {"embed": dev(synth.embed_bf16(shape)), "lm_head": dev(synth.head_bf16(shape)),
         "final_norm": dev(synth.ones_bf16(shape.d_model))}
    for k in ("attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "w_gate", "w_up", "w_down"):
        W[k] = []
    for l in range(shape.layers):
        for k, v in synth.layer_weights_bf16(shape, l).items():
            W[k].append(dev(v))
        W["attn_norm"].append(dev(synth.ones_bf16(shape.d_model)))
        W["ffn_norm"].append(dev(synth.ones_bf16(shape.d_model)))
    m = gf.Model(shape, W, max_batch=w.batch, max_seq=int(lens.max()) + n_dec,
                 max_prefill_tokens=int(lens.sum()) + w.batch * n_dec + 64)
    del W
    inc_d, cand_d = torch.from_numpy(inc).cuda(), torch.from_numpy(cand).cuda()
    s = torch.cuda.current_stream()
    for r in range(a.repeat + 1):
        if r == min(1, a.repeat):  # with --repeat 0 the single run is timed (no warm-up)
            m.profile(1 << gf.GF_PROF_DECODE_STEPS)
            m.profile_read(gf.GF_PROF_DECODE_STEPS)
            e0 = torch.cuda.Event(enable_timing=True)
            e0.record(s)
        m.forecast_batch(inc_d, io, cand_d, co, n_dec, w.verdict_ids, w.tau, want_tokens=False)
    e1 = torch.cuda.Event(enable_timing=True)
    e1.record(s)
    torch.cuda.synchronize()
    m.status()
    ms = e0.elapsed_time(e1) / max(a.repeat, 1)
    d = m.profile_read(gf.GF_PROF_DECODE_STEPS)
    steps = max(a.repeat, 1) * max(n_dec - 1, 1)
    print(f"forecast {a.workload} batch {w.batch} layers {shape.layers} n_decode {n_dec}: {ms:.2f} ms; "
          f"decode step {d['ms'] / steps:.3f} ms, {d['bytes'] / (d['ms'] / 1e3) / 1e9 if d['ms'] else 0:.0f} GB/s")
    m.close()


def main(argv=None):
    root = os.path.dirname(os.path.abspath(__file__))
    if root not in sys.path:
        sys.path.insert(0, root)
    ap = argparse.ArgumentParser()
    ap.add_argument("case", choices=["gemm", "decode_attn", "prefill", "forecast"])
    ap.add_argument("--M", type=int, default=8192)
    ap.add_argument("--N", type=int, default=37888)
    ap.add_argument("--K", type=int, default=3584)
    ap.add_argument("--mode", default="swiglu", choices=["f32", "add", "atomic", "bf16", "swiglu"])
    ap.add_argument("--bn", type=int, default=0)
    ap.add_argument("--splits", type=int, default=0)
    ap.add_argument("--group_m", type=int, default=0)
    ap.add_argument("--B", type=int, default=128)
    ap.add_argument("--ctx", type=int, default=3072)
    ap.add_argument("--n_q", type=int, default=28)
    ap.add_argument("--n_kv", type=int, default=4)
    ap.add_argument("--hd", type=int, default=128)
    ap.add_argument("--workload", default="7b_prefill")
    ap.add_argument("--batch", type=int, default=0)
    ap.add_argument("--layers", type=int, default=0)
    ap.add_argument("--repeat", type=int, default=3)
    ap.add_argument("--n_decode", type=int, default=0)
    a = ap.parse_args(argv)
    from paper_2605_31464_gb300 import _build
    _build.build()
    {"gemm": _gemm, "decode_attn": _decode_attn, "prefill": _prefill, "forecast": _forecast}[a.case](a)


if __name__ == "__main__":
    main()
