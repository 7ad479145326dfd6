"""Micro-benchmark of the token kernels (selection and compaction) through
the C ABI, on inputs cycled beyond twice the L2 size.

    python -m paper_2609_34325_gb300.microbench_tokens [--iters 20] [--cases cfg3,cfg5,shadow1024]

Cases (the deletion step of a pruning block):
  cfg3        DeiT-B shape: 256 images x 197 tokens, D = 768, the first
              pruning block's keep counts
  cfg5        ViT-B/384 shape: 64 images x 577 tokens, D = 768
  shadow1024  1024 sequences x 197 tokens, D = 768 (a training batch with
              its shadows)

For each case it times, with CUDA events on the launching stream over
``iters`` launches that walk R input sets (R sets of rows, moments, ids and
scores whose rows alone exceed 2.5 x the L2 size, so every launch reads
its rows from HBM), the selection (dora_select_keep), the compaction of the
kept rows with their ids and row moments (dora_compact_stats), and the two
fused in one launch (dora_select_compact).  Prints one JSON line per case
and kernel: microseconds per launch, algorithmic bytes (inputs read once,
outputs written once, deleted rows never read) and GB/s.  It is also the
small case for ncu captures of these kernels.
"""
from __future__ import annotations

import argparse
import json
import math

import numpy as np
import torch

import dora_synth as S

from . import dora_compact_stats, dora_select_keep, load_library

CASES = {
    "cfg3": ("cfg3", 256),
    "cfg5": ("cfg5", 64),
    "shadow1024": ("cfg3", 1024),
}


def _fused():
    from . import dora_select_compact
    return dora_select_compact


def _args(argv):
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--iters", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--cases", default="cfg3,cfg5,shadow1024")
    ap.add_argument("--kernels", default="select,compact,fused")
    ap.add_argument("--seed", type=int, default=0)
    return ap.parse_args(argv)


def main(argv=None):
    a = _args(argv)
    load_library()
    dev = torch.device("cuda:0")
    torch.cuda.set_device(dev)
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    g = torch.Generator(device=dev).manual_seed(a.seed)
    stream = torch.cuda.current_stream()
    for case in a.cases.split(","):
        name, batch = CASES[case]
        cfg = S.get_config(name, batch=batch)
        n, d, b = cfg.n_tokens, cfg.dim, cfg.batch
        t = b * n
        keeps = S.keep_schedule(cfg, a.seed)[0][0].astype(np.int32)   # first pruning block
        t_out = int(keeps.sum())
        sets = max(2, math.ceil(2.5 * l2 / (t * d * 2)))
        cu = torch.arange(b + 1, dtype=torch.int32, device=dev) * n
        kc = torch.from_numpy(keeps).to(dev)
        ins = [dict(x=(torch.randn(t, d, generator=g, device=dev)).to(torch.bfloat16),
                    mv=torch.rand(t, 2, generator=g, device=dev),
                    ids=torch.randint(0, n, (t,), generator=g, device=dev, dtype=torch.int32),
                    scores=torch.rand(t, generator=g, device=dev))
               for _ in range(sets)]
        kept = torch.empty(t, dtype=torch.int32, device=dev)
        cu_out = torch.empty(b + 1, dtype=torch.int32, device=dev)
        outs = [dict(x=torch.empty(t, d, dtype=torch.bfloat16, device=dev),
                     mv=torch.empty(t, 2, dtype=torch.float32, device=dev),
                     ids=torch.empty(t, dtype=torch.int32, device=dev)) for _ in range(2)]
        sel_bytes = 4.0 * t + 4.0 * t_out + 8.0 * (b + 1) + 4.0 * b
        cmp_bytes = 2.0 * 2 * d * t_out + 16.0 * t_out + 4.0 * t_out + 8.0 * t_out + 4.0 * (b + 1)
        fused_bytes = (4.0 * t + 2.0 * 2 * d * t_out + 16.0 * t_out + 8.0 * t_out + 4.0 * t_out
                       + 8.0 * (b + 1) + 4.0 * b)
        # kept_idx and cu_out of set 0 for the compaction-only runs
        dora_select_keep(ins[0]["scores"], cu, kc, n, kept, cu_out)
        runs = {
            "select": (sel_bytes, lambda i: dora_select_keep(
                ins[i % sets]["scores"], cu, kc, n, kept, cu_out)),
            "compact": (cmp_bytes, lambda i: dora_compact_stats(
                ins[i % sets]["x"], kept, cu_out, outs[i & 1]["x"], ins[i % sets]["mv"],
                outs[i & 1]["mv"], ids_in=ins[i % sets]["ids"], ids_out=outs[i & 1]["ids"])),
            "fused": (fused_bytes, lambda i: _fused()(
                ins[i % sets]["scores"], cu, kc, n, ins[i % sets]["x"], kept, cu_out,
                outs[i & 1]["x"], ids_in=ins[i % sets]["ids"], ids_out=outs[i & 1]["ids"],
                mv_in=ins[i % sets]["mv"], mv_out=outs[i & 1]["mv"])),
        }
        torch.cuda.synchronize()
        for k in a.kernels.split(","):
            nbytes, fn = runs[k]
            for i in range(a.warmup):
                fn(i)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for i in range(a.iters):
                fn(a.warmup + i)
            e1.record(stream)
            e1.synchronize()
            us = 1000.0 * e0.elapsed_time(e1) / a.iters
            print(json.dumps({"case": case, "kernel": k, "images": b, "tokens": n, "dim": d,
                              "t_in": t, "t_out": t_out, "input_sets": sets,
                              "us_per_launch": round(us, 2), "bytes": int(nbytes),
                              "gbs": round(nbytes / (us * 1e-6) / 1e9, 1)}), flush=True)
        del ins, outs
        torch.cuda.empty_cache()


if __name__ == "__main__":
    main()
