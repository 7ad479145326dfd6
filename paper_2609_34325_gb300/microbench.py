"""Micro-benchmark of one block's kernels through the C ABI.

    python -m paper_2609_34325_gb300.microbench [--images 256] [--iters 20]
    python -m paper_2609_34325_gb300.microbench --mixes cfg6 [--iters 20]

Times, with CUDA events on the launching stream, the QKV linear with
LayerNorm folded in, the projection and fc2 with their residuals (and the
slice moments they write for the next LayerNorm), and fc1 with LayerNorm'
folded in and GELU, at DeiT-B shapes by default, on seeded device-side random
data (any non-degenerate bit pattern serves for timing), then the varlen
attention over `images` images of `tokens` tokens.  Prints one line per
kernel: microseconds per launch and TFLOP/s.  It is also the small case for
profiling one launch of a kernel: the linears run in that order, each
warmup + iters launches, then the attention.

With ``--mixes CFG`` it times only the varlen attention, on the length mixes
of that configuration's seeded deletion schedule (the full-length batch, then
the batch after each pruning block), each twice: with max_seqlen set to the
mix's own longest image and to the configuration's token count N.  The
attention picks its kernel from max_seqlen (the short-image kernel up to 256,
the per-key-half kernel beyond), so the two lines show what a caller that
knows the kept maximum would gain over one that passes N.
"""
from __future__ import annotations

import argparse

import torch

from . import (dora_fold_ln_linear, dora_linear_ln, dora_linear_residual_stats, dora_row_stats,
               dora_varlen_attn, load_library)


def _args(argv):
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--images", type=int, default=256)
    ap.add_argument("--tokens", type=int, default=197)
    ap.add_argument("--dim", type=int, default=768)
    ap.add_argument("--mlp", type=int, default=3072)
    ap.add_argument("--iters", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--mixes", default=None,
                    help="time the attention on this configuration's length mixes instead")
    return ap.parse_args(argv)


def _time(fn, warmup, iters, stream):
    for _ in range(warmup):
        fn()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(iters):
        fn()
    e1.record(stream)
    e1.synchronize()
    return 1000.0 * e0.elapsed_time(e1) / iters


def attention_mixes(a, dev):
    """Varlen attention on each length mix of a configuration's seeded schedule."""
    import numpy as np

    import dora_synth as S

    cfg = S.get_config(a.mixes)
    keeps, _ = S.keep_schedule(cfg, a.seed)
    mixes = [np.full(cfg.batch, cfg.n_tokens, dtype=np.int64)] + [k.astype(np.int64) for k in keeps]
    heads, d = cfg.heads, cfg.dim
    t_cap = cfg.batch * cfg.n_tokens
    g = torch.Generator(device=dev).manual_seed(a.seed)
    qkv = torch.randn(t_cap, 3 * d, generator=g, device=dev).to(torch.bfloat16)
    o = torch.empty(t_cap, d, dtype=torch.bfloat16, device=dev)
    stream = torch.cuda.current_stream()
    for j, lens in enumerate(mixes):
        cu = torch.from_numpy(np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)).to(dev)
        flops = 4.0 * float((lens * lens).sum()) * cfg.head_dim * heads
        label = "full length" if j == 0 else f"after pruning {j}"
        for msl in sorted({int(lens.max()), cfg.n_tokens}):
            us = _time(lambda: dora_varlen_attn(qkv, cu, msl, heads, o), a.warmup, a.iters, stream)
            print(f"{a.mixes} {label:18s} mean {lens.mean():6.1f} max {lens.max():4d} "
                  f"max_seqlen {msl:4d}: {us:8.1f} us  {flops / (us * 1e-6) / 1e12:7.1f} TFLOP/s")


def main(argv=None):
    a = _args(argv)
    load_library()
    dev = torch.device("cuda:0")
    torch.cuda.set_device(dev)
    if a.mixes is not None:
        attention_mixes(a, dev)
        return
    g = torch.Generator(device=dev).manual_seed(a.seed)
    bf16, f32 = torch.bfloat16, torch.float32
    T, D, F = a.images * a.tokens, a.dim, a.mlp
    heads = D // 64

    def rnd(*shape, std=1.0):
        return (torch.randn(*shape, generator=g, device=dev) * std).to(bf16)

    x, r = rnd(T, D), rnd(T, D)
    hid = rnd(T, F)
    w = {"qkv": rnd(3 * D, D, std=0.02), "proj": rnd(D, D, std=0.02),
         "fc1": rnd(F, D, std=0.02), "fc2": rnd(D, F, std=0.02)}
    b = {k: rnd(v.shape[0], std=0.1) for k, v in w.items()}
    gamma, beta = (1 + rnd(D, std=0.1).float()).to(bf16), rnd(D, std=0.1)
    folded = {}
    for k in ("qkv", "fc1"):
        n = w[k].shape[0]
        folded[k] = (torch.empty_like(w[k]), torch.empty(n, dtype=f32, device=dev),
                     torch.empty(n, dtype=f32, device=dev))
        dora_fold_ln_linear(w[k], gamma, beta, *folded[k], bias=b[k])
    mv = torch.empty(T, 2, dtype=f32, device=dev)
    dora_row_stats(x, mv)
    sm = torch.empty(D // 64, T, 2, dtype=f32, device=dev)
    y = {"qkv": torch.empty(T, 3 * D, dtype=bf16, device=dev),
         "proj": torch.empty(T, D, dtype=bf16, device=dev),
         "fc1": torch.empty(T, F, dtype=bf16, device=dev),
         "fc2": torch.empty(T, D, dtype=bf16, device=dev)}
    runs = [
        ("qkv  (LayerNorm folded)", 3 * D, D,
         lambda: dora_linear_ln(x, mv, 1e-6, *folded["qkv"], y["qkv"])),
        ("proj (residual + moments)", D, D,
         lambda: dora_linear_residual_stats(x, w["proj"], r, y["proj"], sm, bias=b["proj"])),
        ("fc1  (LayerNorm folded + GELU)", F, D,
         lambda: dora_linear_ln(x, mv, 1e-6, *folded["fc1"], y["fc1"], gelu=True)),
        ("fc2  (residual + moments)", D, F,
         lambda: dora_linear_residual_stats(hid, w["fc2"], r, y["fc2"], sm, bias=b["fc2"])),
    ]
    cu = torch.arange(a.images + 1, dtype=torch.int32, device=dev) * a.tokens
    o = torch.empty(T, D, dtype=bf16, device=dev)
    attn_flops = 4.0 * a.images * a.tokens * a.tokens * 64 * heads
    runs.append(("varlen attention", None, attn_flops,
                 lambda: dora_varlen_attn(y["qkv"], cu, a.tokens, heads, o)))
    stream = torch.cuda.current_stream()
    torch.cuda.synchronize()
    for name, n, k, fn in runs:
        us = _time(fn, a.warmup, a.iters, stream)
        if n is None:         # attention: k holds its FLOPs
            shape, flops = f"{a.images} x {a.tokens} tokens x {heads} heads", k
        else:
            shape, flops = f"{T} x {n} x {k}", 2.0 * T * n * k
        print(f"{name:32s} {shape}: {us:8.1f} us  {flops / (us * 1e-6) / 1e12:7.1f} TFLOP/s")


if __name__ == "__main__":
    main()
