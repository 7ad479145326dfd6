"""Micro-benchmark of the forward's ends and the training-side kernels
through the C ABI.

    python -m paper_2609_34325_gb300.microbench_ends [--images 256] [--iters 20]

Times, with CUDA events on the launching stream, on seeded device-side random
data: the patch embedding (16- and 14-pixel patches), the CLS classifier
head and DINOv2's LC1 head on a pruned packed batch, the LayerScale fold,
Plackett-Luce sampling, the Plackett-Luce log-probability with its gradient,
the fidelity cost and the shadow branch copy.  Prints one line per call:
microseconds per call and the algorithmic bytes moved per second (reads of
each input once, writes of each output once) or, for the embedding GEMM,
its TFLOP/s.  Inputs are larger than L2 where the call's working set allows.
"""
from __future__ import annotations

import argparse

import torch

from . import (dora_branch, dora_classifier_head, dora_classifier_head_lc1, dora_fold_layerscale,
               dora_kd_cost, dora_patch_embed, dora_pl_logprob, dora_pl_sample, load_library)


def _args(argv):
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--images", type=int, default=256)
    ap.add_argument("--dim", type=int, default=768)
    ap.add_argument("--kept", type=int, default=65, help="rows per image after pruning")
    ap.add_argument("--iters", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--seed", type=int, default=0)
    return ap.parse_args(argv)


def main(argv=None):
    a = _args(argv)
    load_library()
    dev = torch.device("cuda:0")
    torch.cuda.set_device(dev)
    g = torch.Generator(device=dev).manual_seed(a.seed)
    bf16, f32, i32 = torch.bfloat16, torch.float32, torch.int32
    B, D = a.images, a.dim

    def rnd(*shape, std=1.0, dtype=bf16):
        return (torch.randn(*shape, generator=g, device=dev) * std).to(dtype)

    runs = []
    # patch embedding, DeiT (16) and DINOv2 (14) patches at 224 x 224
    imgs = rnd(B, 3, 224, 224)
    for p in (16, 14):
        gsz = (224 // p) ** 2
        k = 3 * p * p
        w_pe, b_pe, cls, pos = rnd(D, k, std=0.02), rnd(D, std=0.02), rnd(D), rnd(gsz + 1, D)
        x0 = torch.empty(B * (gsz + 1), D, dtype=bf16, device=dev)
        ws = dora_patch_embed(imgs, w_pe, b_pe, cls, pos, p, x0)
        flops = 2.0 * B * gsz * k * D
        runs.append((f"patch embed p={p} (K {k})", "flops", flops,
                     lambda w_pe=w_pe, b_pe=b_pe, cls=cls, pos=pos, p=p, x0=x0, ws=ws:
                     dora_patch_embed(imgs, w_pe, b_pe, cls, pos, p, x0, ws)))
    # heads on a pruned packed batch (a.kept rows per image)
    n = a.kept
    cu = torch.arange(B + 1, dtype=i32, device=dev) * n
    x = rnd(B * n, D)
    nw, nb = rnd(D, std=0.1) + 1, rnd(D, std=0.1)
    w_head, b_head = rnd(1024, D, std=0.02), rnd(1024, std=0.02)
    w_lc1 = rnd(1024, 2 * D, std=0.02)
    logits = torch.empty(B, 1024, dtype=bf16, device=dev)
    hws = dora_classifier_head(x, cu, nw, nb, 1e-6, w_head, b_head, logits)
    lws = dora_classifier_head_lc1(x, cu, nw, nb, 1e-6, w_lc1, b_head, logits)
    runs.append(("classifier head (CLS)", "bytes", B * D * 2 + 1024 * D * 2 + B * 1024 * 2,
                 lambda: dora_classifier_head(x, cu, nw, nb, 1e-6, w_head, b_head, logits, hws)))
    runs.append(("LC1 head (all surviving rows)", "bytes",
                 B * n * D * 2 + 1024 * 2 * D * 2 + B * 1024 * 2,
                 lambda: dora_classifier_head_lc1(x, cu, nw, nb, 1e-6, w_lc1, b_head, logits,
                                                  lws)))
    # LayerScale fold of one fc2 weight (3072 -> 768), out of place
    w2, b2, ls = rnd(D, 4 * D, std=0.02), rnd(D, std=0.02), rnd(D, std=0.1)
    w2o, b2o = torch.empty_like(w2), torch.empty_like(b2)
    runs.append(("LayerScale fold (fc2)", "bytes", 2 * D * 4 * D * 2,
                 lambda: dora_fold_layerscale(w2, b2, ls, w2o, b2o)))
    # Plackett-Luce sampling and log-probability at DeiT-B's first pruning block
    N0 = 197
    cu0 = torch.arange(B + 1, dtype=i32, device=dev) * N0
    s = rnd(B * N0, dtype=f32)
    u = torch.rand(B * N0, generator=g, device=dev).clamp_(1e-12, 1 - 1e-7)
    gum = -torch.log(-torch.log(u))
    kk = torch.randint(20, 100, (B,), generator=g, device=dev, dtype=torch.int64).to(i32)
    order = torch.empty(B, N0 - 1, dtype=i32, device=dev)
    keys = torch.empty(B * N0, dtype=f32, device=dev)
    logp = torch.empty(B, dtype=f32, device=dev)
    grad = torch.empty(B * N0, dtype=f32, device=dev)
    adv = rnd(B, dtype=f32)
    dora_pl_sample(s, gum, cu0, kk, order, keys_out=keys)
    runs.append(("Plackett-Luce sample (256 x 196)", "bytes", B * N0 * 4 * 3 + B * (N0 - 1) * 4,
                 lambda: dora_pl_sample(s, gum, cu0, kk, order, keys_out=keys)))
    runs.append(("Plackett-Luce log-prob + grad", "bytes", B * N0 * 4 * 2 + B * (N0 - 1) * 4,
                 lambda: dora_pl_logprob(s, cu0, kk, order, logp, grad=grad, dlogp=adv)))
    # fidelity costs of 4 sequences per image against the Native row
    zs = rnd(4 * B, 1024, std=3.0)
    zn = zs[B:2 * B]
    img = torch.arange(4 * B, dtype=i32, device=dev) % B
    cost = torch.empty(4 * B, dtype=f32, device=dev)
    runs.append(("fidelity cost (1024 seqs x 1000)", "bytes", 2 * 4 * B * 1000 * 2,
                 lambda: dora_kd_cost(zn, zs, cost, 1000, shadow_image=img)))
    # branch: the rollout's 256 images after the first deletion, copied once
    nk = 134
    xb = rnd(2 * B * nk, D)
    cub = torch.arange(B + 1, dtype=i32, device=dev) * nk
    cuo = torch.empty(2 * B + 1, dtype=i32, device=dev)
    src = torch.arange(B, dtype=i32, device=dev)
    runs.append(("shadow branch (256 x 134 rows)", "bytes", 2 * B * nk * D * 2,
                 lambda: dora_branch(xb, cub, src, cuo)))

    stream = torch.cuda.current_stream()
    torch.cuda.synchronize()
    for name, kind, work, fn in runs:
        for _ in range(a.warmup):
            fn()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(a.iters):
            fn()
        e1.record(stream)
        e1.synchronize()
        us = 1000.0 * e0.elapsed_time(e1) / a.iters
        rate = (f"{work / (us * 1e-6) / 1e12:7.1f} TFLOP/s" if kind == "flops"
                else f"{work / (us * 1e-6) / 1e9:7.1f} GB/s")
        print(f"{name:36s} {us:9.1f} us  {rate}")


if __name__ == "__main__":
    main()
