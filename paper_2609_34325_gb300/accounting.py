"""Work accounting for the pruned ViT forward: FLOPs and algorithmic bytes.

FLOPs follow Appendix E.4: one multiply-accumulate counts as two FLOPs, the
count includes patch embedding and the classifier, each image is counted along
its own realised token trajectory, and at a pruning block the attention half
uses the N_l + 1 tokens entering the block while the MLP half uses the
N_l - k_l + 1 survivors.  Selection and memory operations add no FLOPs.

LayerNorm, softmax, GELU and bias terms are not counted; with them the
paper's Native numbers (Table 1) are 0.2-0.4% higher than this count.

Algorithmic bytes are the minimum HBM traffic of each kernel: every input
byte it must read once and every output byte it must write once.
"""
from __future__ import annotations

import numpy as np


def block_flops(n_attn: int | np.ndarray, n_mlp: int | np.ndarray, dim: int, mlp_dim: int):
    """FLOPs of one block for one image: QKV, QK^T, PV, proj on ``n_attn``
    tokens; fc1 and fc2 on ``n_mlp`` tokens."""
    n_attn = np.asarray(n_attn, dtype=np.float64)
    n_mlp = np.asarray(n_mlp, dtype=np.float64)
    qkv = 2.0 * n_attn * dim * 3 * dim
    attn = 4.0 * n_attn * n_attn * dim
    proj = 2.0 * n_attn * dim * dim
    mlp = 2.0 * n_mlp * dim * mlp_dim * 2
    return qkv + attn + proj + mlp


def embed_flops(n_patches: int, patch: int, dim: int, channels: int = 3) -> float:
    return 2.0 * n_patches * patch * patch * channels * dim


def head_flops(dim: int, classes: int = 1000, readout_mult: int = 1) -> float:
    return 2.0 * dim * readout_mult * classes


def native_gflops(n_tokens: int, dim: int, mlp_dim: int, depth: int, patch: int,
                  classes: int = 1000, readout_mult: int = 1) -> float:
    """Complete unpruned forward per image, GFLOPs (Appendix E.4)."""
    f = depth * float(block_flops(n_tokens, n_tokens, dim, mlp_dim))
    f += embed_flops(n_tokens - 1, patch, dim)
    f += head_flops(dim, classes, readout_mult)
    return f / 1e9


def trajectory_flops(depth: int, dim: int, mlp_dim: int, n0: int, schedule: dict,
                     include_embed_head: bool = False, patch: int = 16,
                     readout_mult: int = 1) -> np.ndarray:
    """Per-image FLOPs of the blocks along realised trajectories.

    ``schedule`` maps a pruning block index to the int array of tokens each
    image keeps (CLS included).  Returns a float64 array over images.
    """
    any_keep = next(iter(schedule.values())) if schedule else np.array([n0])
    n = np.full(len(any_keep), n0, dtype=np.float64)
    total = np.zeros_like(n)
    for l in range(depth):
        if l in schedule:
            m = np.asarray(schedule[l], dtype=np.float64)
            total += block_flops(n, m, dim, mlp_dim)
            n = m
        else:
            total += block_flops(n, n, dim, mlp_dim)
    if include_embed_head:
        total += embed_flops(n0 - 1, patch, dim) + head_flops(dim, readout_mult=readout_mult)
    return total


def attention_flops(lengths: np.ndarray, heads: int, head_dim: int = 64) -> float:
    """QK^T + PV FLOPs over the real rows of each image (no padding)."""
    lengths = np.asarray(lengths, dtype=np.float64)
    return float(np.sum(4.0 * lengths * lengths * head_dim * heads))


def attention_bytes(total_rows: int, dim: int) -> float:
    """q, k, v read once and o written once, bf16."""
    return float(total_rows) * dim * 2 * 4


def select_compact_bytes(t_in: int, t_out: int, batch: int, dim: int, fused_ln: bool) -> float:
    """Minimum traffic of one select + compact step.

    Scores read (4 B per input row); kept rows read and written (2D B each);
    kept_idx written and read back (4 B each way); ids read and written
    (4 B each way); cu_seqlens in and out; plus the LayerNorm'
    output (2D B per kept row) when it is fused into compaction.  Deleted rows
    are never read.
    """
    b = 4.0 * t_in + 2.0 * t_out * 2 * dim + 8.0 * t_out + 8.0 * t_out + 8.0 * (batch + 1)
    if fused_ln:
        b += 2.0 * t_out * dim
    return b


def gemm_flops(m: int, n: int, k: int) -> float:
    return 2.0 * m * n * k


def actor_flops(n_tokens: int | np.ndarray, dim: int, n0: int,
                controller: bool | np.ndarray = True) -> np.ndarray:
    """FLOPs of the actor at one block for one image (App. A.1; App. E.4
    counts them): the gate always, and when it opens the controller -- the
    width-128 encoder over the N_l + 1 tokens (input projection, QKV, four
    heads of 32, output projection, 128 -> 256 -> 128 feed-forward), the
    budget head on CLS and the 128 -> 64 -> 1 selector on the visual tokens."""
    n = np.asarray(n_tokens, dtype=np.float64)
    gate = 2.0 * (dim + 19) * 64 + 2.0 * 64
    w = 128.0
    enc = (2.0 * n * dim * w + 2.0 * 3 * w + 2.0 * n * w * 3 * w + 4.0 * n * n * w
           + 2.0 * n * w * w + 2.0 * n * w * 256 * 2)
    budget = 2.0 * w * w + 2.0 * w * ((n0 - 4) // 2)
    selector = 2.0 * (n - 1) * (w * 64 + 64)
    return gate + np.where(np.asarray(controller), enc + budget + selector, 0.0)
