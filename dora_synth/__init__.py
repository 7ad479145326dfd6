"""Seeded synthetic inputs for the DORA deployment hot path.

This module is harness code shared by the CUDA path's tests/bench and by the
fp64 oracle's tests.  It produces *inputs only*: bf16 activations and weights,
fp32 deletion-score tables, per-image keep counts and the workload shapes.  It
holds none of the method's arithmetic (no selection, compaction, attention,
normalisation or linear algebra).

Randomness is counter based: every value is a pure function of
``(seed, tag, index)`` through SplitMix64 (Steele, Lea & Flood, "Fast
splittable pseudorandom number generators", OOPSLA 2014), so any slice of any
tensor can be regenerated independently and identically on any machine.

Workload shapes follow the five configurations of the build:

* ``cfg1`` DeiT-Tiny shape, one pruning block, B=8, N=197, D=192, H=3.
* ``cfg2`` DeiT-Small shape, one pruning block, B=64, N=197, D=384, H=6.
* ``cfg3`` DeiT-Base shape, 12 blocks, B=256, pruning at blocks 3/6/9, per-image
  removal fraction drawn so the batch-mean token-layer compression (Eq. 4) is
  about 0.38 (the paper's DeiT-B FLOPs reduction is 38.4%, Table 1).
* ``cfg4`` ViT-Large shape, 24 blocks, B=128, pruning at 4/8/12/16/20 with a
  heavy-tailed final keep ratio (some images keep everything, many ~20%).
* ``cfg5`` ViT-Base/384 shape, N=577, 12 blocks, B=64, pruning at 2/4/6/8/10,
  deletion scores from a per-image Gaussian spatial bump plus noise.

Removal counts respect the budget legality of Appendix A.2: at least four
visual tokens survive every deletion (Eq. for B_l).  Token counts in this
module *include* CLS unless a name says ``vis``.
"""
from __future__ import annotations

import math
import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field

import numpy as np

__all__ = [
    "Config", "CONFIGS", "get_config", "splitmix64", "hash_u64", "uniform_f64",
    "uniform_f32", "normal_f64", "f32_to_bf16_bits", "bf16_bits_to_f32",
    "activations_bf16", "block_weights", "score_table", "keep_schedule",
    "initial_layout", "compression_from_counts", "actor_weights", "ACTOR_SHAPES",
    "images_bf16", "embed_head_weights",
]

_M64 = np.uint64(0xFFFFFFFFFFFFFFFF)
_GAMMA = np.uint64(0x9E3779B97F4A7C15)
_MUL1 = np.uint64(0xBF58476D1CE4E5B9)
_MUL2 = np.uint64(0x94D049BB133111EB)

# Stream tags: one per kind of tensor so streams never collide.
TAG_ACT = 1
TAG_W = 2          # + (block << 8) + which
TAG_SCORE = 3      # + (block << 8)
TAG_KEEP = 4       # per-image budget law draws
TAG_BUMP = 5       # cfg5 bump centre / width
TAG_LNAFF = 6      # optional random LayerNorm affine (tests)
TAG_ACTOR = 7      # + (which << 8): actor weights
TAG_IMG = 8        # input images
TAG_EMBHEAD = 9    # + (which << 8): patch embedding and classifier weights


def splitmix64(x: np.ndarray) -> np.ndarray:
    """SplitMix64 finaliser applied elementwise to a uint64 array (wraps mod 2^64)."""
    x = np.asarray(x, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = x + _GAMMA
        z = (z ^ (z >> np.uint64(30))) * _MUL1
        z = (z ^ (z >> np.uint64(27))) * _MUL2
        return z ^ (z >> np.uint64(31))


def _stream_key(seed: int, tag: int) -> np.uint64:
    s = splitmix64(np.array([seed & 0xFFFFFFFFFFFFFFFF], dtype=np.uint64))
    k = splitmix64(s ^ np.uint64(tag & 0xFFFFFFFFFFFFFFFF))
    return k[0]


def hash_u64(seed: int, tag: int, idx: np.ndarray) -> np.ndarray:
    """64 random bits for each counter in ``idx`` of stream (seed, tag)."""
    key = _stream_key(seed, tag)
    idx = np.asarray(idx, dtype=np.uint64)
    with np.errstate(over="ignore"):
        return splitmix64(key ^ (idx * _GAMMA))


def uniform_f64(seed: int, tag: int, idx: np.ndarray) -> np.ndarray:
    """U[0,1) doubles from the top 53 bits."""
    h = hash_u64(seed, tag, idx)
    return (h >> np.uint64(11)).astype(np.float64) * (2.0 ** -53)


def uniform_f32(seed: int, tag: int, idx: np.ndarray) -> np.ndarray:
    """U[0,1) floats from the top 24 bits: every value is exact in fp32."""
    h = hash_u64(seed, tag, idx)
    return ((h >> np.uint64(40)).astype(np.float64) * (2.0 ** -24)).astype(np.float32)


def normal_f64(seed: int, tag: int, idx: np.ndarray) -> np.ndarray:
    """Standard normals by Box-Muller on the two 32-bit halves of one hash."""
    h = hash_u64(seed, tag, idx)
    u1 = ((h >> np.uint64(32)).astype(np.float64) + 0.5) * (2.0 ** -32)
    u2 = (h & np.uint64(0xFFFFFFFF)).astype(np.float64) * (2.0 ** -32)
    return np.sqrt(-2.0 * np.log(u1)) * np.cos(2.0 * np.pi * u2)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 (or anything castable) to bf16, nearest-even; returns uint16 bits.

    Inputs produced here are finite, so NaN handling is not needed.
    """
    b = np.ascontiguousarray(np.asarray(x, dtype=np.float32)).view(np.uint32)
    bias = np.uint32(0x7FFF) + ((b >> np.uint32(16)) & np.uint32(1))
    with np.errstate(over="ignore"):
        return ((b + bias) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Widen bf16 bit patterns to fp32 (exact)."""
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def _normal_bf16(seed: int, tag: int, count: int, std: float, base: int = 0) -> np.ndarray:
    """``count`` bf16 bit patterns of N(0, std^2), generated in parallel chunks."""
    out = np.empty(count, dtype=np.uint16)
    chunk = 1 << 22

    def work(lo: int) -> None:
        hi = min(count, lo + chunk)
        idx = np.arange(base + lo, base + hi, dtype=np.uint64)
        out[lo:hi] = f32_to_bf16_bits(normal_f64(seed, tag, idx) * std)

    starts = list(range(0, count, chunk))
    if len(starts) <= 1:
        for s in starts:
            work(s)
    else:
        nthreads = max(1, min(len(starts), len(os.sched_getaffinity(0))))
        with ThreadPoolExecutor(nthreads) as ex:
            list(ex.map(work, starts))
    return out


@dataclass(frozen=True)
class Config:
    name: str
    batch: int
    n_tokens: int          # tokens per image at block 0, CLS included
    dim: int
    heads: int
    mlp_dim: int
    depth: int
    prune_blocks: tuple
    k_law: str
    score_law: str = "uniform"
    k_max: int = 0          # k_law == "uniform"
    f_lo: float = 0.0       # k_law == "fraction"
    f_hi: float = 0.0
    rho_lo: float = 0.0     # k_law == "geometric"
    rho_hi: float = 1.0
    ln_eps: float = 1e-6
    head_dim: int = 64
    grid: int = 14          # patch grid side (N0 = grid^2)
    patch: int = 16         # patch side in pixels
    layerscale: bool = False  # per-channel scales on both residual branches (DINOv2)
    readout: str = "cls"    # "cls", or "lc1": LN(CLS) ++ mean of LN(surviving visual tokens)
    note: str = field(default="", compare=False)

    @property
    def n_vis0(self) -> int:
        return self.n_tokens - 1


CONFIGS = {
    "cfg1": Config("deit_tiny_1block_b8", 8, 197, 192, 3, 768, 1, (0,), "uniform", k_max=98),
    "cfg2": Config("deit_small_1block_b64", 64, 197, 384, 6, 1536, 1, (0,), "uniform", k_max=147),
    # f range calibrated so the batch-mean Eq. 4 compression is 0.38 +- 0.01
    "cfg3": Config("deit_base_12blk_b256", 256, 197, 768, 12, 3072, 12, (3, 6, 9), "fraction",
                   f_lo=0.20, f_hi=0.45),
    "cfg4": Config("vit_large_24blk_b128", 128, 197, 1024, 16, 4096, 24, (4, 8, 12, 16, 20),
                   "heavy_tail"),
    "cfg5": Config("vit_base384_12blk_b64", 64, 577, 768, 12, 3072, 12, (2, 4, 6, 8, 10),
                   "geometric", score_law="bump", rho_lo=0.15, rho_hi=1.0, grid=24),
    # DINOv2-B/14 (Table 3: N0 = 256): LayerScale, LC1 readout, 14-pixel patches;
    # interventions at the blocks the learned gate picks for it (Sec. 4.3: 1, 2, 3, 6)
    # and f range calibrated to its batch-mean compression (Sec. 4.3: 34.8%)
    "cfg6": Config("dinov2_base14_12blk_b256", 256, 257, 768, 12, 3072, 12, (1, 2, 3, 6),
                   "fraction", f_lo=0.09, f_hi=0.19, grid=16, patch=14, layerscale=True, readout="lc1"),
}


def get_config(name: str, **overrides) -> Config:
    """Look up a configuration, optionally overriding fields (e.g. batch=4)."""
    cfg = CONFIGS[name]
    if overrides:
        d = dict(cfg.__dict__)
        d.update(overrides)
        cfg = Config(**d)
    return cfg


def _round_half_up(x: np.ndarray) -> np.ndarray:
    return np.floor(np.asarray(x, dtype=np.float64) + 0.5).astype(np.int64)


def initial_layout(cfg: Config):
    """cu_seqlens (int32 [B+1]) and original token ids (int32 [T]) at block 0."""
    n = cfg.n_tokens
    cu = (np.arange(cfg.batch + 1, dtype=np.int64) * n).astype(np.int32)
    ids = np.tile(np.arange(n, dtype=np.int32), cfg.batch)
    return cu, ids


def activations_bf16(cfg: Config, seed: int = 0, rows: int | None = None) -> np.ndarray:
    """Block-0 residual stream ``x[T, D]`` as bf16 bits, values ~ N(0, 1)."""
    t = cfg.batch * cfg.n_tokens if rows is None else rows
    return _normal_bf16(seed, TAG_ACT, t * cfg.dim, 1.0).reshape(t, cfg.dim)


_W_NAMES = ("w_qkv", "w_proj", "w_fc1", "w_fc2")


def block_weights(cfg: Config, block: int, seed: int = 0, random_affine: bool = False) -> dict:
    """bf16 weights of one block, nn.Linear layout ``W[out, in]``.

    Linear weights ~ N(0, 0.02^2); biases 0; LayerNorm gamma 1, beta 0.  With
    ``random_affine`` the biases and LayerNorm affines are random instead
    (gamma ~ 1 + N(0, 0.1^2), beta and biases ~ N(0, 0.1^2)), which tests use so
    that every term of the block is exercised.
    """
    d, m = cfg.dim, cfg.mlp_dim
    shapes = {"w_qkv": (3 * d, d), "w_proj": (d, d), "w_fc1": (m, d), "w_fc2": (d, m)}
    out = {}
    for which, nm in enumerate(_W_NAMES):
        r, c = shapes[nm]
        tag = TAG_W + (block << 8) + (which << 4)
        out[nm] = _normal_bf16(seed, tag, r * c, 0.02).reshape(r, c)
    vec = {"b_qkv": 3 * d, "b_proj": d, "b_fc1": m, "b_fc2": d,
           "ln1_w": d, "ln1_b": d, "ln2_w": d, "ln2_b": d}
    if cfg.layerscale:
        for which, nm in enumerate(("ls1", "ls2")):
            u = uniform_f64(seed, TAG_LNAFF + (block << 8) + ((10 + which) << 4),
                            np.arange(d, dtype=np.uint64))
            out[nm] = f32_to_bf16_bits(0.05 + 0.45 * u)          # learned scales ~ 0.05-0.5
    for which, (nm, size) in enumerate(vec.items()):
        if random_affine:
            tag = TAG_LNAFF + (block << 8) + (which << 4)
            v = normal_f64(seed, tag, np.arange(size, dtype=np.uint64)) * 0.1
            if nm.endswith("_w"):
                v = v + 1.0
            out[nm] = f32_to_bf16_bits(v)
        else:
            out[nm] = f32_to_bf16_bits(np.ones(size) if nm.endswith("_w") else np.zeros(size))
    return out


def score_table(cfg: Config, block: int, seed: int = 0) -> np.ndarray:
    """fp32 deletion scores ``table[i, j]`` for image i and original token id j.

    Column 0 is CLS; its value is random and must be ignored by selection.
    Higher score = stronger preference for removal (Eq. 2 and Sec. 3.2).
    """
    b, n = cfg.batch, cfg.n_tokens
    idx = np.arange(b * n, dtype=np.uint64)
    tag = TAG_SCORE + (block << 8)
    if cfg.score_law == "uniform":
        return uniform_f32(seed, tag, idx).reshape(b, n)
    if cfg.score_law == "bump":
        g = cfg.grid
        cidx = np.arange(b, dtype=np.uint64)
        cx = uniform_f64(seed, TAG_BUMP, 4 * cidx) * g
        cy = uniform_f64(seed, TAG_BUMP, 4 * cidx + 1) * g
        sig = 2.0 + 4.0 * uniform_f64(seed, TAG_BUMP, 4 * cidx + 2)
        j = np.arange(n) - 1
        px = (j % g).astype(np.float64) + 0.5
        py = (j // g).astype(np.float64) + 0.5
        d2 = (px[None, :] - cx[:, None]) ** 2 + (py[None, :] - cy[:, None]) ** 2
        eps = normal_f64(seed, tag, idx).reshape(b, n)
        s = 1.0 - np.exp(-d2 / (2.0 * sig[:, None] ** 2)) + 0.1 * eps
        return s.astype(np.float32)
    raise ValueError(cfg.score_law)


def keep_schedule(cfg: Config, seed: int = 0):
    """Per pruning block, the number of tokens each image keeps (CLS included).

    Returns a list of int32 arrays ``m[l]`` of shape [B], one per entry of
    ``cfg.prune_blocks``, and the matching token counts before each block.
    Every removal count is >= 0 and leaves >= 4 visual tokens (Appendix A.2),
    except that an image never grows.
    """
    b = cfg.batch
    n_cur = np.full(b, cfg.n_tokens, dtype=np.int64)
    cidx = np.arange(b, dtype=np.uint64)
    keeps, befores = [], []
    law = cfg.k_law
    if law == "fraction":
        f = cfg.f_lo + (cfg.f_hi - cfg.f_lo) * uniform_f64(seed, TAG_KEEP, cidx)
    elif law == "heavy_tail":
        u_all = uniform_f64(seed, TAG_KEEP, 2 * cidx)
        u = uniform_f64(seed, TAG_KEEP, 2 * cidx + 1)
        rho = np.where(u_all < 0.2, 1.0, 0.2 + 0.8 * u ** 3)
    elif law == "geometric":
        rho = cfg.rho_lo + (cfg.rho_hi - cfg.rho_lo) * uniform_f64(seed, TAG_KEEP, cidx)
    for j, blk in enumerate(cfg.prune_blocks):
        befores.append(n_cur.astype(np.int32).copy())
        n_vis = n_cur - 1
        if law == "uniform":
            h = hash_u64(seed, TAG_KEEP + (blk << 8), cidx)
            k = (h % np.uint64(cfg.k_max + 1)).astype(np.int64)
            k = np.minimum(k, np.maximum(n_vis - 4, 0))
        elif law == "fraction":
            k = 2 * _round_half_up(f * n_vis / 2.0)
            k = np.clip(k, 0, np.maximum(n_vis - 4, 0))
        else:
            frac = (j + 1) / len(cfg.prune_blocks)
            target = np.maximum(4, _round_half_up(cfg.n_vis0 * rho ** frac))
            k = np.clip(n_vis - target, 0, None)
        m = n_cur - k
        keeps.append(m.astype(np.int32))
        n_cur = m
    return keeps, befores


def compression_from_counts(cfg: Config, keeps, befores) -> np.ndarray:
    """Per-image token-layer compression C of Eq. 4 from the count schedule.

    ``N_l^post`` counts visual tokens after block l; blocks without pruning
    carry the count forward.  Returns C for each image.
    """
    L, n0 = cfg.depth, cfg.n_vis0
    post = np.full(cfg.batch, n0, dtype=np.float64)
    total = np.zeros(cfg.batch)
    sched = dict(zip(cfg.prune_blocks, keeps))
    for l in range(L):
        if l in sched:
            post = sched[l].astype(np.float64) - 1.0
        total += n0 - post
    return total / (L * n0)


# ---------------------------------------------------------------------------
# actor weights (random init): shapes of Appendix A.1, nn.Linear layout
# ---------------------------------------------------------------------------

def ACTOR_SHAPES(dim: int, depth: int, n0: int) -> dict:
    """Tensor shapes of the actor's parameters for a backbone of width ``dim``,
    ``depth`` blocks and ``n0`` visual tokens: budget head outputs
    M = (n0 - 4) / 2."""
    m = (n0 - 4) // 2
    return {
        "gate_w1": (64, dim + 19), "gate_b1": (64,), "gate_w2": (1, 64), "gate_b2": (1,),
        "gate_emb": (depth, 16),
        "enc_w_in": (128, dim), "enc_b_in": (128,), "enc_emb": (depth, 128), "enc_w_h": (128, 3),
        "enc_ln1_w": (128,), "enc_ln1_b": (128,), "enc_w_qkv": (384, 128), "enc_b_qkv": (384,),
        "enc_w_o": (128, 128), "enc_b_o": (128,), "enc_ln2_w": (128,), "enc_ln2_b": (128,),
        "enc_w_fc1": (256, 128), "enc_b_fc1": (256,), "enc_w_fc2": (128, 256),
        "enc_b_fc2": (128,),
        "bud_ln_w": (128,), "bud_ln_b": (128,), "bud_w1": (128, 128), "bud_b1": (128,),
        "bud_w2": (m, 128), "bud_b2": (m,),
        "sel_w_k": (128,), "sel_w1": (64, 128), "sel_b1": (64,), "sel_w2": (1, 64),
        "sel_b2": (1,),
    }


def actor_weights(dim: int, depth: int, n0: int, seed: int = 0, gate_bias: float = 0.0) -> dict:
    """bf16 bit patterns of a randomly initialised actor.  Matrices ~
    N(0, 1/fan_in), biases and embeddings ~ N(0, 0.1^2), LayerNorm gains
    1 + N(0, 0.1^2) and shifts N(0, 0.1^2); ``gate_bias`` is added to the
    gate's output bias (tests use it to keep gate decisions clear of 0.5)."""
    out = {}
    for which, (name, shape) in enumerate(ACTOR_SHAPES(dim, depth, n0).items()):
        count = int(np.prod(shape))
        tag = TAG_ACTOR + (which << 8)
        if name.endswith("_emb") or len(shape) == 1 or name in ("gate_b2", "sel_b2"):
            v = normal_f64(seed, tag, np.arange(count, dtype=np.uint64)) * 0.1
            if name.endswith("ln1_w") or name.endswith("ln2_w") or name == "bud_ln_w":
                v = v + 1.0
            if name == "gate_b2":
                v = v + gate_bias
            out[name] = f32_to_bf16_bits(v).reshape(shape)
        else:
            out[name] = _normal_bf16(seed, tag, count, 1.0 / np.sqrt(shape[1])).reshape(shape)
    return out


# ---------------------------------------------------------------------------
# input images and the forward's two ends (patch embedding, classifier)
# ---------------------------------------------------------------------------

def images_bf16(cfg: Config, seed: int = 0, patch: int | None = None,
                channels: int = 3) -> np.ndarray:
    """bf16 bit patterns of N(0, 1) images [B, C, H, W] with H = W = patch *
    sqrt(n_vis0) (224 for 196 visual tokens): normalised pixels, as a
    preprocessing pipeline hands them to the model."""
    patch = cfg.patch if patch is None else patch
    g = int(round(np.sqrt(cfg.n_vis0)))
    assert g * g == cfg.n_vis0
    side = g * patch
    count = cfg.batch * channels * side * side
    return _normal_bf16(seed, TAG_IMG, count, 1.0).reshape(cfg.batch, channels, side, side)


def embed_head_weights(cfg: Config, seed: int = 0, patch: int | None = None, channels: int = 3,
                       classes: int = 1000) -> dict:
    """bf16 bit patterns of the patch embedding (w_pe [d, C patch^2], b_pe, cls,
    pos [N, d]) and the classifier (norm_w, norm_b, w_head [classes, d] -- or
    [classes, 2 d] for the LC1 readout -- and b_head), randomly initialised."""
    patch = cfg.patch if patch is None else patch
    d, k = cfg.dim, channels * patch * patch
    hin = 2 * d if cfg.readout == "lc1" else d
    shapes = {"w_pe": (d, k), "b_pe": (d,), "cls": (d,), "pos": (cfg.n_tokens, d),
              "norm_w": (d,), "norm_b": (d,), "w_head": (classes, hin), "b_head": (classes,)}
    out = {}
    for which, (name, shape) in enumerate(shapes.items()):
        count = int(np.prod(shape))
        tag = TAG_EMBHEAD + (which << 8)
        if name in ("w_pe", "w_head"):
            out[name] = _normal_bf16(seed, tag, count, 1.0 / np.sqrt(shape[1])).reshape(shape)
        else:
            v = normal_f64(seed, tag, np.arange(count, dtype=np.uint64)) * (0.1 if name.startswith("norm") else 0.02)
            if name == "norm_w":
                v = v + 1.0
            out[name] = f32_to_bf16_bits(v).reshape(shape)
    return out
