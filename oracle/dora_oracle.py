"""Plain fp64 CPU oracle for DORA's deployment hot path.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import, call or
link this module: only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` use it.  It shares
no code with the CUDA path (no kernels, headers, helpers or tables).

Every function computes the plain definition of one step of the pruned ViT
block of Eq. 1 (Sec. 3.1), in float64, from bf16/fp32 inputs decoded exactly:

* ``select_keep``   deterministic deletion of the k highest selector scores,
                    CLS kept, survivor order kept (Sec. 3.2 "Sampling and
                    deployment"; Appendix A.3).
* ``compact``       hard deletion into a packed buffer with explicit sequence
                    boundaries (Sec. 3.1 pruning operator; Sec. 3.5
                    "Inference").
* ``varlen_attention``  softmax(Q K^T * scale) V within each image only
                    (Sec. 3.5 "Inference": boundaries prevent attention
                    between different images).
* ``layernorm``, ``linear``, ``gelu``  the standard pre-LN ViT block pieces
                    (Eq. 1; backbones of Sec. 4.1).
* ``pruned_block``  Eq. 1: attention over all N_l+1 tokens, residual, delete,
                    LayerNorm', MLP on survivors, residual.
* ``forward``       Eq. 1 applied block after block.
* ``actor_gate``, ``actor_encoder``, ``actor_budget``, ``actor_selector``,
  ``actor_block``   the deterministic actor that produces each block's gate,
                    removal count and deletion scores (Sec. 3.2 "The actor";
                    Appendix A.1-A.3).
* ``patch_embed``, ``classifier_head``  the forward's two ends, which the
                    paper's GFLOPs and throughput include (App. E.4): the
                    strided patch convolution with CLS and position
                    embeddings, and LayerNorm + linear on each CLS row.
* ``pl_sample_gumbel``, ``pl_logprob``, ``pl_logprob_grad``, ``kd_cost``
                    the training side: Plackett-Luce ordered sampling and
                    log-probability (App. A.3) and the shadows' fidelity cost
                    (App. B.2).
* ``lc1_readout``, ``classifier_head_lc1``, LayerScale in the block halves
                    the DINOv2-B/14 backbone (App. E.3): LayerScale on both
                    residual branches and the LC1 readout.

Readings where the paper is silent:

* Ties: among equal scores the lower index is kept (equivalently the higher
  index is removed first).  Scores are ordered by a total order on fp32:
  -0 equals +0, and every NaN sorts above +inf (removed first).
* ``keep_counts`` include CLS; a count outside [1, n] is clamped and status 5
  is reported.
* LayerNorm uses the biased variance; GELU is the exact erf form; the qkv row
  layout is [3][H][head_dim]; the default softmax scale is 1/sqrt(head_dim).
* Actor: LayerNorm epsilon 1e-5; W_k and W_h carry no bias; budget ties go to
  the smaller removal count; the encoder's attention scale is 1/sqrt(32);
  every image gets a budget and selector scores (the gate only decides
  whether they are used); E_<l / (L - 1) divides by 1 when L = 1.
* DINOv2: LayerScale multiplies each branch's output (after its last linear,
  before the residual add) per channel; the LC1 mean runs over the visual
  rows that survive the last deletion, zero when none does.
* Training: the ordered sample is the Gumbel-top-k of the scores (keys
  formed in fp32, noise an input); the fidelity cost runs over the true
  classes only.

Parity pins: every function here is checked in ``tests/test_oracle_pins.py``
against brute force, closed forms, invariants the paper fixes, or an
independent library routine.
"""
from __future__ import annotations

import math

import numpy as np

DORA_OK = 0
DORA_ERR_DEVICE_BAD_COUNT = 5
DORA_ERR_DEVICE_SEQLEN = 6


# ----------------------------------------------------------------------------
# decoding (exact)
# ----------------------------------------------------------------------------

def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact value of bf16 bit patterns (uint16) as float64."""
    u = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return u.view(np.float32).astype(np.float64)


# ----------------------------------------------------------------------------
# O1: selection (Sec. 3.2 "Sampling and deployment"; Appendix A.3)
# ----------------------------------------------------------------------------

def score_order_key(scores: np.ndarray) -> np.ndarray:
    """Map fp32 scores to uint32 keys whose unsigned order is the score order.

    Total order used for the deterministic top-k: -0.0 and +0.0 are equal, every
    NaN is larger than +inf.  For a non-NaN float with bits b the key is
    ``~b`` when the sign bit is set and ``b | 0x80000000`` otherwise, which
    makes unsigned comparison of keys agree with real comparison of values.
    """
    s = np.ascontiguousarray(np.asarray(scores, dtype=np.float32))
    b = s.view(np.uint32).copy()
    b[b == np.uint32(0x80000000)] = np.uint32(0)
    neg = (b >> np.uint32(31)) == 1
    key = np.where(neg, ~b, b | np.uint32(0x80000000)).astype(np.uint32)
    key[np.isnan(s)] = np.uint32(0xFFFFFFFF)
    return key


def select_keep(scores: np.ndarray, cu_in: np.ndarray, keep_counts: np.ndarray):
    """Deterministic deployment selection, one image at a time.

    For image i with rows [cu_in[i], cu_in[i+1]) (n rows, local row 0 = CLS) and
    m = keep_counts[i] tokens to keep (CLS included), the k = n - m visual tokens
    with the highest deletion scores are removed; CLS is never a candidate.
    Equal scores: the lower local index is kept.  Kept rows are emitted in
    ascending order as global row indices of the input packed buffer.

    Returns ``(kept_idx int32[T_out], cu_out int32[B+1], status)``.
    """
    cu_in = np.asarray(cu_in, dtype=np.int64)
    keep_counts = np.asarray(keep_counts, dtype=np.int64)
    batch = len(cu_in) - 1
    key = score_order_key(scores)
    status = DORA_OK
    kept_all = []
    cu_out = np.zeros(batch + 1, dtype=np.int64)
    for i in range(batch):
        lo, hi = int(cu_in[i]), int(cu_in[i + 1])
        n = hi - lo
        m = int(keep_counts[i])
        m_eff = min(max(m, min(1, n)), n)
        if m_eff != m:
            status = DORA_ERR_DEVICE_BAD_COUNT
        if n > 0 and m_eff > 0:
            j = np.arange(1, n, dtype=np.int64)            # visual candidates
            cand_key = key[lo + 1:hi].astype(np.int64)
            order = np.lexsort((j, cand_key))               # by key, then index
            keep_local = np.sort(np.concatenate(([0], j[order[:m_eff - 1]])))
            kept_all.append(lo + keep_local)
        cu_out[i + 1] = cu_out[i] + m_eff
    kept = np.concatenate(kept_all) if kept_all else np.zeros(0, dtype=np.int64)
    return kept.astype(np.int32), cu_out.astype(np.int32), status


# ----------------------------------------------------------------------------
# O2: compaction (Sec. 3.1 pruning operator; Sec. 3.5 "Inference")
# ----------------------------------------------------------------------------

def compact(x: np.ndarray, kept_idx: np.ndarray, ids_in: np.ndarray | None = None):
    """Packed survivors: ``packed[r] = x[kept_idx[r]]`` bit for bit.

    ``x`` may hold raw bf16 bits (uint16) or any dtype; rows are copied
    unchanged.  Original token ids are carried the same way.
    """
    kept_idx = np.asarray(kept_idx, dtype=np.int64)
    packed = np.asarray(x)[kept_idx].copy()
    ids_out = None if ids_in is None else np.asarray(ids_in)[kept_idx].copy()
    return packed, ids_out


def cu_from_counts(counts: np.ndarray) -> np.ndarray:
    """Sequence boundaries of a packed buffer: exclusive prefix sum, int32 [B+1]."""
    out = np.zeros(len(counts) + 1, dtype=np.int64)
    for i, c in enumerate(counts):
        out[i + 1] = out[i] + int(c)
    return out.astype(np.int32)


# ----------------------------------------------------------------------------
# O3: packed variable-length attention (Sec. 3.5 "Inference")
# ----------------------------------------------------------------------------

def attention_single(q: np.ndarray, k: np.ndarray, v: np.ndarray, scale: float):
    """softmax(q k^T * scale) v for one image and one head, float64.

    Returns ``(O, P)`` where P is the row-stochastic attention matrix.
    """
    s = (q @ k.T) * scale
    s = s - s.max(axis=1, keepdims=True)
    e = np.exp(s)
    p = e / e.sum(axis=1, keepdims=True)
    return p @ v, p


def varlen_attention(qkv: np.ndarray, cu: np.ndarray, heads: int, head_dim: int = 64,
                     scale: float | None = None) -> np.ndarray:
    """Multi-head self-attention restricted to each image's rows.

    ``qkv`` is [T, 3*heads*head_dim] (bf16 bits or float); row layout
    [3][heads][head_dim] = (q, k, v).  Output [T, heads*head_dim] float64.
    Rows beyond cu[-1] are left at zero.
    """
    if scale is None or scale == 0.0:
        scale = 1.0 / math.sqrt(head_dim)
    a = bf16_to_f64(qkv) if np.asarray(qkv).dtype == np.uint16 else np.asarray(qkv, np.float64)
    t = a.shape[0]
    a = a.reshape(t, 3, heads, head_dim)
    out = np.zeros((t, heads, head_dim))
    cu = np.asarray(cu, dtype=np.int64)
    for i in range(len(cu) - 1):
        lo, hi = int(cu[i]), int(cu[i + 1])
        if hi <= lo:
            continue
        for h in range(heads):
            o, _ = attention_single(a[lo:hi, 0, h], a[lo:hi, 1, h], a[lo:hi, 2, h], scale)
            out[lo:hi, h] = o
    return out.reshape(t, heads * head_dim)


def padded_masked_attention(qkv: np.ndarray, cu: np.ndarray, heads: int, head_dim: int = 64,
                            scale: float | None = None) -> np.ndarray:
    """The same attention computed the padded way: every image padded to the
    longest, keys beyond each image's length masked with -inf.  Used only to pin
    ``varlen_attention`` (Sec. 3.5: packing removes batch-wide padding but must
    not change the result)."""
    if scale is None or scale == 0.0:
        scale = 1.0 / math.sqrt(head_dim)
    a = bf16_to_f64(qkv) if np.asarray(qkv).dtype == np.uint16 else np.asarray(qkv, np.float64)
    t = a.shape[0]
    a = a.reshape(t, 3, heads, head_dim)
    cu = np.asarray(cu, dtype=np.int64)
    b = len(cu) - 1
    lens = cu[1:] - cu[:-1]
    nmax = int(lens.max()) if b else 0
    pad = np.zeros((b, nmax, 3, heads, head_dim))
    for i in range(b):
        pad[i, :lens[i]] = a[cu[i]:cu[i + 1]]
    q = pad[:, :, 0].transpose(0, 2, 1, 3)        # [B, H, n, d]
    k = pad[:, :, 1].transpose(0, 2, 1, 3)
    v = pad[:, :, 2].transpose(0, 2, 1, 3)
    s = np.einsum("bhqd,bhkd->bhqk", q, k) * scale
    keymask = np.arange(nmax)[None, :] < lens[:, None]          # [B, n]
    s = np.where(keymask[:, None, None, :], s, -np.inf)
    s = s - s.max(axis=-1, keepdims=True)
    e = np.exp(s)
    p = e / e.sum(axis=-1, keepdims=True)
    o = np.einsum("bhqk,bhkd->bhqd", p, v).transpose(0, 2, 1, 3)  # [B, n, H, d]
    out = np.zeros((t, heads, head_dim))
    for i in range(b):
        out[cu[i]:cu[i + 1]] = o[i, :lens[i]]
    return out.reshape(t, heads * head_dim)


# ----------------------------------------------------------------------------
# O4: block pieces and the pruned block (Eq. 1)
# ----------------------------------------------------------------------------

def layernorm(x: np.ndarray, w: np.ndarray, b: np.ndarray, eps: float) -> np.ndarray:
    """Row LayerNorm with biased variance and affine ``w``, ``b`` (float64)."""
    x = np.asarray(x, dtype=np.float64)
    mu = x.mean(axis=1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * w + b


def linear(x: np.ndarray, w: np.ndarray, b: np.ndarray) -> np.ndarray:
    """nn.Linear: ``y = x W^T + b`` with ``W`` stored [out, in]."""
    return np.asarray(x, np.float64) @ np.asarray(w, np.float64).T + b


_ERF = np.vectorize(math.erf, otypes=[np.float64])


def gelu(x: np.ndarray) -> np.ndarray:
    """Exact GELU, 0.5 x (1 + erf(x / sqrt 2))."""
    x = np.asarray(x, dtype=np.float64)
    return 0.5 * x * (1.0 + _ERF(x / math.sqrt(2.0)))


def decode_weights(w: dict) -> dict:
    """bf16-bit weight dict (as produced by the synthetic generator) to float64."""
    return {k: bf16_to_f64(v) for k, v in w.items()}


def block_attention_half(x: np.ndarray, cu: np.ndarray, wf: dict, heads: int, eps: float,
                         head_dim: int = 64) -> np.ndarray:
    """First line of Eq. 1: H_attn = H + Attention(LayerNorm(H)), attention
    including its output projection, over all tokens of each image."""
    xn = layernorm(x, wf["ln1_w"], wf["ln1_b"], eps)
    qkv = linear(xn, wf["w_qkv"], wf["b_qkv"])
    o = varlen_attention(qkv, cu, heads, head_dim)
    a = linear(o, wf["w_proj"], wf["b_proj"])
    if "ls1" in wf:                                   # LayerScale (DINOv2 backbones)
        a = a * wf["ls1"]
    return x + a


def block_mlp_half(h_keep: np.ndarray, wf: dict, eps: float) -> np.ndarray:
    """Second line of Eq. 1: H_{l+1} = H_keep + MLP(LayerNorm'(H_keep))."""
    y = linear(layernorm(h_keep, wf["ln2_w"], wf["ln2_b"], eps), wf["w_fc1"], wf["b_fc1"])
    y = linear(gelu(y), wf["w_fc2"], wf["b_fc2"])
    if "ls2" in wf:                                   # LayerScale (DINOv2 backbones)
        y = y * wf["ls2"]
    return h_keep + y


def pruned_block(x: np.ndarray, cu_in: np.ndarray, ids_in: np.ndarray, wf: dict, heads: int,
                 eps: float, scores: np.ndarray | None = None,
                 keep_counts: np.ndarray | None = None, head_dim: int = 64) -> dict:
    """One ViT block with optional hard pruning, Eq. 1.

    ``x`` is float64 [T_in, D] (decode bf16 inputs first).  Deletion happens
    after the attention residual and before LayerNorm' (Eq. 1; Appendix A.3),
    so deleted tokens take part in this block's attention only.  Returns a dict
    with ``x_out``, ``cu_out``, ``ids_out``, ``kept_idx`` (None without pruning),
    ``h_attn`` and ``status``.
    """
    x = np.asarray(x, dtype=np.float64)
    h_attn = block_attention_half(x, cu_in, wf, heads, eps, head_dim)
    status = DORA_OK
    if scores is None:
        kept, cu_out, h_keep, ids_out = None, np.asarray(cu_in, np.int32), h_attn, ids_in
    else:
        kept, cu_out, status = select_keep(scores, cu_in, keep_counts)
        h_keep, ids_out = compact(h_attn, kept, ids_in)
    x_out = block_mlp_half(h_keep, wf, eps)
    return dict(x_out=x_out, cu_out=cu_out, ids_out=ids_out, kept_idx=kept,
                h_attn=h_attn, status=status)


# ----------------------------------------------------------------------------
# O5: the whole pruned forward (Eq. 1 block after block)
# ----------------------------------------------------------------------------

def gather_scores(table: np.ndarray, cu: np.ndarray, ids: np.ndarray) -> np.ndarray:
    """Row-aligned scores from a per-image table indexed by original token id.

    Stand-in for the actor's selector output (Eq. 2): each surviving row gets
    the score its image's table assigns to that token's original id.
    """
    cu = np.asarray(cu, dtype=np.int64)
    out = np.zeros(int(cu[-1]), dtype=np.float32)
    for i in range(len(cu) - 1):
        out[cu[i]:cu[i + 1]] = table[i, ids[cu[i]:cu[i + 1]]]
    return out


def forward(x: np.ndarray, cu: np.ndarray, ids: np.ndarray, blocks: list, heads: int,
            eps: float, prune: dict | None = None, head_dim: int = 64) -> dict:
    """Eq. 1 over all blocks.  ``blocks`` is a list of float64 weight dicts;
    ``prune`` maps block index to ``(score_table, keep_counts)``.  Returns the
    final ``x``, ``cu``, ``ids`` and the list of per-block ``kept_idx``."""
    prune = prune or {}
    x = np.asarray(x, dtype=np.float64)
    kept_hist = []
    for l, wf in enumerate(blocks):
        if l in prune:
            table, keep = prune[l]
            s = gather_scores(table, cu, ids)
            r = pruned_block(x, cu, ids, wf, heads, eps, s, keep, head_dim)
        else:
            r = pruned_block(x, cu, ids, wf, heads, eps, None, None, head_dim)
        x, cu, ids = r["x_out"], r["cu_out"], r["ids_out"]
        kept_hist.append(r["kept_idx"])
    return dict(x=x, cu=cu, ids=ids, kept=kept_hist)


# ----------------------------------------------------------------------------
# O6: the deployment actor (Sec. 3.2 "The actor"; Appendix A.1-A.3)
# ----------------------------------------------------------------------------
# Widths fixed by Appendix A.1.
ACTOR_WIDTH = 128          # shared encoder width (four heads of 32)
ACTOR_HEADS = 4
ACTOR_FF = 256             # encoder feed-forward 128 -> 256 -> 128
ACTOR_GATE_HIDDEN = 64     # gate (d + 19) -> 64 -> 1
ACTOR_GATE_EMB = 16        # gate block embedding
ACTOR_SEL_HIDDEN = 64      # selector 128 -> 64 -> 1
ACTOR_EPS = 1e-5           # the actor's LayerNorm epsilon (paper silent: PyTorch default)


def sigmoid(x):
    """Logistic function, written through tanh so that it never overflows:
    1 / (1 + e^-x) = (1 + tanh(x / 2)) / 2."""
    return 0.5 * (1.0 + np.tanh(0.5 * np.asarray(x, dtype=np.float64)))


def silu(x):
    """SiLU, x * sigmoid(x)."""
    x = np.asarray(x, dtype=np.float64)
    return x * sigmoid(x)


def budget_grid(n0: int) -> np.ndarray:
    """Candidate removal counts B = {2, 4, ..., N0 - 4} (Appendix A.2)."""
    return np.arange(2, n0 - 4 + 1, 2, dtype=np.int64)


def actor_history(n_l: int, n0: int, rho: float, interventions: int, depth: int) -> np.ndarray:
    """h_l = [N_l / N0, rho_l, E_<l / (L - 1)] (Appendix A.1, history vector);
    for a single-block model (L = 1) the last entry divides by 1."""
    return np.array([n_l / n0, rho, interventions / max(depth - 1, 1)], dtype=np.float64)


def actor_gate(k_cls: np.ndarray, e_gate: np.ndarray, h: np.ndarray, w: dict) -> float:
    """p^G = sigmoid(MLP([K_CLS, e^G_l, h_l])): a (d + 19) -> 64 -> 1 MLP with
    a SiLU hidden layer (Appendix A.1, gate)."""
    z = np.concatenate([np.asarray(k_cls, np.float64), e_gate, h])
    hid = silu(w["gate_w1"] @ z + w["gate_b1"])
    return float(sigmoid(w["gate_w2"][0] @ hid + w["gate_b2"][0]))


def actor_encoder(keys: np.ndarray, e_enc: np.ndarray, h: np.ndarray, w: dict,
                  eps: float = ACTOR_EPS) -> np.ndarray:
    """Z_l for one image (Appendix A.1, shared encoder).  ``keys`` [N_l + 1, d]
    with row 0 the CLS key.  X_j = W_in K_j + b_in + e^C_l, plus W_h h_l on CLS
    only; then one pre-LayerNorm Transformer block of width 128 with four
    attention heads and a 128 -> 256 -> 128 GELU feed-forward sublayer."""
    x = linear(keys, w["enc_w_in"], w["enc_b_in"]) + e_enc
    x[0] += w["enc_w_h"] @ h
    n = x.shape[0]
    qkv = linear(layernorm(x, w["enc_ln1_w"], w["enc_ln1_b"], eps), w["enc_w_qkv"],
                 w["enc_b_qkv"])
    o = varlen_attention(qkv, np.array([0, n]), ACTOR_HEADS, ACTOR_WIDTH // ACTOR_HEADS)
    z1 = x + linear(o, w["enc_w_o"], w["enc_b_o"])
    f = linear(layernorm(z1, w["enc_ln2_w"], w["enc_ln2_b"], eps), w["enc_w_fc1"],
               w["enc_b_fc1"])
    return z1 + linear(gelu(f), w["enc_w_fc2"], w["enc_b_fc2"])


def actor_budget(z_cls: np.ndarray, n_l: int, n0: int, w: dict, eps: float = ACTOR_EPS):
    """Deployment budget (Sec. 3.2; Appendix A.3): LayerNorm(Z_CLS) then a
    128 -> 128 -> M GELU MLP gives one logit per grid entry; budgets that would
    leave fewer than four visual tokens (k > N_l - 4) are masked; the highest
    remaining logit wins (ties: the smaller budget).  Returns (k, logits);
    k = 0 when no budget is feasible."""
    u = layernorm(np.asarray(z_cls, np.float64)[None], w["bud_ln_w"], w["bud_ln_b"], eps)[0]
    logits = w["bud_w2"] @ gelu(w["bud_w1"] @ u + w["bud_b1"]) + w["bud_b2"]
    grid = budget_grid(n0)
    feasible = grid <= n_l - 4
    if not feasible.any():
        return 0, logits
    masked = np.where(feasible, logits, -np.inf)
    return int(grid[int(np.argmax(masked))]), logits


def actor_selector(z_vis: np.ndarray, k: int, n_l: int, w: dict) -> np.ndarray:
    """Eq. 2: s_j = MLP_S(Z_j + W_k k / N_l), a shared 128 -> 64 -> 1 SiLU MLP
    over the visual tokens; higher means remove first."""
    u = np.asarray(z_vis, np.float64) + w["sel_w_k"] * (k / n_l)
    return silu(u @ w["sel_w1"].T + w["sel_b1"]) @ w["sel_w2"][0] + w["sel_b2"][0]


def actor_block(keys: np.ndarray, cu: np.ndarray, block: int, n0: int, depth: int,
                rho: np.ndarray, interventions: np.ndarray, w: dict,
                eps: float = ACTOR_EPS) -> dict:
    """The deterministic actor at one block for every image of a packed batch
    (Sec. 3.2 "Sampling and deployment"; Appendix A.3).

    ``keys`` [T, d] are the block's keys (heads concatenated), row-aligned with
    the packed tokens; ``rho`` and ``interventions`` hold each image's rho_l
    and E_<l.  Every image gets a gate probability, a budget (argmax over its
    feasible grid) and selector scores computed with that budget; the gate
    opens when p >= 0.5 and a budget is feasible, and then k_l = the budget,
    otherwise k_l = 0.  Returns p, gate, budget, k, keep_counts (N_l + 1 - k_l,
    CLS included), scores [T] (CLS rows 0), z [T, 128], logits [B, M], and the
    next block's rho and interventions."""
    keys = bf16_to_f64(keys) if np.asarray(keys).dtype == np.uint16 else np.asarray(keys,
                                                                                   np.float64)
    cu = np.asarray(cu, dtype=np.int64)
    b = len(cu) - 1
    p = np.zeros(b)
    gate = np.zeros(b, dtype=np.int32)
    budget = np.zeros(b, dtype=np.int32)
    k = np.zeros(b, dtype=np.int32)
    scores = np.zeros(int(cu[-1]))
    z = np.zeros((int(cu[-1]), ACTOR_WIDTH))
    logits = np.zeros((b, len(budget_grid(n0))))
    for i in range(b):
        lo, hi = int(cu[i]), int(cu[i + 1])
        n_l = hi - lo - 1
        h = actor_history(n_l, n0, float(rho[i]), int(interventions[i]), depth)
        p[i] = actor_gate(keys[lo], w["gate_emb"][block], h, w)
        zi = actor_encoder(keys[lo:hi], w["enc_emb"][block], h, w, eps)
        z[lo:hi] = zi
        budget[i], logits[i] = actor_budget(zi[0], n_l, n0, w, eps)
        if n_l > 0:                                   # an image of CLS alone has nothing to score
            scores[lo + 1:hi] = actor_selector(zi[1:], int(budget[i]), n_l, w)
        gate[i] = int(p[i] >= 0.5 and budget[i] > 0)
        k[i] = budget[i] if gate[i] else 0
    n_vis = np.diff(cu) - 1
    return dict(p=p, gate=gate, budget=budget, k=k, keep_counts=(n_vis + 1 - k).astype(np.int32),
                scores=scores, z=z, logits=logits,
                rho_next=np.where(gate == 1, k / np.maximum(n_vis, 1), 0.0),
                interventions_next=np.asarray(interventions) + gate)


# ----------------------------------------------------------------------------
# O7: the two ends of the forward (backbones of Sec. 4.1; App. E.4 counts them)
# ----------------------------------------------------------------------------

def patch_embed(images: np.ndarray, w_pe: np.ndarray, b_pe: np.ndarray, cls: np.ndarray,
                pos: np.ndarray, patch: int) -> np.ndarray:
    """ViT input tokens: a patch x patch convolution with stride patch (weights
    [d, C, patch, patch] stored as [d, C * patch * patch]), then each image's
    CLS token prepended and the position embeddings added.  ``images``
    [B, C, H, W] (bf16 bits or float); returns [B * (g_h g_w + 1), d] packed
    image after image, row 0 of each image its CLS token."""
    im = bf16_to_f64(images) if np.asarray(images).dtype == np.uint16 else np.asarray(images,
                                                                                     np.float64)
    b, c, h, w = im.shape
    gh, gw = h // patch, w // patch
    p = im.reshape(b, c, gh, patch, gw, patch).transpose(0, 2, 4, 1, 3, 5)
    p = p.reshape(b * gh * gw, c * patch * patch)
    d = w_pe.shape[0]
    emb = linear(p, w_pe, b_pe).reshape(b, gh * gw, d) + pos[1:]
    out = np.concatenate([np.broadcast_to(cls + pos[0], (b, 1, d)), emb], axis=1)
    return out.reshape(b * (gh * gw + 1), d)


def classifier_head(x: np.ndarray, cu: np.ndarray, ln_w: np.ndarray, ln_b: np.ndarray,
                    eps: float, w_head: np.ndarray, b_head: np.ndarray) -> np.ndarray:
    """The classifier of a CLS-readout ViT: the final LayerNorm on each image's
    CLS row (row cu[i]) and a linear layer to the class logits [B, classes]."""
    x = np.asarray(x, dtype=np.float64)
    rows = np.asarray(cu[:-1], dtype=np.int64)
    return linear(layernorm(x[rows], ln_w, ln_b, eps), w_head, b_head)


def lc1_readout(x: np.ndarray, cu: np.ndarray, ln_w: np.ndarray, ln_b: np.ndarray,
                eps: float) -> np.ndarray:
    """DINOv2's LC1 readout (App. E.3, baseline implementations): the final
    LayerNorm applied to every token, then each image's normalised CLS row
    concatenated with the mean of its normalised surviving visual rows
    ([B, 2 d]; an image without visual tokens contributes a zero mean)."""
    x = np.asarray(x, dtype=np.float64)
    cu = np.asarray(cu, dtype=np.int64)
    d = x.shape[1]
    out = np.zeros((len(cu) - 1, 2 * d))
    for i in range(len(cu) - 1):
        lo, hi = int(cu[i]), int(cu[i + 1])
        if hi <= lo:
            continue
        xn = layernorm(x[lo:hi], ln_w, ln_b, eps)
        out[i, :d] = xn[0]
        if hi - lo > 1:
            out[i, d:] = xn[1:].mean(axis=0)
    return out


def classifier_head_lc1(x: np.ndarray, cu: np.ndarray, ln_w: np.ndarray, ln_b: np.ndarray,
                        eps: float, w_head: np.ndarray, b_head: np.ndarray) -> np.ndarray:
    """Class logits from the LC1 features (App. E.3): the linear layer
    w_head [classes, 2 d] applied to lc1_readout's [B, 2 d] rows."""
    return linear(lc1_readout(x, cu, ln_w, ln_b, eps), w_head, b_head)


# ----------------------------------------------------------------------------
# O8: training side (App. A.3 "Training-time sampling"; App. B.2-B.3 shadow
# evaluation and its fidelity cost)
# ----------------------------------------------------------------------------

def pl_sample_gumbel(scores: np.ndarray, gumbel: np.ndarray, k: int) -> np.ndarray:
    """Ordered removal sequence (i_1, ..., i_k) drawn without replacement from
    the Plackett-Luce distribution of the selector scores (App. A.3), as the
    Gumbel-top-k of the scores: the k largest keys s_j + g_j in decreasing
    order, g_j standard Gumbel noise supplied by the caller.  The keys are
    formed in fp32 (the precision the decision is taken in on both sides);
    -0 equals +0, NaN ranks above +inf, and equal keys go to the higher index
    first -- the tie rule of select_keep, so the first k entries are exactly
    the tokens that deterministic selection on the keys s + g deletes."""
    s = np.asarray(scores, dtype=np.float32)
    g = np.asarray(gumbel, dtype=np.float32)
    keys = score_order_key((s + g).astype(np.float32))
    order = sorted(range(len(s)), key=lambda j: (-int(keys[j]), -j))
    return np.array(order[:k], dtype=np.int64)


def _logsumexp(v: np.ndarray) -> float:
    v = np.asarray(v, dtype=np.float64)
    m = float(np.max(v))
    return m + math.log(float(np.sum(np.exp(v - m))))


def pl_logprob(scores: np.ndarray, order: np.ndarray) -> float:
    """Plackett-Luce log-probability of the ordered sequence (App. A.3):
    sum over t of s_{i_t} - log sum_{j in R_t} exp(s_j), with R_t the indices
    not yet removed before step t."""
    s = np.asarray(scores, dtype=np.float64)
    remaining = list(range(len(s)))
    total = 0.0
    for i in order:
        total += s[int(i)] - _logsumexp(s[remaining])
        remaining.remove(int(i))
    return total


def pl_logprob_grad(scores: np.ndarray, order: np.ndarray) -> np.ndarray:
    """Gradient of pl_logprob with respect to every score: each step t adds 1
    at i_t and subtracts the softmax of the scores over R_t."""
    s = np.asarray(scores, dtype=np.float64)
    grad = np.zeros(len(s))
    remaining = list(range(len(s)))
    for i in order:
        r = np.array(remaining)
        p = np.exp(s[r] - _logsumexp(s[r]))
        grad[r] -= p
        grad[int(i)] += 1.0
        remaining.remove(int(i))
    return grad


def log_softmax(z: np.ndarray) -> np.ndarray:
    z = np.asarray(z, dtype=np.float64)
    return z - _logsumexp(z)


def kd_cost(z_native: np.ndarray, z: np.ndarray, tau: float = 3.0) -> float:
    """Per-image fidelity cost of a shadow (App. B.2): tau^2 times the KL
    divergence from softmax(z_native / tau) to softmax(z / tau), tau = 3."""
    lp_n = log_softmax(np.asarray(z_native, dtype=np.float64) / tau)
    lp = log_softmax(np.asarray(z, dtype=np.float64) / tau)
    return tau * tau * float(np.sum(np.exp(lp_n) * (lp_n - lp)))


def shadow_forwards(x: np.ndarray, cu: np.ndarray, ids: np.ndarray, blocks: list, heads: int,
                    eps: float, prune: dict, head_dim: int = 64) -> dict:
    """Complete-prefix shadows (App. B.2): for each pruning block l of the
    rollout, the forward that replays the rollout's deletions at blocks
    0..l and runs every later block without deletion; key -1 is the empty
    prefix (the Native forward).  Each value is forward()'s result."""
    out = {-1: forward(x, cu, ids, blocks, heads, eps, {}, head_dim)}
    for l in sorted(prune):
        out[l] = forward(x, cu, ids, blocks, heads, eps,
                         {b: v for b, v in prune.items() if b <= l}, head_dim)
    return out


def step_rewards(costs: np.ndarray, removals: np.ndarray, blocks, depth: int, n0: int,
                 a: float) -> np.ndarray:
    """Local rewards of one image's actions (App. B.3): at the l-th acting
    block r_l = 25 Delta C_l - a (D_l - D_{l-1}), Delta C_l = k_l (L - l) /
    (L N0) (Eq. 4's per-block term), D_{-1} = 0.  costs[j] and removals[j]
    belong to blocks[j] (increasing)."""
    out = np.zeros(len(blocks))
    prev = 0.0
    for j, l in enumerate(blocks):
        dc = removals[j] * (depth - l) / (depth * n0)
        out[j] = 25.0 * dc - a * (costs[j] - prev)
        prev = costs[j]
    return out

