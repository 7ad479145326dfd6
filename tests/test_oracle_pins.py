"""Pins for the fp64 oracle: each check comes from outside the oracle itself
(brute force, closed forms, invariants the paper fixes, an independent library
routine, or values the paper prints)."""
import itertools
import math
import os

import numpy as np
import scipy.special
import scipy.stats
import pytest
import torch

import dora_synth as S
import oracle as O

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


# ---------------------------------------------------------------------------
# selection (Sec. 3.2 "Sampling and deployment"; Appendix A.3)
# ---------------------------------------------------------------------------

def _removal_before(a_score, a_idx, b_score, b_idx):
    """True when token a is removed before token b, by the rule written with
    Python float semantics: larger score first, NaN largest of all, equal
    scores (including -0 == +0) remove the higher index first."""
    an, bn = math.isnan(a_score), math.isnan(b_score)
    if an or bn:
        if an and bn:
            return a_idx > b_idx
        return an
    if a_score != b_score:
        return a_score > b_score
    return a_idx > b_idx


def _brute_force_keep(scores, m):
    """Enumerate every subset of visual tokens of size m-1 and return the unique
    one such that every kept token would be removed after every removed one."""
    n = len(scores)
    vis = list(range(1, n))
    valid = []
    for keep in itertools.combinations(vis, m - 1):
        ks = set(keep)
        removed = [j for j in vis if j not in ks]
        if all(_removal_before(scores[r], r, scores[k], k) for r in removed for k in keep):
            valid.append([0] + list(keep))
    assert len(valid) == 1, valid
    return valid[0]


def _select_one(scores, m):
    s = np.asarray(scores, dtype=np.float32)
    kept, cu_out, st = O.select_keep(s, np.array([0, len(s)]), np.array([m]))
    return kept.tolist(), cu_out.tolist(), st


def test_select_brute_force_small():
    rng = np.random.default_rng(1)
    palette = np.array([0.0, -0.0, 0.25, 0.5, -1.0, np.inf, -np.inf, np.nan, 1e-30],
                       dtype=np.float32)
    for trial in range(300):
        n = int(rng.integers(1, 10))
        if trial % 3 == 0:
            s = rng.choice(palette, size=n)
        else:
            s = rng.random(n).astype(np.float32)
        for m in range(1, n + 1):
            kept, cu_out, st = _select_one(s, m)
            assert kept == _brute_force_keep([float(v) for v in s], m)
            assert cu_out == [0, m] and st == 0


def test_select_golden_cases(golden_dir):
    with open(os.path.join(golden_dir, "select_cases.txt")) as f:
        lines = [ln.strip() for ln in f if ln.strip() and not ln.startswith("#")]
    assert len(lines) >= 8
    for ln in lines:
        s_txt, m_txt, k_txt = [p.strip() for p in ln.split("|")]
        s = [float(v) for v in s_txt.split(",")]
        kept, _, st = _select_one(s, int(m_txt))
        assert kept == [int(v) for v in k_txt.split(",")], ln
        assert st == 0


def test_select_distinct_equals_partial_sort():
    rng = np.random.default_rng(2)
    for _ in range(50):
        n = int(rng.integers(2, 600))
        s = rng.permutation(n).astype(np.float32) - n / 2   # distinct
        m = int(rng.integers(1, n + 1))
        kept, _, _ = _select_one(s, m)
        vis = s[1:]
        k = n - m
        removed = set((np.argsort(-vis, kind="stable")[:k] + 1).tolist())
        expect = [j for j in range(n) if j not in removed]
        assert kept == expect


def test_select_all_equal_keeps_prefix():
    for n in (1, 2, 17, 197, 577):
        for m in sorted({1, min(2, n), n // 2 or 1, n}):
            kept, _, _ = _select_one(np.full(n, 0.5), m)
            assert kept == list(range(m))


def test_select_invariants_all_configs():
    for name in ("cfg1", "cfg2", "cfg3", "cfg4", "cfg5"):
        cfg = S.get_config(name, batch=min(S.get_config(name).batch, 32))
        cu, ids = S.initial_layout(cfg)
        keeps, befores = S.keep_schedule(cfg, seed=3)
        table = S.score_table(cfg, cfg.prune_blocks[0], seed=3)
        scores = O.gather_scores(table, cu, ids)
        kept, cu_out, st = O.select_keep(scores, cu, keeps[0])
        assert st == 0
        assert np.array_equal(cu_out, O.cu_from_counts(keeps[0]))
        for i in range(cfg.batch):
            seg = kept[cu_out[i]:cu_out[i + 1]]
            assert len(seg) == keeps[0][i]                 # |kept| = N_i - k_i
            assert seg[0] == cu[i]                         # CLS retained
            assert np.all(np.diff(seg) > 0)                # order preserved
            assert seg[-1] < cu[i + 1]


def test_select_clamps_bad_counts():
    s = np.random.default_rng(4).random(10).astype(np.float32)
    cu = np.array([0, 4, 10])
    kept, cu_out, st = O.select_keep(s, cu, np.array([0, 11]))
    assert st == O.DORA_ERR_DEVICE_BAD_COUNT
    assert cu_out.tolist() == [0, 1, 7]
    assert kept[0] == 0 and kept[1:].tolist() == list(range(4, 10))
    # empty image: nothing kept, count 0 is fine
    kept, cu_out, st = O.select_keep(s[:3], np.array([0, 0, 3]), np.array([0, 2]))
    assert st == 0 and cu_out.tolist() == [0, 0, 2]


# ---------------------------------------------------------------------------
# compaction
# ---------------------------------------------------------------------------

def test_compact_matches_naive_copy():
    rng = np.random.default_rng(5)
    x = rng.integers(0, 65536, size=(50, 24), dtype=np.uint16)
    ids = rng.integers(0, 1000, size=50).astype(np.int32)
    kept = np.sort(rng.choice(50, size=20, replace=False)).astype(np.int32)
    packed, ids_out = O.compact(x, kept, ids)
    for r, src in enumerate(kept):
        assert packed[r].tobytes() == x[src].tobytes()
        assert ids_out[r] == ids[src]


def test_cu_from_counts_closed_form():
    counts = np.array([3, 0, 5, 1])
    assert O.cu_from_counts(counts).tolist() == [0, 3, 3, 8, 9]
    c = np.random.default_rng(6).integers(0, 300, size=200)
    cu = O.cu_from_counts(c)
    assert cu[-1] == c.sum() and np.all(np.diff(cu) == c)


# ---------------------------------------------------------------------------
# attention (Sec. 3.5 "Inference")
# ---------------------------------------------------------------------------

def _rand_qkv(t, h, rng, d=64):
    return rng.standard_normal((t, 3 * h * d))


def test_attention_single_token_returns_v():
    rng = np.random.default_rng(7)
    qkv = _rand_qkv(1, 2, rng)
    out = O.varlen_attention(qkv, np.array([0, 1]), 2)
    v = qkv.reshape(1, 3, 2, 64)[:, 2].reshape(1, 128)
    assert np.allclose(out, v, atol=0, rtol=1e-15)


def test_attention_constant_v_and_identical_keys():
    rng = np.random.default_rng(8)
    n, h = 13, 3
    qkv = _rand_qkv(n, h, rng).reshape(n, 3, h, 64)
    qkv[:, 2] = qkv[0, 2]                      # constant v
    out = O.varlen_attention(qkv.reshape(n, -1), np.array([0, n]), h).reshape(n, h, 64)
    assert np.max(np.abs(out - qkv[0, 2][None])) < 1e-12
    qkv = _rand_qkv(n, h, rng).reshape(n, 3, h, 64)
    qkv[:, 1] = qkv[0, 1]                      # identical keys -> uniform weights
    out = O.varlen_attention(qkv.reshape(n, -1), np.array([0, n]), h).reshape(n, h, 64)
    assert np.max(np.abs(out - qkv[:, 2].mean(axis=0)[None])) < 1e-12


def test_attention_rows_sum_to_one():
    rng = np.random.default_rng(9)
    q, k, v = (rng.standard_normal((40, 64)) * 3 for _ in range(3))
    _, p = O.attention_single(q, k, v, 0.125)
    assert np.max(np.abs(p.sum(axis=1) - 1.0)) < 1e-12
    assert np.all(p >= 0)


def test_attention_matches_torch_sdpa_fp64():
    rng = np.random.default_rng(10)
    lens = [1, 5, 64, 129, 197]
    cu = O.cu_from_counts(lens)
    h = 3
    qkv = _rand_qkv(int(cu[-1]), h, rng)
    out = O.varlen_attention(qkv, cu, h).reshape(-1, h, 64)
    a = torch.from_numpy(qkv.reshape(-1, 3, h, 64))
    for i in range(len(lens)):
        seg = a[cu[i]:cu[i + 1]]
        q, k, v = (seg[:, j].transpose(0, 1) for j in range(3))   # [h, n, d]
        ref = torch.nn.functional.scaled_dot_product_attention(q, k, v).transpose(0, 1)
        assert np.max(np.abs(out[cu[i]:cu[i + 1]] - ref.numpy())) < 1e-12


def test_varlen_equals_per_image_and_padded_mask():
    rng = np.random.default_rng(11)
    lens = rng.integers(1, 80, size=7)
    cu = O.cu_from_counts(lens)
    h = 2
    qkv = _rand_qkv(int(cu[-1]), h, rng)
    packed = O.varlen_attention(qkv, cu, h)
    padded = O.padded_masked_attention(qkv, cu, h)
    assert np.max(np.abs(packed - padded)) < 1e-12
    for i in range(len(lens)):
        sep = O.varlen_attention(qkv[cu[i]:cu[i + 1]], np.array([0, lens[i]]), h)
        assert np.max(np.abs(packed[cu[i]:cu[i + 1]] - sep)) < 1e-12


def test_unpruned_packed_equals_dense_attention():
    """k = 0 for every image: the packed buffer is the dense batch and packed
    attention equals dense batched attention (torch SDPA, fp64)."""
    rng = np.random.default_rng(12)
    b, n, h = 4, 37, 2
    qkv = _rand_qkv(b * n, h, rng)
    packed = O.varlen_attention(qkv, np.arange(b + 1) * n, h)
    a = torch.from_numpy(qkv.reshape(b, n, 3, h, 64))
    q, k, v = (a[:, :, j].permute(0, 2, 1, 3) for j in range(3))
    dense = torch.nn.functional.scaled_dot_product_attention(q, k, v).permute(0, 2, 1, 3)
    assert np.max(np.abs(packed - dense.reshape(b * n, h * 64).numpy())) < 1e-12


# ---------------------------------------------------------------------------
# LayerNorm, linear, GELU
# ---------------------------------------------------------------------------

def test_layernorm_matches_torch_and_invariants():
    rng = np.random.default_rng(13)
    x = rng.standard_normal((33, 96)) * 4 + 2
    w, b = rng.standard_normal(96), rng.standard_normal(96)
    y = O.layernorm(x, w, b, 1e-6)
    ref = torch.nn.functional.layer_norm(torch.from_numpy(x), (96,), torch.from_numpy(w),
                                         torch.from_numpy(b), 1e-6).numpy()
    assert np.max(np.abs(y - ref)) < 1e-12
    y1 = O.layernorm(x, np.ones(96), np.zeros(96), 0.0)
    assert np.max(np.abs(y1.mean(axis=1))) < 1e-12
    assert np.max(np.abs((y1 ** 2).mean(axis=1) - 1)) < 1e-12


def test_linear_matches_loops():
    rng = np.random.default_rng(14)
    x, w, b = rng.standard_normal((3, 5)), rng.standard_normal((4, 5)), rng.standard_normal(4)
    y = O.linear(x, w, b)
    for r in range(3):
        for c in range(4):
            assert abs(y[r, c] - (sum(x[r, i] * w[c, i] for i in range(5)) + b[c])) < 1e-12


def test_gelu_closed_forms_and_torch():
    x = np.linspace(-8, 8, 1001)
    ref = torch.nn.functional.gelu(torch.from_numpy(x), approximate="none").numpy()
    assert np.max(np.abs(O.gelu(x) - ref)) < 1e-14
    assert O.gelu(np.array([0.0]))[0] == 0.0
    assert abs(O.gelu(np.array([10.0]))[0] - 10.0) < 1e-12
    assert abs(O.gelu(np.array([1.0]))[0] - 0.5 * (1 + math.erf(1 / math.sqrt(2)))) < 1e-15


# ---------------------------------------------------------------------------
# the pruned block (Eq. 1) and the forward
# ---------------------------------------------------------------------------

def _small_cfg(**kw):
    base = dict(batch=3, n_tokens=21, dim=128, heads=2, mlp_dim=256, depth=3,
                prune_blocks=(1,), k_law="uniform", k_max=14)
    base.update(kw)
    return S.Config("tiny", **base)


def _torch_block(x, cu, wf, heads, eps, kept=None):
    """The same block written with torch library ops (fp64): F.layer_norm,
    F.linear, per-image SDPA, exact GELU.  Independent of the oracle."""
    F = torch.nn.functional
    t = {k: torch.from_numpy(v) for k, v in wf.items()}
    x = torch.from_numpy(x)
    d = x.shape[1]
    xn = F.layer_norm(x, (d,), t["ln1_w"], t["ln1_b"], eps)
    qkv = F.linear(xn, t["w_qkv"], t["b_qkv"]).reshape(-1, 3, heads, 64)
    o = torch.zeros(x.shape[0], heads, 64, dtype=torch.float64)
    for i in range(len(cu) - 1):
        seg = qkv[cu[i]:cu[i + 1]]
        q, k, v = (seg[:, j].transpose(0, 1) for j in range(3))
        o[cu[i]:cu[i + 1]] = F.scaled_dot_product_attention(q, k, v).transpose(0, 1)
    h = x + F.linear(o.reshape(-1, d), t["w_proj"], t["b_proj"])
    if kept is not None:
        h = h[torch.from_numpy(kept.astype(np.int64))]
    y = F.gelu(F.linear(F.layer_norm(h, (d,), t["ln2_w"], t["ln2_b"], eps), t["w_fc1"], t["b_fc1"]))
    return (h + F.linear(y, t["w_fc2"], t["b_fc2"])).numpy()


def _block_inputs(cfg, seed=0):
    cu, ids = S.initial_layout(cfg)
    x = O.bf16_to_f64(S.activations_bf16(cfg, seed))
    wf = O.decode_weights(S.block_weights(cfg, 0, seed, random_affine=True))
    return x, cu, ids, wf


def test_block_matches_torch_composition():
    cfg = _small_cfg()
    x, cu, ids, wf = _block_inputs(cfg)
    keeps, _ = S.keep_schedule(cfg, 0)
    scores = O.gather_scores(S.score_table(cfg, 1, 0), cu, ids)
    r = O.pruned_block(x, cu, ids, wf, cfg.heads, 1e-6, scores, keeps[0])
    ref = _torch_block(x, cu, wf, cfg.heads, 1e-6, r["kept_idx"])
    assert np.max(np.abs(r["x_out"] - ref)) < 1e-10
    r0 = O.pruned_block(x, cu, ids, wf, cfg.heads, 1e-6)
    assert np.max(np.abs(r0["x_out"] - _torch_block(x, cu, wf, cfg.heads, 1e-6))) < 1e-10


def test_block_pruned_rows_equal_dense_rows():
    """Deletion happens after the attention residual and the MLP is row-wise,
    so the pruned block's output rows are the dense block's output rows at the
    kept positions (Eq. 1)."""
    cfg = _small_cfg()
    x, cu, ids, wf = _block_inputs(cfg, seed=1)
    keeps, _ = S.keep_schedule(cfg, 1)
    scores = O.gather_scores(S.score_table(cfg, 1, 1), cu, ids)
    pr = O.pruned_block(x, cu, ids, wf, cfg.heads, 1e-6, scores, keeps[0])
    dn = O.pruned_block(x, cu, ids, wf, cfg.heads, 1e-6)
    assert np.max(np.abs(pr["x_out"] - dn["x_out"][pr["kept_idx"]])) < 1e-12
    assert np.array_equal(pr["ids_out"], ids[pr["kept_idx"]])


def test_block_keep_all_equals_unpruned():
    cfg = _small_cfg()
    x, cu, ids, wf = _block_inputs(cfg, seed=2)
    scores = np.random.default_rng(0).random(len(ids)).astype(np.float32)
    full = np.full(cfg.batch, cfg.n_tokens)
    pr = O.pruned_block(x, cu, ids, wf, cfg.heads, 1e-6, scores, full)
    dn = O.pruned_block(x, cu, ids, wf, cfg.heads, 1e-6)
    assert np.array_equal(pr["x_out"], dn["x_out"])
    assert np.array_equal(pr["cu_out"], cu)


def test_forward_k0_equals_dense_and_trajectory():
    cfg = _small_cfg(depth=3, prune_blocks=(0, 2))
    cu, ids = S.initial_layout(cfg)
    x = O.bf16_to_f64(S.activations_bf16(cfg, 5))
    blocks = [O.decode_weights(S.block_weights(cfg, l, 5)) for l in range(cfg.depth)]
    full = np.full(cfg.batch, cfg.n_tokens)
    tabs = {l: S.score_table(cfg, l, 5) for l in cfg.prune_blocks}
    k0 = O.forward(x, cu, ids, blocks, cfg.heads, 1e-6, {l: (tabs[l], full) for l in tabs})
    dense = O.forward(x, cu, ids, blocks, cfg.heads, 1e-6)
    assert np.array_equal(k0["x"], dense["x"])
    keeps, befores = S.keep_schedule(cfg, 5)
    pr = O.forward(x, cu, ids, blocks, cfg.heads, 1e-6,
                   {l: (tabs[l], keeps[j]) for j, l in enumerate(cfg.prune_blocks)})
    assert np.array_equal(np.diff(pr["cu"]), keeps[-1])
    for i in range(cfg.batch):
        seg = pr["ids"][pr["cu"][i]:pr["cu"][i + 1]]
        assert seg[0] == 0 and np.all(np.diff(seg) > 0)


# ---------------------------------------------------------------------------
# accounting and generator (Eq. 4, Appendix A.2, Appendix E.4, Table 1, Table 3)
# ---------------------------------------------------------------------------

def test_native_gflops_reproduce_table1(golden_dir):
    from paper_2609_34325_gb300 import accounting as A
    rows = [ln.split() for ln in open(os.path.join(golden_dir, "native_gflops.txt"))
            if ln.strip() and not ln.startswith("#")]
    assert len(rows) == 4
    for name, gf, d, L, n0, mlp, patch, ro in rows:
        ours = A.native_gflops(int(n0) + 1, int(d), int(mlp), int(L), int(patch),
                               readout_mult=int(ro))
        assert abs(ours - float(gf)) / float(gf) < 0.01, (name, ours, gf)


def test_budget_grid_legality(golden_dir):
    rows = [ln.split() for ln in open(os.path.join(golden_dir, "budget_grid.txt"))
            if ln.strip() and not ln.startswith("#")]
    for name, n0, m, gmin, gmax in rows:
        n0, m = int(n0), int(m)
        grid = list(range(2, n0 - 4 + 1, 2))
        assert len(grid) == m and grid[0] == int(gmin) and grid[-1] == int(gmax)
    for name in S.CONFIGS:
        cfg = S.get_config(name)
        keeps, befores = S.keep_schedule(cfg, 0)
        for m, n in zip(keeps, befores):
            k = n - m
            assert np.all(k >= 0)
            assert np.all((k == 0) | (m - 1 >= 4))       # >= 4 visual tokens survive


def test_compression_identity_and_calibration():
    for name in S.CONFIGS:
        cfg = S.get_config(name)
        keeps, befores = S.keep_schedule(cfg, 0)
        c = S.compression_from_counts(cfg, keeps, befores)
        dc = np.zeros(cfg.batch)
        for l, m, n in zip(cfg.prune_blocks, keeps, befores):
            dc += (n - m) * (cfg.depth - l) / (cfg.depth * cfg.n_vis0)
        assert np.max(np.abs(c - dc)) < 1e-12             # C = sum of Delta C_l
    cfg = S.get_config("cfg3")
    for seed in range(3):
        c = S.compression_from_counts(cfg, *S.keep_schedule(cfg, seed))
        assert abs(c.mean() - 0.38) <= 0.01
        assert c.min() < 0.30 and c.max() > 0.45          # per-image spread
    # DINOv2-B: the paper reports 22.9-40.1% compression, mean 34.8% (Sec. 4.3)
    cfg = S.get_config("cfg6")
    for seed in range(3):
        c = S.compression_from_counts(cfg, *S.keep_schedule(cfg, seed))
        assert abs(c.mean() - 0.348) <= 0.01
        assert c.min() < 0.26 and c.max() > 0.40


# ---------------------------------------------------------------------------
# the deployment actor (Sec. 3.2 "The actor"; Appendix A.1-A.3)
# ---------------------------------------------------------------------------

def _actor_w(d=64, depth=4, n0=20, seed=3, **kw):
    return {k: O.bf16_to_f64(v) for k, v in S.actor_weights(d, depth, n0, seed, **kw).items()}


def test_actor_sigmoid_and_silu_closed_forms():
    assert O.sigmoid(0.0) == 0.5
    for x in (-40.0, -2.5, -1e-3, 0.7, 4.0, 40.0):
        ref = 1.0 / (1.0 + math.exp(-x))
        assert abs(O.sigmoid(x) - ref) <= 1e-15 + 1e-14 * ref
        assert abs(O.silu(x) - x * ref) <= 1e-14 * (1 + abs(x))


def test_actor_gate_closed_forms():
    """p = 0.5 exactly with a zero output layer; one-hot first layers read the
    block embedding and the history at the positions Appendix A.1 gives them
    ([K_CLS (d), e^G (16), h (3)])."""
    d = 64
    w = _actor_w(d)
    k_cls = np.linspace(-1, 1, d)
    e_g = w["gate_emb"][2]
    h = O.actor_history(10, 20, 0.25, 2, 4)
    assert np.allclose(h, [0.5, 0.25, 2 / 3], rtol=0, atol=1e-15)
    w0 = dict(w, gate_w2=np.zeros((1, 64)), gate_b2=np.zeros(1))
    assert O.actor_gate(k_cls, e_g, h, w0) == 0.5
    for col, val in ((d, e_g[0]), (d + 15, e_g[15]), (d + 16, h[0]), (d + 18, h[2]), (3, k_cls[3])):
        w1 = np.zeros((64, d + 19))
        w1[0, col] = 1.0
        wv = dict(w, gate_w1=w1, gate_b1=np.zeros(64), gate_w2=np.eye(1, 64), gate_b2=np.array([0.5]))
        silu_v = val / (1 + math.exp(-val))
        assert abs(O.actor_gate(k_cls, e_g, h, wv) - 1 / (1 + math.exp(-(silu_v + 0.5)))) < 1e-14


def test_actor_encoder_reduces_to_its_input_projection():
    """With the attention output and feed-forward output layers zeroed the
    block is the identity, so Z = W_in K + b_in + e^C (+ W_h h on CLS),
    summed out element by element."""
    d, n = 64, 7
    w = _actor_w(d)
    for nm in ("enc_w_o", "enc_b_o", "enc_w_fc2", "enc_b_fc2"):
        w[nm] = np.zeros_like(w[nm])
    rng = np.random.default_rng(1)
    keys = rng.standard_normal((n + 1, d))
    h = np.array([0.3, 0.1, 0.5])
    e_c = w["enc_emb"][1]
    z = O.actor_encoder(keys, e_c, h, w)
    for j in range(n + 1):
        for c in (0, 17, 127):
            ref = sum(w["enc_w_in"][c, t] * keys[j, t] for t in range(d)) + w["enc_b_in"][c] + e_c[c]
            if j == 0:
                ref += sum(w["enc_w_h"][c, t] * h[t] for t in range(3))
            assert abs(z[j, c] - ref) < 1e-12


def test_actor_encoder_is_permutation_equivariant_over_visual_tokens():
    """No positional term enters the encoder (Appendix A.1): permuting the
    visual tokens permutes their outputs and leaves Z_CLS unchanged."""
    d, n = 64, 9
    w = _actor_w(d)
    rng = np.random.default_rng(2)
    keys = rng.standard_normal((n + 1, d))
    h = np.array([0.9, 0.2, 0.0])
    perm = np.concatenate([[0], 1 + rng.permutation(n)])
    z = O.actor_encoder(keys, w["enc_emb"][0], h, w)
    zp = O.actor_encoder(keys[perm], w["enc_emb"][0], h, w)
    assert np.allclose(zp, z[perm], rtol=0, atol=1e-12)


def test_actor_encoder_equal_keys_average_the_values():
    """Equal attention keys (key weights zero) make every head average its
    values uniformly: Z1 = X + W_o mean_j(V_j) + b_o for every token."""
    d, n = 64, 6
    w = _actor_w(d)
    w["enc_w_qkv"] = w["enc_w_qkv"].copy()
    w["enc_w_qkv"][128:256] = 0.0
    for nm in ("enc_w_fc2", "enc_b_fc2"):
        w[nm] = np.zeros_like(w[nm])
    rng = np.random.default_rng(4)
    keys = rng.standard_normal((n + 1, d))
    h = np.array([0.5, 0.0, 0.0])
    e_c = w["enc_emb"][3]
    x = keys @ w["enc_w_in"].T + w["enc_b_in"] + e_c
    x[0] += w["enc_w_h"] @ h
    mu = x.mean(axis=1, keepdims=True)
    xn = (x - mu) / np.sqrt(((x - mu) ** 2).mean(axis=1, keepdims=True) + O.ACTOR_EPS)
    xn = xn * w["enc_ln1_w"] + w["enc_ln1_b"]
    v = xn @ w["enc_w_qkv"][256:].T + w["enc_b_qkv"][256:]
    ref = x + (w["enc_w_o"] @ v.mean(axis=0) + w["enc_b_o"])[None, :]
    assert np.allclose(O.actor_encoder(keys, e_c, h, w), ref, rtol=0, atol=1e-12)


def test_actor_budget_masked_argmax_brute_force():
    """Appendix A.2/A.3: the highest logit among budgets k <= N_l - 4 (at least
    four visual tokens survive), none when N_l < 6; equal logits pick the
    smallest budget."""
    n0 = 196
    w = _actor_w(64, n0=n0)
    grid = list(range(2, n0 - 4 + 1, 2))
    rng = np.random.default_rng(5)
    for n_l in (3, 5, 6, 7, 10, 33, 100, 196):
        z = rng.standard_normal(128)
        k, logits = O.actor_budget(z, n_l, n0, w)
        best = None
        for idx, kk in enumerate(grid):
            if kk <= n_l - 4 and (best is None or logits[idx] > logits[best]):
                best = idx
        assert k == (0 if best is None else grid[best])
        assert k == 0 or n_l - k >= 4
    wt = dict(w, bud_w2=np.zeros_like(w["bud_w2"]), bud_b2=np.full(len(grid), 0.3))
    assert O.actor_budget(rng.standard_normal(128), 50, n0, wt)[0] == 2


def _gelu_lib(x: float) -> float:
    """Exact GELU from PyTorch's float64 routine (independent of the oracle's)."""
    return float(torch.nn.functional.gelu(torch.tensor(x, dtype=torch.float64)))


def test_actor_budget_logits_closed_form():
    """Appendix A.1 budget head: logits = W2 GELU(W1 LN(Z_CLS) + b1) + b2.
    Z_CLS = mu + sigma s with s alternating +-1 over the 128 channels has row
    mean mu and biased variance sigma^2 exactly, so LN(Z_CLS)_c = g_c s_c
    sigma / sqrt(sigma^2 + eps) + beta_c in closed form.  W1 = I and a one-hot
    W2 (logit m reads hidden unit m mod 128 with weight (m + 1) / 10) expose
    every logit.  The large mean (mu = 500) makes a missing LayerNorm fail,
    and the hidden values near +-1 separate GELU from SiLU and ReLU."""
    n0 = 196
    w = _actor_w(64, n0=n0)
    grid = O.budget_grid(n0)
    m = len(grid)
    mu, sigma = 500.0, 0.75
    s = np.array([1.0 if c % 2 == 0 else -1.0 for c in range(128)])
    z = mu + sigma * s
    w1 = np.eye(128)
    w2 = np.zeros((m, 128))
    for j in range(m):
        w2[j, j % 128] = (j + 1) / 10
    wb = dict(w, bud_w1=w1, bud_w2=w2)
    k, logits = O.actor_budget(z, 120, n0, wb)
    scale = sigma / math.sqrt(sigma * sigma + O.ACTOR_EPS)
    for j in range(m):
        c = j % 128
        u = w["bud_ln_w"][c] * s[c] * scale + w["bud_ln_b"][c]
        ref = (j + 1) / 10 * _gelu_lib(u + w["bud_b1"][c]) + w["bud_b2"][j]
        assert abs(logits[j] - ref) < 1e-12, (j, logits[j], ref)
    assert k == int(grid[int(np.argmax(np.where(grid <= 116, logits, -np.inf)))])


def test_actor_encoder_feed_forward_closed_form():
    """Appendix A.1 shared encoder, feed-forward sublayer: with the attention
    output layer zeroed, Z = X + W_fc2 GELU(W_fc1 LN2(X) + b_fc1) + b_fc2,
    pre-LayerNorm.  X is built with a closed-form row mean and variance:
    W_in reads key entry 0 with sign s_c (alternating +-1) and key entry 1
    with weight 1, so X_jc = s_c sigma_j + mu_j (+ h_0 on CLS through W_h),
    and LN2(X)_jc = g_c s_c sigma_j / sqrt(sigma_j^2 + eps) + beta_c.  Hidden
    unit r reads LN2 column r mod 128; output c mixes hidden units c and
    128 + c as 1.5 GELU(.) - 0.5 GELU(.).  The large row means make a missing
    or post-placed LayerNorm fail; the hidden values separate GELU from SiLU
    and ReLU."""
    d, n = 64, 5
    w = _actor_w(d)
    s = np.array([1.0 if c % 2 == 0 else -1.0 for c in range(128)])
    w_in = np.zeros((128, d))
    w_in[:, 0] = s
    w_in[:, 1] = 1.0
    w_h = np.zeros((128, 3))
    w_h[:, 0] = 1.0
    fc1 = np.zeros((256, 128))
    for r in range(256):
        fc1[r, r % 128] = 1.0
    fc2 = np.zeros((128, 256))
    for c in range(128):
        fc2[c, c] = 1.5
        fc2[c, 128 + c] = -0.5
    we = dict(w, enc_w_in=w_in, enc_b_in=np.zeros(128), enc_w_h=w_h,
              enc_w_o=np.zeros_like(w["enc_w_o"]), enc_b_o=np.zeros_like(w["enc_b_o"]),
              enc_w_fc1=fc1, enc_w_fc2=fc2)
    e_c = np.zeros(128)
    h = np.array([7.0, 0.2, 0.1])
    sig = [0.5, 1.0, 1.7, 2.5, 0.9, 3.0]
    mus = [40.0 + 25.0 * j for j in range(n + 1)]
    keys = np.zeros((n + 1, d))
    for j in range(n + 1):
        keys[j, 0], keys[j, 1] = sig[j], mus[j]
    z = O.actor_encoder(keys, e_c, h, we)
    g, beta = w["enc_ln2_w"], w["enc_ln2_b"]
    b1, b2 = w["enc_b_fc1"], w["enc_b_fc2"]
    for j in range(n + 1):
        mu = mus[j] + (h[0] if j == 0 else 0.0)
        scale = sig[j] / math.sqrt(sig[j] ** 2 + O.ACTOR_EPS)
        for c in range(128):
            x = s[c] * sig[j] + mu
            u = g[c] * s[c] * scale + beta[c]
            ref = x + 1.5 * _gelu_lib(u + b1[c]) - 0.5 * _gelu_lib(u + b1[128 + c]) + b2[c]
            assert abs(z[j, c] - ref) < 1e-11, (j, c, z[j, c], ref)


def test_actor_selector_closed_form():
    """Eq. 2 with a one-hot first layer: s_j = silu(Z_j[0] + 2 k / N_l) + 0.25."""
    w = _actor_w(64)
    w1 = np.zeros((64, 128))
    w1[0, 0] = 1.0
    wk = np.zeros(128)
    wk[0] = 2.0
    ws = dict(w, sel_w1=w1, sel_b1=np.zeros(64), sel_w2=np.eye(1, 64), sel_b2=np.array([0.25]),
              sel_w_k=wk)
    rng = np.random.default_rng(6)
    z = rng.standard_normal((5, 128))
    s = O.actor_selector(z, 8, 40, ws)
    for j in range(5):
        a = z[j, 0] + 2 * 8 / 40
        assert abs(s[j] - (a / (1 + math.exp(-a)) + 0.25)) < 1e-14


def test_actor_block_decisions_and_history():
    """Deployment rules (Appendix A.3): the gate opens when p >= 0.5 and a
    budget is feasible; k_l = the budget then, 0 otherwise; keep = N_l + 1 -
    k_l; rho_{l+1} = k_l / N_l and E counts the interventions."""
    d, n0, depth = 64, 20, 4
    lens = np.array([21, 5, 9, 13, 21])             # N_l + 1 tokens; 5 -> N_l = 4: no budget
    cu = O.cu_from_counts(lens)
    rng = np.random.default_rng(7)
    keys = rng.standard_normal((int(cu[-1]), d))
    rho = np.array([0.0, 0.1, 0.2, 0.0, 0.3])
    e_prev = np.array([0, 1, 2, 0, 1])
    for gb, want in ((9.0, 1), (-9.0, 0)):
        w = _actor_w(d, depth, n0, gate_bias=gb)
        r = O.actor_block(keys, cu, 2, n0, depth, rho, e_prev, w)
        n_vis = lens - 1
        feasible = n_vis >= 6
        assert np.array_equal(r["gate"], (want * feasible).astype(np.int32))
        assert np.array_equal(r["gate"], ((r["p"] >= 0.5) & (r["budget"] > 0)).astype(np.int32))
        assert np.array_equal(r["k"], r["budget"] * r["gate"])
        assert np.array_equal(r["keep_counts"], lens - r["k"])
        assert np.all((r["k"] == 0) | (r["keep_counts"] - 1 >= 4))
        assert np.allclose(r["rho_next"], r["k"] / n_vis)
        assert np.array_equal(r["interventions_next"], e_prev + r["gate"])
        assert np.all(r["scores"][cu[:-1]] == 0.0)


# ---------------------------------------------------------------------------
# patch embedding and classifier (the ends of the forward that App. E.4 counts)
# ---------------------------------------------------------------------------

def test_patch_embed_is_a_strided_convolution():
    """Every token against a direct convolution written as loops, plus the CLS
    row and the position embeddings."""
    rng = np.random.default_rng(11)
    b, c, h, w, p, d = 2, 2, 8, 12, 4, 3
    im = rng.standard_normal((b, c, h, w))
    wc = rng.standard_normal((d, c, p, p))
    bias = rng.standard_normal(d)
    cls = rng.standard_normal(d)
    gh, gw = h // p, w // p
    pos = rng.standard_normal((gh * gw + 1, d))
    out = O.patch_embed(im, wc.reshape(d, -1), bias, cls, pos, p)
    assert out.shape == (b * (gh * gw + 1), d)
    for i in range(b):
        base = i * (gh * gw + 1)
        assert np.allclose(out[base], cls + pos[0], rtol=0, atol=1e-14)
        for py in range(gh):
            for px in range(gw):
                for o in range(d):
                    acc = bias[o]
                    for ch in range(c):
                        for ky in range(p):
                            for kx in range(p):
                                acc += wc[o, ch, ky, kx] * im[i, ch, py * p + ky, px * p + kx]
                    tok = 1 + py * gw + px
                    assert abs(out[base + tok, o] - (acc + pos[tok, o])) < 1e-12


def test_classifier_reads_only_cls_rows():
    """Logits depend on each image's CLS row alone (LayerNorm then linear):
    changing every other row leaves them unchanged; with a unit LayerNorm and
    an identity head the logits are the normalised CLS row."""
    rng = np.random.default_rng(12)
    d = 8
    cu = np.array([0, 5, 6, 10])
    x = rng.standard_normal((10, d))
    g, be = 1 + 0.1 * rng.standard_normal(d), 0.1 * rng.standard_normal(d)
    wh, bh = rng.standard_normal((4, d)), rng.standard_normal(4)
    a = O.classifier_head(x, cu, g, be, 1e-6, wh, bh)
    x2 = x.copy()
    mask = np.ones(10, bool)
    mask[cu[:-1]] = False
    x2[mask] = rng.standard_normal((mask.sum(), d))
    assert np.array_equal(a, O.classifier_head(x2, cu, g, be, 1e-6, wh, bh))
    ident = O.classifier_head(x, cu, np.ones(d), np.zeros(d), 0.0, np.eye(d), np.zeros(d))
    r = x[cu[:-1]]
    ref = (r - r.mean(1, keepdims=True)) / r.std(1, keepdims=True)
    assert np.allclose(ident, ref, rtol=0, atol=1e-12)


# ---------------------------------------------------------------------------
# DINOv2 pieces: LayerScale and the LC1 readout (App. E.3; Table 3)
# ---------------------------------------------------------------------------

def test_layerscale_zero_leaves_the_residual_stream():
    """With both LayerScales zero the block passes its (compacted) input
    through: x_out = x[kept]; with both equal to one it is the plain block."""
    cfg = S.get_config("cfg1", batch=3)
    cu, ids = S.initial_layout(cfg)
    x = O.bf16_to_f64(S.activations_bf16(cfg, 5))
    wf = O.decode_weights(S.block_weights(cfg, 0, 5, random_affine=True))
    keeps, _ = S.keep_schedule(cfg, 5)
    sc = O.gather_scores(S.score_table(cfg, 0, 5), cu, ids)
    z = dict(wf, ls1=np.zeros(cfg.dim), ls2=np.zeros(cfg.dim))
    r = O.pruned_block(x, cu, ids, z, cfg.heads, cfg.ln_eps, sc, keeps[0])
    assert np.array_equal(r["x_out"], x[r["kept_idx"]])
    one = dict(wf, ls1=np.ones(cfg.dim), ls2=np.ones(cfg.dim))
    a = O.pruned_block(x, cu, ids, one, cfg.heads, cfg.ln_eps, sc, keeps[0])
    b = O.pruned_block(x, cu, ids, wf, cfg.heads, cfg.ln_eps, sc, keeps[0])
    assert np.array_equal(a["x_out"], b["x_out"])


def test_lc1_readout_loops_and_invariants():
    """Element by element against loops; a single visual token's mean is that
    token; the mean does not depend on the order of the visual tokens."""
    rng = np.random.default_rng(21)
    d = 6
    cu = np.array([0, 4, 6, 7, 11])
    x = rng.standard_normal((11, d)) * 2 + 1
    g, be = 1 + 0.1 * rng.standard_normal(d), 0.1 * rng.standard_normal(d)
    r = O.lc1_readout(x, cu, g, be, 1e-6)
    for i in range(4):
        lo, hi = cu[i], cu[i + 1]
        rows = []
        for j in range(lo, hi):
            mu = sum(x[j]) / d
            var = sum((v - mu) ** 2 for v in x[j]) / d
            rows.append([(x[j][c] - mu) / math.sqrt(var + 1e-6) * g[c] + be[c] for c in range(d)])
        assert np.allclose(r[i, :d], rows[0], rtol=0, atol=1e-12)
        mean = [sum(rw[c] for rw in rows[1:]) / max(len(rows) - 1, 1) for c in range(d)]
        assert np.allclose(r[i, d:], mean if len(rows) > 1 else np.zeros(d), rtol=0, atol=1e-12)
    # image 1 has one visual token: its mean is that token's normalised row
    assert np.allclose(r[1, d:], O.layernorm(x[5:6], g, be, 1e-6)[0], rtol=0, atol=1e-12)
    xp = x.copy()
    xp[8:11] = x[[10, 8, 9]]
    assert np.allclose(O.lc1_readout(xp, cu, g, be, 1e-6), r, rtol=0, atol=1e-12)


# ---------------------------------------------------------------------------
# training side: Plackett-Luce sampling / log-probability (App. A.3), the
# shadows' fidelity cost (App. B.2)
# ---------------------------------------------------------------------------

def test_pl_logprob_is_a_distribution_over_ordered_sequences():
    """exp(log pi) summed over every ordered k-sequence of n items is 1, and a
    sequential draw's probabilities multiply out to it."""
    rng = np.random.default_rng(3)
    for n, k in ((4, 1), (5, 2), (5, 3), (4, 4)):
        s = rng.standard_normal(n) * 2
        tot = sum(math.exp(O.pl_logprob(s, np.array(p)))
                  for p in itertools.permutations(range(n), k))
        assert abs(tot - 1) < 1e-12
        # hand product for one sequence
        seq = list(itertools.permutations(range(n), k))[-1]
        prob, rem = 1.0, list(range(n))
        for i in seq:
            prob *= math.exp(s[i]) / sum(math.exp(s[j]) for j in rem)
            rem.remove(i)
        assert abs(math.log(prob) - O.pl_logprob(s, np.array(seq))) < 1e-12


def test_pl_logprob_closed_forms():
    rng = np.random.default_rng(4)
    s = rng.standard_normal(9)
    # k = 1: the log-softmax entry; equal scores: -sum_t log(n - t + 1)
    for i in range(9):
        assert abs(O.pl_logprob(s, np.array([i])) - scipy.special.log_softmax(s)[i]) < 1e-12
    order = np.array([4, 0, 7, 2])
    assert abs(O.pl_logprob(np.full(9, 0.3), order) + sum(math.log(9 - t) for t in range(4))) \
        < 1e-12
    # shift invariance; a full permutation's last step contributes 0
    assert abs(O.pl_logprob(s + 5.0, order) - O.pl_logprob(s, order)) < 1e-12
    full = np.array([3, 1, 8, 0, 2, 5, 4, 7, 6])
    assert abs(O.pl_logprob(s, full) - O.pl_logprob(s, full[:-1])) < 1e-12


def test_pl_logprob_grad_matches_finite_differences():
    rng = np.random.default_rng(5)
    s = rng.standard_normal(7)
    order = np.array([2, 6, 0])
    g = O.pl_logprob_grad(s, order)
    h = 1e-6
    for j in range(7):
        e = np.zeros(7)
        e[j] = h
        fd = (O.pl_logprob(s + e, order) - O.pl_logprob(s - e, order)) / (2 * h)
        assert abs(fd - g[j]) < 1e-8
    assert abs(g.sum()) < 1e-12                       # shift invariance


def test_gumbel_top_k_is_a_plackett_luce_sample():
    """The Gumbel-top-k order has the Plackett-Luce law: empirical frequencies
    of every ordered pair of 4 items against exp(log pi), within 5 sigma."""
    rng = np.random.default_rng(6)
    s = np.array([0.8, -0.4, 0.1, 1.5], dtype=np.float32)
    draws = 40000
    counts = {}
    u = rng.random((draws, 4))
    gum = -np.log(-np.log(u))
    for r in range(draws):
        key = tuple(O.pl_sample_gumbel(s, gum[r], 2))
        counts[key] = counts.get(key, 0) + 1
    for seq in itertools.permutations(range(4), 2):
        p = math.exp(O.pl_logprob(s.astype(np.float64), np.array(seq)))
        f = counts.get(seq, 0) / draws
        assert abs(f - p) <= 5 * math.sqrt(p * (1 - p) / draws), (seq, f, p)


def test_gumbel_top_k_order_rules():
    s = np.array([0.5, 2.0, -1.0, 2.0, 0.0, -0.0, np.nan], dtype=np.float32)
    z = np.zeros(7, dtype=np.float32)
    # NaN first, equal keys by higher index (as deployment deletes), -0 == +0
    assert O.pl_sample_gumbel(s, z, 7).tolist() == [6, 3, 1, 0, 5, 4, 2]
    assert O.pl_sample_gumbel(s[:6], z[:6], 2).tolist() == [3, 1]
    # keys are fp32 sums: 1 + 2^-24 rounds to 1, so index order decides
    a = np.array([1.0, 1.0], dtype=np.float32)
    g = np.array([0.0, 2.0 ** -24], dtype=np.float32)
    assert O.pl_sample_gumbel(a, g, 2).tolist() == [1, 0]


def test_sampled_set_is_what_selection_deletes_on_the_keys():
    """The first k of the Gumbel-top-k order are exactly the tokens that the
    deterministic selection removes when given the keys s + g (ties
    included), so a training rollout deletes its sampled set."""
    rng = np.random.default_rng(8)
    for trial in range(200):
        n = int(rng.integers(1, 30))
        s = rng.integers(-3, 4, n).astype(np.float32)
        g = (rng.integers(-2, 3, n) * 0.5).astype(np.float32)
        k = int(rng.integers(0, n + 1))
        removed = set(O.pl_sample_gumbel(s, g, k).tolist())
        keys = np.concatenate([[0.0], s + g]).astype(np.float32)   # CLS row first
        kept, _, st = O.select_keep(keys, np.array([0, n + 1]), np.array([n + 1 - k]))
        assert st == 0
        assert removed == set(range(n)) - set((kept[1:] - 1).tolist())


def test_kd_cost_pins():
    rng = np.random.default_rng(7)
    zn, z = rng.standard_normal(10) * 4, rng.standard_normal(10) * 4
    assert O.kd_cost(zn, zn) == 0.0
    assert O.kd_cost(zn, z) > 0                        # Gibbs
    pn = scipy.special.softmax(zn / 3)
    q = scipy.special.softmax(z / 3)
    assert abs(O.kd_cost(zn, z) - 9 * scipy.stats.entropy(pn, q)) < 1e-12
    # two classes: tau^2 [p log(p/q) + (1-p) log((1-p)/(1-q))] with logistic p, q
    a, b = 1.7, -0.6
    p, qq = 1 / (1 + math.exp(-a / 3)), 1 / (1 + math.exp(-b / 3))
    closed = 9 * (p * math.log(p / qq) + (1 - p) * math.log((1 - p) / (1 - qq)))
    assert abs(O.kd_cost(np.array([a, 0.0]), np.array([b, 0.0])) - closed) < 1e-12
    # invariant to a constant added to either logit vector
    assert abs(O.kd_cost(zn + 3, z - 2) - O.kd_cost(zn, z)) < 1e-12


def test_shadow_prefixes_end_at_native_and_rollout():
    """The empty prefix is the dense forward, the full prefix the rollout; a
    prefix ending at block l equals the rollout through block l."""
    cfg = S.get_config("cfg1", batch=2, depth=3, prune_blocks=(0, 2))
    cu, ids = S.initial_layout(cfg)
    x = O.bf16_to_f64(S.activations_bf16(cfg, 8))
    blocks = [O.decode_weights(S.block_weights(cfg, l, 8)) for l in range(3)]
    keeps, _ = S.keep_schedule(cfg, 8)
    prune = {l: (S.score_table(cfg, l, 8), keeps[j]) for j, l in enumerate(cfg.prune_blocks)}
    sh = O.shadow_forwards(x, cu, ids, blocks, cfg.heads, cfg.ln_eps, prune)
    dense = O.forward(x, cu, ids, blocks, cfg.heads, cfg.ln_eps)
    roll = O.forward(x, cu, ids, blocks, cfg.heads, cfg.ln_eps, prune)
    assert np.array_equal(sh[-1]["x"], dense["x"])
    assert np.array_equal(sh[2]["x"], roll["x"])
    assert np.array_equal(sh[0]["kept"][0], roll["kept"][0])
    assert np.array_equal(sh[0]["cu"], O.cu_from_counts(keeps[0]))


def test_step_rewards_telescope():
    """Sum over an episode of the local rewards = 25 C - a D_final (App. B.3),
    with C from the definition C = (1 / L N0) sum_l (N0 - N_l^post) and the
    per-block counts written out."""
    rng = np.random.default_rng(10)
    depth, n0 = 12, 196
    blocks = [1, 3, 6, 9]
    k = rng.integers(0, 40, len(blocks))
    d = np.cumsum(rng.uniform(-0.2, 0.5, len(blocks)))
    a = 30.0
    r = O.step_rewards(d, k, blocks, depth, n0, a)
    post, n = [], n0
    for l in range(depth):
        if l in blocks:
            n -= k[blocks.index(l)]
        post.append(n)
    c = sum(n0 - p for p in post) / (depth * n0)
    assert abs(r.sum() - (25 * c - a * d[-1])) < 1e-12
    # a gate-off step (k = 0, D unchanged) earns nothing
    k0, d0 = k.copy(), d.copy()
    k0[2], d0[2] = 0, d0[1]
    assert O.step_rewards(d0, k0, blocks, depth, n0, a)[2] == 0.0
