"""GPU parity of the training side (App. A.3 sampling and log-probability;
App. B.2 complete-prefix shadows and their fidelity cost) through the C ABI,
against the fp64 oracle on the same seeded inputs.  Sampled orders, sequence
boundaries, ids and branched rows must match bit for bit; log-probabilities,
gradients and costs within the fp32 bounds stated in each test."""
import numpy as np
import pytest
import scipy.special
import torch

import __graft_entry__ as G
import dora_synth as S
import oracle as O
import paper_2609_34325_gb300 as P
from helpers import assert_close, bf, bits, dev, f32, f64, i32
from paper_2609_34325_gb300.shadow import ShadowRollout

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    G.build()
    P.load_library()
    torch.cuda.set_device(0)


def _status():
    return torch.zeros(1, dtype=torch.int32, device=dev())


def _gumbel(rng, t):
    u = rng.random(t)
    return (-np.log(-np.log(u))).astype(np.float32)


def _pruned_layout(name, seed, block=-1):
    cfg = S.get_config(name)
    keeps, _ = S.keep_schedule(cfg, seed)
    lens = np.asarray(keeps[block]) if block is not None else np.full(cfg.batch, cfg.n_tokens)
    return O.cu_from_counts(lens)


def _run_sample(scores, gumbel, cu, k, k_cap):
    b = len(cu) - 1
    order = torch.full((b, k_cap), 77, dtype=torch.int32, device=dev())
    st = _status()
    P.dora_pl_sample(f32(scores), f32(gumbel), i32(cu), i32(k), order, status=st)
    torch.cuda.synchronize()
    return order.cpu().numpy(), int(st.item())


def _oracle_orders(scores, gumbel, cu, k, k_cap):
    out = np.full((len(cu) - 1, k_cap), -1, dtype=np.int64)
    for i in range(len(cu) - 1):
        lo, hi = int(cu[i]), int(cu[i + 1])
        n = max(hi - lo - 1, 0)
        if n == 0 or k[i] == 0:
            continue
        out[i, :k[i]] = O.pl_sample_gumbel(scores[lo + 1:hi], gumbel[lo + 1:hi], int(k[i]))
    return out


@pytest.mark.parametrize("name,block", [("cfg1", None), ("cfg3", 0), ("cfg3", -1),
                                        ("cfg5", None)])
def test_pl_sample_bit_exact(name, block):
    cu = _pruned_layout(name, 3, block)
    t = int(cu[-1])
    rng = np.random.default_rng(t)
    scores = rng.standard_normal(t).astype(np.float32) * 2
    gumbel = _gumbel(rng, t)
    n = np.diff(cu) - 1
    k = np.array([rng.integers(0, m + 1) for m in n])
    k[0] = n[0]                                         # a full permutation
    k_cap = int(n.max())
    got, st = _run_sample(scores, gumbel, cu, k, k_cap)
    assert st == 0
    assert np.array_equal(got, _oracle_orders(scores, gumbel, cu, k, k_cap))


def test_pl_sample_ties_nan_signed_zero_and_counts():
    lens = [9, 1, 0, 12, 6, 40]
    cu = O.cu_from_counts(lens)
    t = int(cu[-1])
    rng = np.random.default_rng(9)
    scores = rng.integers(-2, 3, t).astype(np.float32)   # many exact ties
    gumbel = np.zeros(t, dtype=np.float32)
    scores[cu[0] + 3] = np.nan
    scores[cu[3] + 2], scores[cu[3] + 5] = -0.0, 0.0
    gumbel[cu[5] + 1:cu[5] + 20] = rng.integers(-1, 2, 19).astype(np.float32) * 0.5
    k = np.array([8, 0, 0, 11, 3, 39])
    got, st = _run_sample(scores, gumbel, cu, k, 40)
    assert st == 0
    assert np.array_equal(got, _oracle_orders(scores, gumbel, cu, k, 40))
    # k above the visual count, and above k_cap: clamped and flagged
    got, st = _run_sample(scores, gumbel, cu, np.array([9, 1, 0, 11, 3, 39]), 39)
    assert st == O.DORA_ERR_DEVICE_BAD_COUNT
    assert np.array_equal(got[0, :8], _oracle_orders(scores, gumbel, cu, [8] + [0] * 5, 39)[0, :8])


def _check_logprob(scores, cu, orders, k, dlogp, grad_rtol=2e-4):
    b = len(cu) - 1
    k_cap = orders.shape[1]
    logp = torch.full((b,), 5.0, dtype=torch.float32, device=dev())
    grad = torch.full((int(cu[-1]),), 5.0, dtype=torch.float32, device=dev())
    st = _status()
    P.dora_pl_logprob(f32(scores), i32(cu), i32(k), i32(orders), logp, grad=grad,
                      dlogp=f32(dlogp), status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    lp, g = logp.cpu().numpy().astype(np.float64), grad.cpu().numpy().astype(np.float64)
    for i in range(b):
        lo, hi = int(cu[i]), int(cu[i + 1])
        if hi - lo < 1:
            continue
        s = scores[lo + 1:hi].astype(np.float64)
        seq = orders[i, :k[i]]
        ref = O.pl_logprob(s, seq)
        # fp32 bound: every term s_{i_t} - L_t carries ~1e-6 of its magnitude
        scale = sum(abs(s[j]) + abs(scipy.special.logsumexp(np.delete(s, seq[:t])))
                    for t, j in enumerate(seq)) if len(seq) else 0.0
        assert abs(lp[i] - ref) <= 1e-5 * scale + 1e-6, (i, lp[i], ref)
        gref = dlogp[i] * O.pl_logprob_grad(s, seq)
        assert g[lo] == 0.0
        err = np.abs(g[lo + 1:hi] - gref)
        assert np.all(err <= grad_rtol * (1 + np.abs(gref))), (i, err.max())


@pytest.mark.parametrize("scale", [1.0, 30.0])
def test_pl_logprob_and_gradient_match_oracle(scale):
    cu = _pruned_layout("cfg3", 4, 0)[:65]               # 64 images after the first deletion
    t = int(cu[-1])
    rng = np.random.default_rng(int(scale))
    scores = (rng.standard_normal(t) * scale).astype(np.float32)
    n = np.diff(cu) - 1
    k = np.array([rng.integers(0, m + 1) for m in n])
    k[1], k[2] = 0, n[2]
    k_cap = int(n.max())
    orders, st = _run_sample(scores, _gumbel(rng, t), cu, k, k_cap)
    assert st == 0
    _check_logprob(scores, cu, orders, k, rng.uniform(-2, 2, len(k)))


def test_pl_logprob_bad_sequences_give_nan_and_status():
    cu = O.cu_from_counts([6, 6])
    scores = np.arange(12, dtype=np.float32)
    orders = np.array([[0, 0, -1], [1, 7, -1]], dtype=np.int32)   # repeat; out of range
    logp = torch.zeros(2, dtype=torch.float32, device=dev())
    st = _status()
    P.dora_pl_logprob(f32(scores), i32(cu), i32([2, 2]), i32(orders), logp, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == O.DORA_ERR_DEVICE_BAD_COUNT
    assert torch.isnan(logp).all()


def test_kd_cost_matches_oracle():
    rng = np.random.default_rng(11)
    b, shadows, classes, ld = 16, 40, 1000, 1024
    zn = np.zeros((b, ld), np.float32)
    zn[:, :classes] = rng.standard_normal((b, classes)) * 3
    z = np.zeros((shadows, ld), np.float32)
    img = rng.integers(0, b, shadows)
    z[:, :classes] = zn[img, :classes] + rng.standard_normal((shadows, classes)) * \
        rng.uniform(0, 2, (shadows, 1))
    z[:, classes:] = 50.0                                # padding must be ignored
    zn_b, z_b = S.f32_to_bf16_bits(zn), S.f32_to_bf16_bits(z)
    cost = torch.zeros(shadows, dtype=torch.float32, device=dev())
    st = _status()
    P.dora_kd_cost(bf(zn_b), bf(z_b), cost, classes, shadow_image=i32(img), tau=3.0, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    got = cost.cpu().numpy().astype(np.float64)
    zn64, z64 = O.bf16_to_f64(zn_b), O.bf16_to_f64(z_b)
    for s in range(shadows):
        ref = O.kd_cost(zn64[img[s], :classes], z64[s, :classes], 3.0)
        assert abs(got[s] - ref) <= 1e-4 * (1 + ref), (s, got[s], ref)


def test_branch_copies_rows_ids_and_moments_bit_exact():
    rng = np.random.default_rng(12)
    lens = [5, 0, 9, 3]
    cu = O.cu_from_counts(lens)
    t, d, t_cap = int(cu[-1]), 192, 64
    x = S.f32_to_bf16_bits(rng.standard_normal((t_cap, d)))
    ids = rng.integers(0, 1000, t_cap).astype(np.int32)
    mv = rng.standard_normal((t_cap, 2)).astype(np.float32)
    src = np.array([2, 1, 0, 2], dtype=np.int32)
    xt, it, mt = bf(x), i32(ids), f32(mv)
    cu_out = torch.full((len(lens) + 1 + len(src),), -5, dtype=torch.int32, device=dev())
    lens_out = torch.zeros(len(src), dtype=torch.int32, device=dev())
    st = _status()
    P.dora_branch(xt, i32(cu), i32(src), cu_out, ids=it, x_moments=mt, len_out=lens_out, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    want_lens = [lens[s] for s in src]
    want_cu = np.concatenate([cu, cu[-1] + np.cumsum(want_lens)])
    assert np.array_equal(cu_out.cpu().numpy(), want_cu)
    assert lens_out.cpu().numpy().tolist() == want_lens
    rows = np.concatenate([np.arange(cu[s], cu[s + 1]) for s in src]).astype(np.int64)
    end = t + len(rows)
    xb = bits(xt)
    assert np.array_equal(xb[:t], x[:t]) and np.array_equal(xb[end:], x[end:])
    assert np.array_equal(xb[t:end], x[rows])
    assert np.array_equal(it.cpu().numpy()[t:end], ids[rows])
    assert np.array_equal(mt.cpu().numpy()[t:end], mv[rows])
    # no room: the overflowing sequence gets length 0 and the status says so
    cu_small = torch.zeros(len(lens) + 2, dtype=torch.int32, device=dev())
    st = _status()
    P.dora_branch(bf(x[:t + 4]), i32(cu), i32([2]), cu_small, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == O.DORA_ERR_DEVICE_SEQLEN
    assert cu_small.cpu().numpy()[-1] == t


def _shadow_case(batch=4, depth=4, prune=(0, 2, 3), seed=13):
    cfg = S.get_config("cfg1", batch=batch, depth=depth, prune_blocks=prune)
    cu, ids = S.initial_layout(cfg)
    x = S.activations_bf16(cfg, seed)
    wbs = [S.block_weights(cfg, l, seed, random_affine=True) for l in range(depth)]
    keeps, _ = S.keep_schedule(cfg, seed)
    tables = [S.score_table(cfg, l, seed) for l in prune]
    return cfg, cu, ids, x, wbs, keeps, tables


def _run_shadows(cfg, cu, ids, x, wbs, keeps, tables):
    blocks = [P.BlockWeights({k: bf(v) for k, v in w.items()}, cfg.dim, cfg.heads, cfg.mlp_dim,
                             cfg.ln_eps) for w in wbs]
    sr = ShadowRollout(blocks, cfg.batch, cfg.n_tokens, cfg.prune_blocks, dev())
    xo, cuo, ido = sr.forward(bf(x), i32(cu), i32(ids), [f32(t) for t in tables],
                              [i32(k) for k in keeps])
    torch.cuda.synchronize()
    assert int(sr.status.item()) == 0
    assert P.dora_read_status(P.dora_workspace_status(sr.ws)) == 0
    return sr, xo, cuo.cpu().numpy(), ido.cpu().numpy()


def test_shadow_rollout_matches_oracle_prefixes():
    """Rollout, Native and the shadows of prefixes 0 and 2 in one packed
    batch: the integer trajectory of every sequence (boundaries, ids) bit for
    bit against the oracle's forward of each prefix run on its own."""
    cfg, cu, ids, x, wbs, keeps, tables = _shadow_case()
    sr, xo, cuo, ido = _run_shadows(cfg, cu, ids, x, wbs, keeps, tables)
    b = cfg.batch
    prune = {l: (tables[j], keeps[j]) for j, l in enumerate(cfg.prune_blocks)}
    ref = O.shadow_forwards(O.bf16_to_f64(x), cu, ids, [O.decode_weights(w) for w in wbs],
                            cfg.heads, cfg.ln_eps, prune)
    groups = [("rollout", cfg.prune_blocks[-1]), ("native", -1)] + \
        [(l, l) for l in cfg.prune_blocks[:-1]]
    assert len(cuo) == b * len(groups) + 1
    for name, key in groups:
        g0 = sr.groups[name]
        r = ref[key]
        lens = np.diff(cuo)[g0:g0 + b]
        assert np.array_equal(lens, np.diff(r["cu"])), name
        rows = np.concatenate([np.arange(cuo[g0 + i], cuo[g0 + i + 1]) for i in range(b)])
        assert np.array_equal(ido[rows], r["ids"]), name


def test_shadow_rollout_blocks_match_oracle():
    """Each block of the batched forward (rollout pruned, Native and shadows
    kept whole, branches after the pruning blocks) against the oracle block
    fed the same bf16 input: rows within the block tolerance, boundaries,
    ids and branched copies bit for bit."""
    cfg, cu, ids, x, wbs, keeps, tables = _shadow_case()
    blocks = [P.BlockWeights({k: bf(v) for k, v in w.items()}, cfg.dim, cfg.heads, cfg.mlp_dim,
                             cfg.ln_eps) for w in wbs]
    sr = ShadowRollout(blocks, cfg.batch, cfg.n_tokens, cfg.prune_blocks, dev())
    b = cfg.batch

    def state(stop):
        xs, cs, i_s = sr.forward(bf(x), i32(cu), i32(ids), [f32(t) for t in tables],
                                 [i32(k) for k in keeps], stop=stop)
        torch.cuda.synchronize()
        cs = cs.cpu().numpy()
        t = int(cs[-1])
        return bits(xs)[:t], cs, i_s.cpu().numpy()[:t]

    x_in, cu_in, ids_in = state(0)
    assert np.array_equal(cu_in, cu)
    for l in range(cfg.depth):
        x_out, cu_out, ids_out = state(l + 1)
        wf = O.decode_weights(wbs[l])
        if l == cfg.prune_blocks[0]:                     # the Native copies branch off here
            rows = np.arange(cu_in[0], cu_in[b])
            x_in = np.concatenate([x_in, x_in[rows]])
            ids_in = np.concatenate([ids_in, ids_in[rows]])
            cu_in = np.concatenate([cu_in, cu_in[-1] + cu_in[1:b + 1]])
        if l in cfg.prune_blocks:
            j = cfg.prune_blocks.index(l)
            scores = np.zeros(len(ids_in))
            scores[:cu_in[b]] = O.gather_scores(tables[j], cu_in[:b + 1], ids_in[:cu_in[b]])
            kc = np.concatenate([keeps[j], np.diff(cu_in)[b:]])
            r = O.pruned_block(O.bf16_to_f64(x_in), cu_in, ids_in, wf, cfg.heads, cfg.ln_eps,
                               scores, kc)
            rx, rcu, rids = r["x_out"], r["cu_out"], r["ids_out"]
            if l in cfg.prune_blocks[:-1]:               # the rollout's images branch off
                rows = np.arange(rcu[0], rcu[b])
                rx = np.concatenate([rx, rx[rows]])
                rids = np.concatenate([rids, rids[rows]])
                rcu = np.concatenate([rcu, rcu[-1] + rcu[1:b + 1]])
        else:
            r = O.pruned_block(O.bf16_to_f64(x_in), cu_in, ids_in, wf, cfg.heads, cfg.ln_eps)
            rx, rcu, rids = r["x_out"], cu_in, ids_in
        assert np.array_equal(cu_out, rcu), l
        assert np.array_equal(ids_out, rids), l
        assert_close(O.bf16_to_f64(x_out), rx, f"batched shadow forward, block {l}")
        if l in cfg.prune_blocks[:-1]:                   # branched rows are exact copies
            t0 = int(rcu[-b - 1])
            assert np.array_equal(x_out[t0:], x_out[rcu[0]:rcu[b]])
        x_in, cu_in, ids_in = x_out, cu_out, ids_out


def test_shadow_equals_the_prefix_run_alone_bit_for_bit():
    """A shadow riding in the big batch has the bits of the same prefix run as
    a rollout on its own (rows never interact across sequences)."""
    cfg, cu, ids, x, wbs, keeps, tables = _shadow_case()
    sr, xo, cuo, _ = _run_shadows(cfg, cu, ids, x, wbs, keeps, tables)
    b = cfg.batch
    g0 = sr.groups[0]
    shadow_rows = bits(xo)[cuo[g0]:cuo[g0 + b]]
    alone = S.get_config("cfg1", batch=b, depth=cfg.depth, prune_blocks=(0,))
    _, xa, cua, _ = _run_shadows(alone, cu, ids, x, wbs, keeps[:1], tables[:1])
    assert np.array_equal(bits(xa)[cua[0]:cua[b]], shadow_rows)


def test_shadow_costs_match_oracle_on_the_logits():
    cfg, cu, ids, x, wbs, keeps, tables = _shadow_case()
    sr, xo, cuo, _ = _run_shadows(cfg, cu, ids, x, wbs, keeps, tables)
    wh = S.embed_head_weights(cfg, 13)
    w_head = np.zeros((1024, cfg.dim), np.uint16)
    w_head[:1000] = wh["w_head"]
    b_head = np.zeros(1024, np.uint16)
    b_head[:1000] = wh["b_head"]
    logits, cost = sr.head_and_costs(xo, i32(cuo), bf(wh["norm_w"]), bf(wh["norm_b"]), 1e-6,
                                     bf(w_head), bf(b_head))
    torch.cuda.synchronize()
    assert int(sr.status.item()) == 0
    lg = f64(logits)
    c = cost.cpu().numpy().astype(np.float64)
    b = cfg.batch
    ref_logits = O.classifier_head(f64(xo), cuo, O.bf16_to_f64(wh["norm_w"]),
                                   O.bf16_to_f64(wh["norm_b"]), 1e-6, O.bf16_to_f64(w_head),
                                   O.bf16_to_f64(b_head))
    assert_close(lg, ref_logits, "shadow logits")
    for s in range(len(c)):
        ref = O.kd_cost(lg[b + s % b, :1000], lg[s, :1000], 3.0)
        assert abs(c[s] - ref) <= 1e-4 * (1 + ref), (s, c[s], ref)
    assert np.all(c[b:2 * b] == 0.0)                     # Native against itself
    assert np.all(c[:b] > 0) and np.all(c[2 * b:] > 0)


def test_training_rollout_deletes_its_sampled_sets():
    """Training mode: at each pruning block the removal order is sampled
    (Gumbel-top-k of the gathered scores) and the block deletes exactly the
    sampled set -- the rollout's trajectory equals the oracle forward whose
    score tables are the fp32 keys s + g; the orders' log-probabilities and
    gradients match the oracle's on the same scores."""
    cfg, cu, ids, x, wbs, keeps, tables = _shadow_case(seed=17)
    rng = np.random.default_rng(17)
    gtabs = [_gumbel(rng, t.size).reshape(t.shape) for t in tables]
    _, befores = S.keep_schedule(cfg, 17)
    removals = [np.asarray(bf_) - np.asarray(k) for bf_, k in zip(befores, keeps)]
    blocks = [P.BlockWeights({k: bf(v) for k, v in w.items()}, cfg.dim, cfg.heads, cfg.mlp_dim,
                             cfg.ln_eps) for w in wbs]
    sr = ShadowRollout(blocks, cfg.batch, cfg.n_tokens, cfg.prune_blocks, dev())
    xo, cuo, ido = sr.forward(bf(x), i32(cu), i32(ids), [f32(t) for t in tables],
                              [i32(k) for k in keeps], gumbel=[f32(g) for g in gtabs],
                              removals=[i32(r) for r in removals])
    adv = rng.uniform(-1, 1, cfg.batch)
    logp, grads = sr.logprob([i32(r) for r in removals], dlogp=f32(adv))
    torch.cuda.synchronize()
    assert int(sr.status.item()) == 0
    b = cfg.batch
    keyed = {l: ((tables[j] + gtabs[j]).astype(np.float32), keeps[j])
             for j, l in enumerate(cfg.prune_blocks)}
    ref = O.forward(O.bf16_to_f64(x), cu, ids, [O.decode_weights(w) for w in wbs], cfg.heads,
                    cfg.ln_eps, keyed)
    cuo = cuo.cpu().numpy()
    assert np.array_equal(np.diff(cuo)[:b], np.diff(ref["cu"]))
    assert np.array_equal(ido.cpu().numpy()[:cuo[b]], ref["ids"])
    orders = sr.order.cpu().numpy()
    lp = logp.cpu().numpy()
    for j, l in enumerate(cfg.prune_blocks):
        cuj = sr.cu_hist[j].cpu().numpy()
        sj = sr.s_hist[j].cpu().numpy()
        gj = grads[j].cpu().numpy()
        kept = ref["kept"][l]
        for i in range(b):
            lo, hi = int(cuj[i]), int(cuj[i + 1])
            k = int(removals[j][i])
            seq = orders[j, i, :k]
            kept_local = set((kept[(kept > lo) & (kept < hi)] - lo - 1).tolist())
            assert set(seq.tolist()) == set(range(hi - lo - 1)) - kept_local, (l, i)
            s = sj[lo + 1:hi].astype(np.float64)
            r = O.pl_logprob(s, seq)
            assert abs(lp[j, i] - r) <= 1e-5 * (abs(r) + k * (1 + np.abs(s).max())), (l, i)
            gref = adv[i] * O.pl_logprob_grad(s, seq)
            assert np.all(np.abs(gj[lo + 1:hi] - gref) <= 2e-4 * (1 + np.abs(gref)))


def test_branch_scan_across_chunks_and_overflow():
    """More appended sequences than one 1024-wide scan chunk: boundaries carried
    across chunks bit for bit; the first sequence past t_cap and every later
    one get length 0 with the status set."""
    rng = np.random.default_rng(14)
    lens = rng.integers(0, 6, 300)
    cu = O.cu_from_counts(lens)
    src = rng.integers(0, 300, 2500).astype(np.int32)
    want = np.concatenate([cu, cu[-1] + np.cumsum(lens[src])])
    d = 64
    t_cap = int(want[-1]) + 3
    x = S.f32_to_bf16_bits(rng.standard_normal((t_cap, d)))
    xt = bf(x)
    cu_out = torch.zeros(301 + len(src), dtype=torch.int32, device=dev())
    st = _status()
    P.dora_branch(xt, i32(cu), i32(src), cu_out, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert np.array_equal(cu_out.cpu().numpy(), want)
    rows = np.concatenate([np.arange(cu[s], cu[s + 1]) for s in src]).astype(np.int64)
    assert np.array_equal(bits(xt)[int(cu[-1]):int(want[-1])], x[rows])
    # room for the sequences up to index 1500 only
    cap = int(want[301 + 1500])
    lens_out = torch.zeros(len(src), dtype=torch.int32, device=dev())
    st = _status()
    P.dora_branch(bf(x[:cap]), i32(cu), i32(src), cu_out, len_out=lens_out, status=st)
    torch.cuda.synchronize()
    got = cu_out.cpu().numpy()
    fits = want[301:] <= cap
    assert np.array_equal(got[301:][fits], want[301:][fits])
    assert np.all(got[301:][~fits] == cap) and got[-1] == cap
    lo = lens_out.cpu().numpy()
    assert np.array_equal(lo[fits], lens[src][fits]) and np.all(lo[~fits] == 0)
    assert int(st.item()) == (O.DORA_ERR_DEVICE_SEQLEN if (lens[src][~fits] > 0).any() else 0)


def test_pl_sample_and_logprob_at_the_largest_image():
    """2048 visual tokens (the kernels' shared-memory limit), k up to 2048."""
    cu = O.cu_from_counts([2049, 2049, 300])
    t = int(cu[-1])
    rng = np.random.default_rng(15)
    scores = (rng.standard_normal(t) * 3).astype(np.float32)
    gumbel = _gumbel(rng, t)
    k = np.array([2048, 1000, 150])
    got, st = _run_sample(scores, gumbel, cu, k, 2048)
    assert st == 0
    assert np.array_equal(got, _oracle_orders(scores, gumbel, cu, k, 2048))
    _check_logprob(scores, cu, got.astype(np.int32), k, np.ones(3))


def _kd_first_order_bound(zn, z, dzn, dz, tau=3.0):
    """First-order bound on the change of D = tau^2 KL(softmax(zn/tau) ||
    softmax(z/tau)) when the logits move by at most dzn (Native) and dz
    (shadow) in every entry: dD/dz_c = tau (p_c - pn_c) and dD/dzn_c =
    tau pn_c (log(pn_c / p_c) - D / tau^2)."""
    lpn = O.log_softmax(zn / tau)
    lp = O.log_softmax(z / tau)
    pn, p = np.exp(lpn), np.exp(lp)
    d = tau * tau * float(np.sum(pn * (lpn - lp)))
    return (tau * float(np.abs(p - pn).sum()) * dz
            + tau * float(np.sum(pn * np.abs(lpn - lp - d / (tau * tau)))) * dzn)


def test_step_rewards_from_the_shadow_costs():
    """Local rewards (App. B.3) from the batched forward's fidelity costs,
    against the oracle's rewards on the same costs.  The costs are taken by
    the sequence groups of the batch, whose prefixes are pinned against the
    oracle's forwards elsewhere; each image's episode sum is checked against
    the telescoping identity 25 C - a D_final with C from the count schedule
    (Eq. 4) and D_final the rollout's own cost; and the first shadow's cost
    against the oracle's complete-prefix shadow (App. B.2) run end to end in
    fp64, within the first-order bound of the measured logit error."""
    cfg, cu, ids, x, wbs, keeps, tables = _shadow_case()
    sr, xo, cuo, _ = _run_shadows(cfg, cu, ids, x, wbs, keeps, tables)
    wh = S.embed_head_weights(cfg, 13)
    w_head = np.zeros((1024, cfg.dim), np.uint16)
    w_head[:1000] = wh["w_head"]
    logits, cost = sr.head_and_costs(xo, i32(cuo), bf(wh["norm_w"]), bf(wh["norm_b"]), 1e-6,
                                     bf(w_head), None)
    _, befores = S.keep_schedule(cfg, 13)
    rem = np.stack([np.asarray(b_) - np.asarray(k) for b_, k in zip(befores, keeps)])
    b, npb = cfg.batch, len(cfg.prune_blocks)
    reward = torch.zeros(npb, b, dtype=torch.float32, device=dev())
    ret = torch.zeros(b, dtype=torch.float32, device=dev())
    sr.rewards(i32(rem), 30.0, reward, ret=ret)
    torch.cuda.synchronize()
    c = cost.cpu().numpy().astype(np.float64)
    r = reward.cpu().numpy().astype(np.float64)
    comp = S.compression_from_counts(cfg, keeps, befores)
    g_roll = sr.groups["rollout"]
    for i in range(b):
        d = [c[sr.groups[l] + i] for l in cfg.prune_blocks[:-1]] + [c[g_roll + i]]
        ref = O.step_rewards(np.array(d), rem[:, i], cfg.prune_blocks, cfg.depth,
                             cfg.n_vis0, 30.0)
        assert np.allclose(r[:, i], ref, rtol=1e-5, atol=1e-5), (i, r[:, i], ref)
        assert abs(ret[i].item() - ref.sum()) <= 1e-5 * (1 + abs(ref.sum()))
        tele = 25.0 * comp[i] - 30.0 * c[g_roll + i]
        assert abs(ret[i].item() - tele) <= 1e-5 * (1 + abs(tele)), (i, ret[i].item(), tele)
    # the first shadow's cost against the oracle's own complete-prefix forward
    prune = {l: (tables[j], keeps[j]) for j, l in enumerate(cfg.prune_blocks)}
    l0 = cfg.prune_blocks[0]
    fw = O.shadow_forwards(O.bf16_to_f64(x), cu, ids, [O.decode_weights(w) for w in wbs],
                           cfg.heads, cfg.ln_eps, {l0: prune[l0]})
    head = (O.bf16_to_f64(wh["norm_w"]), O.bf16_to_f64(wh["norm_b"]), 1e-6,
            O.bf16_to_f64(w_head[:1000]), np.zeros(1000))
    zn = O.classifier_head(fw[-1]["x"], fw[-1]["cu"], *head)
    zs = O.classifier_head(fw[l0]["x"], fw[l0]["cu"], *head)
    lg = f64(logits)[:, :1000]
    g_nat, g_sh = sr.groups["native"], sr.groups[l0]
    for i in range(b):
        dzn = float(np.abs(lg[g_nat + i] - zn[i]).max())
        dz = float(np.abs(lg[g_sh + i] - zs[i]).max())
        want = O.kd_cost(zn[i], zs[i], 3.0)
        tol = 2.0 * _kd_first_order_bound(zn[i], zs[i], dzn, dz) + 1e-4 * (1 + want)
        assert abs(c[g_sh + i] - want) <= tol, (i, c[g_sh + i], want, tol)
