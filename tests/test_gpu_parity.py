"""GPU parity: every entry point of include/dora.h, called through the C ABI,
against the fp64 oracle on the same seeded inputs.  Integer and byte outputs
(kept_idx, cu_seqlens, ids, packed rows) must match bit for bit; floating
outputs within |err| <= 2e-2 or |err| <= 1e-2 |ref|."""
import numpy as np
import pytest
import torch

import __graft_entry__ as G
import dora_synth as S
import oracle as O
import paper_2609_34325_gb300 as P
from helpers import assert_close, bf, bits, dev, f32, f64, i32, sub_batch

pytestmark = pytest.mark.gpu

CFGS = ("cfg1", "cfg2", "cfg3", "cfg4", "cfg5")
SENT = -7


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    G.build()
    P.load_library()
    torch.cuda.set_device(0)


def _status():
    return torch.zeros(1, dtype=torch.int32, device=dev())


# ---------------------------------------------------------------------------
# select_keep
# ---------------------------------------------------------------------------

def _run_select(scores, cu, keeps, max_seqlen):
    t_in = int(cu[-1])
    b = len(cu) - 1
    kept = torch.full((max(t_in, 1),), SENT, dtype=torch.int32, device=dev())
    cu_out = torch.full((b + 1,), SENT, dtype=torch.int32, device=dev())
    st = _status()
    P.dora_select_keep(f32(scores), i32(cu), i32(keeps), max_seqlen, kept, cu_out, st)
    torch.cuda.synchronize()
    return kept.cpu().numpy(), cu_out.cpu().numpy(), int(st.item())


def _check_select(scores, cu, keeps, max_seqlen=None):
    lens = np.diff(cu)
    ms = int(lens.max()) if max_seqlen is None else max_seqlen
    kept, cu_out, st = _run_select(scores, cu, keeps, ms)
    rk, rcu, rst = O.select_keep(scores, cu, keeps)
    assert np.array_equal(cu_out, rcu)
    t_out = int(rcu[-1])
    assert np.array_equal(kept[:t_out], rk)
    assert np.all(kept[t_out:] == SENT)            # nothing written past T_out
    assert st == rst
    return t_out


@pytest.mark.parametrize("name", CFGS)
def test_select_keep_configs(name):
    cfg = S.get_config(name)
    cu, ids = S.initial_layout(cfg)
    keeps, _ = S.keep_schedule(cfg, 0)
    for j, blk in enumerate(cfg.prune_blocks[:2]):
        table = S.score_table(cfg, blk, 0)
        # the second step uses the packed layout produced by the first
        if j == 0:
            lcu, lids = cu, ids
        scores = O.gather_scores(table, lcu, lids)
        _check_select(scores, lcu, keeps[j], cfg.n_tokens)
        rk, rcu, _ = O.select_keep(scores, lcu, keeps[j])
        lcu, lids = rcu, lids[rk]


def _edge_lengths():
    return np.array([1, 2, 15, 16, 17, 31, 32, 33, 64, 127, 128, 129, 197, 255, 256, 257, 577])


def _edge_scores(rng, t, kind):
    """Scores of one edge-case kind for t tokens."""
    if kind == "uniform":
        return rng.random(t).astype(np.float32)
    if kind == "ties":
        return rng.choice(np.array([0.0, 0.25, 0.5], np.float32), size=t)
    if kind == "allequal":
        return np.full(t, 0.125, np.float32)
    if kind == "prefixes":
        # positive floats whose bit patterns share their top one, two or
        # three bytes, with exact duplicates: the threshold's prefix is
        # unique after the first, second or third 8-bit pass, or never
        b3 = rng.choice(np.array([0x3E, 0x3F], np.uint32), size=t)
        b2 = rng.choice(np.array([0x00, 0x80], np.uint32), size=t)
        b1 = rng.choice(np.array([0x10, 0x20, 0x30], np.uint32), size=t)
        b0 = rng.integers(0, 256, size=t).astype(np.uint32)
        s = ((b3 << 24) | (b2 << 16) | (b1 << 8) | b0).view(np.float32)
        dup = rng.random(t) < 0.1
        s[dup] = np.roll(s, 1)[dup]
        return s
    pal = np.array([0.0, -0.0, np.nan, -np.nan, np.inf, -np.inf, 1.0, -1.0, 1e-38, -1e-38],
                   dtype=np.float32)
    return rng.choice(pal, size=t)


@pytest.mark.parametrize("kind", ["uniform", "ties", "special", "allequal", "prefixes"])
def test_select_keep_edges(kind):
    rng = np.random.default_rng(42)
    lens = _edge_lengths()
    cu = O.cu_from_counts(lens)
    t = int(cu[-1])
    s = _edge_scores(rng, t, kind)
    if kind == "special":
        s[rng.random(t) < 0.02] = np.float32(np.nan)
    for mode in ("one", "all", "random"):
        if mode == "one":
            keeps = np.ones_like(lens)
        elif mode == "all":
            keeps = lens.copy()
        else:
            keeps = np.array([rng.integers(1, n + 1) for n in lens])
        _check_select(s, cu, keeps)


def test_select_keep_bad_counts_and_empty_images():
    lens = np.array([5, 0, 9, 3, 12])
    cu = O.cu_from_counts(lens)
    s = np.random.default_rng(3).random(int(cu[-1])).astype(np.float32)
    keeps = np.array([0, 0, 20, 3, -4])       # 0 (<1), empty ok, >n, ok, negative
    _check_select(s, cu, keeps)
    _, _, st = _run_select(s, cu, keeps, 12)
    assert st == O.DORA_ERR_DEVICE_BAD_COUNT


def test_select_keep_longer_than_max_seqlen_flags():
    lens = np.array([10, 40, 10])
    cu = O.cu_from_counts(lens)
    s = np.random.default_rng(4).random(60).astype(np.float32)
    kept, cu_out, st = _run_select(s, cu, np.array([5, 5, 5]), 32)
    assert st == 6
    assert cu_out.tolist() == [0, 5, 5, 10]     # the long image keeps nothing


def test_select_keep_large_batch_b1024():
    rng = np.random.default_rng(5)
    lens = rng.integers(1, 198, size=1024)
    cu = O.cu_from_counts(lens)
    s = rng.random(int(cu[-1])).astype(np.float32)
    keeps = np.array([rng.integers(1, n + 1) for n in lens])
    _check_select(s, cu, keeps, 197)


# ---------------------------------------------------------------------------
# compaction
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("name", CFGS)
def test_compact_bit_exact(name):
    cfg = S.get_config(name)
    cu, ids = S.initial_layout(cfg)
    keeps, _ = S.keep_schedule(cfg, 1)
    scores = O.gather_scores(S.score_table(cfg, cfg.prune_blocks[0], 1), cu, ids)
    rk, rcu, _ = O.select_keep(scores, cu, keeps[0])
    t_in, t_out = int(cu[-1]), int(rcu[-1])
    rng = np.random.default_rng(6)
    x = rng.integers(0, 65536, size=(t_in, cfg.dim), dtype=np.uint16)   # any bit pattern
    packed = torch.zeros(t_in, cfg.dim, dtype=torch.bfloat16, device=dev())
    packed.view(torch.int16).fill_(SENT)
    ids_out = torch.full((t_in,), SENT, dtype=torch.int32, device=dev())
    st = _status()
    kept_d = torch.zeros(t_in, dtype=torch.int32, device=dev())
    kept_d[:t_out] = i32(rk)
    P.dora_compact(bf(x), kept_d, i32(rcu), packed, ids_in=i32(ids), ids_out=ids_out, status=st)
    torch.cuda.synchronize()
    ref_packed, ref_ids = O.compact(x, rk, ids)
    got = bits(packed)
    assert np.array_equal(got[:t_out], ref_packed)
    assert np.all(got[t_out:].view(np.int16) == SENT)
    assert np.array_equal(ids_out.cpu().numpy()[:t_out], ref_ids)
    assert int(st.item()) == 0


@pytest.mark.parametrize("name", ["cfg1", "cfg3", "cfg4"])
def test_compact_ln_fused(name):
    cfg = S.get_config(name)
    cu, ids = S.initial_layout(cfg)
    keeps, _ = S.keep_schedule(cfg, 2)
    scores = O.gather_scores(S.score_table(cfg, cfg.prune_blocks[0], 2), cu, ids)
    rk, rcu, _ = O.select_keep(scores, cu, keeps[0])
    t_in, t_out = int(cu[-1]), int(rcu[-1])
    x = S.activations_bf16(cfg, 2)
    wb = S.block_weights(cfg, 0, 2, random_affine=True)
    packed = torch.zeros(t_in, cfg.dim, dtype=torch.bfloat16, device=dev())
    ln = torch.zeros_like(packed)
    kept_d = torch.zeros(t_in, dtype=torch.int32, device=dev())
    kept_d[:t_out] = i32(rk)
    P.dora_compact_ln(bf(x), kept_d, i32(rcu), bf(wb["ln2_w"]), bf(wb["ln2_b"]), cfg.ln_eps,
                      packed, ln)
    torch.cuda.synchronize()
    assert np.array_equal(bits(packed)[:t_out], x[rk])
    ref = O.layernorm(O.bf16_to_f64(x[rk]), O.bf16_to_f64(wb["ln2_w"]),
                      O.bf16_to_f64(wb["ln2_b"]), cfg.ln_eps)
    assert_close(f64(ln[:t_out]), ref, "compact_ln")


def test_compact_empty_output():
    cu_out = i32(np.zeros(4))
    x = torch.zeros(10, 64, dtype=torch.bfloat16, device=dev())
    packed = torch.full_like(x, 3.0)
    P.dora_compact(x, torch.zeros(10, dtype=torch.int32, device=dev()), cu_out, packed)
    torch.cuda.synchronize()
    assert torch.all(packed == 3.0)


# ---------------------------------------------------------------------------
# selection fused with the compaction (one launch)
# ---------------------------------------------------------------------------

def _run_select_compact(scores, cu, keeps, max_seqlen, x, ids=None, mv=None, t_cap=None,
                        extra=0):
    """dora_select_compact with sentinel-filled outputs of t_cap + extra rows."""
    t_cap = int(cu[-1]) if t_cap is None else t_cap
    b = len(cu) - 1
    dim = x.shape[1]
    rows = max(t_cap + extra, 1)
    kept = torch.full((rows,), SENT, dtype=torch.int32, device=dev())
    cu_out = torch.full((b + 1,), SENT, dtype=torch.int32, device=dev())
    packed = torch.zeros(rows, dim, dtype=torch.bfloat16, device=dev())
    packed.view(torch.int16).fill_(SENT)
    ids_out = mv_out = None
    if ids is not None:
        ids_out = torch.full((rows,), SENT, dtype=torch.int32, device=dev())
    if mv is not None:
        mv_out = torch.full((rows, 2), float(SENT), dtype=torch.float32, device=dev())
    st = _status()
    xd = bf(x[:t_cap]) if t_cap > 0 else torch.zeros(0, dim, dtype=torch.bfloat16, device=dev())
    P.dora_select_compact(f32(scores), i32(cu), i32(keeps), max_seqlen, xd, kept, cu_out, packed,
                          ids_in=None if ids is None else i32(ids[:t_cap]), ids_out=ids_out,
                          mv_in=None if mv is None else f32(mv[:t_cap]), mv_out=mv_out, status=st)
    torch.cuda.synchronize()
    return dict(kept=kept.cpu().numpy(), cu=cu_out.cpu().numpy(), packed=bits(packed),
                ids=None if ids_out is None else ids_out.cpu().numpy(),
                mv=None if mv_out is None else mv_out.cpu().numpy(), status=int(st.item()))


def _check_select_compact(scores, cu, keeps, x, ids=None, mv=None, max_seqlen=None):
    lens = np.diff(cu)
    ms = int(lens.max()) if max_seqlen is None else max_seqlen
    g = _run_select_compact(scores, cu, keeps, ms, x, ids, mv)
    rk, rcu, rst = O.select_keep(scores, cu, keeps)
    t_out = int(rcu[-1])
    assert np.array_equal(g["cu"], rcu)
    assert np.array_equal(g["kept"][:t_out], rk)
    assert np.all(g["kept"][t_out:] == SENT)
    assert g["status"] == rst
    ref_packed, ref_ids = O.compact(x, rk, ids if ids is not None else np.zeros(len(x), np.int32))
    assert np.array_equal(g["packed"][:t_out], ref_packed)
    assert np.all(g["packed"][t_out:].view(np.int16) == SENT)
    if ids is not None:
        assert np.array_equal(g["ids"][:t_out], ref_ids)
        assert np.all(g["ids"][t_out:] == SENT)
    if mv is not None:
        assert np.array_equal(g["mv"][:t_out].view(np.uint32), mv[rk].view(np.uint32))
        assert np.all(g["mv"][t_out:] == SENT)
    return t_out


def _row_inputs(rng, t, dim):
    x = rng.integers(0, 65536, size=(t, dim), dtype=np.uint16)      # any bit pattern
    ids = rng.integers(0, 1 << 20, size=t).astype(np.int32)
    mv = rng.standard_normal((t, 2)).astype(np.float32)
    return x, ids, mv


@pytest.mark.parametrize("name", CFGS)
def test_select_compact_configs(name):
    """Kept rows, ids, row moments, kept_idx and boundaries of one launch,
    bit for bit against the oracle's selection and compaction, on the first
    two pruning steps of every workload."""
    cfg = S.get_config(name)
    cu, ids = S.initial_layout(cfg)
    keeps, _ = S.keep_schedule(cfg, 3)
    rng = np.random.default_rng(30)
    lcu, lids = cu, ids
    for j, blk in enumerate(cfg.prune_blocks[:2]):
        scores = O.gather_scores(S.score_table(cfg, blk, 3), lcu, lids)
        x, _, mv = _row_inputs(rng, int(lcu[-1]), cfg.dim)
        _check_select_compact(scores, lcu, keeps[j], x, lids, mv, cfg.n_tokens)
        rk, rcu, _ = O.select_keep(scores, lcu, keeps[j])
        lcu, lids = rcu, lids[rk]


@pytest.mark.parametrize("dim", [64, 192, 384, 768, 1024, 2048])
@pytest.mark.parametrize("kind", ["uniform", "ties", "special", "allequal", "prefixes"])
def test_select_compact_edges(kind, dim):
    """Lengths 1..577 around the 16/32/128/256 boundaries, ties, signed
    zeros, NaN and infinities, keep one / all / random, every row width class
    (1 to 8 16-byte chunks a lane); ids and moments given or not."""
    rng = np.random.default_rng(43)
    lens = _edge_lengths()
    cu = O.cu_from_counts(lens)
    t = int(cu[-1])
    s = _edge_scores(rng, t, kind)
    x, ids, mv = _row_inputs(rng, t, dim)
    for n, mode in enumerate(("one", "all", "random")):
        if mode == "one":
            keeps = np.ones_like(lens)
        elif mode == "all":
            keeps = lens.copy()
        else:
            keeps = np.array([rng.integers(1, k + 1) for k in lens])
        with_side = n != 1
        _check_select_compact(s, cu, keeps, x, ids if with_side else None,
                              mv if with_side else None)


def test_select_compact_bad_counts_and_max_seqlen():
    rng = np.random.default_rng(44)
    lens = np.array([5, 0, 9, 3, 12])
    cu = O.cu_from_counts(lens)
    s = rng.random(int(cu[-1])).astype(np.float32)
    x, ids, mv = _row_inputs(rng, int(cu[-1]), 192)
    keeps = np.array([0, 0, 20, 3, -4])
    _check_select_compact(s, cu, keeps, x, ids, mv)
    lens = np.array([10, 40, 10])
    cu = O.cu_from_counts(lens)
    x, ids, mv = _row_inputs(rng, 60, 192)
    g = _run_select_compact(rng.random(60).astype(np.float32), cu, np.array([5, 5, 5]), 32, x,
                            ids, mv)
    assert g["status"] == O.DORA_ERR_DEVICE_SEQLEN
    assert g["cu"].tolist() == [0, 5, 5, 10]               # the long image keeps nothing
    assert np.all(g["packed"][10:].view(np.int16) == SENT)


def test_select_compact_overlapping_boundaries_stay_in_capacity():
    """Boundaries that are not increasing ([0, 100, 50, 150]: the second
    image has negative length, the third overlaps the first) keep the outputs
    inside the input's 150 rows: rows past them are dropped and the status
    says so."""
    rng = np.random.default_rng(45)
    cu = np.array([0, 100, 50, 150], np.int32)
    s = rng.random(150).astype(np.float32)
    x, ids, mv = _row_inputs(rng, 150, 128)
    keeps = np.array([90, 0, 80])
    g = _run_select_compact(s, cu, keeps, 100, x, ids, mv, t_cap=150, extra=64)
    # the first error recorded wins: the negative length or the overflow
    assert g["status"] in (O.DORA_ERR_DEVICE_BAD_COUNT, O.DORA_ERR_DEVICE_SEQLEN)
    assert g["cu"].tolist() == [0, 90, 90, 170]
    assert np.all(g["kept"][150:] == SENT)
    assert np.all(g["packed"][150:].view(np.int16) == SENT)
    assert np.all(g["ids"][150:] == SENT) and np.all(g["mv"][150:] == SENT)
    # the first image's 90 rows are exact
    rk, _, _ = O.select_keep(s[:100], np.array([0, 100]), np.array([90]))
    assert np.array_equal(g["kept"][:90], rk)
    assert np.array_equal(g["packed"][:90], x[rk])


def test_select_compact_large_batch_b1024():
    rng = np.random.default_rng(46)
    lens = rng.integers(1, 198, size=1024)
    cu = O.cu_from_counts(lens)
    t = int(cu[-1])
    s = rng.random(t).astype(np.float32)
    x, ids, mv = _row_inputs(rng, t, 768)
    keeps = np.array([rng.integers(1, n + 1) for n in lens])
    _check_select_compact(s, cu, keeps, x, ids, mv, 197)


def test_select_compact_longest_images():
    """Images of 8192 tokens (the selection's shared-memory limit), every
    image the same length and a mix."""
    rng = np.random.default_rng(47)
    lens = np.array([8192, 1, 8192, 4097])
    cu = O.cu_from_counts(lens)
    t = int(cu[-1])
    s = rng.random(t).astype(np.float32)
    pick = rng.random(t) < 0.4                        # ties and NaN among random scores
    s[pick] = rng.choice(np.array([0.0, 0.5, 1.0, np.nan], np.float32), size=int(pick.sum()))
    x, ids, mv = _row_inputs(rng, t, 64)
    keeps = np.array([4000, 1, 8192, 17])
    _check_select_compact(s, cu, keeps, x, ids, mv, 8192)


# ---------------------------------------------------------------------------
# LayerNorm
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("dim", [64, 192, 384, 768, 1024, 2048])
def test_layernorm(dim):
    rng = np.random.default_rng(dim)
    rows_cap, rows = 1000, 777
    x = S.f32_to_bf16_bits(rng.standard_normal((rows_cap, dim)) * 3 + 1)
    w = S.f32_to_bf16_bits(1 + 0.1 * rng.standard_normal(dim))
    b = S.f32_to_bf16_bits(0.1 * rng.standard_normal(dim))
    y = torch.full((rows_cap, dim), 5.0, dtype=torch.bfloat16, device=dev())
    P.dora_layernorm(bf(x), bf(w), bf(b), 1e-6, y, rows_dev=i32([rows]))
    torch.cuda.synchronize()
    ref = O.layernorm(O.bf16_to_f64(x[:rows]), O.bf16_to_f64(w), O.bf16_to_f64(b), 1e-6)
    assert_close(f64(y[:rows]), ref, f"layernorm d={dim}")
    assert torch.all(y[rows:] == 5.0)


# ---------------------------------------------------------------------------
# linear (tcgen05 GEMM)
# ---------------------------------------------------------------------------

LINEAR_CASES = [
    # m_cap, m_live, k, n, epilogue
    (128, 128, 64, 128, 0),
    (300, 300, 192, 576, 0),       # ragged M, N not a multiple of 256
    (1576, 1576, 192, 576, 0),     # cfg1 QKV
    (1576, 1200, 192, 768, 1),     # cfg1 fc1 after a deletion
    (1576, 1200, 768, 192, 2),     # cfg1 fc2
    (12608, 7904, 384, 1152, 0),   # cfg2 QKV shape, fewer live rows
    (2000, 1999, 768, 2304, 0),
    (2000, 1001, 768, 3072, 1),
    (2000, 1500, 3072, 768, 2),
    (777, 777, 1024, 4096, 1),
    (777, 640, 4096, 1024, 2),
    (129, 1, 64, 32, 2),
    (256, 0, 64, 256, 0),
]


@pytest.mark.parametrize("m_cap,m_live,k,n,epi", LINEAR_CASES)
def test_linear(m_cap, m_live, k, n, epi):
    rng = np.random.default_rng(m_cap * 7 + n + epi)
    x = S.f32_to_bf16_bits(rng.standard_normal((m_cap, k)))
    w = S.f32_to_bf16_bits(0.02 * rng.standard_normal((n, k)))
    b = S.f32_to_bf16_bits(0.1 * rng.standard_normal(n))
    r = S.f32_to_bf16_bits(rng.standard_normal((m_cap, n)))
    y = torch.full((m_cap, n), 7.0, dtype=torch.bfloat16, device=dev())
    st = _status()
    P.dora_linear(bf(x), bf(w), y, bias=bf(b), residual=bf(r) if epi == 2 else None,
                  epilogue=epi, m_dev=i32([m_live]), status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    ref = O.linear(O.bf16_to_f64(x[:m_live]), O.bf16_to_f64(w), O.bf16_to_f64(b))
    if epi == 1:
        ref = O.gelu(ref)
    if epi == 2:
        ref = ref + O.bf16_to_f64(r[:m_live])
    assert_close(f64(y[:m_live]), ref, f"linear {m_cap}x{n}x{k} epi{epi}")
    assert torch.all(y[m_live:] == 7.0)


def test_linear_gelu_epilogue_within_one_bf16_ulp():
    """The GELU epilogue against exact-erf GELU on a dense grid: x has one
    nonzero column and W routes it to every output, so each output is
    GELU(v) of an exactly known v; the result must be within one bf16 ulp,
    plus the approximation's absolute bound (|x| * 0.75e-7 <= 1e-6 here) that
    matters only in the far tail where GELU itself is below 1e-6."""
    m, k, n = 4096, 64, 32
    v = S.bf16_bits_to_f32(S.f32_to_bf16_bits(np.linspace(-9.0, 9.0, m))).astype(np.float64)
    x = np.zeros((m, k))
    x[:, 0] = v
    w = np.zeros((n, k))
    w[:, 0] = 1.0
    y = torch.zeros(m, n, dtype=torch.bfloat16, device=dev())
    P.dora_linear(bf(S.f32_to_bf16_bits(x)), bf(S.f32_to_bf16_bits(w)), y,
                  epilogue=P.EPI_BIAS_GELU)
    torch.cuda.synchronize()
    ref = O.gelu(v)[:, None]
    err = np.abs(f64(y) - ref)
    assert np.all(err <= 2.0 ** -7 * np.abs(ref) + 1e-6), float(err.max())


def test_linear_no_bias_full_rows():
    rng = np.random.default_rng(9)
    x = S.f32_to_bf16_bits(rng.standard_normal((512, 256)))
    w = S.f32_to_bf16_bits(0.05 * rng.standard_normal((512, 256)))
    y = torch.zeros(512, 512, dtype=torch.bfloat16, device=dev())
    P.dora_linear(bf(x), bf(w), y)
    torch.cuda.synchronize()
    ref = O.bf16_to_f64(x) @ O.bf16_to_f64(w).T
    assert_close(f64(y), ref, "linear no bias")


# ---------------------------------------------------------------------------
# LayerNorm folded into the linear after it
# ---------------------------------------------------------------------------

def _row_moments_ref(x_bits):
    """fp64 row moments (mean, biased variance) of bf16 rows."""
    v = O.bf16_to_f64(x_bits)
    mean = v.mean(axis=1)
    return mean, ((v - mean[:, None]) ** 2).mean(axis=1)


def _check_row_moments(got, x_bits, what):
    """got [rows, 2] against fp64: fp32 sums of dim terms, a few roundings of
    the largest partial sum."""
    mean, var = _row_moments_ref(x_bits)
    scale = np.abs(O.bf16_to_f64(x_bits)).max(axis=1)
    assert np.all(np.abs(got[:, 0] - mean) <= 4e-6 * scale + 1e-30), what
    assert np.all(np.abs(got[:, 1] - var) <= 1e-5 * var + 1e-6 * scale ** 2 + 1e-30), what


def _ln_rows(rng, rows, dim):
    """Rows with their own offset and spread, as a residual stream has."""
    off = rng.uniform(-8, 8, (rows, 1))
    sd = np.exp(rng.uniform(-1.5, 1.5, (rows, 1)))
    return S.f32_to_bf16_bits(off + sd * rng.standard_normal((rows, dim)))


@pytest.mark.parametrize("slices", [1, 3, 12, 16, 17, 32])
def test_merge_moments_slice_counts(slices):
    """Row moments merged from 64-column slice moments: the held path (up to
    16 slices in registers) and the streaming one past it, rows past the live
    count untouched."""
    rng = np.random.default_rng(40 + slices)
    rows, live = 300, 257
    xb = _ln_rows(rng, rows, 64 * slices)
    v = O.bf16_to_f64(xb).reshape(rows, slices, 64)
    s_mean = v.mean(axis=2)
    s_m2 = ((v - s_mean[..., None]) ** 2).sum(axis=2)
    sm = np.stack([s_mean, s_m2], axis=2).transpose(1, 0, 2).astype(np.float32)   # [S, rows, 2]
    sm_d = torch.from_numpy(np.ascontiguousarray(sm)).to(dev())
    mv = torch.full((rows, 2), -3.0, dtype=torch.float32, device=dev())
    P.dora_merge_moments(sm_d, mv, rows_dev=i32([live]))
    torch.cuda.synchronize()
    got = mv.cpu().numpy().astype(np.float64)
    assert np.all(got[live:] == -3.0)
    _check_row_moments(got[:live], xb[:live], f"merged moments, {slices} slices")


@pytest.mark.parametrize("dim", [64, 192, 768, 1024, 2048])
def test_row_stats(dim):
    rng = np.random.default_rng(dim + 1)
    rows_cap, rows = 1000, 777
    x = _ln_rows(rng, rows_cap, dim)
    mv = torch.full((rows_cap, 2), -3.0, dtype=torch.float32, device=dev())
    P.dora_row_stats(bf(x), mv, rows_dev=i32([rows]))
    torch.cuda.synchronize()
    got = mv.cpu().numpy().astype(np.float64)
    _check_row_moments(got[:rows], x[:rows], f"row_stats d={dim}")
    assert np.all(got[rows:] == -3.0)


@pytest.mark.parametrize("n,k", [(576, 192), (3072, 768), (32, 2048)])
def test_fold_ln_linear(n, k):
    rng = np.random.default_rng(n + k)
    w = S.f32_to_bf16_bits(0.02 * rng.standard_normal((n, k)))
    g = S.f32_to_bf16_bits(1 + 0.3 * rng.standard_normal(k))
    be = S.f32_to_bf16_bits(0.1 * rng.standard_normal(k))
    b = S.f32_to_bf16_bits(0.1 * rng.standard_normal(n))
    w_out = torch.zeros(n, k, dtype=torch.bfloat16, device=dev())
    cs = torch.zeros(n, dtype=torch.float32, device=dev())
    cb = torch.zeros(n, dtype=torch.float32, device=dev())
    P.dora_fold_ln_linear(bf(w), bf(g), bf(be), w_out, cs, cb, bias=bf(b))
    torch.cuda.synchronize()
    wf, gf, bef, bf_ = (O.bf16_to_f64(a) for a in (w, g, be, b))
    # the product of two bf16 values is exact in fp32: one nearest-even rounding
    want = S.f32_to_bf16_bits(wf * gf[None, :])
    assert np.array_equal(bits(w_out), want)
    c_ref = O.bf16_to_f64(want).sum(axis=1)
    d_ref = wf @ bef + bf_
    mag = np.abs(O.bf16_to_f64(want)).sum(axis=1)
    # fp32 accumulation: k/32 terms per lane, then a 32-lane tree (a dropped
    # term would be ~1/k of mag)
    assert np.all(np.abs(cs.cpu().numpy() - c_ref) <= 8e-6 * mag + 1e-7)
    mag_d = np.abs(wf) @ np.abs(bef) + np.abs(bf_)
    assert np.all(np.abs(cb.cpu().numpy() - d_ref) <= 8e-6 * mag_d + 1e-7)


@pytest.mark.parametrize("name", ["cfg1", "cfg3"])
def test_compact_stats(name):
    """Compaction carrying row moments: packed rows bit-exact (as
    dora_compact) and mv_out[r] = mv_in[kept[r]] bit for bit."""
    cfg = S.get_config(name)
    cu, ids = S.initial_layout(cfg)
    t_in = int(cu[-1])
    rng = np.random.default_rng(5)
    x = _ln_rows(rng, t_in, cfg.dim)
    mv_in = rng.standard_normal((t_in, 2)).astype(np.float32)
    keeps, _ = S.keep_schedule(cfg, 5)
    scores = O.gather_scores(S.score_table(cfg, cfg.prune_blocks[0], 5), cu, ids)
    rk, rcu, _ = O.select_keep(scores, cu, keeps[0])
    t_out = int(rcu[-1])
    packed = torch.zeros(t_in, cfg.dim, dtype=torch.bfloat16, device=dev())
    mv_out = torch.full((t_in, 2), -3.0, dtype=torch.float32, device=dev())
    ids_out = torch.full((t_in,), SENT, dtype=torch.int32, device=dev())
    P.dora_compact_stats(bf(x), i32(rk), i32(rcu), packed, f32(mv_in), mv_out, ids_in=i32(ids),
                         ids_out=ids_out)
    torch.cuda.synchronize()
    assert np.array_equal(bits(packed[:t_out]), x[rk])
    assert np.array_equal(ids_out.cpu().numpy()[:t_out], ids[rk])
    got = mv_out.cpu().numpy()
    assert np.array_equal(got[:t_out].view(np.uint32), mv_in[rk].view(np.uint32))
    assert np.all(got[t_out:] == -3.0)


LINEAR_LN_CASES = [
    # m_cap, m_live, k, n, gelu
    (300, 300, 64, 128, False),      # one slice, ragged M
    (1576, 1576, 192, 576, False),   # cfg1 QKV
    (1576, 1200, 192, 768, True),    # cfg1 fc1 after a deletion
    (2000, 1999, 768, 2304, False),  # DeiT-B QKV
    (2000, 1001, 768, 3072, True),   # DeiT-B fc1
    (777, 640, 1024, 4096, True),
    (129, 1, 2048, 32, False),
    (256, 0, 768, 256, True),
]


@pytest.mark.parametrize("m_cap,m_live,k,n,gelu", LINEAR_LN_CASES)
def test_linear_ln(m_cap, m_live, k, n, gelu):
    """row moments -> fold -> GEMM with the folded LayerNorm, against the
    oracle's LayerNorm then linear (then GELU) in fp64."""
    rng = np.random.default_rng(m_cap + 3 * n + k)
    eps = 1e-6
    x = _ln_rows(rng, m_cap, k)
    g = S.f32_to_bf16_bits(1 + 0.3 * rng.standard_normal(k))
    be = S.f32_to_bf16_bits(0.2 * rng.standard_normal(k))
    w = S.f32_to_bf16_bits(0.02 * rng.standard_normal((n, k)))
    b = S.f32_to_bf16_bits(0.1 * rng.standard_normal(n))
    mv = torch.zeros(m_cap, 2, dtype=torch.float32, device=dev())
    w_out = torch.zeros(n, k, dtype=torch.bfloat16, device=dev())
    cs = torch.zeros(n, dtype=torch.float32, device=dev())
    cb = torch.zeros(n, dtype=torch.float32, device=dev())
    y = torch.full((m_cap, n), 7.0, dtype=torch.bfloat16, device=dev())
    st = _status()
    m_dev = i32([m_live])
    P.dora_row_stats(bf(x), mv, rows_dev=m_dev)
    P.dora_fold_ln_linear(bf(w), bf(g), bf(be), w_out, cs, cb, bias=bf(b))
    P.dora_linear_ln(bf(x), mv, eps, w_out, cs, cb, y, gelu=gelu, m_dev=m_dev, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    ref = O.linear(O.layernorm(O.bf16_to_f64(x[:m_live]), O.bf16_to_f64(g), O.bf16_to_f64(be),
                               eps), O.bf16_to_f64(w), O.bf16_to_f64(b))
    if gelu:
        ref = O.gelu(ref)
    assert_close(f64(y[:m_live]), ref, f"linear_ln {m_cap}x{n}x{k} gelu={gelu}")
    assert torch.all(y[m_live:] == 7.0)


@pytest.mark.parametrize("m_cap,m_live,k,n", [(1576, 1200, 768, 192), (2000, 1500, 3072, 768),
                                              (129, 1, 64, 64), (777, 640, 4096, 1024)])
def test_linear_residual_stats(m_cap, m_live, k, n):
    """The residual epilogue's output equals dora_linear's bit for bit; its
    slice moments match fp64 slice moments of that output, and merged they
    match the fp64 row moments (and dora_row_stats) within fp32 rounding."""
    rng = np.random.default_rng(m_cap + n)
    x = S.f32_to_bf16_bits(rng.standard_normal((m_cap, k)))
    w = S.f32_to_bf16_bits(0.02 * rng.standard_normal((n, k)))
    b = S.f32_to_bf16_bits(0.1 * rng.standard_normal(n))
    r = _ln_rows(rng, m_cap, n)
    m_dev = i32([m_live])
    y = torch.full((m_cap, n), 7.0, dtype=torch.bfloat16, device=dev())
    y2 = torch.full((m_cap, n), 7.0, dtype=torch.bfloat16, device=dev())
    sm = torch.full((n // 64, m_cap, 2), -3.0, dtype=torch.float32, device=dev())
    mv = torch.full((m_cap, 2), -3.0, dtype=torch.float32, device=dev())
    st = _status()
    P.dora_linear_residual_stats(bf(x), bf(w), bf(r), y, sm, bias=bf(b), m_dev=m_dev, status=st)
    P.dora_linear(bf(x), bf(w), y2, bias=bf(b), residual=bf(r), epilogue=P.EPI_BIAS_RESIDUAL,
                  m_dev=m_dev)
    P.dora_merge_moments(sm, mv, rows_dev=m_dev)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert torch.equal(y, y2)
    yb = bits(y[:m_live])
    got = sm.cpu().numpy().astype(np.float64).transpose(1, 0, 2)     # slice-major -> rows
    assert np.all(got[m_live:] == -3.0)
    v = O.bf16_to_f64(yb).reshape(m_live, n // 64, 64)
    s_mean = v.mean(axis=2)
    s_m2 = ((v - s_mean[..., None]) ** 2).sum(axis=2)
    s_scale = np.abs(v).max(axis=2)
    assert np.all(np.abs(got[:m_live, :, 0] - s_mean) <= 4e-6 * s_scale + 1e-30)
    assert np.all(np.abs(got[:m_live, :, 1] - s_m2) <= 1e-5 * s_m2 + 64e-6 * s_scale ** 2 + 1e-30)
    _check_row_moments(mv.cpu().numpy().astype(np.float64)[:m_live], yb, "merged moments")


@pytest.mark.parametrize("m_cap,m_live", [(20000, 19999), (20224, 20224)])
def test_linear_residual_long_k_many_tiles(m_cap, m_live):
    """A long-K residual linear (K = 3072, the fc2 shape) over enough rows
    that every CTA pair runs several tiles, so each warp's two staging
    buffers are reloaded within a tile and reused across tiles: sampled rows
    against the fp64 oracle, every row and slice moment against the plain
    residual entry point bit for bit, and the rows past the live count
    untouched."""
    k, n = 3072, 768
    rng = np.random.default_rng(m_cap + 31)
    x = S.f32_to_bf16_bits(rng.standard_normal((m_cap, k)))
    w = S.f32_to_bf16_bits(0.02 * rng.standard_normal((n, k)))
    b = S.f32_to_bf16_bits(0.1 * rng.standard_normal(n))
    r = _ln_rows(rng, m_cap, n)
    m_dev = i32([m_live])
    y = torch.full((m_cap, n), 7.0, dtype=torch.bfloat16, device=dev())
    y2 = torch.full((m_cap, n), 7.0, dtype=torch.bfloat16, device=dev())
    sm = torch.full((n // 64, m_cap, 2), -3.0, dtype=torch.float32, device=dev())
    st = _status()
    P.dora_linear_residual_stats(bf(x), bf(w), bf(r), y, sm, bias=bf(b), m_dev=m_dev, status=st)
    P.dora_linear(bf(x), bf(w), y2, bias=bf(b), residual=bf(r), epilogue=P.EPI_BIAS_RESIDUAL,
                  m_dev=m_dev)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert torch.equal(y, y2)
    assert torch.all(y[m_live:] == 7.0)
    assert torch.all(sm[:, m_live:] == -3.0)
    rows = np.unique(np.concatenate([rng.integers(0, m_live, 250), [0, m_live - 1]]))
    ref = O.linear(O.bf16_to_f64(x[rows]), O.bf16_to_f64(w), O.bf16_to_f64(b)) + O.bf16_to_f64(r[rows])
    assert_close(f64(y[torch.from_numpy(rows).to(dev())]), ref, f"long-K residual {m_cap}")
    v = O.bf16_to_f64(bits(y[torch.from_numpy(rows).to(dev())])).reshape(len(rows), n // 64, 64)
    got = sm.cpu().numpy().astype(np.float64).transpose(1, 0, 2)[rows]
    s_mean = v.mean(axis=2)
    s_scale = np.abs(v).max(axis=2)
    assert np.all(np.abs(got[:, :, 0] - s_mean) <= 4e-6 * s_scale + 1e-30)


# ---------------------------------------------------------------------------
# varlen attention (tcgen05)
# ---------------------------------------------------------------------------

def _run_attn(qkv_bits, cu, heads, max_seqlen, t_cap=None):
    t = qkv_bits.shape[0] if t_cap is None else t_cap
    out = torch.full((t, heads * 64), 9.0, dtype=torch.bfloat16, device=dev())
    st = _status()
    P.dora_varlen_attn(bf(qkv_bits), i32(cu), max_seqlen, heads, out, status=st)
    torch.cuda.synchronize()
    return out, int(st.item())


def _check_attn(lens, heads, seed, tail_nan=0):
    rng = np.random.default_rng(seed)
    cu = O.cu_from_counts(lens)
    t = int(cu[-1])
    qkv = S.f32_to_bf16_bits(rng.standard_normal((t + tail_nan, 3 * heads * 64)))
    if tail_nan:
        qkv[t:] = 0x7FC0            # NaN rows past the last image
    out, st = _run_attn(qkv, cu, heads, int(max(lens)))
    assert st == 0
    ref = O.varlen_attention(qkv[:t], cu, heads)
    assert_close(f64(out[:t]), ref, f"attn lens={list(lens)[:6]}")
    if tail_nan:
        assert torch.all(out[t:] == 9.0)


@pytest.mark.parametrize("name", ["cfg1", "cfg2", "cfg3", "cfg4"])
def test_attention_configs(name):
    cfg = S.get_config(name)
    keeps, _ = S.keep_schedule(cfg, 3)
    _check_attn(np.full(cfg.batch, cfg.n_tokens), cfg.heads, 1)      # dense blocks
    _check_attn(keeps[0], cfg.heads, 2)                               # after a deletion


def test_attention_cfg5_long_sequences():
    cfg = S.get_config("cfg5", batch=12)
    keeps, _ = S.keep_schedule(cfg, 4)
    _check_attn(np.full(4, 577), cfg.heads, 3)
    _check_attn(keeps[1], cfg.heads, 4)


def test_attention_edge_lengths_and_nan_tail():
    _check_attn(np.array([1]), 1, 5)
    _check_attn(np.array([1, 1, 1]), 2, 6)
    _check_attn(np.array([16, 17, 31, 32, 33, 127, 128, 129]), 3, 7)
    _check_attn(np.array([255, 256, 257, 383, 384, 385, 600]), 2, 8)
    _check_attn(np.array([197, 5, 130]), 12, 9, tail_nan=70)


def test_attention_running_maximum_moves_between_key_chunks():
    """Keys of later 128-key chunks scaled up (image 0: x4 then x8; image 2:
    x6) so that the row maximum of a later chunk lies far above the first
    chunk's and the online softmax has to move its reference; image 1 is the
    reverse (first chunk dominant, later probabilities underflow)."""
    lens = np.array([300, 200, 140])
    heads = 2
    rng = np.random.default_rng(13)
    cu = O.cu_from_counts(lens)
    t = int(cu[-1])
    x = rng.standard_normal((t, 3 * heads * 64))
    kcols = slice(heads * 64, 2 * heads * 64)
    x[cu[0] + 128:cu[0] + 256, kcols] *= 4.0
    x[cu[0] + 256:cu[1], kcols] *= 8.0
    x[cu[1]:cu[1] + 128, kcols] *= 6.0
    x[cu[2] + 128:cu[3], kcols] *= 6.0
    qkv = S.f32_to_bf16_bits(x)
    out, st = _run_attn(qkv, cu, heads, int(max(lens)))
    assert st == 0
    assert_close(f64(out), O.varlen_attention(qkv, cu, heads), "attn rescale")


def test_attention_empty_images_and_long_image_flag():
    lens = np.array([0, 20, 0, 33])
    _check_attn(lens, 2, 10)
    cu = O.cu_from_counts(np.array([10, 300]))
    qkv = S.f32_to_bf16_bits(np.random.default_rng(11).standard_normal((310, 3 * 64)))
    _, st = _run_attn(qkv, cu, 1, 128)
    assert st == 6


@pytest.mark.parametrize("mix", ["many_images", "skewed", "few_image_heads"])
def test_attention_range_split_over_many_images(mix):
    """The split of image-heads over the persistent CTAs (each lane of the
    range search reading a block of image bounds): batches above 256 images
    (several rounds of loads per lane), skewed costs with many empty and
    one-token images beside a few of 300 tokens (the kernel for images past
    256 tokens), and fewer image-heads than SMs.  Every row of every
    image is compared with the oracle, so an image-head given to no CTA (its
    rows keep the fill value) or to two fails."""
    rng = np.random.default_rng({"many_images": 21, "skewed": 22, "few_image_heads": 23}[mix])
    if mix == "many_images":
        lens = rng.integers(0, 201, 1100)
        lens[rng.random(1100) < 0.2] = 0
        heads = 2
    elif mix == "skewed":
        lens = rng.integers(0, 4, 700)
        lens[rng.choice(700, 9, replace=False)] = 300    # the per-key-half kernel
        heads = 3
    else:
        lens = rng.integers(0, 257, 40)
        heads = 1
    _check_attn(lens, heads, 24)


def test_attention_matches_dense_when_unpruned():
    """k = 0: packed attention equals dense batched attention (torch SDPA on
    the same bf16 values, fp64) on the GPU path too."""
    b, n, h = 4, 197, 3
    rng = np.random.default_rng(12)
    qkv = S.f32_to_bf16_bits(rng.standard_normal((b * n, 3 * h * 64)))
    out, _ = _run_attn(qkv, np.arange(b + 1) * n, h, n)
    a = torch.from_numpy(O.bf16_to_f64(qkv).reshape(b, n, 3, h, 64))
    q, k, v = (a[:, :, j].permute(0, 2, 1, 3) for j in range(3))
    dense = torch.nn.functional.scaled_dot_product_attention(q, k, v).permute(0, 2, 1, 3)
    assert_close(f64(out), dense.reshape(b * n, h * 64).numpy(), "dense")


# ---------------------------------------------------------------------------
# the pruned block and the forward
# ---------------------------------------------------------------------------

def _device_weights(cfg, wb):
    return P.BlockWeights({k: bf(v) for k, v in wb.items()}, cfg.dim, cfg.heads, cfg.mlp_dim,
                          cfg.ln_eps)


def _run_block(cfg, x_bits, cu, ids, w, scores=None, keeps=None, t_cap=None):
    t_cap = t_cap or x_bits.shape[0]
    ws = P.alloc_workspace(t_cap, cfg.batch, w)
    x_out = torch.zeros(t_cap, cfg.dim, dtype=torch.bfloat16, device=dev())
    cu_out = torch.zeros(len(cu), dtype=torch.int32, device=dev())
    ids_out = torch.full((t_cap,), SENT, dtype=torch.int32, device=dev())
    kept = torch.full((t_cap,), SENT, dtype=torch.int32, device=dev())
    xin = torch.zeros(t_cap, cfg.dim, dtype=torch.bfloat16, device=dev())
    xin[:x_bits.shape[0]] = bf(x_bits)
    P.dora_pruned_block(xin, i32(cu), w, int(np.diff(cu).max()), x_out, ws, ids_in=i32(ids),
                        scores=None if scores is None else f32(scores),
                        keep_counts=None if keeps is None else i32(keeps), cu_out=cu_out,
                        ids_out=ids_out, kept_idx=kept)
    torch.cuda.synchronize()
    st = P.dora_read_status(P.dora_workspace_status(ws))
    return dict(x_out=x_out, cu_out=cu_out.cpu().numpy(), ids_out=ids_out.cpu().numpy(),
                kept=kept.cpu().numpy(), status=st)


def _check_block_images(cfg, x_bits, cu, ids, wb, scores, keeps, r, images):
    """Oracle on a sub-batch of images (images are independent)."""
    rows, lcu = sub_batch(cu, images)
    wf = O.decode_weights(wb)
    sub_scores = None if scores is None else scores[rows]
    sub_keeps = None if keeps is None else np.asarray(keeps)[list(images)]
    ref = O.pruned_block(O.bf16_to_f64(x_bits[rows]), lcu, ids[rows], wf, cfg.heads, cfg.ln_eps,
                         sub_scores, sub_keeps)
    cu_out = r["cu_out"] if scores is not None else cu
    got_rows = np.concatenate([np.arange(cu_out[i], cu_out[i + 1]) for i in images])
    assert_close(f64(r["x_out"])[got_rows], ref["x_out"], f"block {cfg.name} imgs {images}")


@pytest.mark.parametrize("name", ["cfg1", "cfg2"])
def test_block_full_oracle(name):
    cfg = S.get_config(name)
    cu, ids = S.initial_layout(cfg)
    x = S.activations_bf16(cfg, 20)
    wb = S.block_weights(cfg, 0, 20, random_affine=True)
    keeps, _ = S.keep_schedule(cfg, 20)
    scores = O.gather_scores(S.score_table(cfg, 0, 20), cu, ids)
    w = _device_weights(cfg, wb)
    r = _run_block(cfg, x, cu, ids, w, scores, keeps[0])
    assert r["status"] == 0
    ref = O.pruned_block(O.bf16_to_f64(x), cu, ids, O.decode_weights(wb), cfg.heads, cfg.ln_eps,
                         scores, keeps[0])
    t_out = int(ref["cu_out"][-1])
    assert np.array_equal(r["cu_out"], ref["cu_out"])
    assert np.array_equal(r["kept"][:t_out], ref["kept_idx"])
    assert np.array_equal(r["ids_out"][:t_out], ref["ids_out"])
    assert_close(f64(r["x_out"][:t_out]), ref["x_out"], f"block {name}")
    # no deletion: the output boundaries are the input's and every row is computed
    r0 = _run_block(cfg, x, cu, ids, w)
    ref0 = O.pruned_block(O.bf16_to_f64(x), cu, ids, O.decode_weights(wb), cfg.heads, cfg.ln_eps)
    assert_close(f64(r0["x_out"][:int(cu[-1])]), ref0["x_out"], f"dense block {name}")
    # pruned rows equal the dense block's rows at the kept positions (Eq. 1)
    assert np.array_equal(bits(r["x_out"][:t_out]), bits(r0["x_out"])[ref["kept_idx"]])


@pytest.mark.parametrize("name", ["cfg1", "cfg3"])
def test_block_tiny_batch(name):
    """Fewer rows than one 256-row tile pair, before and after the deletion
    (the linears' row walks, forward and from the last row block, meet a
    single partial row block), with a one-token image; the one-CTA-pair path
    (D = 768) and the one-CTA path (D = 192)."""
    cfg = S.get_config(name, batch=3)
    lens = np.array([5, 1, 40])
    cu = O.cu_from_counts(lens)
    ids = np.concatenate([np.arange(n) for n in lens]).astype(np.int32)
    rng = np.random.default_rng(61)
    x = S.f32_to_bf16_bits(rng.standard_normal((int(cu[-1]), cfg.dim)))
    wb = S.block_weights(cfg, 0, 61, random_affine=True)
    w = _device_weights(cfg, wb)
    scores = rng.random(int(cu[-1])).astype(np.float32)
    keeps = np.array([2, 1, 7], dtype=np.int32)
    wf = O.decode_weights(wb)
    for sc, kp in ((scores, keeps), (None, None)):
        r = _run_block(cfg, x, cu, ids, w, sc, kp)
        assert r["status"] == 0
        ref = O.pruned_block(O.bf16_to_f64(x), cu, ids, wf, cfg.heads, cfg.ln_eps, sc, kp)
        t_out = int(ref["cu_out"][-1]) if sc is not None else int(cu[-1])
        if sc is not None:
            assert np.array_equal(r["cu_out"], ref["cu_out"])
            assert np.array_equal(r["kept"][:t_out], ref["kept_idx"])
        assert_close(f64(r["x_out"][:t_out]), ref["x_out"], f"tiny block {name}")


def test_block_prefolded_weights_give_the_same_bits():
    """Weights folded once (dora_fold_block_weights) and weights folded inside
    every call produce the same block output bit for bit."""
    cfg = S.get_config("cfg1")
    cu, ids = S.initial_layout(cfg)
    x = S.activations_bf16(cfg, 23)
    wb = S.block_weights(cfg, 1, 23, random_affine=True)
    keeps, _ = S.keep_schedule(cfg, 23)
    scores = O.gather_scores(S.score_table(cfg, 1, 23), cu, ids)
    w = _device_weights(cfg, wb)
    wf = _device_weights(cfg, wb).fold()
    assert P.dora_workspace_size(100, 1, wf) < P.dora_workspace_size(100, 1, w)
    for sc, kp in ((scores, keeps[0]), (None, None)):
        a = _run_block(cfg, x, cu, ids, w, sc, kp)
        b = _run_block(cfg, x, cu, ids, wf, sc, kp)
        assert a["status"] == 0 and b["status"] == 0
        assert torch.equal(a["x_out"], b["x_out"])
        assert np.array_equal(a["cu_out"], b["cu_out"])


@pytest.mark.parametrize("name,scored", [("cfg1", False), ("cfg1", True), ("cfg2", True)])
def test_block_equals_its_public_entry_points(name, scored):
    """The block gives the same bits as its steps run one by one through the
    public entries: row moments, QKV linear with LayerNorm folded in, varlen
    attention, projection + residual with slice moments, their merge,
    [selection, compaction carrying the moments,] fc1 with LayerNorm' folded
    in + GELU, fc2 + residual with slice moments, their merge.  The block
    runs twice on one workspace and gives the same bits both times."""
    cfg = S.get_config(name)
    cu, ids = S.initial_layout(cfg)
    t = int(cu[-1])
    d, m, h = cfg.dim, cfg.mlp_dim, cfg.heads
    x = S.activations_bf16(cfg, 26)
    wb = S.block_weights(cfg, 2, 26, random_affine=True)
    W = {k: bf(v) for k, v in wb.items()}
    wf = _device_weights(cfg, wb).fold()
    ws = P.alloc_workspace(t, cfg.batch, wf)
    keeps, _ = S.keep_schedule(cfg, 26)
    scores = O.gather_scores(S.score_table(cfg, 0, 26), cu, ids) if scored else None
    f32t = lambda *shape, v=0.0: torch.full(shape, v, dtype=torch.float32, device=dev())
    bf16t = lambda *shape: torch.zeros(*shape, dtype=torch.bfloat16, device=dev())
    xin = bf(x)
    outs = []
    for _ in range(2):
        x_out, mo = bf16t(t, d), f32t(t, 2, v=-3.0)
        cu_out = torch.zeros(len(cu), dtype=torch.int32, device=dev())
        ids_out = torch.zeros(t, dtype=torch.int32, device=dev())
        P.dora_pruned_block(xin, i32(cu), wf, cfg.n_tokens, x_out, ws, ids_in=i32(ids),
                            scores=None if scores is None else f32(scores),
                            keep_counts=i32(keeps[0]) if scored else None, cu_out=cu_out,
                            ids_out=ids_out, x_out_moments=mo)
        torch.cuda.synchronize()
        assert P.dora_read_status(P.dora_workspace_status(ws)) == 0
        outs.append((x_out, mo, cu_out))
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])

    def fold(wname, g, b, bias, n):
        w_, c_, d_ = bf16t(n, d), f32t(n), f32t(n)
        P.dora_fold_ln_linear(W[wname], W[g], W[b], w_, c_, d_, bias=W[bias])
        return w_, c_, d_
    st = _status()
    rows = i32([t])
    mv = f32t(t, 2)
    P.dora_row_stats(xin, mv, rows_dev=rows)
    qkv = bf16t(t, 3 * d)
    P.dora_linear_ln(xin, mv, cfg.ln_eps, *fold("w_qkv", "ln1_w", "ln1_b", "b_qkv", 3 * d), qkv,
                     m_dev=rows, status=st)
    o = bf16t(t, d)
    P.dora_varlen_attn(qkv, i32(cu), cfg.n_tokens, h, o, status=st)
    hattn, sm = bf16t(t, d), f32t(d // 64, t, 2)
    P.dora_linear_residual_stats(o, W["w_proj"], xin, hattn, sm, bias=W["b_proj"], m_dev=rows,
                                 status=st)
    P.dora_merge_moments(sm, mv, rows_dev=rows)
    hk, mv2, rows2 = hattn, mv, rows
    if scored:
        kept = torch.zeros(t, dtype=torch.int32, device=dev())
        cu2 = torch.zeros(len(cu), dtype=torch.int32, device=dev())
        P.dora_select_keep(f32(scores), i32(cu), i32(keeps[0]), cfg.n_tokens, kept, cu2, status=st)
        hk, mv2 = bf16t(t, d), f32t(t, 2)
        P.dora_compact_stats(hattn, kept, cu2, hk, mv, mv2, ids_in=i32(ids),
                             ids_out=torch.zeros(t, dtype=torch.int32, device=dev()), status=st)
        rows2 = cu2[-1:].contiguous()
    u = bf16t(t, m)
    P.dora_linear_ln(hk, mv2, cfg.ln_eps, *fold("w_fc1", "ln2_w", "ln2_b", "b_fc1", m), u,
                     gelu=True, m_dev=rows2, status=st)
    y, sm2, mo = bf16t(t, d), f32t(d // 64, t, 2), f32t(t, 2, v=-3.0)
    P.dora_linear_residual_stats(u, W["w_fc2"], hk, y, sm2, bias=W["b_fc2"], m_dev=rows2,
                                 status=st)
    P.dora_merge_moments(sm2, mo, rows_dev=rows2)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    t_out = int(rows2.item())
    assert torch.equal(outs[0][0][:t_out], y[:t_out])
    assert torch.equal(outs[0][1], mo)


def test_block_chained_row_moments():
    """Two blocks chained through x_out_moments -> x_in_moments: the moments
    each block hands on match the fp64 row moments of its output, and the
    second block's output matches the oracle on its input (and the unchained
    run within rounding)."""
    cfg = S.get_config("cfg1")
    cu, ids = S.initial_layout(cfg)
    t_cap = int(cu[-1])
    x = S.activations_bf16(cfg, 24)
    keeps, _ = S.keep_schedule(cfg, 24)
    wb = [S.block_weights(cfg, l, 24, random_affine=True) for l in range(2)]
    ws_ = [_device_weights(cfg, w).fold() for w in wb]
    ws = P.alloc_workspace(t_cap, cfg.batch, ws_[0])
    scores = O.gather_scores(S.score_table(cfg, 1, 24), cu, ids)
    x0 = bf(x)
    mids = [torch.zeros(t_cap, cfg.dim, dtype=torch.bfloat16, device=dev()) for _ in range(2)]
    outs = [torch.zeros(t_cap, cfg.dim, dtype=torch.bfloat16, device=dev()) for _ in range(2)]
    m1 = torch.full((t_cap, 2), -3.0, dtype=torch.float32, device=dev())
    m2 = torch.full((t_cap, 2), -3.0, dtype=torch.float32, device=dev())
    cu_out = torch.zeros(len(cu), dtype=torch.int32, device=dev())
    ids_out = torch.zeros(t_cap, dtype=torch.int32, device=dev())
    for k, chained in enumerate((False, True)):
        P.dora_pruned_block(x0, i32(cu), ws_[0], cfg.n_tokens, mids[k], ws, ids_in=i32(ids),
                            x_out_moments=m1 if chained else None)
        P.dora_pruned_block(mids[k], i32(cu), ws_[1], cfg.n_tokens, outs[k], ws, ids_in=i32(ids),
                            scores=f32(scores), keep_counts=i32(keeps[0]), cu_out=cu_out,
                            ids_out=ids_out, x_in_moments=m1 if chained else None,
                            x_out_moments=m2 if chained else None)
        torch.cuda.synchronize()
        assert P.dora_read_status(P.dora_workspace_status(ws)) == 0
    t_out = int(cu_out.cpu().numpy()[-1])
    _check_row_moments(m1.cpu().numpy().astype(np.float64)[:t_cap], bits(mids[1]), "block 0 out")
    _check_row_moments(m2.cpu().numpy().astype(np.float64)[:t_out], bits(outs[1][:t_out]),
                       "block 1 out")
    assert np.all(m2.cpu().numpy()[t_out:] == -3.0)
    ref = O.pruned_block(O.bf16_to_f64(bits(mids[1])), cu, ids, O.decode_weights(wb[1]),
                         cfg.heads, cfg.ln_eps, scores, keeps[0])
    assert_close(f64(outs[1][:t_out]), ref["x_out"], "chained block")
    assert_close(f64(outs[1][:t_out]), f64(outs[0][:t_out]), "chained vs unchained")


@pytest.mark.parametrize("name", ["cfg3", "cfg4", "cfg5", "cfg6"])
def test_block_full_size_sampled_images(name):
    cfg = S.get_config(name)
    cu, ids = S.initial_layout(cfg)
    x = S.activations_bf16(cfg, 21)
    blk = cfg.prune_blocks[0]
    wb = S.block_weights(cfg, blk, 21, random_affine=True)
    keeps, _ = S.keep_schedule(cfg, 21)
    scores = O.gather_scores(S.score_table(cfg, blk, 21), cu, ids)
    r = _run_block(cfg, x, cu, ids, _device_weights(cfg, wb), scores, keeps[0])
    assert r["status"] == 0
    rk, rcu, _ = O.select_keep(scores, cu, keeps[0])
    assert np.array_equal(r["cu_out"], rcu)
    assert np.array_equal(r["kept"][:int(rcu[-1])], rk)
    assert np.array_equal(r["ids_out"][:int(rcu[-1])], ids[rk])
    b = cfg.batch
    _check_block_images(cfg, x, cu, ids, wb, scores, keeps[0], r, [0, b // 2, b - 1])


def test_forward_deit_b_shape_per_block():
    """Twelve DeiT-B-shape blocks pruned at 3/6/9 through the C ABI.  The token
    trajectory (cu, ids, kept) must equal the oracle's bit for bit end to end;
    each block's output is checked against the oracle fed the same block input
    on sampled images."""
    cfg = S.get_config("cfg3", batch=16)
    cu, ids = S.initial_layout(cfg)
    t_cap = int(cu[-1])
    x = S.activations_bf16(cfg, 22)
    keeps, _ = S.keep_schedule(cfg, 22)
    sched = dict(zip(cfg.prune_blocks, keeps))
    cur = torch.zeros(t_cap, cfg.dim, dtype=torch.bfloat16, device=dev())
    cur[:] = bf(x)
    cu_d, ids_d = i32(cu), i32(ids)
    host_cu, host_ids = cu.copy(), ids.copy()
    for l in range(cfg.depth):
        wb = S.block_weights(cfg, l, 22)
        w = _device_weights(cfg, wb)
        ws = P.alloc_workspace(t_cap, cfg.batch, w)
        nxt = torch.zeros_like(cur)
        x_in_bits = bits(cur)
        kw = {}
        if l in sched:
            table = S.score_table(cfg, l, 22)
            sc = torch.zeros(t_cap, dtype=torch.float32, device=dev())
            P.dora_gather_scores(f32(table), ids_d, cu_d, sc)
            cu_o = torch.zeros_like(cu_d)
            ids_o = torch.zeros_like(ids_d)
            kept = torch.zeros_like(ids_d)
            kw = dict(scores=sc, keep_counts=i32(sched[l]), cu_out=cu_o, ids_out=ids_o,
                      kept_idx=kept)
        P.dora_pruned_block(cur, cu_d, w, cfg.n_tokens, nxt, ws, ids_in=ids_d, **kw)
        torch.cuda.synchronize()
        assert P.dora_read_status(P.dora_workspace_status(ws)) == 0
        scores = None
        if l in sched:
            scores = O.gather_scores(table, host_cu, host_ids)
            assert np.array_equal(sc.cpu().numpy()[:int(host_cu[-1])], scores)
            rk, rcu, _ = O.select_keep(scores, host_cu, sched[l])
            assert np.array_equal(cu_o.cpu().numpy(), rcu)
            assert np.array_equal(kept.cpu().numpy()[:int(rcu[-1])], rk)
            assert np.array_equal(ids_o.cpu().numpy()[:int(rcu[-1])], host_ids[rk])
        r = dict(x_out=nxt, cu_out=(cu_o.cpu().numpy() if l in sched else host_cu))
        imgs = [l % cfg.batch]
        _check_block_images(cfg, x_in_bits, host_cu, host_ids, wb, scores,
                            sched.get(l), r, imgs)
        if l in sched:
            host_cu, host_ids = rcu, host_ids[rk]
            cu_d, ids_d = cu_o, ids_o
        cur = nxt
    assert np.array_equal(np.diff(host_cu), keeps[-1])


# ---------------------------------------------------------------------------
# the deployment actor (Sec. 3.2 "The actor"; Appendix A.1-A.3)
# ---------------------------------------------------------------------------

def _actor_case(cfg, seed, gate_bias=0.0, lens=None):
    """Packed qkv rows with the given image lengths, per-image history, and the
    actor's weights (host bits and prepared device copy)."""
    rng = np.random.default_rng(seed)
    if lens is None:
        lens = np.full(cfg.batch, cfg.n_tokens)
    cu = O.cu_from_counts(lens)
    t = int(cu[-1])
    qkv = S.f32_to_bf16_bits(rng.standard_normal((t, 3 * cfg.dim)))
    rho = rng.uniform(0, 0.5, len(lens)).astype(np.float32)
    e_prev = rng.integers(0, 3, len(lens)).astype(np.int32)
    wa = S.actor_weights(cfg.dim, cfg.depth, cfg.n_vis0, seed, gate_bias=gate_bias)
    aw = P.ActorWeights({k_: bf(v) for k_, v in wa.items()}, cfg.dim, cfg.depth, cfg.n_vis0)
    return cu, qkv, rho, e_prev, wa, aw.prepare()


def _run_actor(cfg, cu, qkv, rho, e_prev, aw, block, max_seqlen):
    b, t = len(cu) - 1, int(cu[-1])
    out = {n: torch.full((b,), -7, dtype=torch.int32, device=dev())
           for n in ("gate", "budget", "k", "keep", "e_next")}
    p = torch.zeros(b, dtype=torch.float32, device=dev())
    rho_next = torch.zeros(b, dtype=torch.float32, device=dev())
    scores = torch.full((t,), 5.0, dtype=torch.float32, device=dev())
    z = torch.zeros(t, 128, dtype=torch.bfloat16, device=dev())
    ws = P.alloc_actor_workspace(t, b, aw)
    P.dora_actor(bf(qkv), i32(cu), aw, block, max_seqlen, f32(rho), i32(e_prev), out["gate"],
                 out["budget"], out["k"], out["keep"], scores, ws, p_gate=p, rho_next=rho_next,
                 interventions_next=out["e_next"], z_out=z)
    torch.cuda.synchronize()
    assert P.dora_read_status(P.dora_workspace_status(ws)) == 0
    r = {n: v.cpu().numpy() for n, v in out.items()}
    r.update(p=p.cpu().numpy(), rho_next=rho_next.cpu().numpy(), scores=scores.cpu().numpy(),
             z=f64(z))
    return r


# The encoder's residual stream is rounded to bf16 three times (X, Z1, Z),
# each by at most 2^-9 of the value, before the GEMM and attention errors the
# block tolerance already allows for: 3e-2 absolute or 2e-2 relative.  (At the
# block's 2e-2 / 1e-2, 4 of 47,872 Z elements of the cfg1 case fall outside,
# by at most 2.7e-2 absolute: about 1.6 bf16 ulps at |Z| near 2.3.)
ACTOR_ATOL, ACTOR_RTOL = 3e-2, 2e-2


def _check_actor(cfg, cu, qkv, rho, e_prev, wa, got, block, images):
    """Oracle on a sub-batch of images (the actor treats images independently)."""
    wf = O.decode_weights(wa)
    rows, lcu = sub_batch(cu, images)
    ref = O.actor_block(qkv[rows][:, cfg.dim:2 * cfg.dim], lcu, block, cfg.n_vis0, cfg.depth,
                        rho[images], e_prev[images], wf)
    n_vis = np.diff(cu)[images] - 1
    # encoder output within the block tolerance; gate probability in fp32
    assert_close(got["z"][rows], ref["z"], "actor Z", atol=ACTOR_ATOL, rtol=ACTOR_RTOL)
    assert np.all(np.abs(got["p"][images] - ref["p"]) <= 1e-4)
    # decisions agree wherever the oracle's margin exceeds the arithmetic's error,
    # and the filter leaves out only near-ties: all but 5% (at least one) of
    # the gate decisions are compared, and all but 15% (at least one) of the
    # budgets equal the oracle's own argmax (the rest are within 0.05 of its
    # best logit)
    clear = np.abs(ref["p"] - 0.5) > 1e-4
    assert np.array_equal((got["p"][images] >= 0.5)[clear], (ref["p"] >= 0.5)[clear])
    skipped = int((~clear).sum())
    assert skipped <= max(1, int(0.05 * clear.size)), f"gate decisions skipped: {skipped}"
    grid = O.budget_grid(cfg.n_vis0)
    exact = total = 0
    for j, i in enumerate(images):
        bud = int(got["budget"][i])
        feas = grid <= n_vis[j] - 4
        if not feas.any():
            assert bud == 0
            continue
        assert bud in grid[feas]
        best = ref["logits"][j][feas].max()
        assert ref["logits"][j][list(grid).index(bud)] >= best - 0.05, (i, bud, ref["budget"][j])
        total += 1
        exact += int(bud == int(ref["budget"][j]))
    assert exact >= total - max(1, int(0.15 * total)), (
        f"budgets equal to the oracle's: {exact}/{total}")
    # the integer bookkeeping is exact given the GPU's own decisions
    g, bud = got["gate"][images], got["budget"][images]
    assert np.array_equal(g, ((got["p"][images] >= 0.5) & (bud > 0)).astype(np.int32))
    assert np.array_equal(got["k"][images], bud * g)
    assert np.array_equal(got["keep"][images], n_vis + 1 - bud * g)
    assert np.array_equal(got["e_next"][images], e_prev[images] + g)
    assert np.allclose(got["rho_next"][images], bud * g / np.maximum(n_vis, 1), rtol=1e-6)
    # selector scores: the oracle's selector on the oracle's Z with the GPU's budget
    for j, i in enumerate(images):
        lo, hi = int(lcu[j]), int(lcu[j + 1])
        assert got["scores"][cu[i]] == 0.0
        if n_vis[j] == 0:
            continue
        ref_s = O.actor_selector(ref["z"][lo + 1:hi], int(got["budget"][i]), int(n_vis[j]), wf)
        assert_close(got["scores"][cu[i] + 1:cu[i + 1]], ref_s, f"actor scores image {i}",
                     atol=ACTOR_ATOL, rtol=ACTOR_RTOL)


@pytest.mark.parametrize("name,block,seed", [("cfg1", 0, 31), ("cfg2", 0, 32), ("cfg3", 5, 33)])
def test_actor_matches_oracle(name, block, seed):
    cfg = S.get_config(name)
    lens = None
    if name == "cfg3":
        keeps, _ = S.keep_schedule(cfg, seed)
        lens = keeps[1]                              # token counts after two deletions
    cu, qkv, rho, e_prev, wa, aw = _actor_case(cfg, seed, lens=lens)
    got = _run_actor(cfg, cu, qkv, rho, e_prev, aw, block, int(np.diff(cu).max()))
    b = len(cu) - 1
    images = list(range(b)) if b <= 64 else [0, 1, 77, 128, b - 2, b - 1]
    _check_actor(cfg, cu, qkv, rho, e_prev, wa, got, block, images)


def test_actor_edges_short_images_and_gate_bias():
    """Images too short for any budget (N_l < 6) keep everything; an empty
    image is skipped; a strongly positive or negative gate bias opens or
    closes every feasible gate."""
    cfg = S.get_config("cfg1")
    lens = np.array([197, 6, 7, 1, 10, 0, 150, 3])
    for gb, want in ((8.0, 1), (-8.0, 0)):
        cu, qkv, rho, e_prev, wa, aw = _actor_case(cfg, 41, gate_bias=gb, lens=lens)
        got = _run_actor(cfg, cu, qkv, rho, e_prev, aw, 0, int(lens.max()))
        n_vis = lens - 1
        feasible = n_vis >= 6
        assert np.array_equal(got["gate"], (want * feasible).astype(np.int32))
        assert np.array_equal(got["keep"], lens - got["k"])
        assert np.all(got["k"][~feasible] == 0)
        _check_actor(cfg, cu, qkv, rho, e_prev, wa, got, 0, [0, 1, 2, 3, 4, 6, 7])


@pytest.mark.parametrize("given_counts", [True, False])
def test_block_with_actor_equals_actor_then_block(given_counts):
    """dora_pruned_block_actor gives the same bits as running dora_actor on the
    block's QKV output (computed through the public entries) and then
    dora_pruned_block with the actor's scores and the given (or the actor's)
    keep counts."""
    cfg = S.get_config("cfg2")
    cu, ids = S.initial_layout(cfg)
    t = int(cu[-1])
    x = S.activations_bf16(cfg, 27)
    wb = S.block_weights(cfg, 0, 27, random_affine=True)
    wf = _device_weights(cfg, wb).fold()
    wa = S.actor_weights(cfg.dim, cfg.depth, cfg.n_vis0, 27, gate_bias=1.0)
    aw = P.ActorWeights({k_: bf(v) for k_, v in wa.items()}, cfg.dim, cfg.depth, cfg.n_vis0).prepare()
    keeps, _ = S.keep_schedule(cfg, 27)
    b = cfg.batch
    i32z = lambda n: torch.zeros(n, dtype=torch.int32, device=dev())
    rho = torch.zeros(b, dtype=torch.float32, device=dev())
    e0 = i32z(b)
    ws = P.alloc_workspace(t, b, wf)
    aws = P.alloc_actor_workspace(t, b, aw)
    # the block with the actor inside
    out = {n: i32z(b) for n in ("gate", "budget", "k", "keep")}
    scores = torch.zeros(t, dtype=torch.float32, device=dev())
    x_out = torch.zeros(t, cfg.dim, dtype=torch.bfloat16, device=dev())
    cu_out, ids_out = i32z(b + 1), i32z(t)
    P.dora_pruned_block_actor(bf(x), i32(cu), wf, cfg.n_tokens, x_out, ws, aw, 0, rho, e0,
                              out["gate"], out["budget"], out["k"], out["keep"], scores, aws,
                              i32(ids), cu_out, ids_out,
                              keep_counts=i32(keeps[0]) if given_counts else None)
    torch.cuda.synchronize()
    assert P.dora_read_status(P.dora_workspace_status(ws)) == 0
    assert P.dora_read_status(P.dora_workspace_status(aws)) == 0
    # the same through the public entries
    W = {k_: bf(v) for k_, v in wb.items()}
    mv = torch.zeros(t, 2, dtype=torch.float32, device=dev())
    P.dora_row_stats(bf(x), mv)
    wq = torch.zeros(3 * cfg.dim, cfg.dim, dtype=torch.bfloat16, device=dev())
    cq = torch.zeros(3 * cfg.dim, dtype=torch.float32, device=dev())
    dq = torch.zeros(3 * cfg.dim, dtype=torch.float32, device=dev())
    P.dora_fold_ln_linear(W["w_qkv"], W["ln1_w"], W["ln1_b"], wq, cq, dq, bias=W["b_qkv"])
    qkv = torch.zeros(t, 3 * cfg.dim, dtype=torch.bfloat16, device=dev())
    P.dora_linear_ln(bf(x), mv, cfg.ln_eps, wq, cq, dq, qkv)
    ref = {n: i32z(b) for n in ("gate", "budget", "k", "keep")}
    scores2 = torch.zeros(t, dtype=torch.float32, device=dev())
    P.dora_actor(qkv, i32(cu), aw, 0, cfg.n_tokens, rho, e0, ref["gate"], ref["budget"], ref["k"],
                 ref["keep"], scores2, P.alloc_actor_workspace(t, b, aw))
    for n in ref:
        assert torch.equal(out[n], ref[n]), n
    assert torch.equal(scores, scores2)
    x_out2 = torch.zeros(t, cfg.dim, dtype=torch.bfloat16, device=dev())
    cu2, ids2 = i32z(b + 1), i32z(t)
    P.dora_pruned_block(bf(x), i32(cu), wf, cfg.n_tokens, x_out2, P.alloc_workspace(t, b, wf),
                        ids_in=i32(ids), scores=scores2,
                        keep_counts=i32(keeps[0]) if given_counts else ref["keep"],
                        cu_out=cu2, ids_out=ids2)
    torch.cuda.synchronize()
    assert torch.equal(cu_out, cu2) and torch.equal(ids_out, ids2)
    t_out = int(cu2[-1].item())
    assert torch.equal(x_out[:t_out], x_out2[:t_out])
    if not given_counts:
        assert torch.equal(torch.diff(cu_out), out["keep"])


# ---------------------------------------------------------------------------
# patch embedding and classifier head (the ends of the forward, App. E.4)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("b,c,h,w,patch,d", [(8, 3, 224, 224, 16, 192), (3, 3, 64, 96, 16, 768),
                                             (2, 4, 32, 32, 8, 128),
                                             (2, 3, 224, 224, 14, 768),    # DINOv2: K 588 -> 640
                                             (3, 1, 42, 28, 7, 128),       # K 49 -> 64
                                             (1, 4, 24, 40, 4, 64),        # even path, K 64
                                             (2, 3, 36, 48, 6, 64)])       # even, K 108 -> 128
def test_patch_embed_matches_oracle(b, c, h, w, patch, d):
    rng = np.random.default_rng(b * 100 + d)
    g = (h // patch) * (w // patch)
    k = c * patch * patch
    im = S.f32_to_bf16_bits(rng.standard_normal((b, c, h, w)))
    wpe = S.f32_to_bf16_bits(rng.standard_normal((d, k)) / np.sqrt(k))
    bpe = S.f32_to_bf16_bits(0.02 * rng.standard_normal(d))
    cls = S.f32_to_bf16_bits(0.02 * rng.standard_normal(d))
    pos = S.f32_to_bf16_bits(0.02 * rng.standard_normal((g + 1, d)))
    x0 = torch.full((b * (g + 1), d), 9.0, dtype=torch.bfloat16, device=dev())
    ws = P.dora_patch_embed(bf(im), bf(wpe), bf(bpe), bf(cls), bf(pos), patch, x0)
    torch.cuda.synchronize()
    assert P.dora_read_status(P.dora_workspace_status(ws)) == 0
    ref = O.patch_embed(im, O.bf16_to_f64(wpe), O.bf16_to_f64(bpe), O.bf16_to_f64(cls),
                        O.bf16_to_f64(pos), patch)
    assert_close(f64(x0), ref, f"patch embed {b}x{c}x{h}x{w}/{patch} d={d}")


@pytest.mark.parametrize("name", ["cfg1", "cfg3"])
def test_classifier_head_matches_oracle(name):
    cfg = S.get_config(name)
    keeps, _ = S.keep_schedule(cfg, 13)
    lens = keeps[-1]
    cu = O.cu_from_counts(lens)
    t = int(cu[-1])
    rng = np.random.default_rng(13)
    x = S.f32_to_bf16_bits(rng.uniform(-3, 3, (t, 1)) + rng.standard_normal((t, cfg.dim)))
    wh = S.embed_head_weights(cfg, 13)
    classes = 1024                                   # 1000 padded with zero rows
    w_head = np.zeros((classes, cfg.dim), np.uint16)
    w_head[:1000] = wh["w_head"]
    b_head = np.zeros(classes, np.uint16)
    b_head[:1000] = wh["b_head"]
    logits = torch.full((cfg.batch, classes), 9.0, dtype=torch.bfloat16, device=dev())
    ws = P.dora_classifier_head(bf(x), i32(cu), bf(wh["norm_w"]), bf(wh["norm_b"]), 1e-6,
                                bf(w_head), bf(b_head), logits)
    torch.cuda.synchronize()
    assert P.dora_read_status(P.dora_workspace_status(ws)) == 0
    ref = O.classifier_head(O.bf16_to_f64(x), cu, O.bf16_to_f64(wh["norm_w"]),
                            O.bf16_to_f64(wh["norm_b"]), 1e-6, O.bf16_to_f64(w_head),
                            O.bf16_to_f64(b_head))
    assert_close(f64(logits), ref, f"classifier {name}")
    assert torch.all(logits[:, 1000:] == 0)


# ---------------------------------------------------------------------------
# DINOv2 backbone: LayerScale fold, LayerScale blocks, LC1 readout
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("n,k,bias,inplace", [(768, 768, True, False), (768, 3072, True, True),
                                              (96, 40, False, False)])
def test_fold_layerscale_bit_exact(n, k, bias, inplace):
    """A bf16 x bf16 product is exact in fp32, so the fold is the
    round-to-nearest-even of gamma_i * w_ij: checked bit for bit."""
    rng = np.random.default_rng(n + k)
    w = S.f32_to_bf16_bits(rng.standard_normal((n, k)) * 0.05)
    b = S.f32_to_bf16_bits(rng.standard_normal(n) * 0.02)
    g = S.f32_to_bf16_bits(rng.uniform(0.05, 0.5, n) * np.where(rng.random(n) < 0.1, -1, 1))
    wt, bt, gt = bf(w), bf(b) if bias else None, bf(g)
    wo, bo = P.dora_fold_layerscale(wt, bt, gt, w_out=wt if inplace else None,
                                    b_out=bt if inplace and bias else None)
    torch.cuda.synchronize()
    gf = O.bf16_to_f64(g).astype(np.float32)
    want_w = S.f32_to_bf16_bits(gf[:, None] * O.bf16_to_f64(w).astype(np.float32))
    got_w = wo.cpu().view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(got_w, want_w)
    if bias:
        want_b = S.f32_to_bf16_bits(gf * O.bf16_to_f64(b).astype(np.float32))
        assert np.array_equal(bo.cpu().view(torch.int16).numpy().view(np.uint16), want_b)


def test_dinov2_block_with_layerscale():
    """A DINOv2-B/14 block (257 tokens, LayerScale on both branches) pruned
    by scores: the block on folded weights against the oracle's block with
    the scales applied to the branch outputs."""
    cfg = S.get_config("cfg6", batch=6)
    cu, ids = S.initial_layout(cfg)
    x = S.activations_bf16(cfg, 41)
    wb = S.block_weights(cfg, 3, 41, random_affine=True)
    assert "ls1" in wb and "ls2" in wb
    keeps, _ = S.keep_schedule(cfg, 41)
    scores = O.gather_scores(S.score_table(cfg, 3, 41), cu, ids)
    w = _device_weights(cfg, wb)
    r = _run_block(cfg, x, cu, ids, w, scores, keeps[0])
    assert r["status"] == 0
    ref = O.pruned_block(O.bf16_to_f64(x), cu, ids, O.decode_weights(wb), cfg.heads, cfg.ln_eps,
                         scores, keeps[0])
    t_out = int(ref["cu_out"][-1])
    assert np.array_equal(r["cu_out"], ref["cu_out"])
    assert np.array_equal(r["kept"][:t_out], ref["kept_idx"])
    assert_close(f64(r["x_out"][:t_out]), ref["x_out"], "dinov2 block")


@pytest.mark.parametrize("name,dim", [("cfg6", 768), ("cfg1", 192), ("cfg4", 1024),
                                      ("cfg1", 2048)])
def test_classifier_head_lc1_matches_oracle(name, dim):
    cfg = S.get_config(name, batch=24)
    keeps, _ = S.keep_schedule(cfg, 17)
    lens = np.array(keeps[-1])
    lens[3] = 1                                      # CLS only: zero visual mean
    lens[5] = 2                                      # one visual token
    lens[7] = 0                                      # empty image
    cu = O.cu_from_counts(lens)
    t = int(cu[-1])
    rng = np.random.default_rng(17)
    x = S.f32_to_bf16_bits(rng.uniform(-3, 3, (t, 1)) + rng.standard_normal((t, dim)))
    nw = S.f32_to_bf16_bits(1 + 0.1 * rng.standard_normal(dim))
    nb = S.f32_to_bf16_bits(0.1 * rng.standard_normal(dim))
    classes = 1024
    w_head = np.zeros((classes, 2 * dim), np.uint16)
    w_head[:1000] = S.f32_to_bf16_bits(rng.standard_normal((1000, 2 * dim)) / np.sqrt(2 * dim))
    b_head = np.zeros(classes, np.uint16)
    b_head[:1000] = S.f32_to_bf16_bits(0.02 * rng.standard_normal(1000))
    logits = torch.full((cfg.batch, classes), 9.0, dtype=torch.bfloat16, device=dev())
    ws = P.dora_classifier_head_lc1(bf(x), i32(cu), bf(nw), bf(nb), 1e-6, bf(w_head), bf(b_head),
                                    logits)
    torch.cuda.synchronize()
    assert P.dora_read_status(P.dora_workspace_status(ws)) == 0
    ref = O.classifier_head_lc1(O.bf16_to_f64(x), cu, O.bf16_to_f64(nw), O.bf16_to_f64(nb), 1e-6,
                                O.bf16_to_f64(w_head), O.bf16_to_f64(b_head))
    assert_close(f64(logits), ref, f"lc1 head {name}")
    assert torch.all(logits[:, 1000:] == 0)

