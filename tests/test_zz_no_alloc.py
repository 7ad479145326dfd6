"""dora_pruned_block_noalloc: the block entry point for callers that cannot
allocate device memory when they run it (its intermediates live in a scratch
array the library holds).  It must give the same outputs as
dora_pruned_block with a caller-allocated workspace, on consecutive calls
that share the library's scratch, and refuse blocks that do not fit.

This file is named so that pytest collects it last."""
import ctypes

import numpy as np
import pytest
import torch

import __graft_entry__ as G
import dora_synth as S
import oracle as O
import paper_2609_34325_gb300 as P
from helpers import assert_close, bf, f32, i32

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    G.build()
    P.load_library()
    torch.cuda.set_device(0)


def _inputs(cfg, seed, prune):
    cu, ids = S.initial_layout(cfg)
    x = S.activations_bf16(cfg, seed)
    wb = S.block_weights(cfg, 0, seed, random_affine=True)
    w = P.BlockWeights({k: bf(v) for k, v in wb.items()}, cfg.dim, cfg.heads, cfg.mlp_dim,
                       cfg.ln_eps)
    kw = {}
    if prune:
        keeps, _ = S.keep_schedule(cfg, seed)
        scores = O.gather_scores(S.score_table(cfg, 0, seed), cu, ids)
        kw = dict(scores=f32(scores), keep_counts=i32(keeps[0]))
    return bf(x), i32(cu), i32(ids), w, kw


def _outputs(t, b, dim):
    dev = torch.device("cuda:0")
    return dict(x_out=torch.zeros(t, dim, dtype=torch.bfloat16, device=dev),
                cu_out=torch.zeros(b + 1, dtype=torch.int32, device=dev),
                ids_out=torch.zeros(t, dtype=torch.int32, device=dev),
                kept_idx=torch.zeros(t, dtype=torch.int32, device=dev))


def _check_consecutive_calls(cfg, seeds):
    """Calls in a row through the scratch-array entry point against the
    workspace entry point on the same inputs: the same kernels run on the same
    data, so every output must match bit for bit.  The first call is also
    checked against the fp64 oracle within the block tolerance."""
    t = cfg.batch * cfg.n_tokens
    for n, (seed, prune) in enumerate(seeds):
        x, cu, ids, w, kw = _inputs(cfg, seed, prune)
        assert P.dora_workspace_size(t, cfg.batch, w) <= P.NOALLOC_SCRATCH_BYTES
        ref = _outputs(t, cfg.batch, cfg.dim)
        ws = P.alloc_workspace(t, cfg.batch, w)
        P.dora_pruned_block(x, cu, w, cfg.n_tokens, ref["x_out"], ws, ids_in=ids,
                            cu_out=ref["cu_out"], ids_out=ref["ids_out"],
                            kept_idx=ref["kept_idx"], **kw)
        got = _outputs(t, cfg.batch, cfg.dim)
        status = torch.full((1,), -1, dtype=torch.int32, device="cuda:0")
        P.dora_pruned_block_noalloc(x, cu, w, cfg.n_tokens, got["x_out"], ids_in=ids,
                                    cu_out=got["cu_out"], ids_out=got["ids_out"],
                                    kept_idx=got["kept_idx"], status=status, **kw)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        assert P.dora_read_status(P.dora_workspace_status(ws)) == 0
        if prune:
            t_out = int(ref["cu_out"][-1].item())
            assert torch.equal(got["cu_out"], ref["cu_out"])
            assert torch.equal(got["kept_idx"][:t_out], ref["kept_idx"][:t_out])
            assert torch.equal(got["ids_out"][:t_out], ref["ids_out"][:t_out])
        else:
            t_out = t
        assert torch.equal(got["x_out"][:t_out], ref["x_out"][:t_out]), f"seed {seed}"
        if n == 0:
            cu_h, ids_h = S.initial_layout(cfg)
            wb = S.block_weights(cfg, 0, seed, random_affine=True)
            sc = kp = None
            if prune:
                keeps, _ = S.keep_schedule(cfg, seed)
                sc = O.gather_scores(S.score_table(cfg, 0, seed), cu_h, ids_h)
                kp = keeps[0]
            o = O.pruned_block(O.bf16_to_f64(S.activations_bf16(cfg, seed)), cu_h, ids_h,
                               O.decode_weights(wb), cfg.heads, cfg.ln_eps, sc, kp)
            assert np.array_equal(got["cu_out"].cpu().numpy(), o["cu_out"])
            assert_close(got["x_out"][:t_out].float().cpu().numpy(), o["x_out"],
                         f"noalloc vs oracle, seed {seed}")


def test_noalloc_matches_workspace_entry_on_consecutive_calls():
    # DeiT-Tiny shape, 8 x 197 tokens, D = 192: about 7 MB of scratch
    _check_consecutive_calls(S.get_config("cfg1"), ((31, True), (32, True), (33, False)))


def test_noalloc_matches_workspace_entry_deit_small_sub_batch():
    # DeiT-Small shape, 16 of its 64 images (3152 rows, D = 384): about 26 MB
    _check_consecutive_calls(S.get_config("cfg2", batch=16), ((41, True), (42, True)))


def test_noalloc_rejects_blocks_larger_than_its_scratch():
    cfg = S.get_config("cfg3", batch=16)              # 3152 rows x ~17 KB > 32 MiB
    t = cfg.batch * cfg.n_tokens
    dev = torch.device("cuda:0")
    x = torch.zeros(t, cfg.dim, dtype=torch.bfloat16, device=dev)
    cu = i32(np.arange(cfg.batch + 1) * cfg.n_tokens)
    wt = {n: torch.zeros(s, dtype=torch.bfloat16, device=dev) for n, s in (
        ("ln1_w", cfg.dim), ("ln1_b", cfg.dim), ("w_qkv", (3 * cfg.dim, cfg.dim)),
        ("w_proj", (cfg.dim, cfg.dim)), ("ln2_w", cfg.dim), ("ln2_b", cfg.dim),
        ("w_fc1", (cfg.mlp_dim, cfg.dim)), ("w_fc2", (cfg.dim, cfg.mlp_dim)))}
    w = P.BlockWeights(wt, cfg.dim, cfg.heads, cfg.mlp_dim)
    assert P.dora_workspace_size(t, cfg.batch, w) > P.NOALLOC_SCRATCH_BYTES
    out = torch.full_like(x, 2.0)
    lib = P.load_library()
    rc = lib.dora_pruned_block_noalloc(x.data_ptr(), cu.data_ptr(), None, cfg.batch,
                                       cfg.n_tokens, t, ctypes.byref(w.c), None, None,
                                       out.data_ptr(), None, None, None, None, None, None,
                                       torch.cuda.current_stream().cuda_stream)
    assert rc == 7 and P.dora_status_string(rc).startswith("block needs more scratch")
    torch.cuda.synchronize()
    assert torch.all(out == 2.0)                      # nothing was launched
