"""Host-only checks of the C ABI: the library builds, loads, exports every
symbol the header declares, and rejects bad arguments before touching a GPU."""
import ctypes
import os
import re

import pytest

import __graft_entry__ as G
import paper_2609_34325_gb300 as P

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    G.build()
    return P.load_library()


def _declared_functions():
    src = open(os.path.join(ROOT, "include", "dora.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(dora_[a-z0-9_]+)\s*\(", src)))


def test_header_declares_the_entry_points():
    decl = _declared_functions()
    for name in ("dora_select_keep", "dora_compact", "dora_varlen_attn", "dora_pruned_block",
                 "dora_workspace_size", "dora_read_status"):
        assert name in decl
    assert sorted(P.EXPORTED_SYMBOLS) == decl


def test_library_exports_every_declared_symbol(lib):
    for name in _declared_functions():
        assert hasattr(lib, name), name


def test_status_strings(lib):
    assert P.dora_version() == 2
    assert P.dora_status_string(0) == "ok"
    assert "timed out" in P.dora_status_string(4)
    assert P.dora_status_string(99) == "unknown status"


def test_host_validation_without_gpu(lib):
    # every failure below is decided from the arguments, before any CUDA call
    assert lib.dora_select_keep(None, None, None, 1, 197, None, None, None, None) == 1
    assert lib.dora_select_keep(None, 8, 8, 1, 1 << 20, 8, 8, None, None) == 1
    assert lib.dora_varlen_attn(16, 16, 1, 197, 197, 3, 32, 0.0, 16, None, None) == 2
    assert lib.dora_varlen_attn(16, 16, 1, 197, 197, 3, 64, -1.0, 16, None, None) == 1
    assert lib.dora_varlen_attn(17, 16, 1, 197, 197, 3, 64, 0.0, 16, None, None) == 1
    assert lib.dora_linear(16, 128, None, 100, 16, 128, None, None, 0, 16, None, None) == 1
    assert lib.dora_linear(16, 128, None, 128, 16, 100, None, None, 0, 16, None, None) == 1
    assert lib.dora_linear(16, 128, None, 128, 16, 128, None, None, 2, 16, None, None) == 1
    assert lib.dora_linear(16, 128, None, 128, 16, 128, None, None, 7, 16, None, None) == 1
    assert lib.dora_compact(16, 12, 16, 16, 1, 10, None, 16, None, None, None) == 1
    # dora_select_compact: dim % 8, ids given without ids_out, mv_out misaligned
    assert lib.dora_select_compact(16, 16, 16, 1, 197, 16, 12, 197, None, None, 16, 16, 16,
                                   None, None, None, None) == 1
    assert lib.dora_select_compact(16, 16, 16, 1, 197, 16, 64, 197, 16, None, 16, 16, 16,
                                   None, None, None, None) == 1
    assert lib.dora_select_compact(16, 16, 16, 1, 197, 16, 64, 197, None, 16, 16, 16, 16,
                                   None, 12, None, None) == 1
    assert lib.dora_select_compact(16, 16, 16, 1, 1 << 20, 16, 64, 197, None, None, 16, 16, 16,
                                   None, None, None, None) == 1
    assert lib.dora_layernorm(16, 4, None, 4096, 16, 16, 1e-6, 16, None) == 1
    assert lib.dora_gather_scores(16, 0, 16, 16, 1, 16, None, None) == 1
    assert lib.dora_read_status(None, None) == 1
    assert lib.dora_pruned_block(None, None, None, 1, 197, 197, None, None, None, None, None,
                                 None, None, None, None, None, 0, None) == 1
    assert lib.dora_row_stats(16, 4, None, 100, 16, None) == 1           # dim % 8
    assert lib.dora_row_stats(16, 4, None, 128, 12, None) == 1            # mv alignment
    assert lib.dora_merge_moments(16, 4, None, 0, 16, None) == 1          # no slices
    assert lib.dora_compact_stats(16, 64, 16, 16, 1, 10, None, None, 16, None, 16, None,
                                  None) == 1                              # mv_in missing
    assert lib.dora_fold_ln_linear(16, 8, 12, 16, 16, None, 16, 16, 16, None) == 1   # k % 8
    assert lib.dora_linear_ln(16, 128, None, 96, 16, 1e-6, 16, 128, 16, 16, 0, 16, None,
                              None) == 1                                 # k % 64
    assert lib.dora_linear_ln(16, 128, None, 128, 16, -1.0, 16, 128, 16, 16, 0, 16, None,
                              None) == 1                                 # eps < 0
    assert lib.dora_linear_residual_stats(16, 128, None, 128, 16, 96, None, 32, 16, 16, None,
                                          None) == 1                     # n % 64
    assert lib.dora_fold_block_weights(None, 256, 1 << 20, None) == 1


def test_block_weights_struct_and_workspace(lib):
    # per row: slice moments (dim/64 x 8 B), two row moments (8 B each), qkv,
    # attention output, H_attn, H_keep, kept index, MLP hidden; plus the
    # folded QKV and fc1 weights
    # (bf16 W', fp32 c and d) when the caller has not folded them
    t, d, m = 50432, 768, 3072
    w = P._BlockWeightsC(*([16] * 12), d, 12, m, 1e-6, None)
    per_rows = t * (d // 64 * 8 + 16 + 3 * d * 2 + 3 * d * 2 + 4 + m * 2)
    fold = (3 * d + m) * d * 2 + 2 * (3 * d + m) * 4
    folded_size = lib.dora_folded_weights_size(ctypes.byref(w))
    assert fold <= folded_size < fold + 8 * 256
    n = lib.dora_workspace_size(t, 256, ctypes.byref(w))
    assert per_rows + folded_size <= n < per_rows + folded_size + 16 * 256
    w.folded = 256
    assert lib.dora_workspace_size(t, 256, ctypes.byref(w)) == n - folded_size
    assert lib.dora_workspace_size(-1, 1, ctypes.byref(w)) == 0


def test_python_binding_rejects_cpu_tensors(lib):
    import torch
    x = torch.zeros(4, 8, dtype=torch.bfloat16)
    with pytest.raises(TypeError):
        P.dora_layernorm(x, x[0], x[0], 1e-6, x)


def test_actor_struct_sizes_and_host_checks(lib):
    w = P._ActorWeightsC(*([16] * len(P.ActorWeights.NAMES)), 768, 12, 196, 1e-5, None)
    prep = lib.dora_actor_prepared_size(ctypes.byref(w))
    assert prep > 0
    # per row: X, Z1, Z (128 bf16 each), padded qkv (768), attention out (256),
    # feed-forward (256), selector hidden (64), row moments and two slice
    # moments; per image the gate logit
    t, b = 50000, 256
    per_rows = t * (3 * 256 + 1536 + 512 + 512 + 128 + 8 + 16) + 4 * b
    n = lib.dora_actor_workspace_size(t, b, ctypes.byref(w))
    assert per_rows + prep <= n < per_rows + prep + 16 * 256
    w.prepared = 256
    assert lib.dora_actor_workspace_size(t, b, ctypes.byref(w)) == n - prep
    w.prepared = None
    n = lib.dora_actor_workspace_size(1000, 4, ctypes.byref(w))
    args = [16, 16, 4, 197, 1000, 0, ctypes.byref(w), 16, 16, None, 16, 16, 16, 16, 16, None, None,
            None, 256, n, None]
    bad = []
    for i, v in ((5, 12),):                       # block >= depth
        a = list(args); a[i] = v; bad.append(a)
    a = list(args); a[6] = None; bad.append(a)    # no weights
    a = list(args); a[18] = 264; bad.append(a)    # misaligned workspace
    a = list(args); a[19] = n - 1; bad.append(a)  # workspace too small
    for a in bad:
        assert lib.dora_actor(*a) == 1
    for field, v in (("dim", 100), ("n0", 4), ("n0", 2000), ("depth", 0)):
        w2 = P._ActorWeightsC(*([16] * len(P.ActorWeights.NAMES)), 768, 12, 196, 1e-5, None)
        setattr(w2, field, v)
        a = list(args); a[6] = ctypes.byref(w2)
        assert lib.dora_actor(*a) == 1
        assert lib.dora_actor_prepare(ctypes.byref(w2), 256, 1 << 20, None) == 1


def test_dinov2_entry_points_host_checks(lib):
    # LC1 head: dim above the kernel's register-held row (2048)
    assert lib.dora_classifier_head_lc1(16, 16, 4, 100, 4096, 16, 16, ctypes.c_float(1e-6), 16,
                                        16, 1024, 16, 256, 1 << 20, None) == 1
    # LC1 head: classes not a multiple of 32
    assert lib.dora_classifier_head_lc1(16, 16, 4, 100, 768, 16, 16, ctypes.c_float(1e-6), 16,
                                        16, 1000, 16, 256, 1 << 20, None) == 1
    assert lib.dora_head_lc1_workspace_size(4, 768) >= 256 + 4 * 2 * 768 * 2
    # LayerScale fold: k % 8, bias without its output
    assert lib.dora_fold_layerscale(16, None, 16, 8, 12, 16, None, None) == 1
    assert lib.dora_fold_layerscale(16, 16, 16, 8, 16, 16, None, None) == 1
    # patch embedding: patch 0, image side not a multiple of the patch
    assert lib.dora_patch_embed(16, 1, 3, 224, 224, 0, 768, 16, 16, 16, 16, 16, 256, 1 << 30,
                                None) == 1
    assert lib.dora_patch_embed(16, 1, 3, 225, 224, 14, 768, 16, 16, 16, 16, 16, 256, 1 << 30,
                                None) == 1
    # the 14-pixel patch workspace holds the K-padded (588 -> 640) patches and weight copy
    n = lib.dora_embed_workspace_size(2, 3, 224, 224, 14, 768)
    assert n >= 256 + 2 * 256 * 640 * 2 + 2 * 256 * 768 * 2 + 768 * 640 * 2


def test_training_entry_points_host_checks(lib):
    # Plackett-Luce: k_cap outside [1, 2048], missing buffers
    assert lib.dora_pl_sample(16, 16, 16, 4, 100, 16, 0, 16, None, None, None) == 1
    assert lib.dora_pl_sample(16, 16, 16, 4, 100, 16, 4096, 16, None, None, None) == 1
    assert lib.dora_pl_sample(16, None, 16, 4, 100, 16, 8, 16, None, None, None) == 1
    assert lib.dora_pl_logprob(16, 16, 4, 100, 16, 16, 0, 16, None, None, None, None) == 1
    assert lib.dora_pl_logprob(16, 16, 4, 100, 16, 16, 8, None, None, None, None, None) == 1
    # branch: dim % 8, misaligned rows, sources missing
    assert lib.dora_branch(16, None, None, 16, 4, 100, 12, 16, 2, 16, None, None, None) == 1
    assert lib.dora_branch(24, None, None, 16, 4, 100, 16, 16, 2, 16, None, None, None) == 1
    assert lib.dora_branch(16, None, None, 16, 4, 100, 16, None, 2, 16, None, None, None) == 1
    # fidelity cost: row pitch below the class count, tau <= 0
    assert lib.dora_kd_cost(16, 16, None, 8, 4, 1000, 999, ctypes.c_float(3.0), 16, None,
                            None) == 1
    assert lib.dora_kd_cost(16, 16, None, 8, 4, 1000, 1024, ctypes.c_float(0.0), 16, None,
                            None) == 1


def test_step_rewards_host_checks(lib):
    assert lib.dora_step_rewards(16, 16, 16, 0, 4, 12, 196, ctypes.c_float(30.0), 16, None,
                                 None) == 1
    assert lib.dora_step_rewards(16, None, 16, 3, 4, 12, 196, ctypes.c_float(30.0), 16, None,
                                 None) == 1


def test_shadow_rollout_rejects_bad_schedules():
    from paper_2609_34325_gb300.shadow import ShadowRollout
    for prune in ((), (2, 1), (0, 5), (-1, 2), (1, 1)):
        with pytest.raises(ValueError):
            ShadowRollout([object()] * 3, 4, 197, prune, "cpu")
