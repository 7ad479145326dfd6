"""GB300 (sm_103a) deployment hot path of DORA's pruned ViT forward.

A thin ctypes binding over ``libdora.so`` (C ABI in ``include/dora.h``).  The
Python functions carry the C names and only marshal arguments: torch tensors
supply device pointers and the current CUDA stream; every step of the path
runs in the library's CUDA kernels.  There is no fallback: when the library
is missing or the device is not sm_103 the calls raise.
"""
from __future__ import annotations

import ctypes
import os

import torch

__all__ = [
    "DoraError", "load_library", "library_path", "EPI_BIAS", "EPI_BIAS_GELU",
    "EPI_BIAS_RESIDUAL", "EXPORTED_SYMBOLS", "dora_status_string", "dora_version",
    "dora_select_keep", "dora_select_compact", "dora_compact", "dora_compact_ln", "dora_layernorm", "dora_linear",
    "dora_varlen_attn", "dora_gather_scores", "BlockWeights", "dora_workspace_size",
    "dora_pruned_block", "dora_workspace_status", "dora_read_status", "alloc_workspace",
    "dora_pruned_block_noalloc", "NOALLOC_SCRATCH_BYTES", "dora_row_stats",
    "dora_fold_ln_linear", "dora_linear_ln", "dora_linear_residual_stats",
    "dora_folded_weights_size", "dora_fold_block_weights", "dora_compact_stats",
    "dora_merge_moments", "ActorWeights", "dora_actor", "dora_actor_workspace_size",
    "alloc_actor_workspace", "dora_pruned_block_actor", "dora_patch_embed",
    "dora_classifier_head", "dora_classifier_head_lc1", "dora_fold_layerscale",
    "dora_pl_sample", "dora_pl_logprob", "dora_branch", "dora_kd_cost", "dora_step_rewards",
]

_HERE = os.path.dirname(os.path.abspath(__file__))
EPI_BIAS, EPI_BIAS_GELU, EPI_BIAS_RESIDUAL = 0, 1, 2
STATUS_NAMES = {0: "DORA_OK", 1: "DORA_ERR_INVALID_ARG", 2: "DORA_ERR_UNSUPPORTED",
                3: "DORA_ERR_CUDA", 4: "DORA_ERR_TIMEOUT", 5: "DORA_ERR_DEVICE_BAD_COUNT",
                6: "DORA_ERR_DEVICE_SEQLEN", 7: "DORA_ERR_SCRATCH_TOO_SMALL"}
NOALLOC_SCRATCH_BYTES = 32 << 20

_vp, _i32, _f32, _sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_float, ctypes.c_size_t
_SIGS = {
    "dora_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "dora_version": (ctypes.c_int, []),
    "dora_select_keep": (ctypes.c_int, [_vp, _vp, _vp, _i32, _i32, _vp, _vp, _vp, _vp]),
    "dora_select_compact": (ctypes.c_int, [_vp, _vp, _vp, _i32, _i32, _vp, _i32, _i32, _vp, _vp,
                                           _vp, _vp, _vp, _vp, _vp, _vp, _vp]),
    "dora_compact": (ctypes.c_int, [_vp, _i32, _vp, _vp, _i32, _i32, _vp, _vp, _vp, _vp, _vp]),
    "dora_compact_ln": (ctypes.c_int, [_vp, _i32, _vp, _vp, _i32, _i32, _vp, _vp, _vp, _f32,
                                       _vp, _vp, _vp, _vp, _vp]),
    "dora_layernorm": (ctypes.c_int, [_vp, _i32, _vp, _i32, _vp, _vp, _f32, _vp, _vp]),
    "dora_linear": (ctypes.c_int, [_vp, _i32, _vp, _i32, _vp, _i32, _vp, _vp, _i32, _vp, _vp,
                                   _vp]),
    "dora_varlen_attn": (ctypes.c_int, [_vp, _vp, _i32, _i32, _i32, _i32, _i32, _f32, _vp, _vp,
                                        _vp]),
    "dora_gather_scores": (ctypes.c_int, [_vp, _i32, _vp, _vp, _i32, _vp, _vp, _vp]),
    "dora_workspace_size": (_sz, [_i32, _i32, _vp]),
    "dora_pruned_block": (ctypes.c_int, [_vp, _vp, _vp, _i32, _i32, _i32, _vp, _vp, _vp, _vp,
                                         _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "dora_workspace_status": (_vp, [_vp]),
    "dora_pruned_block_noalloc": (ctypes.c_int, [_vp, _vp, _vp, _i32, _i32, _i32, _vp, _vp, _vp,
                                                 _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp]),
    "dora_read_status": (ctypes.c_int, [_vp, _vp]),
    "dora_row_stats": (ctypes.c_int, [_vp, _i32, _vp, _i32, _vp, _vp]),
    "dora_fold_ln_linear": (ctypes.c_int, [_vp, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _vp]),
    "dora_linear_ln": (ctypes.c_int, [_vp, _i32, _vp, _i32, _vp, _f32, _vp, _i32, _vp, _vp, _i32,
                                      _vp, _vp, _vp]),
    "dora_linear_residual_stats": (ctypes.c_int, [_vp, _i32, _vp, _i32, _vp, _i32, _vp, _vp, _vp,
                                                  _vp, _vp, _vp]),
    "dora_folded_weights_size": (_sz, [_vp]),
    "dora_fold_block_weights": (ctypes.c_int, [_vp, _vp, _sz, _vp]),
    "dora_compact_stats": (ctypes.c_int, [_vp, _i32, _vp, _vp, _i32, _i32, _vp, _vp, _vp, _vp,
                                          _vp, _vp, _vp]),
    "dora_merge_moments": (ctypes.c_int, [_vp, _i32, _vp, _i32, _vp, _vp]),
    "dora_actor_prepared_size": (_sz, [_vp]),
    "dora_actor_workspace_size": (_sz, [_i32, _i32, _vp]),
    "dora_actor_prepare": (ctypes.c_int, [_vp, _vp, _sz, _vp]),
    "dora_actor": (ctypes.c_int, [_vp, _vp, _i32, _i32, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _vp,
                                  _vp, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "dora_embed_workspace_size": (_sz, [_i32, _i32, _i32, _i32, _i32, _i32]),
    "dora_patch_embed": (ctypes.c_int, [_vp, _i32, _i32, _i32, _i32, _i32, _i32, _vp, _vp, _vp,
                                        _vp, _vp, _vp, _sz, _vp]),
    "dora_head_workspace_size": (_sz, [_i32, _i32]),
    "dora_head_lc1_workspace_size": (_sz, [_i32, _i32]),
    "dora_classifier_head_lc1": (ctypes.c_int, [_vp, _vp, _i32, _i32, _i32, _vp, _vp, _f32, _vp,
                                                _vp, _i32, _vp, _vp, _sz, _vp]),
    "dora_fold_layerscale": (ctypes.c_int, [_vp, _vp, _vp, _i32, _i32, _vp, _vp, _vp]),
    "dora_pl_sample": (ctypes.c_int, [_vp, _vp, _vp, _i32, _i32, _vp, _i32, _vp, _vp, _vp, _vp]),
    "dora_pl_logprob": (ctypes.c_int, [_vp, _vp, _i32, _i32, _vp, _vp, _i32, _vp, _vp, _vp, _vp,
                                       _vp]),
    "dora_branch": (ctypes.c_int, [_vp, _vp, _vp, _vp, _i32, _i32, _i32, _vp, _i32, _vp, _vp, _vp,
                                   _vp]),
    "dora_kd_cost": (ctypes.c_int, [_vp, _vp, _vp, _i32, _i32, _i32, _i32, _f32, _vp, _vp, _vp]),
    "dora_step_rewards": (ctypes.c_int, [_vp, _vp, _vp, _i32, _i32, _i32, _i32, _f32, _vp, _vp,
                                         _vp]),
    "dora_classifier_head": (ctypes.c_int, [_vp, _vp, _i32, _i32, _i32, _vp, _vp, _f32, _vp, _vp,
                                            _i32, _vp, _vp, _sz, _vp]),
    "dora_pruned_block_actor": (ctypes.c_int, [_vp, _vp, _vp, _i32, _i32, _i32, _vp, _vp, _vp,
                                               _vp, _vp, _vp, _vp, _vp, _sz, _vp, _i32, _vp, _vp,
                                               _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _sz,
                                               _vp]),
}
EXPORTED_SYMBOLS = tuple(_SIGS)

_lib = None


class DoraError(RuntimeError):
    """A libdora entry point returned a nonzero host status."""


class _BlockWeightsC(ctypes.Structure):
    _fields_ = [(n, _vp) for n in ("ln1_w", "ln1_b", "w_qkv", "b_qkv", "w_proj", "b_proj",
                                   "ln2_w", "ln2_b", "w_fc1", "b_fc1", "w_fc2", "b_fc2")] + [
        ("dim", _i32), ("heads", _i32), ("mlp_dim", _i32), ("ln_eps", _f32), ("folded", _vp)]


def library_path() -> str:
    return os.path.join(_HERE, "libdora.so")


def load_library():
    """Load libdora.so (built by ``__graft_entry__.build()``); raise if absent."""
    global _lib
    if _lib is not None:
        return _lib
    path = library_path()
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is not built; run __graft_entry__.build() first")
    lib = ctypes.CDLL(path)
    for name, (res, args) in _SIGS.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream):
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def _req(t, dtype, name, optional=False):
    if t is None:
        if optional:
            return
        raise TypeError(f"{name} is required")
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise TypeError(f"{name} must be contiguous")


def _check(code, name):
    if code != 0:
        raise DoraError(f"{name}: {dora_status_string(code)} ({STATUS_NAMES.get(code, code)})")


def dora_status_string(code: int) -> str:
    return load_library().dora_status_string(int(code)).decode()


def dora_version() -> int:
    return load_library().dora_version()


def dora_select_keep(scores, cu_in, keep_counts, max_seqlen, kept_idx, cu_out, status=None,
                     stream=None):
    _req(scores, torch.float32, "scores")
    for n, t in (("cu_in", cu_in), ("keep_counts", keep_counts), ("kept_idx", kept_idx),
                 ("cu_out", cu_out)):
        _req(t, torch.int32, n)
    _req(status, torch.int32, "status", optional=True)
    batch = cu_in.numel() - 1
    _check(load_library().dora_select_keep(_ptr(scores), _ptr(cu_in), _ptr(keep_counts), batch,
                                           int(max_seqlen), _ptr(kept_idx), _ptr(cu_out),
                                           _ptr(status), _stream(stream)), "dora_select_keep")


def dora_select_compact(scores, cu_in, keep_counts, max_seqlen, x, kept_idx, cu_out, packed,
                        ids_in=None, ids_out=None, mv_in=None, mv_out=None, status=None,
                        stream=None):
    """dora_select_keep and the compaction of the kept rows in one launch:
    kept_idx and cu_out as dora_select_keep writes them, packed[r] =
    x[kept_idx[r]], and (when given) ids_out[r] = ids_in[kept_idx[r]],
    mv_out[r] = mv_in[kept_idx[r]]."""
    _req(scores, torch.float32, "scores")
    _req(x, torch.bfloat16, "x")
    _req(packed, torch.bfloat16, "packed")
    for n, t in (("cu_in", cu_in), ("keep_counts", keep_counts), ("kept_idx", kept_idx),
                 ("cu_out", cu_out)):
        _req(t, torch.int32, n)
    for n, t in (("ids_in", ids_in), ("ids_out", ids_out), ("status", status)):
        _req(t, torch.int32, n, optional=True)
    _req(mv_in, torch.float32, "mv_in", optional=True)
    _req(mv_out, torch.float32, "mv_out", optional=True)
    t_in_cap, dim = x.shape
    if packed.shape[0] < t_in_cap or packed.shape[1] != dim:
        raise ValueError("packed must hold at least as many rows as x")
    for n, t in (("mv_in", mv_in), ("mv_out", mv_out)):
        if t is not None and t.numel() < t_in_cap * 2:
            raise ValueError(f"{n} must hold [t_in_cap, 2] floats")
    _check(load_library().dora_select_compact(
        _ptr(scores), _ptr(cu_in), _ptr(keep_counts), cu_in.numel() - 1, int(max_seqlen),
        _ptr(x), dim, t_in_cap, _ptr(ids_in), _ptr(mv_in), _ptr(kept_idx), _ptr(cu_out),
        _ptr(packed), _ptr(ids_out), _ptr(mv_out), _ptr(status), _stream(stream)),
        "dora_select_compact")


def dora_compact(x, kept_idx, cu_out, packed, ids_in=None, ids_out=None, status=None,
                 stream=None):
    _req(x, torch.bfloat16, "x")
    _req(packed, torch.bfloat16, "packed")
    _req(kept_idx, torch.int32, "kept_idx")
    _req(cu_out, torch.int32, "cu_out")
    _req(ids_in, torch.int32, "ids_in", optional=True)
    _req(ids_out, torch.int32, "ids_out", optional=True)
    _req(status, torch.int32, "status", optional=True)
    t_in_cap, dim = x.shape
    if packed.shape[0] < t_in_cap or packed.shape[1] != dim:
        raise ValueError("packed must hold at least as many rows as x")
    _check(load_library().dora_compact(_ptr(x), dim, _ptr(kept_idx), _ptr(cu_out),
                                       cu_out.numel() - 1, t_in_cap, _ptr(ids_in), _ptr(packed),
                                       _ptr(ids_out), _ptr(status), _stream(stream)),
           "dora_compact")


def dora_compact_stats(x, kept_idx, cu_out, packed, mv_in, mv_out, ids_in=None, ids_out=None,
                       status=None, stream=None):
    """dora_compact that also carries the row moments: mv_out[r] = mv_in[kept_idx[r]]."""
    _req(x, torch.bfloat16, "x")
    _req(packed, torch.bfloat16, "packed")
    _req(mv_in, torch.float32, "mv_in")
    _req(mv_out, torch.float32, "mv_out")
    _req(kept_idx, torch.int32, "kept_idx")
    _req(cu_out, torch.int32, "cu_out")
    _req(ids_in, torch.int32, "ids_in", optional=True)
    _req(ids_out, torch.int32, "ids_out", optional=True)
    _req(status, torch.int32, "status", optional=True)
    t_in_cap, dim = x.shape
    if packed.shape[0] < t_in_cap or packed.shape[1] != dim:
        raise ValueError("packed must hold at least as many rows as x")
    if mv_in.numel() < t_in_cap * 2 or mv_out.numel() < t_in_cap * 2:
        raise ValueError("mv_in and mv_out must hold [t_in_cap, 2] floats")
    _check(load_library().dora_compact_stats(_ptr(x), dim, _ptr(kept_idx), _ptr(cu_out),
                                             cu_out.numel() - 1, t_in_cap, _ptr(ids_in),
                                             _ptr(mv_in), _ptr(packed), _ptr(ids_out),
                                             _ptr(mv_out), _ptr(status), _stream(stream)),
           "dora_compact_stats")


def dora_compact_ln(x, kept_idx, cu_out, ln_w, ln_b, eps, packed, ln_out, ids_in=None,
                    ids_out=None, status=None, stream=None):
    for n, t in (("x", x), ("packed", packed), ("ln_out", ln_out), ("ln_w", ln_w),
                 ("ln_b", ln_b)):
        _req(t, torch.bfloat16, n)
    _req(kept_idx, torch.int32, "kept_idx")
    _req(cu_out, torch.int32, "cu_out")
    _req(ids_in, torch.int32, "ids_in", optional=True)
    _req(ids_out, torch.int32, "ids_out", optional=True)
    _req(status, torch.int32, "status", optional=True)
    t_in_cap, dim = x.shape
    if packed.shape[0] < t_in_cap or ln_out.shape[0] < t_in_cap:
        raise ValueError("packed and ln_out must hold at least as many rows as x")
    _check(load_library().dora_compact_ln(_ptr(x), dim, _ptr(kept_idx), _ptr(cu_out),
                                          cu_out.numel() - 1, t_in_cap, _ptr(ids_in), _ptr(ln_w),
                                          _ptr(ln_b), float(eps), _ptr(packed), _ptr(ids_out),
                                          _ptr(ln_out), _ptr(status), _stream(stream)),
           "dora_compact_ln")


def dora_layernorm(x, w, b, eps, y, rows_dev=None, stream=None):
    for n, t in (("x", x), ("w", w), ("b", b), ("y", y)):
        _req(t, torch.bfloat16, n)
    _req(rows_dev, torch.int32, "rows_dev", optional=True)
    rows, dim = x.shape
    _check(load_library().dora_layernorm(_ptr(x), rows, _ptr(rows_dev), dim, _ptr(w), _ptr(b),
                                         float(eps), _ptr(y), _stream(stream)), "dora_layernorm")


def dora_linear(x, w, y, bias=None, residual=None, epilogue=EPI_BIAS, m_dev=None, status=None,
                stream=None):
    _req(x, torch.bfloat16, "x")
    _req(w, torch.bfloat16, "w")
    _req(y, torch.bfloat16, "y")
    _req(bias, torch.bfloat16, "bias", optional=True)
    _req(residual, torch.bfloat16, "residual", optional=True)
    _req(m_dev, torch.int32, "m_dev", optional=True)
    _req(status, torch.int32, "status", optional=True)
    m_cap, k = x.shape
    n = w.shape[0]
    if w.shape[1] != k or tuple(y.shape) != (m_cap, n):
        raise ValueError("shape mismatch: x [M,K], w [N,K], y [M,N]")
    _check(load_library().dora_linear(_ptr(x), m_cap, _ptr(m_dev), k, _ptr(w), n, _ptr(bias),
                                      _ptr(residual), int(epilogue), _ptr(y), _ptr(status),
                                      _stream(stream)), "dora_linear")


def dora_row_stats(x, mv, rows_dev=None, stream=None):
    """Row moments (mean, biased variance) of the rows of x [rows, dim] into
    mv (fp32 [rows, 2])."""
    _req(x, torch.bfloat16, "x")
    _req(mv, torch.float32, "mv")
    _req(rows_dev, torch.int32, "rows_dev", optional=True)
    rows, dim = x.shape
    if mv.numel() < rows * 2:
        raise ValueError("mv must hold [rows, 2] floats")
    _check(load_library().dora_row_stats(_ptr(x), rows, _ptr(rows_dev), dim, _ptr(mv),
                                         _stream(stream)), "dora_row_stats")


def dora_merge_moments(sm, mv, rows_dev=None, stream=None):
    """Row moments mv (fp32 [rows, 2]) from slice moments sm (fp32 [S, rows, 2])."""
    _req(sm, torch.float32, "sm")
    _req(mv, torch.float32, "mv")
    _req(rows_dev, torch.int32, "rows_dev", optional=True)
    slices, rows = sm.shape[0], sm.shape[1]
    if mv.numel() < rows * 2:
        raise ValueError("mv must hold [rows, 2] floats")
    _check(load_library().dora_merge_moments(_ptr(sm), rows, _ptr(rows_dev), slices, _ptr(mv),
                                             _stream(stream)), "dora_merge_moments")


def dora_fold_ln_linear(w, gamma, beta, w_out, colsum, colbias, bias=None, stream=None):
    """LayerNorm affine into the linear after it: w_out = bf16(w diag(gamma)),
    colsum = w_out 1, colbias = w beta + bias."""
    for n, t in (("w", w), ("gamma", gamma), ("beta", beta), ("w_out", w_out)):
        _req(t, torch.bfloat16, n)
    _req(bias, torch.bfloat16, "bias", optional=True)
    _req(colsum, torch.float32, "colsum")
    _req(colbias, torch.float32, "colbias")
    n_out, k = w.shape
    if tuple(w_out.shape) != (n_out, k) or colsum.numel() < n_out or colbias.numel() < n_out:
        raise ValueError("shape mismatch: w, w_out [n,k]; colsum, colbias [n]")
    _check(load_library().dora_fold_ln_linear(_ptr(w), n_out, k, _ptr(gamma), _ptr(beta),
                                              _ptr(bias), _ptr(w_out), _ptr(colsum),
                                              _ptr(colbias), _stream(stream)),
           "dora_fold_ln_linear")


def dora_linear_ln(x, mv, eps, w_folded, colsum, colbias, y, gelu=False, m_dev=None,
                   status=None, stream=None):
    """y = LayerNorm(x) W^T + b (GELU of it when gelu) from folded weights and
    the row moments mv of x."""
    _req(x, torch.bfloat16, "x")
    _req(w_folded, torch.bfloat16, "w_folded")
    _req(y, torch.bfloat16, "y")
    _req(mv, torch.float32, "mv")
    _req(colsum, torch.float32, "colsum")
    _req(colbias, torch.float32, "colbias")
    _req(m_dev, torch.int32, "m_dev", optional=True)
    _req(status, torch.int32, "status", optional=True)
    m_cap, k = x.shape
    n = w_folded.shape[0]
    if w_folded.shape[1] != k or tuple(y.shape) != (m_cap, n):
        raise ValueError("shape mismatch: x [M,K], w_folded [N,K], y [M,N]")
    _check(load_library().dora_linear_ln(_ptr(x), m_cap, _ptr(m_dev), k, _ptr(mv), float(eps),
                                         _ptr(w_folded), n, _ptr(colsum), _ptr(colbias),
                                         1 if gelu else 0, _ptr(y), _ptr(status),
                                         _stream(stream)), "dora_linear_ln")


def dora_linear_residual_stats(x, w, residual, y, stats_out, bias=None, m_dev=None, status=None,
                               stream=None):
    """y = residual + x W^T + b, plus the slice moments of y's rows."""
    for n_, t in (("x", x), ("w", w), ("residual", residual), ("y", y)):
        _req(t, torch.bfloat16, n_)
    _req(bias, torch.bfloat16, "bias", optional=True)
    _req(stats_out, torch.float32, "stats_out")
    _req(m_dev, torch.int32, "m_dev", optional=True)
    _req(status, torch.int32, "status", optional=True)
    m_cap, k = x.shape
    n = w.shape[0]
    if w.shape[1] != k or tuple(y.shape) != (m_cap, n) or tuple(residual.shape) != (m_cap, n):
        raise ValueError("shape mismatch: x [M,K], w [N,K], residual, y [M,N]")
    _check(load_library().dora_linear_residual_stats(
        _ptr(x), m_cap, _ptr(m_dev), k, _ptr(w), n, _ptr(bias), _ptr(residual), _ptr(y),
        _ptr(stats_out), _ptr(status), _stream(stream)), "dora_linear_residual_stats")


def dora_varlen_attn(qkv, cu_seqlens, max_seqlen, heads, out, head_dim=64, softmax_scale=0.0,
                     status=None, stream=None):
    _req(qkv, torch.bfloat16, "qkv")
    _req(out, torch.bfloat16, "out")
    _req(cu_seqlens, torch.int32, "cu_seqlens")
    _req(status, torch.int32, "status", optional=True)
    t_cap = qkv.shape[0]
    _check(load_library().dora_varlen_attn(_ptr(qkv), _ptr(cu_seqlens), cu_seqlens.numel() - 1,
                                           int(max_seqlen), t_cap, int(heads), int(head_dim),
                                           float(softmax_scale), _ptr(out), _ptr(status),
                                           _stream(stream)), "dora_varlen_attn")


def dora_gather_scores(table, ids, cu, scores, status=None, stream=None):
    _req(table, torch.float32, "table")
    _req(scores, torch.float32, "scores")
    _req(ids, torch.int32, "ids")
    _req(cu, torch.int32, "cu")
    _req(status, torch.int32, "status", optional=True)
    _check(load_library().dora_gather_scores(_ptr(table), table.shape[-1], _ptr(ids), _ptr(cu),
                                             cu.numel() - 1, _ptr(scores), _ptr(status),
                                             _stream(stream)), "dora_gather_scores")


class BlockWeights:
    """Device weights of one block plus the C struct that points at them.

    ``tensors`` maps the names of ``dora_block_weights`` to bf16 CUDA tensors
    (linears in nn.Linear layout).  The tensors are kept alive here.
    """

    NAMES = ("ln1_w", "ln1_b", "w_qkv", "b_qkv", "w_proj", "b_proj", "ln2_w", "ln2_b", "w_fc1",
             "b_fc1", "w_fc2", "b_fc2")

    def __init__(self, tensors: dict, dim: int, heads: int, mlp_dim: int, ln_eps: float = 1e-6,
                 stream=None):
        """Optional ``ls1``/``ls2`` (bf16 [dim], DINOv2 LayerScale) are folded
        here, on ``stream``, into scaled copies of w_proj/b_proj and
        w_fc2/b_fc2 (dora_fold_layerscale); the given tensors are not changed."""
        self.tensors = {}
        for n in self.NAMES:
            t = tensors.get(n)
            _req(t, torch.bfloat16, n, optional=n.startswith("b_"))
            self.tensors[n] = t
        for ls, wn, bn in (("ls1", "w_proj", "b_proj"), ("ls2", "w_fc2", "b_fc2")):
            g = tensors.get(ls)
            if g is None:
                continue
            _req(g, torch.bfloat16, ls)
            w, b = self.tensors[wn], self.tensors[bn]
            if g.numel() != w.shape[0]:
                raise ValueError(f"{ls} must have {w.shape[0]} entries")
            self.tensors[wn], self.tensors[bn] = dora_fold_layerscale(w, b, g, stream=stream)
        self.dim, self.heads, self.mlp_dim, self.ln_eps = dim, heads, mlp_dim, ln_eps
        self.folded = None
        self.c = _BlockWeightsC(*[_ptr(self.tensors[n]) for n in self.NAMES], dim, heads, mlp_dim,
                                float(ln_eps), None)

    def fold(self, stream=None):
        """Fold both LayerNorms into the QKV and fc1 weights once
        (dora_fold_block_weights); later blocks run on the folded copy.
        Call again after changing any of the weights."""
        n = int(load_library().dora_folded_weights_size(ctypes.byref(self.c)))
        buf = torch.empty(n + 256, dtype=torch.uint8, device=self.tensors["w_qkv"].device)
        off = (-buf.data_ptr()) % 256
        folded = buf[off:off + n]
        self.c.folded = None
        _check(load_library().dora_fold_block_weights(ctypes.byref(self.c), _ptr(folded), n,
                                                      _stream(stream)),
               "dora_fold_block_weights")
        self.folded = folded
        self.c.folded = _ptr(folded)
        return self


def dora_workspace_size(t_cap, batch, weights: BlockWeights) -> int:
    return int(load_library().dora_workspace_size(int(t_cap), int(batch), ctypes.byref(weights.c)))


def alloc_workspace(t_cap, batch, weights: BlockWeights, device=None) -> torch.Tensor:
    """Zero-filled uint8 workspace (torch allocation, 256-byte aligned)."""
    n = dora_workspace_size(t_cap, batch, weights)
    return torch.zeros(n, dtype=torch.uint8, device=device or "cuda")


def dora_pruned_block(x_in, cu_in, weights: BlockWeights, max_seqlen, x_out, workspace,
                      ids_in=None, scores=None, keep_counts=None, cu_out=None, ids_out=None,
                      kept_idx=None, x_in_moments=None, x_out_moments=None, stream=None):
    """One block of Eq. 1 (dora_pruned_block).  x_in_moments / x_out_moments
    (fp32 [t_cap, 2], optional) carry the row moments from block to block so
    that the next block skips its pass over x_in."""
    _req(x_in, torch.bfloat16, "x_in")
    _req(x_out, torch.bfloat16, "x_out")
    _req(cu_in, torch.int32, "cu_in")
    _req(workspace, torch.uint8, "workspace")
    for n, t in (("ids_in", ids_in), ("keep_counts", keep_counts), ("cu_out", cu_out),
                 ("ids_out", ids_out), ("kept_idx", kept_idx)):
        _req(t, torch.int32, n, optional=True)
    _req(scores, torch.float32, "scores", optional=True)
    _req(x_in_moments, torch.float32, "x_in_moments", optional=True)
    _req(x_out_moments, torch.float32, "x_out_moments", optional=True)
    t_cap = x_in.shape[0]
    for t in (x_in_moments, x_out_moments):
        if t is not None and t.numel() < 2 * t_cap:
            raise ValueError("row moments must hold [t_cap, 2] floats")
    _check(load_library().dora_pruned_block(
        _ptr(x_in), _ptr(cu_in), _ptr(ids_in), cu_in.numel() - 1, int(max_seqlen), t_cap,
        ctypes.byref(weights.c), _ptr(scores), _ptr(keep_counts), _ptr(x_out), _ptr(cu_out),
        _ptr(ids_out), _ptr(kept_idx), _ptr(x_in_moments), _ptr(x_out_moments),
        _ptr(workspace), workspace.numel(), _stream(stream)),
        "dora_pruned_block")


def dora_pruned_block_noalloc(x_in, cu_in, weights: BlockWeights, max_seqlen, x_out,
                              ids_in=None, scores=None, keep_counts=None, cu_out=None,
                              ids_out=None, kept_idx=None, x_in_moments=None,
                              x_out_moments=None, status=None, stream=None):
    """dora_pruned_block without a workspace argument, for callers that cannot
    allocate device memory when they run the block: the intermediates live in
    a 32 MiB scratch array the library holds on each GPU.  Blocks needing more
    raise DoraError (DORA_ERR_SCRATCH_TOO_SMALL).  Calls on one device share
    that scratch, so keep them ordered on one stream.  ``status`` (optional
    int32 CUDA tensor) receives the block's device status word."""
    _req(x_in, torch.bfloat16, "x_in")
    _req(x_out, torch.bfloat16, "x_out")
    _req(cu_in, torch.int32, "cu_in")
    for n, t in (("ids_in", ids_in), ("keep_counts", keep_counts), ("cu_out", cu_out),
                 ("ids_out", ids_out), ("kept_idx", kept_idx), ("status", status)):
        _req(t, torch.int32, n, optional=True)
    _req(scores, torch.float32, "scores", optional=True)
    _req(x_in_moments, torch.float32, "x_in_moments", optional=True)
    _req(x_out_moments, torch.float32, "x_out_moments", optional=True)
    t_cap = x_in.shape[0]
    _check(load_library().dora_pruned_block_noalloc(
        _ptr(x_in), _ptr(cu_in), _ptr(ids_in), cu_in.numel() - 1, int(max_seqlen), t_cap,
        ctypes.byref(weights.c), _ptr(scores), _ptr(keep_counts), _ptr(x_out), _ptr(cu_out),
        _ptr(ids_out), _ptr(kept_idx), _ptr(x_in_moments), _ptr(x_out_moments), _ptr(status),
        _stream(stream)),
        "dora_pruned_block_noalloc")


def dora_workspace_status(workspace) -> int:
    """Device address of the status word inside a block workspace."""
    return int(load_library().dora_workspace_status(_ptr(workspace)))


def dora_read_status(status) -> int:
    """Synchronise and read a device status word (tensor or device address)."""
    code = ctypes.c_int32(0)
    _check(load_library().dora_read_status(_ptr(status), ctypes.byref(code)), "dora_read_status")
    return int(code.value)


# ---------------------------------------------------------------------------
# the deployment actor
# ---------------------------------------------------------------------------
_ACTOR_NAMES = ("gate_w1", "gate_b1", "gate_w2", "gate_b2", "gate_emb", "enc_w_in", "enc_b_in",
                "enc_emb", "enc_w_h", "enc_ln1_w", "enc_ln1_b", "enc_w_qkv", "enc_b_qkv",
                "enc_w_o", "enc_b_o", "enc_ln2_w", "enc_ln2_b", "enc_w_fc1", "enc_b_fc1",
                "enc_w_fc2", "enc_b_fc2", "bud_ln_w", "bud_ln_b", "bud_w1", "bud_b1", "bud_w2",
                "bud_b2", "sel_w_k", "sel_w1", "sel_b1", "sel_w2", "sel_b2")


class _ActorWeightsC(ctypes.Structure):
    _fields_ = [(n, _vp) for n in _ACTOR_NAMES] + [
        ("dim", _i32), ("depth", _i32), ("n0", _i32), ("eps", _f32), ("prepared", _vp)]


class ActorWeights:
    """Device weights of the actor (dora_actor_weights) plus the C struct that
    points at them.  ``tensors`` maps the struct's names to bf16 CUDA tensors;
    ``prepare()`` builds the encoder's folded and padded weights once."""

    NAMES = _ACTOR_NAMES

    def __init__(self, tensors: dict, dim: int, depth: int, n0: int, eps: float = 1e-5):
        self.tensors = {}
        for n in self.NAMES:
            t = tensors.get(n)
            _req(t, torch.bfloat16, n)
            self.tensors[n] = t.contiguous()
        self.dim, self.depth, self.n0, self.eps = dim, depth, n0, eps
        self.prepared = None
        self.c = _ActorWeightsC(*[_ptr(self.tensors[n]) for n in self.NAMES], dim, depth, n0,
                                float(eps), None)

    def prepare(self, stream=None):
        n = int(load_library().dora_actor_prepared_size(ctypes.byref(self.c)))
        buf = torch.empty(n + 256, dtype=torch.uint8, device=self.tensors["enc_w_in"].device)
        off = (-buf.data_ptr()) % 256
        prep = buf[off:off + n]
        self.c.prepared = None
        _check(load_library().dora_actor_prepare(ctypes.byref(self.c), _ptr(prep), n,
                                                 _stream(stream)), "dora_actor_prepare")
        self.prepared = buf
        self.c.prepared = _ptr(prep)
        return self


def dora_actor_workspace_size(t_cap, batch, weights: ActorWeights) -> int:
    return int(load_library().dora_actor_workspace_size(int(t_cap), int(batch),
                                                        ctypes.byref(weights.c)))


def alloc_actor_workspace(t_cap, batch, weights: ActorWeights, device=None) -> torch.Tensor:
    n = dora_actor_workspace_size(t_cap, batch, weights)
    return torch.zeros(n, dtype=torch.uint8, device=device or "cuda")


def dora_actor(qkv, cu, weights: ActorWeights, block, max_seqlen, rho, interventions, gate,
               budget, k, keep_counts, scores, workspace, p_gate=None, rho_next=None,
               interventions_next=None, z_out=None, stream=None):
    """The deterministic actor at one block (dora_actor): gate, budget, k,
    keep counts and deletion scores for every image of the packed batch."""
    _req(qkv, torch.bfloat16, "qkv")
    _req(cu, torch.int32, "cu")
    _req(workspace, torch.uint8, "workspace")
    for n, t, dt, opt in (("rho", rho, torch.float32, False),
                          ("interventions", interventions, torch.int32, False),
                          ("gate", gate, torch.int32, False), ("budget", budget, torch.int32, False),
                          ("k", k, torch.int32, False), ("keep_counts", keep_counts, torch.int32, False),
                          ("scores", scores, torch.float32, False),
                          ("p_gate", p_gate, torch.float32, True),
                          ("rho_next", rho_next, torch.float32, True),
                          ("interventions_next", interventions_next, torch.int32, True),
                          ("z_out", z_out, torch.bfloat16, True)):
        _req(t, dt, n, optional=opt)
    t_cap = qkv.shape[0]
    batch = cu.numel() - 1
    if qkv.shape[1] != 3 * weights.dim or scores.numel() < t_cap:
        raise ValueError("qkv must be [t_cap, 3 dim] and scores hold t_cap floats")
    if z_out is not None and tuple(z_out.shape) != (t_cap, 128):
        raise ValueError("z_out must be [t_cap, 128]")
    _check(load_library().dora_actor(
        _ptr(qkv), _ptr(cu), batch, int(max_seqlen), t_cap, int(block), ctypes.byref(weights.c),
        _ptr(rho), _ptr(interventions), _ptr(p_gate), _ptr(gate), _ptr(budget), _ptr(k),
        _ptr(keep_counts), _ptr(scores), _ptr(rho_next), _ptr(interventions_next), _ptr(z_out),
        _ptr(workspace), workspace.numel(), _stream(stream)), "dora_actor")


def dora_pruned_block_actor(x_in, cu_in, weights: BlockWeights, max_seqlen, x_out, workspace,
                            actor: ActorWeights, block, rho, interventions, gate, budget, k,
                            actor_keep, scores, actor_workspace, ids_in, cu_out, ids_out,
                            keep_counts=None, kept_idx=None, rho_next=None,
                            interventions_next=None, x_in_moments=None, x_out_moments=None,
                            stream=None):
    """dora_pruned_block with the actor deciding the deletion at this block
    (its scores; its keep counts unless ``keep_counts`` is given)."""
    _req(x_in, torch.bfloat16, "x_in")
    _req(x_out, torch.bfloat16, "x_out")
    for n, t in (("cu_in", cu_in), ("ids_in", ids_in), ("cu_out", cu_out), ("ids_out", ids_out),
                 ("interventions", interventions), ("gate", gate), ("budget", budget), ("k", k),
                 ("actor_keep", actor_keep)):
        _req(t, torch.int32, n)
    for n, t in (("keep_counts", keep_counts), ("kept_idx", kept_idx),
                 ("interventions_next", interventions_next)):
        _req(t, torch.int32, n, optional=True)
    _req(rho, torch.float32, "rho")
    _req(scores, torch.float32, "scores")
    for n, t in (("rho_next", rho_next), ("x_in_moments", x_in_moments),
                 ("x_out_moments", x_out_moments)):
        _req(t, torch.float32, n, optional=True)
    _req(workspace, torch.uint8, "workspace")
    _req(actor_workspace, torch.uint8, "actor_workspace")
    t_cap = x_in.shape[0]
    _check(load_library().dora_pruned_block_actor(
        _ptr(x_in), _ptr(cu_in), _ptr(ids_in), cu_in.numel() - 1, int(max_seqlen), t_cap,
        ctypes.byref(weights.c), _ptr(x_out), _ptr(cu_out), _ptr(ids_out), _ptr(kept_idx),
        _ptr(x_in_moments), _ptr(x_out_moments), _ptr(workspace), workspace.numel(),
        ctypes.byref(actor.c), int(block), _ptr(rho), _ptr(interventions), _ptr(keep_counts),
        _ptr(gate), _ptr(budget), _ptr(k), _ptr(actor_keep), _ptr(scores), _ptr(rho_next),
        _ptr(interventions_next), _ptr(actor_workspace), actor_workspace.numel(),
        _stream(stream)), "dora_pruned_block_actor")


# ---------------------------------------------------------------------------
# the forward's two ends
# ---------------------------------------------------------------------------

def dora_patch_embed(images, w_pe, b_pe, cls, pos, patch, x0, workspace=None, stream=None):
    """Packed tokens x0 [B * (g + 1), d] from images [B, C, H, W]: strided patch
    convolution (w_pe [d, C * patch^2]), CLS first, position embeddings added.

    The C entry point never allocates.  This wrapper does when ``workspace``
    is None: it then makes a zero-filled uint8 tensor of
    ``dora_embed_workspace_size`` bytes with torch on every such call.  The
    workspace used is returned; pass it back on later calls to keep a loop
    free of allocations."""
    for n, t in (("images", images), ("w_pe", w_pe), ("cls", cls), ("pos", pos), ("x0", x0)):
        _req(t, torch.bfloat16, n)
    _req(b_pe, torch.bfloat16, "b_pe", optional=True)
    b, c, h, w = images.shape
    d = w_pe.shape[0]
    n = int(load_library().dora_embed_workspace_size(b, c, h, w, int(patch), d))
    if workspace is None:
        workspace = torch.zeros(n, dtype=torch.uint8, device=images.device)
    _req(workspace, torch.uint8, "workspace")
    g = (h // patch) * (w // patch)
    if tuple(x0.shape) != (b * (g + 1), d) or tuple(pos.shape) != (g + 1, d):
        raise ValueError("x0 must be [B * (g + 1), d] and pos [g + 1, d]")
    _check(load_library().dora_patch_embed(_ptr(images), b, c, h, w, int(patch), d, _ptr(w_pe),
                                           _ptr(b_pe), _ptr(cls), _ptr(pos), _ptr(x0),
                                           _ptr(workspace), workspace.numel(), _stream(stream)),
           "dora_patch_embed")
    return workspace


def dora_fold_layerscale(w, b, gamma, w_out=None, b_out=None, stream=None):
    """(bf16(gamma_i w[i, :]), bf16(gamma_i b_i)): LayerScale folded into a
    linear's rows.  Outputs are allocated when not given; b may be None."""
    _req(w, torch.bfloat16, "w")
    _req(gamma, torch.bfloat16, "gamma")
    _req(b, torch.bfloat16, "b", optional=True)
    n, k = w.shape
    w_out = torch.empty_like(w) if w_out is None else w_out
    if b is not None and b_out is None:
        b_out = torch.empty_like(b)
    _check(load_library().dora_fold_layerscale(_ptr(w), _ptr(b), _ptr(gamma), n, k, _ptr(w_out),
                                               _ptr(b_out) if b is not None else None,
                                               _stream(stream)), "dora_fold_layerscale")
    return w_out, b_out


def dora_classifier_head_lc1(x, cu, norm_w, norm_b, eps, w_head, b_head, logits, workspace=None,
                             stream=None):
    """logits [B, classes] from DINOv2's LC1 features [LN(CLS), mean LN(visual
    rows)] of each image (w_head [classes, 2 d], classes a multiple of 32).

    With ``workspace`` None a zero-filled workspace of
    ``dora_head_lc1_workspace_size`` bytes is allocated with torch on that
    call; the workspace used is returned for reuse (the C entry point itself
    never allocates)."""
    for n, t in (("x", x), ("norm_w", norm_w), ("norm_b", norm_b), ("w_head", w_head),
                 ("logits", logits)):
        _req(t, torch.bfloat16, n)
    _req(b_head, torch.bfloat16, "b_head", optional=True)
    _req(cu, torch.int32, "cu")
    t_cap, d = x.shape
    b = cu.numel() - 1
    classes = w_head.shape[0]
    if tuple(w_head.shape) != (classes, 2 * d) or tuple(logits.shape) != (b, classes):
        raise ValueError("w_head must be [classes, 2 d] and logits [B, classes]")
    n = int(load_library().dora_head_lc1_workspace_size(b, d))
    if workspace is None:
        workspace = torch.zeros(n, dtype=torch.uint8, device=x.device)
    _req(workspace, torch.uint8, "workspace")
    _check(load_library().dora_classifier_head_lc1(_ptr(x), _ptr(cu), b, t_cap, d, _ptr(norm_w),
                                                   _ptr(norm_b), float(eps), _ptr(w_head),
                                                   _ptr(b_head), classes, _ptr(logits),
                                                   _ptr(workspace), workspace.numel(),
                                                   _stream(stream)), "dora_classifier_head_lc1")
    return workspace


def dora_classifier_head(x, cu, norm_w, norm_b, eps, w_head, b_head, logits, workspace=None,
                         stream=None):
    """logits [B, classes] = LayerNorm(x[cu[i]]) W_head^T + b_head per image
    (classes a multiple of 32: pad the head with zero rows).

    With ``workspace`` None a zero-filled workspace of
    ``dora_head_workspace_size`` bytes is allocated with torch on that call;
    the workspace used is returned for reuse (the C entry point itself never
    allocates)."""
    for n, t in (("x", x), ("norm_w", norm_w), ("norm_b", norm_b), ("w_head", w_head),
                 ("logits", logits)):
        _req(t, torch.bfloat16, n)
    _req(b_head, torch.bfloat16, "b_head", optional=True)
    _req(cu, torch.int32, "cu")
    t_cap, d = x.shape
    b = cu.numel() - 1
    classes = w_head.shape[0]
    n = int(load_library().dora_head_workspace_size(b, d))
    if workspace is None:
        workspace = torch.zeros(n, dtype=torch.uint8, device=x.device)
    _req(workspace, torch.uint8, "workspace")
    if tuple(logits.shape) != (b, classes):
        raise ValueError("logits must be [B, classes]")
    _check(load_library().dora_classifier_head(_ptr(x), _ptr(cu), b, t_cap, d, _ptr(norm_w),
                                               _ptr(norm_b), float(eps), _ptr(w_head),
                                               _ptr(b_head), classes, _ptr(logits),
                                               _ptr(workspace), workspace.numel(),
                                               _stream(stream)), "dora_classifier_head")
    return workspace


# ---------------------------------------------------------------------------
# training side: Plackett-Luce sampling and log-probability, shadow branching,
# fidelity cost
# ---------------------------------------------------------------------------

def dora_pl_sample(scores, gumbel, cu, k, order, keys_out=None, status=None, stream=None):
    """Gumbel-top-k removal sequences: order int32 [B, k_cap] (-1 past k_i);
    keys_out (fp32, row-aligned) receives the perturbed keys s + g."""
    _req(scores, torch.float32, "scores")
    _req(gumbel, torch.float32, "gumbel")
    _req(cu, torch.int32, "cu")
    _req(k, torch.int32, "k")
    _req(order, torch.int32, "order")
    _req(keys_out, torch.float32, "keys_out", optional=True)
    b = cu.numel() - 1
    if order.dim() != 2 or order.shape[0] != b or k.numel() != b:
        raise ValueError("order must be [B, k_cap] and k [B]")
    _check(load_library().dora_pl_sample(_ptr(scores), _ptr(gumbel), _ptr(cu), b, scores.numel(),
                                         _ptr(k), order.shape[1], _ptr(order), _ptr(keys_out),
                                         _ptr(status), _stream(stream)), "dora_pl_sample")
    return order


def dora_pl_logprob(scores, cu, k, order, logp, grad=None, dlogp=None, status=None, stream=None):
    """Plackett-Luce log-probabilities logp [B] and, optionally, their gradient
    with respect to the row-aligned scores (times dlogp)."""
    _req(scores, torch.float32, "scores")
    _req(cu, torch.int32, "cu")
    _req(k, torch.int32, "k")
    _req(order, torch.int32, "order")
    _req(logp, torch.float32, "logp")
    _req(grad, torch.float32, "grad", optional=True)
    _req(dlogp, torch.float32, "dlogp", optional=True)
    b = cu.numel() - 1
    if order.dim() != 2 or order.shape[0] != b or logp.numel() != b:
        raise ValueError("order must be [B, k_cap] and logp [B]")
    if grad is not None and grad.numel() != scores.numel():
        raise ValueError("grad must match scores")
    _check(load_library().dora_pl_logprob(_ptr(scores), _ptr(cu), b, scores.numel(), _ptr(k),
                                          _ptr(order), order.shape[1], _ptr(logp), _ptr(grad),
                                          _ptr(dlogp), _ptr(status), _stream(stream)),
           "dora_pl_logprob")
    return logp


def dora_branch(x, cu, src, cu_out, ids=None, x_moments=None, len_out=None, status=None,
                stream=None):
    """Append copies of sequences src (device int32) after row cu[-1] of x,
    in place; cu_out [B + 1 + len(src)]."""
    _req(x, torch.bfloat16, "x")
    _req(cu, torch.int32, "cu")
    _req(src, torch.int32, "src")
    _req(cu_out, torch.int32, "cu_out")
    _req(ids, torch.int32, "ids", optional=True)
    _req(x_moments, torch.float32, "x_moments", optional=True)
    _req(len_out, torch.int32, "len_out", optional=True)
    b, nb = cu.numel() - 1, src.numel()
    if cu_out.numel() < b + 1 + nb:
        raise ValueError("cu_out needs B + 1 + len(src) entries")
    t_cap, d = x.shape
    _check(load_library().dora_branch(_ptr(x), _ptr(ids), _ptr(x_moments), _ptr(cu), b, t_cap, d,
                                      _ptr(src), nb, _ptr(cu_out), _ptr(len_out), _ptr(status),
                                      _stream(stream)), "dora_branch")
    return cu_out


def dora_kd_cost(z_native, z, cost, classes, shadow_image=None, tau=3.0, status=None,
                 stream=None):
    """Fidelity costs [S]: tau^2 KL(softmax(z_native[img] / tau) || softmax(z[s] / tau))
    over the first `classes` logits of each row."""
    _req(z_native, torch.bfloat16, "z_native")
    _req(z, torch.bfloat16, "z")
    _req(cost, torch.float32, "cost")
    _req(shadow_image, torch.int32, "shadow_image", optional=True)
    if z.shape[1] != z_native.shape[1] or cost.numel() != z.shape[0]:
        raise ValueError("z and z_native need the same row pitch; cost one entry per row of z")
    _check(load_library().dora_kd_cost(_ptr(z_native), _ptr(z), _ptr(shadow_image), z.shape[0],
                                       z_native.shape[0], int(classes), z.shape[1], float(tau),
                                       _ptr(cost), _ptr(status), _stream(stream)), "dora_kd_cost")
    return cost


def dora_step_rewards(cost, removals, blocks, depth, n0, a, reward, ret=None, stream=None):
    """Local rewards [P, B] (and episode sums [B]) from a batched shadow
    forward's fidelity costs (rollout, Native, shadows) and the removal
    counts [P, B] at the pruning blocks (device int32 [P])."""
    _req(cost, torch.float32, "cost")
    _req(removals, torch.int32, "removals")
    _req(blocks, torch.int32, "blocks")
    _req(reward, torch.float32, "reward")
    _req(ret, torch.float32, "ret", optional=True)
    p, b = removals.shape
    if blocks.numel() != p or tuple(reward.shape) != (p, b) or cost.numel() < (p + 1) * b:
        raise ValueError("removals and reward must be [P, B], blocks [P], cost >= (P + 1) B")
    _check(load_library().dora_step_rewards(_ptr(cost), _ptr(removals), _ptr(blocks), p, b,
                                            int(depth), int(n0), float(a), _ptr(reward),
                                            _ptr(ret), _stream(stream)), "dora_step_rewards")
    return reward

