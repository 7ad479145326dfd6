"""Shared helpers for the GPU parity tests: host<->device marshalling of the
seeded inputs and the tolerance rule."""
import numpy as np
import torch

ATOL = 2e-2   # absolute bound for bf16-in / fp32-accumulate outputs
RTOL = 1e-2   # relative bound; an element passes if either holds


def dev():
    return torch.device("cuda:0")


def bf(a: np.ndarray) -> torch.Tensor:
    """uint16 bf16 bits (numpy) -> bfloat16 CUDA tensor, bit for bit."""
    a = np.ascontiguousarray(a, dtype=np.uint16)
    return torch.from_numpy(a.view(np.int16)).view(torch.bfloat16).to(dev())


def i32(a) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.int32)).to(dev())


def f32(a) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(dev())


def bits(t: torch.Tensor) -> np.ndarray:
    """bfloat16 CUDA tensor -> numpy uint16 bits."""
    return t.detach().cpu().view(torch.int16).numpy().view(np.uint16)


def f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().astype(np.float64)


def assert_close(got: np.ndarray, ref: np.ndarray, what: str = "", atol=ATOL, rtol=RTOL):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (what, got.shape, ref.shape)
    err = np.abs(got - ref)
    ok = (err <= atol) | (err <= rtol * np.abs(ref))
    big = np.abs(ref) >= 1e-3
    max_rel = float((err[big] / np.abs(ref[big])).max()) if big.any() else 0.0
    if not ok.all():
        idx = np.argwhere(~ok)[:5]
        raise AssertionError(
            f"{what}: {int((~ok).sum())} of {ok.size} outside tolerance; max abs "
            f"{err.max():.3e}, max rel {max_rel:.3e}; first bad {idx.tolist()} "
            f"got {got[tuple(idx[0])]:.5f} ref {ref[tuple(idx[0])]:.5f}")
    return float(err.max()) if err.size else 0.0, max_rel


def sub_batch(cu: np.ndarray, images):
    """Rows of the chosen images and their local cu_seqlens."""
    rows = np.concatenate([np.arange(cu[i], cu[i + 1]) for i in images]).astype(np.int64)
    lens = [int(cu[i + 1] - cu[i]) for i in images]
    lcu = np.zeros(len(images) + 1, dtype=np.int64)
    lcu[1:] = np.cumsum(lens)
    return rows, lcu
