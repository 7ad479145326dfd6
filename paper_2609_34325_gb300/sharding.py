"""Split a packed batch across ranks by image.

Images never attend to one another (Sec. 3.5: sequence boundaries prevent
attention between different images) and every later step is per row, so a
packed batch shards into contiguous image ranges with no exchange: each rank
runs the whole hot path on its own images and nothing is communicated on the
data path.
"""
from __future__ import annotations

import numpy as np


def image_range(batch: int, rank: int, world: int) -> tuple:
    """Contiguous [lo, hi) image range of ``rank``; sizes differ by at most 1."""
    if world <= 0 or not 0 <= rank < world:
        raise ValueError("bad rank/world")
    base, extra = divmod(batch, world)
    lo = rank * base + min(rank, extra)
    return lo, lo + base + (1 if rank < extra else 0)


def shard_packed(cu: np.ndarray, rank: int, world: int) -> dict:
    """The rank's images, its row range in the packed buffer and its local
    ``cu_seqlens`` (rebased to start at 0)."""
    cu = np.asarray(cu, dtype=np.int64)
    lo, hi = image_range(len(cu) - 1, rank, world)
    r0, r1 = int(cu[lo]), int(cu[hi])
    return {"images": (lo, hi), "rows": (r0, r1),
            "cu_local": (cu[lo:hi + 1] - r0).astype(np.int32)}
