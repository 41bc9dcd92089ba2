"""Partition of the (b, h) slices of one forward call across ranks.

The (b, h) problems of Eq. attention are independent two-dimensional problems (the Remark in
Section 4.2, Eq. batched_mm), so a call over B*H slices splits across G ranks with no exchange
step: rank r owns a contiguous range [lo, hi) of the flattened B*H axis of Q, K, V and O
([B, H, N, d] contiguous, so a slice range is one contiguous block of each tensor) and runs the
forward on that block alone.  This module holds only that index arithmetic, no attention step.
"""
from __future__ import annotations


def bh_range(n_slices: int, world: int, rank: int) -> tuple[int, int]:
    """[lo, hi) of the slices rank `rank` of `world` owns: contiguous, sizes differing by at most
    one, the larger ranges first; empty when there are more ranks than slices."""
    if n_slices < 0 or world < 1 or not 0 <= rank < world:
        raise ValueError(f"bad partition request: {n_slices} slices, rank {rank} of {world}")
    base, extra = divmod(n_slices, world)
    lo = rank * base + min(rank, extra)
    return lo, lo + base + (1 if rank < extra else 0)


def bh_ranges(n_slices: int, world: int) -> list[tuple[int, int]]:
    """The ranges of every rank, in rank order."""
    return [bh_range(n_slices, world, r) for r in range(world)]


def slice_offset(lo: int, rows: int, d: int) -> int:
    """Element offset of slice `lo` in a contiguous [B*H, rows, d] tensor."""
    return lo * rows * d


def slice_numel(lo: int, hi: int, rows: int, d: int) -> int:
    """Elements of slices [lo, hi) of a contiguous [B*H, rows, d] tensor."""
    return (hi - lo) * rows * d


def block(arr, lo: int, hi: int):
    """Slices [lo, hi) of a [B, H, N, d] array as a contiguous [1, hi - lo, N, d] array (a numpy
    copy; for a contiguous torch tensor use block_view)."""
    import numpy as np
    a = np.asarray(arr)
    bh = a.shape[0] * a.shape[1]
    return np.ascontiguousarray(a.reshape(bh, *a.shape[2:])[lo:hi].reshape(1, hi - lo, *a.shape[2:]))


def block_view(t, lo: int, hi: int):
    """Slices [lo, hi) of a contiguous [B, H, N, d] torch tensor as a [1, hi - lo, N, d] view: the
    same memory at element offset slice_offset(lo, N, d), no copy."""
    B, H, N, d = t.shape
    if not t.is_contiguous():
        raise ValueError("block_view needs a contiguous tensor")
    return t.view(B * H, N, d)[lo:hi].view(1, hi - lo, N, d)
