"""Splitting a batch of rows over ranks (one GPU each).

Rows are independent, so a batch splits into contiguous blocks of rows with
no exchange between ranks: dense rows into blocks of near-equal row counts,
ragged rows into blocks of near-equal element counts (cut where the running
length crosses k/world of the total), each with its offsets rebased to start
at 0 so the block is a ragged batch of its own.  Host logic only: the blocks
are views of the caller's arrays and no device memory is touched.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np


def dense_block(rows: int, world: int, rank: int) -> tuple[int, int]:
    """Rows [lo, hi) of `rank` among `world` ranks: counts differ by at most
    one, lower ranks take the extra rows."""
    if world < 1 or not 0 <= rank < world or rows < 0:
        raise ValueError("need world >= 1, 0 <= rank < world and rows >= 0")
    base, extra = divmod(rows, world)
    lo = rank * base + min(rank, extra)
    return lo, lo + base + (1 if rank < extra else 0)


@dataclass
class RaggedBlock:
    row_lo: int          # first row of the block in the whole batch
    row_hi: int          # one past its last row
    elem_lo: int         # offsets[row_lo]: where its elements start
    elem_hi: int         # offsets[row_hi]
    offsets: np.ndarray  # int64 [row_hi - row_lo + 1], rebased to start at 0

    @property
    def rows(self) -> int:
        return self.row_hi - self.row_lo

    @property
    def elements(self) -> int:
        return self.elem_hi - self.elem_lo


def ragged_cuts(offsets, world: int) -> np.ndarray:
    """Row boundaries [world + 1] that split the rows into `world` contiguous
    blocks of near-equal element counts: boundary k is the first row whose
    start is at or past k/world of the elements (so a block's elements differ
    from the even share by less than one row's length)."""
    off = np.asarray(offsets, dtype=np.int64).reshape(-1)
    if world < 1:
        raise ValueError("world must be >= 1")
    if off.shape[0] < 1 or np.any(np.diff(off) < 0):
        raise ValueError("offsets must be a non-decreasing array of rows + 1 entries")
    rows = off.shape[0] - 1
    total = int(off[-1] - off[0])
    targets = off[0] + (np.arange(world + 1, dtype=np.int64) * total) // world
    cuts = np.searchsorted(off[:rows], targets, side="left").astype(np.int64)
    cuts[0], cuts[-1] = 0, rows
    return np.maximum.accumulate(np.minimum(cuts, rows))


def ragged_block(offsets, world: int, rank: int) -> RaggedBlock:
    """The block of `rank` among `world` ranks (see ragged_cuts)."""
    if not 0 <= rank < world:
        raise ValueError("need 0 <= rank < world")
    off = np.asarray(offsets, dtype=np.int64).reshape(-1)
    cuts = ragged_cuts(off, world)
    lo, hi = int(cuts[rank]), int(cuts[rank + 1])
    return RaggedBlock(lo, hi, int(off[lo]), int(off[hi]), off[lo:hi + 1] - off[lo])
