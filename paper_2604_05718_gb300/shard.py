"""Splitting a packed batch of images across ranks (one GPU per rank).

Images are independent (Section 3.1 of the paper: batches are processed
independently), so a batch shards by images with no exchange on the data
path: each rank merges, composes and gathers its own images, and the
per-rank outputs concatenate to the single-GPU result.  Ranges are
contiguous, so a rank's tokens, maps and offsets are plain slices of the
global packed arrays.  Work per image grows like N_b^2 * D (the affinity
pass), so ranges are balanced on sum(N_b^2) rather than on image count.
"""

from __future__ import annotations

from dataclasses import dataclass

import numpy as np


@dataclass(frozen=True)
class Shard:
    """Rank's share of a packed batch: images [image_start, image_end)."""

    image_start: int
    image_end: int
    row_start: int
    row_end: int

    def local_offsets(self, offsets: np.ndarray) -> np.ndarray:
        """Offsets of the shard's images relative to its first row."""
        return np.asarray(offsets[self.image_start:self.image_end + 1], dtype=np.int64) - self.row_start


def partition_images(sizes, world: int) -> list:
    """Contiguous image ranges, one per rank, balanced on sum(N_b^2).

    Greedy over the prefix of costs: rank r ends where the prefix first
    reaches (r + 1) / world of the total.  Every image goes to exactly one
    rank; a rank may be empty when there are fewer images than ranks.
    """
    if world < 1:
        raise ValueError("world must be >= 1")
    sizes = np.asarray(sizes, dtype=np.float64)
    cost = np.cumsum(sizes * sizes)
    total = cost[-1] if cost.size else 0.0
    bounds = [0]
    for r in range(1, world):
        target = total * r / world
        cut = int(np.searchsorted(cost, target, side="left")) + 1 if total > 0 else 0
        cut = min(max(cut, bounds[-1]), len(sizes))
        bounds.append(cut)
    bounds.append(len(sizes))
    return [(bounds[r], bounds[r + 1]) for r in range(world)]


def shard_for_rank(offsets, rank: int, world: int) -> Shard:
    """The shard of `rank` for a packed batch with the given offsets."""
    offsets = np.asarray(offsets, dtype=np.int64)
    ranges = partition_images(np.diff(offsets), world)
    a, b = ranges[rank]
    return Shard(a, b, int(offsets[a]), int(offsets[b]))
