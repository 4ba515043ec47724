"""Host-side sharding of the routing path across GPUs (one process per GPU).

Under snapshot semantics every request of a batch is routed independently,
so a batch splits across ranks by request with no exchange on the data path:
each rank holds a replica of the index, routes its contiguous slice of
requests and writes its slice of the outputs. These helpers compute the
slices; they hold no routing arithmetic.
"""

from __future__ import annotations

import numpy as np


def request_range(n_requests: int, rank: int, world: int) -> tuple[int, int]:
    """Contiguous request slice [lo, hi) of `rank`; sizes differ by at most one."""
    if world < 1 or not 0 <= rank < world:
        raise ValueError("rank must be in [0, world)")
    base, extra = divmod(n_requests, world)
    lo = rank * base + min(rank, extra)
    return lo, lo + base + (1 if rank < extra else 0)


def shard_batch(tokens: np.ndarray, offsets: np.ndarray, rank: int, world: int):
    """This rank's sub-batch: (tokens view, offsets rebased to 0, request lo, hi)."""
    lo, hi = request_range(len(offsets) - 1, rank, world)
    t0, t1 = int(offsets[lo]), int(offsets[hi])
    return tokens[t0:t1], (offsets[lo:hi + 1] - t0).astype(np.int64), lo, hi


def rank_batches(rank: int, world: int, count: int) -> list[int]:
    """Ids of the `count` batches rank routes when every rank streams its own
    batches (weak scaling): rank, rank + world, rank + 2 world, ..."""
    return [rank + world * i for i in range(count)]
