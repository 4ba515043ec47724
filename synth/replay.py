"""Replay driver for the multi-batch agent traces (configs 1-3).

Between batches the serving cluster changes state: the routed requests'
blocks enter the chosen instance's local KV$ tier (and the global tier when
the workload has one), capped tiers evict least-recently-used blocks, and the
instances drain their queues. This module is that workload policy. It is not
part of the routing method: it only turns one batch's routing outputs into the
next batch's inputs (index insert/evict lists and the per-instance load), so a
GPU replay and an oracle replay each drive their own copy from their own
outputs.

Recency order: a block touched by request r of batch k at block position b
has stamp (k, r, -b); the smallest stamp is evicted first, so within one
request the deepest blocks leave first and prefixes survive.
"""

from __future__ import annotations

from collections import OrderedDict
from typing import Optional

import numpy as np

GLOBAL_TIER = -1


class ReplayDriver:
    def __init__(self, num_instances: int, block_size: int, *, local_cap: Optional[int] = None,
                 global_policy: str = "none", global_cap: Optional[int] = None):
        if global_policy not in ("none", "all", "lru"):
            raise ValueError(global_policy)
        self.N = num_instances
        self.B = block_size
        self.local_cap = local_cap
        self.global_policy = global_policy
        self.global_cap = global_cap
        self.load = np.zeros(num_instances, dtype=np.int64)
        self.local_lru = [OrderedDict() for _ in range(num_instances)]
        self.global_lru: OrderedDict = OrderedDict()
        self.batch_index = 0

    def after_batch(self, offsets: np.ndarray, instance: np.ndarray, local_hit: np.ndarray,
                    block_hashes: np.ndarray):
        """Consume one batch's routing outputs.

        offsets:      int64 [n+1] token offsets of the batch
        instance:     int32 [n] chosen instance per request
        local_hit:    int32 [n] local-hit tokens on the chosen instance
        block_hashes: uint64 [sum n_r] full-block hashes, request-major

        Returns (insert_keys, insert_tiers, evict_keys, evict_tiers); apply the
        inserts, then the evictions. Updates self.load in place with the
        drain rule load_i <- (load_i + sum over requests routed to i of the
        tokens i must prefill or fetch) >> 1.
        """
        B = self.B
        lens = np.diff(offsets)
        nblk = lens // B
        bstart = np.concatenate([[0], np.cumsum(nblk)])
        ins_keys, ins_tiers = [], []
        for r in range(len(lens)):
            keys = block_hashes[bstart[r]:bstart[r + 1]]
            if len(keys) == 0:
                continue
            i = int(instance[r])
            rev = keys[::-1].tolist()  # deepest block first: oldest stamp within r
            lru = self.local_lru[i]
            for key in rev:
                lru.pop(key, None)
                lru[key] = None
            ins_keys.append(keys)
            ins_tiers.append(np.full(len(keys), i, dtype=np.int32))
            if self.global_policy != "none":
                if self.global_policy == "lru":
                    g = self.global_lru
                    for key in rev:
                        g.pop(key, None)
                        g[key] = None
                ins_keys.append(keys)
                ins_tiers.append(np.full(len(keys), GLOBAL_TIER, dtype=np.int32))
        ev_keys, ev_tiers = [], []
        if self.local_cap is not None:
            for i, lru in enumerate(self.local_lru):
                over = len(lru) - self.local_cap
                if over > 0:
                    victims = [lru.popitem(last=False)[0] for _ in range(over)]
                    ev_keys.append(np.array(victims, dtype=np.uint64))
                    ev_tiers.append(np.full(over, i, dtype=np.int32))
        if self.global_policy == "lru" and self.global_cap is not None:
            over = len(self.global_lru) - self.global_cap
            if over > 0:
                victims = [self.global_lru.popitem(last=False)[0] for _ in range(over)]
                ev_keys.append(np.array(victims, dtype=np.uint64))
                ev_tiers.append(np.full(over, GLOBAL_TIER, dtype=np.int32))
        # queue drain: tokens the chosen instance must prefill or fetch
        work = lens - np.asarray(local_hit, dtype=np.int64)
        added = np.bincount(np.asarray(instance, dtype=np.int64), weights=work,
                            minlength=self.N).astype(np.int64)
        self.load = (self.load + added) >> 1
        self.batch_index += 1
        cat = lambda xs, dt: np.concatenate(xs).astype(dt) if xs else np.zeros(0, dtype=dt)
        return (cat(ins_keys, np.uint64), cat(ins_tiers, np.int32),
                cat(ev_keys, np.uint64), cat(ev_tiers, np.int32))
