"""Helpers for the GPU parity tests: run the CUDA path through the C ABI and
the CPU oracle on the same seeded inputs and compare element by element."""

from __future__ import annotations

import itertools

import numpy as np
import torch

import oracle
import paper_2607_08565_gb300 as pkg
from synth import ReplayDriver
from synth.traces import pack

DEV = torch.device("cuda:0")
FIELDS = ("instance", "local_hit", "global_hit", "session_key")


def T(a, dtype=None):
    t = torch.from_numpy(np.ascontiguousarray(a))
    return t.to(DEV) if dtype is None else t.to(DEV, dtype)


def make_index(N, B, S, cap=1 << 14, max_req=4096, max_tok=1 << 22, seed=0, host_staging=False):
    return pkg.SMetricIndex(N, B, S, capacity_slots=cap, max_batch_requests=max_req,
                            max_batch_tokens=max_tok, hash_seed=seed, host_staging=host_staging)


def n_blocks(offsets, B):
    return int((np.diff(offsets) // B).sum())


def gpu_route(ix, tokens, offsets, load, w, want_hashes=True):
    out = ix.route_batch(T(tokens), T(offsets), T(np.asarray(load, np.int64)), w, want_hashes)
    ix.check()
    res = {k: v.cpu().numpy() for k, v in out.items()}
    if want_hashes:
        res["block_hashes"] = res["block_hashes"][:n_blocks(offsets, ix.B)]
    return res


def gpu_hashes(ix, tokens, offsets):
    hb, sk = ix.block_hashes(T(tokens), T(offsets))
    ix.check()
    return hb.cpu().numpy()[:n_blocks(offsets, ix.B)], sk.cpu().numpy()


def assert_outputs_equal(g, o, fields=FIELDS + ("block_hashes",), ctx=""):
    for f in fields:
        if f not in o:
            continue
        a = np.asarray(g[f]).astype(o[f].dtype)
        b = o[f]
        assert a.shape == b.shape, (ctx, f, a.shape, b.shape)
        bad = np.nonzero(a != b)[0]
        assert len(bad) == 0, f"{ctx} field {f}: {len(bad)} mismatches, first at {bad[:5]}: " \
                              f"gpu {a[bad[:5]]} oracle {b[bad[:5]]}"


def replay_both(trace, n_batches=None, cap=None, n_threads=8, shared_driver=False):
    """Replay an agent trace through the GPU and through the oracle, each
    side driving its own index from its own outputs; compare every batch.

    With shared_driver, one replay driver serves both sides: every batch's
    outputs are asserted equal before the driver consumes them, so the two
    drivers would receive identical inputs and produce identical insert and
    evict lists; sharing halves the host-side LRU work of the long replays."""
    p = trace.params
    batches = list(itertools.islice(trace.batches(), n_batches))
    total_blocks = sum(n_blocks(b.offsets, p.block_size) for b in batches)
    cap = cap or max(1024, int(total_blocks / 0.5))
    ix = make_index(p.num_instances, p.block_size, p.session_blocks, cap=cap,
                    max_req=max(b.n_requests for b in batches),
                    max_tok=max(b.n_tokens for b in batches), seed=p.hash_seed)
    ox = oracle.OracleIndex(p.num_instances)
    kw = dict(local_cap=trace.local_cap, global_policy=trace.global_policy, global_cap=trace.global_cap)
    dg = ReplayDriver(p.num_instances, p.block_size, **kw)
    do = dg if shared_driver else ReplayDriver(p.num_instances, p.block_size, **kw)
    w = (p.w_load, p.w_miss, p.w_glob)
    stats = dict(batches=0, requests=0, local=0, glob=0, evicted=0)
    for k, bt in enumerate(batches):
        g = gpu_route(ix, bt.tokens, bt.offsets, dg.load, w)
        o = ox.route_batch(p.block_size, p.session_blocks, p.hash_seed, bt.tokens, bt.offsets,
                           do.load, *w, want_hashes=True, n_threads=n_threads)
        assert_outputs_equal(g, o, ctx=f"{trace.name} batch {k}")
        ik, it_, ek, et = dg.after_batch(bt.offsets, g["instance"], g["local_hit"], g["block_hashes"])
        if len(ik):
            ix.insert(T(ik), T(it_))
        if len(ek):
            ix.evict(T(ek), T(et))
        ix.check()
        if not shared_driver:
            ik, it_, ek, et = do.after_batch(bt.offsets, o["instance"], o["local_hit"], o["block_hashes"])
        ox.insert(ik, it_)
        ox.evict(ek, et)
        assert np.array_equal(dg.load, do.load)
        stats["batches"] += 1
        stats["requests"] += bt.n_requests
        stats["local"] += int(o["local_hit"].sum())
        stats["glob"] += int(o["global_hit"].sum())
        stats["evicted"] += len(ek)
    ix.close()
    return stats


def tiny_alphabet_case(rng, N, B, n_req, alphabet=3, max_blocks=10, n_stored=3):
    """Prompts over a tiny alphabet so that block prefixes are widely shared.
    Returns (stored prompts per tier, request list)."""
    base = rng.integers(0, alphabet, size=max_blocks * B, dtype=np.int32)

    def mutate(n_tokens):
        keep = int(rng.integers(0, min(len(base), n_tokens) + 1))
        return np.concatenate([base[:keep],
                               rng.integers(0, alphabet, size=n_tokens - keep, dtype=np.int32)])

    stored = {t: [mutate(int(rng.integers(0, (max_blocks + 1) * B)))
                  for _ in range(int(rng.integers(0, n_stored + 1)))] for t in range(-1, N)}
    reqs = [mutate(int(rng.integers(0, (max_blocks + 1) * B))) for _ in range(n_req)]
    return stored, reqs


def populate_both(ix, ox, stored, B, seed=0):
    """Insert every stored prompt's full blocks into its tier: the GPU index
    with hashes from the CUDA path, the oracle index with its own hashes."""
    keys_g, tiers_g = [], []
    for t, prompts in stored.items():
        for pr in prompts:
            if len(pr) < B:
                continue
            tok, off = pack([pr])
            hb, _ = gpu_hashes(ix, tok, off)
            keys_g.append(hb)
            tiers_g.append(np.full(len(hb), t, np.int32))
            ox.insert(oracle.block_hashes(pr, B, seed), t)
    if keys_g:
        ix.insert(T(np.concatenate(keys_g)), T(np.concatenate(tiers_g)))
        ix.check()
