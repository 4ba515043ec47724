"""ctypes binding of the CPU oracle (``smetric_oracle.c``).

TEST INFRASTRUCTURE ONLY: the test suite, the package smoke check and the
benchmark's CPU-baseline leg may import this module; the product path never
does. The oracle shares no code with the CUDA path. ``build()`` compiles it
with gcc into ``oracle/_build/liboracle.so``.
"""

from __future__ import annotations

import ctypes as C
import os
import subprocess
import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "smetric_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB = os.path.join(_BUILD, "liboracle.so")
_lib = None

u64p = np.ctypeslib.ndpointer(dtype=np.uint64, flags="C_CONTIGUOUS")
i64p = np.ctypeslib.ndpointer(dtype=np.int64, flags="C_CONTIGUOUS")
i32p = np.ctypeslib.ndpointer(dtype=np.int32, flags="C_CONTIGUOUS")


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (plain C11, OpenMP for the optional
    request-parallel loop)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-Wall", "-Wextra", "-fopenmp",
                               "-shared", "-fPIC", _SRC, "-o", tmp])
        os.replace(tmp, _LIB)
    return _LIB


def load_library(path: str):
    """Load an oracle build from `path` and declare its prototypes."""
    L = C.CDLL(path)
    L.oracle_mix64.restype = C.c_uint64
    L.oracle_mix64.argtypes = [C.c_uint64]
    L.oracle_block_hashes.restype = C.c_int64
    L.oracle_block_hashes.argtypes = [i32p, C.c_int64, C.c_int32, C.c_uint64, u64p]
    L.oracle_index_create.restype = C.c_void_p
    L.oracle_index_create.argtypes = [C.c_int32]
    L.oracle_index_destroy.restype = None
    L.oracle_index_destroy.argtypes = [C.c_void_p]
    for f in (L.oracle_index_insert, L.oracle_index_evict):
        f.restype = C.c_int
        f.argtypes = [C.c_void_p, u64p, i32p, C.c_int64]
    L.oracle_index_contains.restype = C.c_int
    L.oracle_index_contains.argtypes = [C.c_void_p, C.c_uint64, C.c_int32]
    L.oracle_prefix_hits.restype = None
    L.oracle_prefix_hits.argtypes = [C.c_void_p, u64p, C.c_int64, i64p, i64p]
    L.oracle_route_batch.restype = C.c_int
    L.oracle_route_batch.argtypes = [
        C.c_void_p, C.c_int32, C.c_int32, C.c_uint64, i32p, i64p, C.c_int32, i64p,
        C.c_int64, C.c_int64, C.c_int64, i32p, i32p, i32p, u64p, C.c_void_p, C.c_int32]
    L.oracle_route_batch_policy.restype = C.c_int
    L.oracle_route_batch_policy.argtypes = [
        C.c_void_p, C.c_int32, C.c_int32, C.c_uint64, i32p, i64p, C.c_int32, i64p, i32p, i64p,
        C.c_int64, C.c_int64, C.c_int64, C.c_int64, C.c_int64, C.c_int64, C.c_int32,
        i32p, i32p, i32p, i32p, u64p]
    L.oracle_route_batch_coloc.restype = C.c_int
    L.oracle_route_batch_coloc.argtypes = [
        C.c_void_p, C.c_int32, C.c_int32, C.c_uint64, i32p, i64p, C.c_int32, i64p, i64p, i64p, i32p, i64p,
        C.c_int64, C.c_int64, C.c_int64, C.c_int64, C.c_int64, C.c_int64, C.c_int32,
        i32p, i32p, i32p, i32p, u64p]
    L.oracle_route_batch_baseline.restype = C.c_int
    L.oracle_route_batch_baseline.argtypes = [
        C.c_void_p, C.c_int32, C.c_int32, C.c_uint64, i32p, i64p, C.c_int32, C.c_int32, i64p, i64p,
        C.c_int64, C.c_int64, i32p, i32p, i32p, u64p]
    L.oracle_route_batch_sequential.restype = C.c_int
    L.oracle_route_batch_sequential.argtypes = [
        C.c_void_p, C.c_int32, C.c_int32, C.c_uint64, i32p, i64p, C.c_int32, i64p,
        C.c_int64, C.c_int64, C.c_int64, i32p, i32p, i32p, u64p, i64p]
    L.oracle_reuse_breakdown.restype = C.c_int
    L.oracle_reuse_breakdown.argtypes = [C.c_int32, C.c_uint64, i32p, i64p, C.c_int32, i32p, i32p,
                                         i32p, i32p, i32p, i32p]
    L.oracle_window_imbalance.restype = C.c_int
    L.oracle_window_imbalance.argtypes = [C.c_int32, C.c_int64, C.c_int32, i32p, i64p, i64p, C.c_int32, i64p, i32p,
                                          i64p]
    L.oracle_link_sessions.restype = C.c_int
    L.oracle_link_sessions.argtypes = [C.c_int32, C.c_uint64, i32p, i64p, C.c_int32, i64p, i32p, i32p, i32p]
    return L


def lib():
    global _lib
    if _lib is None:
        _lib = load_library(build())
    return _lib


def mix64(z: int, L=None) -> int:
    return int((L or lib()).oracle_mix64(C.c_uint64(z & 0xFFFFFFFFFFFFFFFF)))


def block_hashes(tokens: np.ndarray, block_size: int, seed: int = 0, L=None) -> np.ndarray:
    t = np.ascontiguousarray(tokens, dtype=np.int32)
    out = np.zeros(max(len(t) // block_size, 1), dtype=np.uint64)
    n = (L or lib()).oracle_block_hashes(t if len(t) else np.zeros(1, np.int32), len(t), block_size,
                                  seed & 0xFFFFFFFFFFFFFFFF, out)
    if n < 0:
        raise ValueError("invalid block size")
    return out[:n]


def link_sessions(block_size: int, seed: int, tokens, offsets, users, turns, L=None):
    """Session reconstruction (Appendix A). Returns (parent, session), int32 per request."""
    t = np.ascontiguousarray(tokens, dtype=np.int32)
    o = np.ascontiguousarray(offsets, dtype=np.int64)
    n = len(o) - 1
    u = np.ascontiguousarray(users, dtype=np.int64)
    tu = np.ascontiguousarray(turns, dtype=np.int32)
    parent = np.zeros(max(n, 1), np.int32)
    session = np.zeros(max(n, 1), np.int32)
    rc = (L or lib()).oracle_link_sessions(block_size, seed & 0xFFFFFFFFFFFFFFFF,
                                           t if len(t) else np.zeros(1, np.int32), o, n,
                                           u if n else np.zeros(1, np.int64), tu if n else np.zeros(1, np.int32),
                                           parent, session)
    if rc != 0:
        raise ValueError(f"oracle_link_sessions: {rc}")
    return parent[:n], session[:n]


def reuse_breakdown(block_size: int, seed: int, tokens, offsets, sessions, sys_blocks, L=None):
    """Reuse against an unbounded store of every earlier request's blocks:
    dict(hit, sys, intra, inter), int32 blocks per request."""
    t = np.ascontiguousarray(tokens, dtype=np.int32)
    o = np.ascontiguousarray(offsets, dtype=np.int64)
    n = len(o) - 1
    ss = np.ascontiguousarray(sessions, dtype=np.int32)
    sb = np.ascontiguousarray(sys_blocks, dtype=np.int32)
    outs = [np.zeros(max(n, 1), np.int32) for _ in range(4)]
    rc = (L or lib()).oracle_reuse_breakdown(block_size, seed & 0xFFFFFFFFFFFFFFFF,
                                             t if len(t) else np.zeros(1, np.int32), o, n,
                                             ss if n else np.zeros(1, np.int32), sb if n else np.zeros(1, np.int32),
                                             *outs)
    if rc != 0:
        raise ValueError(f"oracle_reuse_breakdown: {rc}")
    return dict(zip(("hit", "sys", "intra", "inter"), (x[:n] for x in outs)))


def window_imbalance(num_instances: int, window: int, n_windows: int, instance, start, end, L=None):
    """Per window of `window` ticks: dict(max, argmax, sum) of the instances'
    running-request ticks; the imbalance is num_instances * max / sum."""
    inst = np.ascontiguousarray(instance, dtype=np.int32)
    st = np.ascontiguousarray(start, dtype=np.int64)
    en = np.ascontiguousarray(end, dtype=np.int64)
    n = len(inst)
    m = max(n_windows, 1)
    mx, am, sm = np.zeros(m, np.int64), np.zeros(m, np.int32), np.zeros(m, np.int64)
    rc = (L or lib()).oracle_window_imbalance(num_instances, window, n_windows,
                                              inst if n else np.zeros(1, np.int32),
                                              st if n else np.zeros(1, np.int64),
                                              en if n else np.zeros(1, np.int64), n, mx, am, sm)
    if rc != 0:
        raise ValueError(f"oracle_window_imbalance: {rc}")
    return dict(max=mx[:n_windows], argmax=am[:n_windows], sum=sm[:n_windows])


class OracleLRU:
    """Contents of capped KV$ tiers under least-recently-used eviction
    (Section 2: each instance's local KV$ and the global store are bounded).

    Plain and slow, written from the recency rule itself: every commit k
    touches, for each committed request r (in order) and each of its full
    blocks b, the block's key in the request's local tier (and in the global
    tier when asked) with stamp (k, r, -b), so that later commits, later
    requests and, within a request, leading blocks are more recent. A key's
    stamp in a tier is its largest; after the commit each capped tier keeps
    its `cap` keys of largest stamp. Tier -1 is the global tier."""

    def __init__(self, num_instances: int, local_cap: int = 0, global_cap: int = 0):
        self.N = num_instances
        self.caps = {t: local_cap for t in range(num_instances)}
        self.caps[-1] = global_cap
        self.stamp = {t: {} for t in range(-1, num_instances)}  # tier -> key -> stamp
        self.k = 0

    def commit(self, n_blocks, instance, hashes, also_global: bool):
        """n_blocks[r] full blocks of request r (its hashes in order, request
        after request); instance[r] < 0 commits nothing for r. Returns the
        evicted (keys, tiers)."""
        hashes = [int(x) for x in np.asarray(hashes, dtype=np.uint64)]
        pos = 0
        for r, (nb, i) in enumerate(zip(np.asarray(n_blocks).tolist(), np.asarray(instance).tolist())):
            keys = hashes[pos:pos + nb]
            pos += nb
            if i < 0:
                continue
            for t in ([i, -1] if also_global else [i]):
                if self.caps[t] <= 0:
                    continue
                tier = self.stamp[t]
                for b, key in enumerate(keys):
                    st = (self.k, r, -b)
                    if key not in tier or tier[key] < st:
                        tier[key] = st
        self.k += 1
        ev_k, ev_t = [], []
        for t, tier in self.stamp.items():
            over = len(tier) - self.caps[t]
            if self.caps[t] > 0 and over > 0:
                for key, _ in sorted(tier.items(), key=lambda kv: kv[1])[:over]:
                    del tier[key]
                    ev_k.append(key)
                    ev_t.append(t)
        return np.array(ev_k, dtype=np.uint64), np.array(ev_t, dtype=np.int32)

    def holds(self, key: int, tier: int) -> bool:
        return int(key) in self.stamp[tier]

    def size(self, tier: int) -> int:
        return len(self.stamp[tier]) if self.caps[tier] > 0 else 0


class OracleIndex:
    """Two-tier KV$ index: local tier per instance plus one global tier (-1)."""

    def __init__(self, num_instances: int, L=None):
        self.N = num_instances
        self._L = L or lib()
        self._h = self._L.oracle_index_create(num_instances)
        if not self._h:
            raise ValueError("oracle_index_create failed")

    def close(self):
        if getattr(self, "_h", None):
            self._L.oracle_index_destroy(self._h)
            self._h = None

    __del__ = close

    def insert(self, keys, tiers):
        k = np.ascontiguousarray(keys, dtype=np.uint64)
        t = np.ascontiguousarray(np.broadcast_to(tiers, k.shape), dtype=np.int32)
        if len(k) == 0:
            return
        rc = self._L.oracle_index_insert(self._h, k, t, len(k))
        if rc != 0:
            raise ValueError(f"oracle_index_insert: {rc}")

    def evict(self, keys, tiers):
        k = np.ascontiguousarray(keys, dtype=np.uint64)
        t = np.ascontiguousarray(np.broadcast_to(tiers, k.shape), dtype=np.int32)
        if len(k) == 0:
            return
        rc = self._L.oracle_index_evict(self._h, k, t, len(k))
        if rc != 0:
            raise ValueError(f"oracle_index_evict: {rc}")

    def contains(self, key: int, tier: int) -> bool:
        return bool(self._L.oracle_index_contains(self._h, C.c_uint64(int(key)), tier))

    def prefix_hits(self, hashes: np.ndarray):
        h = np.ascontiguousarray(hashes, dtype=np.uint64)
        c = np.zeros(self.N, dtype=np.int64)
        g = np.zeros(1, dtype=np.int64)
        self._L.oracle_prefix_hits(self._h, h if len(h) else np.zeros(1, np.uint64), len(h), c, g)
        return c, int(g[0])

    def route_batch(self, block_size: int, session_blocks: int, seed: int, tokens, offsets,
                    load, w_load: int, w_miss: int, w_glob: int, want_hashes: bool = False,
                    n_threads: int = 1):
        """Returns dict(instance, local_hit, global_hit, session_key[, block_hashes])."""
        t = np.ascontiguousarray(tokens, dtype=np.int32)
        o = np.ascontiguousarray(offsets, dtype=np.int64)
        ld = np.ascontiguousarray(load, dtype=np.int64)
        if len(ld) != self.N:
            raise ValueError("load must have one entry per instance")
        n = len(o) - 1
        inst = np.zeros(max(n, 1), np.int32)
        lh = np.zeros(max(n, 1), np.int32)
        gh = np.zeros(max(n, 1), np.int32)
        sk = np.zeros(max(n, 1), np.uint64)
        nblk = int((np.diff(o) // block_size).sum()) if n > 0 else 0
        hb = np.zeros(max(nblk, 1), np.uint64) if want_hashes else None
        rc = self._L.oracle_route_batch(
            self._h, block_size, session_blocks, seed & 0xFFFFFFFFFFFFFFFF,
            t if len(t) else np.zeros(1, np.int32), o, n, ld, w_load, w_miss, w_glob,
            inst, lh, gh, sk, hb.ctypes.data if hb is not None else None, n_threads)
        if rc != 0:
            raise ValueError(f"oracle_route_batch: {rc}")
        out = dict(instance=inst[:n], local_hit=lh[:n], global_hit=gh[:n], session_key=sk[:n])
        if want_hashes:
            out["block_hashes"] = hb[:nblk]
        return out

    def route_batch_policy(self, block_size: int, session_blocks: int, seed: int, tokens, offsets,
                           queued, turn, est_hit, c_lin: int, c_att: int, d0: int, d1: int,
                           hit_num: int, hit_den: int, rr_base: int = 0):
        """The session-centric policy of Figure 10. Returns dict(instance,
        local_hit, global_hit, stick, session_key)."""
        t = np.ascontiguousarray(tokens, dtype=np.int32)
        o = np.ascontiguousarray(offsets, dtype=np.int64)
        q = np.ascontiguousarray(queued, dtype=np.int64)
        n = len(o) - 1
        tu = np.ascontiguousarray(turn, dtype=np.int32)
        eh = np.ascontiguousarray(est_hit, dtype=np.int64)
        if len(q) != self.N or len(tu) != n or len(eh) != n:
            raise ValueError("queued has one entry per instance; turn and est_hit one per request")
        outs = [np.zeros(max(n, 1), np.int32) for _ in range(4)]
        sk = np.zeros(max(n, 1), np.uint64)
        rc = self._L.oracle_route_batch_policy(
            self._h, block_size, session_blocks, seed & 0xFFFFFFFFFFFFFFFF,
            t if len(t) else np.zeros(1, np.int32), o, n, q,
            tu if n else np.zeros(1, np.int32), eh if n else np.zeros(1, np.int64),
            c_lin, c_att, d0, d1, hit_num, hit_den, rr_base, *outs, sk)
        if rc != 0:
            raise ValueError(f"oracle_route_batch_policy: {rc}")
        inst, lh, gh, st = outs
        return dict(instance=inst[:n], local_hit=lh[:n], global_hit=gh[:n], stick=st[:n],
                    session_key=sk[:n])

    def route_batch_coloc(self, block_size: int, session_blocks: int, seed: int, tokens, offsets,
                          queued, tpot_budget, num_requests, turn, est_hit, c_lin: int, c_att: int,
                          d0: int, d1: int, hit_num: int, hit_den: int, rr_base: int = 0):
        """The session-centric policy under PD colocation (Appendix B).
        Returns dict(instance, local_hit, global_hit, stick, session_key)."""
        t = np.ascontiguousarray(tokens, dtype=np.int32)
        o = np.ascontiguousarray(offsets, dtype=np.int64)
        n = len(o) - 1
        per_inst = [np.ascontiguousarray(a, dtype=np.int64) for a in (queued, tpot_budget, num_requests)]
        tu = np.ascontiguousarray(turn, dtype=np.int32)
        eh = np.ascontiguousarray(est_hit, dtype=np.int64)
        if any(len(a) != self.N for a in per_inst) or len(tu) != n or len(eh) != n:
            raise ValueError("queued, tpot_budget, num_requests: one per instance; turn, est_hit: one per request")
        outs = [np.zeros(max(n, 1), np.int32) for _ in range(4)]
        sk = np.zeros(max(n, 1), np.uint64)
        rc = self._L.oracle_route_batch_coloc(
            self._h, block_size, session_blocks, seed & 0xFFFFFFFFFFFFFFFF,
            t if len(t) else np.zeros(1, np.int32), o, n, *per_inst,
            tu if n else np.zeros(1, np.int32), eh if n else np.zeros(1, np.int64),
            c_lin, c_att, d0, d1, hit_num, hit_den, rr_base, *outs, sk)
        if rc != 0:
            raise ValueError(f"oracle_route_batch_coloc: {rc}")
        inst, lh, gh, st = outs
        return dict(instance=inst[:n], local_hit=lh[:n], global_hit=gh[:n], stick=st[:n],
                    session_key=sk[:n])

    def route_batch_baseline(self, block_size: int, session_blocks: int, seed: int, tokens, offsets,
                             scorer: int, queued, batch, lam_num: int = 1, lam_den: int = 2):
        """Baseline scorers of Section 5.1: scorer 1 = Bailian, 2 = LMetric.
        Returns dict(instance, local_hit, global_hit, session_key)."""
        t = np.ascontiguousarray(tokens, dtype=np.int32)
        o = np.ascontiguousarray(offsets, dtype=np.int64)
        n = len(o) - 1
        q = np.ascontiguousarray(queued, dtype=np.int64)
        b = np.ascontiguousarray(batch, dtype=np.int64)
        if len(q) != self.N or len(b) != self.N:
            raise ValueError("queued and batch have one entry per instance")
        outs = [np.zeros(max(n, 1), np.int32) for _ in range(3)]
        sk = np.zeros(max(n, 1), np.uint64)
        rc = self._L.oracle_route_batch_baseline(
            self._h, block_size, session_blocks, seed & 0xFFFFFFFFFFFFFFFF,
            t if len(t) else np.zeros(1, np.int32), o, n, scorer, q, b, lam_num, lam_den, *outs, sk)
        if rc != 0:
            raise ValueError(f"oracle_route_batch_baseline: {rc}")
        inst, lh, gh = outs
        return dict(instance=inst[:n], local_hit=lh[:n], global_hit=gh[:n], session_key=sk[:n])

    def route_batch_sequential(self, block_size: int, session_blocks: int, seed: int, tokens, offsets, load,
                               w_load: int, w_miss: int, w_glob: int):
        """The argmin cost with loads updated request by request. Returns
        dict(instance, local_hit, global_hit, session_key, load_after)."""
        t = np.ascontiguousarray(tokens, dtype=np.int32)
        o = np.ascontiguousarray(offsets, dtype=np.int64)
        ld = np.ascontiguousarray(load, dtype=np.int64)
        n = len(o) - 1
        outs = [np.zeros(max(n, 1), np.int32) for _ in range(3)]
        sk = np.zeros(max(n, 1), np.uint64)
        after = np.zeros(self.N, np.int64)
        rc = self._L.oracle_route_batch_sequential(
            self._h, block_size, session_blocks, seed & 0xFFFFFFFFFFFFFFFF,
            t if len(t) else np.zeros(1, np.int32), o, n, ld, w_load, w_miss, w_glob, *outs, sk, after)
        if rc != 0:
            raise ValueError(f"oracle_route_batch_sequential: {rc}")
        inst, lh, gh = outs
        return dict(instance=inst[:n], local_hit=lh[:n], global_hit=gh[:n], session_key=sk[:n],
                    load_after=after)
