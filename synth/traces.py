"""Workload recipes for the five trace configurations.

Every generator is seeded and deterministic. Token IDs are int32, uniform in
[0, VOCAB) with VOCAB = 151936 (the Qwen3 vocabulary the paper serves).

Agent traces (configs 1-3) model the append-only agent loop of Section 2
("Agentic workflow and the agent session"): turn t of a session resends the
whole history of turn t-1 plus the new tool output / reply. Requests are
issued in turn waves: all sessions' turn t before any turn t+1.

The burst trace (configs 4-5) models many concurrent sessions with skewed
popularity (Finding 5: the top quarter of sessions hold most tokens), each
request resending its session's cached prefix plus a small fresh suffix.
"""

from __future__ import annotations

import math
import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field
from typing import Iterator, List, Optional, Sequence

import numpy as np

VOCAB = 151936

# Distinct stream tags so that no two generator purposes share a stream.
_TAG_PREFIX = 0x5E55_0001
_TAG_TAIL = 0x5E55_0002
_TAG_BATCH = 0x5E55_0003
_TAG_FILL = 0x5E55_0004


@dataclass(frozen=True)
class RouteParams:
    """Index and scoring parameters of one workload."""

    num_instances: int
    block_size: int
    session_blocks: int
    hash_seed: int = 0
    w_load: int = 1
    w_miss: int = 4
    w_glob: int = 2


@dataclass
class Batch:
    """One routing batch: flat ragged tokens plus request offsets."""

    tokens: np.ndarray  # int32 [offsets[-1]]
    offsets: np.ndarray  # int64 [n + 1], offsets[0] == 0
    sessions: np.ndarray  # int64 [n]
    turns: np.ndarray  # int32 [n]
    load: Optional[np.ndarray] = None  # int64 [N] when the workload draws it

    @property
    def n_requests(self) -> int:
        return int(self.offsets.shape[0] - 1)

    @property
    def n_tokens(self) -> int:
        return int(self.offsets[-1])

    def lengths(self) -> np.ndarray:
        return np.diff(self.offsets)


def _stream(*key: int) -> np.random.Generator:
    """An independent PCG64 stream for a tuple of non-negative integer keys."""
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([int(k) for k in key])))


def _tokens(rng: np.random.Generator, n: int) -> np.ndarray:
    return rng.integers(0, VOCAB, size=int(n), dtype=np.int32)


def _parallel(fn, n_items: int, threads: int = 0):
    """Run fn(lo, hi) over [0, n_items) split into contiguous ranges on a
    thread pool (numpy releases the GIL while generating and copying)."""
    threads = threads or min(16, os.cpu_count() or 1)
    if n_items == 0:
        return
    step = max(1, (n_items + threads * 4 - 1) // (threads * 4))
    ranges = [(lo, min(n_items, lo + step)) for lo in range(0, n_items, step)]
    if threads == 1 or len(ranges) == 1:
        for lo, hi in ranges:
            fn(lo, hi)
        return
    with ThreadPoolExecutor(threads) as ex:
        for f in [ex.submit(fn, lo, hi) for lo, hi in ranges]:
            f.result()


def pack(requests: Sequence[np.ndarray], out: Optional[np.ndarray] = None
         ) -> tuple[np.ndarray, np.ndarray]:
    """Concatenate per-request token arrays into (tokens, offsets). With `out`
    (an int32 buffer at least as long as the total), tokens is a view of it,
    which avoids touching fresh memory for every batch."""
    lens = np.fromiter((len(r) for r in requests), dtype=np.int64, count=len(requests))
    offsets = np.zeros(len(requests) + 1, dtype=np.int64)
    np.cumsum(lens, out=offsets[1:])
    total = int(offsets[-1])
    if out is not None and len(out) >= total:
        tokens = out[:total]
    else:
        tokens = np.empty(total, dtype=np.int32)
    for r, a in enumerate(requests):
        tokens[offsets[r]:offsets[r + 1]] = a
    return tokens, offsets


# ---------------------------------------------------------------------------
# Agent traces (configs 1-3)
# ---------------------------------------------------------------------------


@dataclass
class AgentTrace:
    """Multi-turn agent sessions replayed in turn waves.

    growth: ("uniform", lo, hi)     new tokens per turn ~ U{lo..hi}
            ("loguniform", lo, hi)  new tokens per turn ~ exp(U[ln lo, ln hi])
            ("target", lo, hi)      per-session target T ~ U{lo..hi}; each turn
                                    appends T // n_turns tokens
    truncate_prob: per-turn probability that the request drops the oldest
                   floor(|H| * truncate_frac) tokens of its history (the history
                   itself is kept whole).
    local_cap / global_cap: LRU capacity in blocks per tier (None = unbounded).
    global_policy: "none" (empty global tier), "all" (every inserted block is
                   also in the global tier), "lru" (global tier with global_cap).
    """

    params: RouteParams
    n_sessions: int
    n_turns: int
    batch_size: int
    n_system_prompts: int
    system_prompt_len: int
    growth: tuple
    truncate_prob: float = 0.0
    truncate_frac: float = 0.25
    local_cap: Optional[int] = None
    global_policy: str = "none"
    global_cap: Optional[int] = None
    seed: int = 0
    name: str = "agent"

    def batches(self) -> Iterator[Batch]:
        rng = np.random.Generator(np.random.PCG64(self.seed))
        sys_prompts = [_tokens(rng, self.system_prompt_len) for _ in range(self.n_system_prompts)]
        pick = rng.integers(0, self.n_system_prompts, size=self.n_sessions)
        kind = self.growth[0]
        if kind == "target":
            target = rng.integers(self.growth[1], self.growth[2] + 1, size=self.n_sessions)
            per_turn = target // self.n_turns
        history: List[List[np.ndarray]] = [[sys_prompts[p]] for p in pick]
        hist_len = np.full(self.n_sessions, self.system_prompt_len, dtype=np.int64)
        for turn in range(self.n_turns):
            if kind == "uniform":
                g = rng.integers(self.growth[1], self.growth[2] + 1, size=self.n_sessions)
            elif kind == "loguniform":
                u = rng.uniform(math.log(self.growth[1]), math.log(self.growth[2]), size=self.n_sessions)
                g = np.floor(np.exp(u)).astype(np.int64)
            elif kind == "target":
                g = per_turn
            else:
                raise ValueError(kind)
            fresh = _tokens(rng, int(g.sum()))
            cut = np.concatenate([[0], np.cumsum(g)])
            trunc = rng.random(self.n_sessions) < self.truncate_prob
            for s in range(self.n_sessions):
                history[s].append(fresh[cut[s]:cut[s + 1]])
            hist_len += g
            for b0 in range(0, self.n_sessions, self.batch_size):
                sess = np.arange(b0, min(b0 + self.batch_size, self.n_sessions))
                reqs = []
                for s in sess:
                    h = np.concatenate(history[s])
                    if trunc[s]:
                        h = h[int(len(h) * self.truncate_frac):]
                    reqs.append(h)
                tokens, offsets = pack(reqs)
                yield Batch(tokens=tokens, offsets=offsets, sessions=sess.astype(np.int64),
                            turns=np.full(len(sess), turn, dtype=np.int32))

    @property
    def n_batches(self) -> int:
        return self.n_turns * ((self.n_sessions + self.batch_size - 1) // self.batch_size)


def agent_trace(config: str, scale: float = 1.0, seed: int = 0) -> AgentTrace:
    """Configs 1-3. scale < 1 shrinks sessions, turns, lengths and caps together
    (for tests that must finish quickly); scale = 1 is the full workload."""

    def S(x, lo=1):
        return max(lo, int(round(x * scale)))

    if config == "c1_tiny":
        p = RouteParams(num_instances=4, block_size=16, session_blocks=2048 // 16 + 1)
        return AgentTrace(params=p, n_sessions=S(64, 2), n_turns=S(8, 2), batch_size=S(64, 2),
                          n_system_prompts=1, system_prompt_len=2048,
                          growth=("uniform", 128, 1024), global_policy="none",
                          seed=seed, name=config)
    if config == "c2_medium":
        p = RouteParams(num_instances=16, block_size=16, session_blocks=4096 // 16 + 1)
        return AgentTrace(params=p, n_sessions=S(1024, 4), n_turns=S(16, 2), batch_size=S(256, 2),
                          n_system_prompts=4, system_prompt_len=4096,
                          growth=("loguniform", 256, 4096), local_cap=S(200_000, 64),
                          global_policy="all", seed=seed, name=config)
    if config == "c3_long":
        p = RouteParams(num_instances=32, block_size=64, session_blocks=4096 // 64 + 1)
        return AgentTrace(params=p, n_sessions=S(4096, 4), n_turns=S(32, 2), batch_size=S(1024, 2),
                          n_system_prompts=1, system_prompt_len=4096,
                          growth=("target", S(32768, 256), S(131072, 512)),
                          truncate_prob=0.5, truncate_frac=0.25,
                          local_cap=S(1_000_000, 64), global_policy="lru",
                          global_cap=S(16_000_000, 256), seed=seed, name=config)
    raise KeyError(config)


# ---------------------------------------------------------------------------
# Burst trace (configs 4-5)
# ---------------------------------------------------------------------------


@dataclass
class BurstTrace:
    """Many concurrent sessions with Zipf popularity and a pre-populated index.

    Session s has a prompt length L_s ~ U{len_lo..len_hi} and a cached prefix of
    floor(prefix_frac * L_s) tokens. A request for s is that prefix followed by
    L_s - prefix fresh tokens. The index holds every full block of each
    session's prefix in the global tier, in the local tier of the session's
    home instance with probability p_home, and in one other instance's local
    tier with probability p_second. Per-instance queued load is redrawn
    uniformly in [0, load_hi] for every batch.
    """

    params: RouteParams
    n_sessions: int = 65536
    batch_size: int = 8192
    zipf_s: float = 1.1
    len_lo: int = 8000
    len_hi: int = 40000
    prefix_frac: float = 0.95
    p_home: float = 0.8
    p_second: float = 0.2
    load_hi: int = 2_000_000
    seed: int = 0
    name: str = "burst"
    _cache: dict = field(default_factory=dict, repr=False)

    def __post_init__(self):
        rng = np.random.Generator(np.random.PCG64(self.seed))
        n, N = self.n_sessions, self.params.num_instances
        self.session_len = rng.integers(self.len_lo, self.len_hi + 1, size=n).astype(np.int64)
        self.prefix_len = np.floor(self.prefix_frac * self.session_len).astype(np.int64)
        self.home = rng.integers(0, N, size=n).astype(np.int32)
        self.in_home = rng.random(n) < self.p_home
        off = rng.integers(1, max(N, 2), size=n) if N > 1 else np.zeros(n, dtype=np.int64)
        self.second = ((self.home + off) % N).astype(np.int32)
        self.in_second = (rng.random(n) < self.p_second) & (N > 1)
        self.perm = rng.permutation(n)  # popularity rank -> session id
        w = np.arange(1, n + 1, dtype=np.float64) ** (-self.zipf_s)
        self.cdf = np.cumsum(w) / w.sum()

    # -- sessions -----------------------------------------------------------
    def _gen_prefix(self, s: int) -> np.ndarray:
        return _tokens(_stream(_TAG_PREFIX, self.seed, int(s)), self.prefix_len[int(s)])

    def session_prefix(self, s: int) -> np.ndarray:
        s = int(s)
        got = self._cache.get(s)
        if got is None:
            got = self._gen_prefix(s)
            if len(self._cache) < 16384:
                self._cache[s] = got
        return got

    def session_tiers(self, s: int) -> List[int]:
        """Tiers holding session s's prefix blocks: -1 = global, i = local of i."""
        t = [-1]
        if self.in_home[s]:
            t.append(int(self.home[s]))
        if self.in_second[s]:
            t.append(int(self.second[s]))
        return t

    def prepopulation(self, sessions: Optional[np.ndarray] = None, chunk: int = 2048,
                      out: Optional[np.ndarray] = None):
        """Yield (session ids, tokens, offsets) chunks covering `sessions`
        (default: all). The consumer hashes each prefix and inserts its full
        blocks into session_tiers(s). With `out`, every chunk's tokens are a
        view of that one buffer, valid until the next chunk."""
        if sessions is None:
            sessions = np.arange(self.n_sessions)
        sessions = np.asarray(sessions, dtype=np.int64)
        for c0 in range(0, len(sessions), chunk):
            ids = sessions[c0:c0 + chunk]
            offsets = np.zeros(len(ids) + 1, dtype=np.int64)
            np.cumsum(self.prefix_len[ids], out=offsets[1:])
            total = int(offsets[-1])
            tokens = out[:total] if out is not None and len(out) >= total else np.empty(total, np.int32)

            def fill(lo, hi):
                for j in range(lo, hi):
                    tokens[offsets[j]:offsets[j + 1]] = self._gen_prefix(ids[j])

            _parallel(fill, len(ids))
            yield ids, tokens, offsets

    def n_prefix_blocks(self, sessions: Optional[np.ndarray] = None) -> int:
        pl = self.prefix_len if sessions is None else self.prefix_len[np.asarray(sessions)]
        return int((pl // self.params.block_size).sum())

    # -- batches ------------------------------------------------------------
    def batch_sessions(self, k: int, batch_size: Optional[int] = None) -> np.ndarray:
        bs = self.batch_size if batch_size is None else batch_size
        rng = _stream(_TAG_BATCH, self.seed, k)
        u = rng.random(bs)
        rank = np.minimum(np.searchsorted(self.cdf, u, side="right"), self.n_sessions - 1)
        return self.perm[rank].astype(np.int64)

    def batch(self, k: int, batch_size: Optional[int] = None,
              out: Optional[np.ndarray] = None) -> Batch:
        bs = self.batch_size if batch_size is None else batch_size
        sess = self.batch_sessions(k, bs)
        rng = _stream(_TAG_BATCH, self.seed, k)
        rng.random(bs)  # skip the session draws (same stream as batch_sessions)
        load = rng.integers(0, self.load_hi + 1, size=self.params.num_instances).astype(np.int64)
        tail_rng = _stream(_TAG_TAIL, self.seed, k)
        tails = self.session_len[sess] - self.prefix_len[sess]
        fresh = _tokens(tail_rng, int(tails.sum()))
        cut = np.concatenate([[0], np.cumsum(tails)])
        offsets = np.zeros(bs + 1, dtype=np.int64)
        np.cumsum(self.session_len[sess], out=offsets[1:])
        total = int(offsets[-1])
        tokens = out[:total] if out is not None and len(out) >= total else np.empty(total, np.int32)
        uniq = np.unique(sess)
        prefixes = {}

        def gen(lo, hi):
            for j in range(lo, hi):
                prefixes[int(uniq[j])] = self.session_prefix(uniq[j])

        _parallel(gen, len(uniq))

        def fill(lo, hi):
            for r in range(lo, hi):
                a = offsets[r]
                s = int(sess[r])
                pl = int(self.prefix_len[s])
                tokens[a:a + pl] = prefixes[s]
                tokens[a + pl:offsets[r + 1]] = fresh[cut[r]:cut[r + 1]]

        _parallel(fill, bs)
        return Batch(tokens=tokens, offsets=offsets, sessions=sess,
                     turns=np.ones(bs, dtype=np.int32), load=load)

    def filler_keys(self, n: int, k: int = 0):
        """n random 64-bit keys (>= 2) with random tiers, for padding a table
        to a target size (config 5). Returns (keys uint64, tiers int32)."""
        rng = _stream(_TAG_FILL, self.seed, k)
        keys = rng.integers(2, np.iinfo(np.uint64).max, size=n, dtype=np.uint64, endpoint=True)
        tiers = rng.integers(-1, self.params.num_instances, size=n).astype(np.int32)
        return keys, tiers


def burst_trace(config: str = "c4_burst", *, num_instances: int = 64, block_size: int = 32,
                n_sessions: int = 65536, batch_size: int = 8192, seed: int = 0,
                len_lo: int = 8000, len_hi: int = 40000) -> BurstTrace:
    """Config 4 (defaults) and the config-5 sweep points (other N, B, batch)."""
    p = RouteParams(num_instances=num_instances, block_size=block_size,
                    session_blocks=1)
    # The burst sessions share no system prompt, so the session key is the
    # hash of the first block.
    return BurstTrace(params=p, n_sessions=n_sessions, batch_size=batch_size, seed=seed,
                      len_lo=len_lo, len_hi=len_hi, name=config)


TRACE_CONFIGS = {
    "c1_tiny": lambda scale=1.0, seed=0: agent_trace("c1_tiny", scale, seed),
    "c2_medium": lambda scale=1.0, seed=0: agent_trace("c2_medium", scale, seed),
    "c3_long": lambda scale=1.0, seed=0: agent_trace("c3_long", scale, seed),
    "c4_burst": lambda seed=0, **kw: burst_trace("c4_burst", seed=seed, **kw),
}
