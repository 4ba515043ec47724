"""Pins for the CPU oracle: checks against what the paper and mathematics fix.

Each check takes an oracle library handle so the same checks can be run
against deliberately broken oracle builds (test_oracle_mutants.py) to show
that a plausible mistake anywhere in the oracle fails at least one of them.
"""

from __future__ import annotations

import json
import os
from fractions import Fraction

import numpy as np

import oracle

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
M64 = (1 << 64) - 1
GAMMA = 0x9E3779B97F4A7C15


def _golden_hex(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return [int(x, 16) for x in f.read().split("\n") if x and not x.startswith("#")]


def _golden_json(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


# ---------------------------------------------------------------------------
# mix64
# ---------------------------------------------------------------------------

def check_published_vector(L):
    """The SplitMix64 generator's published first outputs for seed 0."""
    want = _golden_hex("splitmix64_seed0.txt")
    state = 0
    for w in want:
        state = (state + GAMMA) & M64
        assert oracle.mix64(state, L) == w, hex(w)


def _py_mix64(z):
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & M64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & M64
    return z ^ (z >> 31)


def _unxorshift(z, s):
    x = z
    for _ in range(64 // s + 1):
        x = z ^ (x >> s)
    return x


def py_mix64_inverse(z):
    """Inverse of the SplitMix64 output function (each step is a bijection:
    xor-shift right by s >= 1, and multiplication by an odd constant)."""
    z = _unxorshift(z, 31)
    z = (z * pow(0x94D049BB133111EB, -1, 1 << 64)) & M64
    z = _unxorshift(z, 27)
    z = (z * pow(0xBF58476D1CE4E5B9, -1, 1 << 64)) & M64
    return _unxorshift(z, 30)


def check_bijection(L):
    rng = np.random.default_rng(7)
    for z in rng.integers(0, 2**63, size=64).tolist() + [0, 1, M64]:
        assert py_mix64_inverse(oracle.mix64(z, L)) == z


# ---------------------------------------------------------------------------
# chain hash
# ---------------------------------------------------------------------------

def check_prefix_locality(L):
    """h_b depends on exactly tokens [0, (b+1)B): flipping token p leaves
    every h_b with b < p // B unchanged and changes every later one."""
    rng = np.random.default_rng(1)
    for B in (2, 4, 16):
        t = rng.integers(0, 151936, size=B * 9 + B // 2, dtype=np.int32)
        h = oracle.block_hashes(t, B, 0, L)
        assert len(h) == 9
        for p in rng.choice(len(t), size=12, replace=False):
            u = t.copy()
            u[p] ^= 0x55
            hu = oracle.block_hashes(u, B, 0, L)
            j = p // B
            assert np.array_equal(h[:min(j, 9)], hu[:min(j, 9)])
            assert np.all(h[j:] != hu[j:])
        # every block position matters, not only its content: repeating one
        # block's tokens must not repeat its hash
        rep = np.tile(t[:B], 6)
        hr = oracle.block_hashes(rep, B, 0, L)
        assert len(set(hr.tolist())) == 6


def check_tail_and_empty(L):
    rng = np.random.default_rng(2)
    B = 8
    t = rng.integers(0, 151936, size=5 * B, dtype=np.int32)
    base = oracle.block_hashes(t, B, 0, L)
    for extra in range(B):
        u = np.concatenate([t, rng.integers(0, 151936, size=extra, dtype=np.int32)])
        assert np.array_equal(oracle.block_hashes(u, B, 0, L), base)
    assert len(oracle.block_hashes(t[:B - 1], B, 0, L)) == 0
    assert len(oracle.block_hashes(t[:0], B, 0, L)) == 0


def check_seed_and_block_size(L):
    rng = np.random.default_rng(3)
    t = rng.integers(0, 151936, size=64, dtype=np.int32)
    a = oracle.block_hashes(t, 16, 0, L)
    b = oracle.block_hashes(t, 16, 12345, L)
    assert np.all(a != b)
    c = oracle.block_hashes(t, 32, 0, L)
    assert c[0] != a[1] and c[0] != a[0]


def sentinel_tokens(target_pre_remap: int, seed: int = 0):
    """Two tokens (B = 2) whose block-0 chain value before the remap equals
    `target_pre_remap`, constructed by inverting the definition."""
    h_init = _py_mix64((seed + GAMMA) & M64)
    # h_0 = mix64((h_init + GAMMA) ^ d_0); want h_0 == target
    d0 = py_mix64_inverse(target_pre_remap) ^ ((h_init + GAMMA) & M64)
    # d_0 = mix64(mix64(seed ^ B) ^ w_0), B = 2
    w0 = py_mix64_inverse(d0) ^ _py_mix64(seed ^ 2)
    lo, hi = w0 & 0xFFFFFFFF, w0 >> 32
    return np.array([lo, hi], dtype=np.uint32).view(np.int32)


def check_sentinel_remap(L):
    """0 and 1 are reserved: a chain value of 0 becomes 2, 1 becomes 3, and the
    remapped value is what the next block chains from."""
    rng = np.random.default_rng(4)
    for target, want in ((0, 2), (1, 3)):
        for seed in (0, 99):
            t = sentinel_tokens(target, seed)
            h = oracle.block_hashes(t, 2, seed, L)
            assert len(h) == 1 and int(h[0]) == want
            more = np.concatenate([t, rng.integers(0, 151936, size=2, dtype=np.int32)])
            h2 = oracle.block_hashes(more, 2, seed, L)
            w1 = int(more[2].astype(np.uint32)) | (int(more[3].astype(np.uint32)) << 32)
            d1 = _py_mix64(_py_mix64(seed ^ 2) ^ w1)
            assert int(h2[1]) == _py_mix64(((want + GAMMA) & M64) ^ d1)


def _fold(x, words):
    for w in words:
        x = _py_mix64(x ^ w)
    return x


def _words_to_tokens(words):
    out = []
    for w in words:
        out += [w & 0xFFFFFFFF, w >> 32]
    return np.array(out, dtype=np.uint32).view(np.int32)


def multiword_tokens(targets, B, seed, rng):
    """Tokens of len(targets) blocks of B tokens (B/2 >= 2 words each) whose
    chain values h_0, h_1, ... before the remap are the given targets. Every
    word of a block but the last is random; the last is solved for by
    inverting mix64, the chain step and the digest's final fold step, so the
    construction relies on the words being folded first to last from
    mix64(seed ^ B)."""
    hb = B // 2
    h = _py_mix64((seed + GAMMA) & M64)
    words = []
    for target in targets:
        d = py_mix64_inverse(target) ^ ((h + GAMMA) & M64)  # h_b = mix64((h + G) ^ d_b)
        head = [int(x) for x in rng.integers(0, 1 << 63, size=hb - 1, dtype=np.uint64)]
        x = _fold(_py_mix64(seed ^ B), head)  # fold of every word but the last
        words += head + [py_mix64_inverse(d) ^ x]  # d_b = mix64(x ^ w_last)
        h = target if target >= 2 else target | 2
    return _words_to_tokens(words)


def check_multiword_digest(L):
    """Blocks of several words: the digest folds the block's words in order,
    first to last, each into the running value. Tokens built backwards from
    chosen chain values (the last word of each block solved for through the
    inverse of mix64) must hash to exactly those values, for B = 4, 6, 16 and
    two seeds, including a chain value of 0 (remapped to 2) inside the run."""
    rng = np.random.default_rng(12)
    for B in (4, 6, 16):
        for seed in (0, (1 << 63) + 5):
            targets = [int(x) | 2 for x in rng.integers(0, 1 << 63, size=3, dtype=np.uint64)]
            targets.insert(1, 0)
            t = multiword_tokens(targets, B, seed, rng)
            h = oracle.block_hashes(t, B, seed, L)
            want = [x if x >= 2 else x | 2 for x in targets]
            assert [int(v) for v in h] == want, (B, seed)
            # one word of the first block moved: every chain value changes
            u = t.copy()
            u[[0, 2]] = u[[2, 0]]
            hu = oracle.block_hashes(u, B, seed, L)
            assert all(int(a) != int(b) for a, b in zip(hu, h)), (B, seed)


# ---------------------------------------------------------------------------
# routing
# ---------------------------------------------------------------------------

def _route(ix, B, S, tokens_list, load, w=(1, 4, 2), seed=0):
    from synth.traces import pack
    tokens, offsets = pack(tokens_list)
    return ix.route_batch(B, S, seed, tokens, offsets, np.asarray(load, np.int64), *w,
                          want_hashes=True)


def check_session_key(L):
    rng = np.random.default_rng(5)
    B = 4
    for S in (1, 3, 7):
        ix = oracle.OracleIndex(2, L)
        shared = rng.integers(0, 151936, size=S * B, dtype=np.int32)
        reqs = [np.concatenate([shared, rng.integers(0, 151936, size=k, dtype=np.int32)])
                for k in (0, 3, 9, 40)]
        reqs += [shared[:B * (S - 1)] if S > 1 else shared[:0], shared[:2]]
        out = _route(ix, B, S, reqs, [0, 0])
        sk = out["session_key"]
        assert len(set(sk[:4].tolist())) == 1 and sk[0] != 0
        for r, t in enumerate(reqs):
            h = oracle.block_hashes(t, B, 0, L)
            want = 0 if len(h) == 0 else h[min(len(h), S) - 1]
            assert sk[r] == want
        assert sk[-1] == 0  # fewer than B tokens: no full block
        other = np.concatenate([shared[:B * (S - 1)], shared[B * (S - 1):] ^ 1])
        assert _route(ix, B, S, [other], [0, 0])["session_key"][0] != sk[0]


def brute_hit(req, stored, B):
    """Longest k such that every request prefix of 1..k blocks equals a
    block-aligned prefix of some stored prompt, by token comparison."""
    prefixes = set()
    for p in stored:
        for j in range(1, len(p) // B + 1):
            prefixes.add(tuple(p[:j * B].tolist()))
    k = 0
    while k < len(req) // B and tuple(req[:(k + 1) * B].tolist()) in prefixes:
        k += 1
    return k


def _mutate(rng, base, n_tokens):
    """A prompt sharing a random-length prefix with base (alphabet {0,1,2})."""
    keep = int(rng.integers(0, min(len(base), n_tokens) + 1))
    return np.concatenate([base[:keep], rng.integers(0, 3, size=n_tokens - keep, dtype=np.int32)])


def check_brute_force_prefix(L):
    rng = np.random.default_rng(6)
    for trial in range(60):
        B = int(rng.choice([2, 4]))
        N = int(rng.integers(1, 6))
        base = rng.integers(0, 3, size=8 * B, dtype=np.int32)
        stored = {t: [_mutate(rng, base, int(rng.integers(0, 9 * B)))
                      for _ in range(int(rng.integers(0, 4)))] for t in range(-1, N)}
        ix = oracle.OracleIndex(N, L)
        for t, prompts in stored.items():
            for p in prompts:
                ix.insert(oracle.block_hashes(p, B, 0, L), t)
        for _ in range(6):
            req = _mutate(rng, base, int(rng.integers(0, 9 * B)))
            h = oracle.block_hashes(req, B, 0, L)
            c, g = ix.prefix_hits(h)
            assert g == brute_hit(req, stored[-1], B)
            for i in range(N):
                assert c[i] == brute_hit(req, stored[i], B), (trial, i)
            # the routing outputs agree with these hits
            load = rng.integers(0, 50, size=N)
            out = _route(ix, B, 2, [req], load)
            i = int(out["instance"][0])
            gi = max(c[i], g)
            assert out["local_hit"][0] == B * c[i]
            assert out["global_hit"][0] == B * (gi - c[i])
            cost = [1 * load[j] + 4 * (len(req) - B * max(c[j], g)) + 2 * B * (max(c[j], g) - c[j])
                    for j in range(N)]
            assert i == int(np.argmin(cost))


def check_non_prefix_closed(L):
    """A tier that holds a deep block but not an earlier one stops at the gap."""
    rng = np.random.default_rng(8)
    B = 4
    t = rng.integers(0, 151936, size=10 * B, dtype=np.int32)
    h = oracle.block_hashes(t, B, 0, L)
    ix = oracle.OracleIndex(2, L)
    ix.insert(h[[0, 1, 2, 4, 5]], 0)
    ix.insert(h[[1, 2, 3]], 1)
    ix.insert(h[:7], -1)
    c, g = ix.prefix_hits(h)
    assert list(c) == [3, 0] and g == 7


def check_jsq_when_index_empty(L):
    """Empty index: cost_i = w_load*load_i + w_miss*L, so routing is
    join-the-shortest-queue (Section 4.1, 'Load-balance-only'), ties to the
    lowest id."""
    rng = np.random.default_rng(9)
    for N in (1, 3, 8, 33):
        ix = oracle.OracleIndex(N, L)
        reqs = [rng.integers(0, 151936, size=int(rng.integers(0, 200)), dtype=np.int32)
                for _ in range(20)]
        for _ in range(5):
            load = rng.integers(0, 4, size=N)  # many ties
            out = _route(ix, 8, 3, reqs, load)
            assert np.all(out["instance"] == int(np.argmin(load)))
            assert np.all(out["local_hit"] == 0) and np.all(out["global_hit"] == 0)


def check_argmax_hit_when_load_ignored(L):
    """w_load = 0 and an empty global tier: cost_i = w_miss*(L - B*c_i), so
    routing picks the instance with the longest local hit (the sticky choice
    of Figure 10), ties to the lowest id."""
    rng = np.random.default_rng(10)
    B = 2
    for trial in range(30):
        N = int(rng.integers(1, 7))
        base = rng.integers(0, 3, size=10 * B, dtype=np.int32)
        stored = {i: [_mutate(rng, base, int(rng.integers(0, 11 * B)))
                      for _ in range(int(rng.integers(0, 3)))] for i in range(N)}
        ix = oracle.OracleIndex(N, L)
        for i, ps in stored.items():
            for p in ps:
                ix.insert(oracle.block_hashes(p, B, 0, L), i)
        req = _mutate(rng, base, int(rng.integers(0, 11 * B)))
        c = [brute_hit(req, stored[i], B) for i in range(N)]
        out = _route(ix, B, 1, [req], rng.integers(0, 1000, size=N), w=(0, 3, 5))
        assert int(out["instance"][0]) == int(np.argmax(c))


def check_equal_costs_pick_zero(L):
    ix = oracle.OracleIndex(5, L)
    rng = np.random.default_rng(11)
    reqs = [rng.integers(0, 151936, size=50, dtype=np.int32) for _ in range(4)]
    out = _route(ix, 4, 1, reqs, [7] * 5)
    assert np.all(out["instance"] == 0)


def check_paper_examples(L):
    ex = _golden_json("paper_examples.json")
    rng = np.random.default_rng(12)
    a = ex["three_token_two_hits"]
    B = a["block_size"]
    t = rng.integers(0, 151936, size=a["prompt_len"], dtype=np.int32)
    ix = oracle.OracleIndex(1, L)
    ix.insert(oracle.block_hashes(t, B, 0, L)[:a["cached_blocks"]], 0)
    out = _route(ix, B, 1, [t], [0])
    assert out["local_hit"][0] == a["expect_local_hit"]
    assert a["prompt_len"] - out["local_hit"][0] - out["global_hit"][0] == a["expect_tokens_to_compute"]

    b = ex["reuse_70_to_80"]
    B = b["block_size"]
    t = rng.integers(0, 151936, size=b["prompt_len"], dtype=np.int32)
    h = oracle.block_hashes(t, B, 0, L)
    comp = []
    for k in (b["cached_blocks_low"], b["cached_blocks_high"]):
        ix = oracle.OracleIndex(1, L)
        ix.insert(h[:k], 0)
        out = _route(ix, B, 1, [t], [0])
        comp.append(b["prompt_len"] - int(out["local_hit"][0]))
    assert comp == [b["expect_compute_low"], b["expect_compute_high"]]
    assert Fraction(comp[0] - comp[1], comp[0]) == Fraction(b["expect_cut_num"], b["expect_cut_den"])


def check_hand_costs(L):
    ex = _golden_json("hand_costs.json")
    B, Lp, N = ex["block_size"], ex["prompt_len"], ex["num_instances"]
    rng = np.random.default_rng(13)
    t = rng.integers(0, 151936, size=Lp, dtype=np.int32)
    h = oracle.block_hashes(t, B, 0, L)
    ix = oracle.OracleIndex(N, L)
    ix.insert(h[:ex["global_blocks"]], -1)
    for i, k in enumerate(ex["local_blocks"]):
        ix.insert(h[:k], i)
    for case in ex["cases"]:
        out = _route(ix, B, 1, [t], case["load"], w=tuple(ex["weights"]))
        assert int(out["instance"][0]) == case["instance"], case
        assert int(out["local_hit"][0]) == case["local_hit"], case
        assert int(out["global_hit"][0]) == case["global_hit"], case


def check_batch_invariants(L):
    """Invariants on a synthetic multi-turn batch: hits never exceed the full
    blocks, and a session's key is the same on every turn."""
    from synth import agent_trace, ReplayDriver
    tr = agent_trace("c1_tiny", scale=0.25, seed=3)
    p = tr.params
    ix = oracle.OracleIndex(p.num_instances, L)
    drv = ReplayDriver(p.num_instances, p.block_size)
    keys_by_session = {}
    for bt in tr.batches():
        out = ix.route_batch(p.block_size, p.session_blocks, 0, bt.tokens, bt.offsets, drv.load,
                             p.w_load, p.w_miss, p.w_glob, want_hashes=True)
        lens = bt.lengths()
        nfull = (lens // p.block_size) * p.block_size
        assert np.all(out["local_hit"] + out["global_hit"] <= nfull)
        assert np.all(out["local_hit"] >= 0) and np.all(out["global_hit"] >= 0)
        for s, k in zip(bt.sessions.tolist(), out["session_key"].tolist()):
            assert keys_by_session.setdefault(s, k) == k
        ins_k, ins_t, ev_k, ev_t = drv.after_batch(bt.offsets, out["instance"], out["local_hit"],
                                                   out["block_hashes"])
        ix.insert(ins_k, ins_t)
        ix.evict(ev_k, ev_t)
    assert len(keys_by_session) == tr.n_sessions


def check_lru_recency(L):
    """The LRU oracle against recency worked out by hand, the rule's special
    cases (one slot keeps the most recent touch: the last committed
    request's first block; a cap above every key evicts nothing), and a
    second formulation of the rule (move-to-back ordered dicts, deepest
    block first within a request)."""
    from collections import OrderedDict
    # hand example: N = 2, local cap 3, global cap 0
    lru = oracle.OracleLRU(2, local_cap=3)
    ek, et = lru.commit([4], [1], [11, 12, 13, 14], also_global=False)
    # stamps (0,0,0) (0,0,-1) (0,0,-2) (0,0,-3): the deepest block (14) leaves
    assert ek.tolist() == [14] and et.tolist() == [1]
    assert [lru.holds(k, 1) for k in (11, 12, 13, 14)] == [True, True, True, False]
    ek, et = lru.commit([1, 2], [1, 0], [21, 31, 32], also_global=False)
    # tier 1 now: 21 (1,0,0), 11 (0,0,0), 12 (0,0,-1), 13 (0,0,-2): 13 leaves
    assert ek.tolist() == [13] and lru.size(1) == 3 and lru.size(0) == 2
    ek, et = lru.commit([2, 1], [1, 1], [12, 41, 11], also_global=False)
    # request 1 touches 11 at (2,1,0), request 0 touches 12 at (2,0,0) and 41
    # at (2,0,-1): tier 1 holds 11, 12, 41, 21 by recency; 21 leaves
    assert ek.tolist() == [21] and all(lru.holds(k, 1) for k in (11, 12, 41))
    # one slot: the last committed request's first block
    one = oracle.OracleLRU(3, local_cap=1, global_cap=1)
    one.commit([3, 2, 2], [2, 0, 2], [1, 2, 3, 4, 5, 6, 7], also_global=True)
    assert one.holds(6, 2) and one.size(2) == 1 and one.holds(4, 0) and one.holds(6, -1)
    # a cap above every key: nothing leaves
    big = oracle.OracleLRU(2, local_cap=100, global_cap=100)
    ek, _ = big.commit([3, 3], [0, 1], [1, 2, 3, 1, 2, 3], also_global=True)
    assert len(ek) == 0 and big.size(-1) == 3
    # the second formulation, on random commits with repeated keys
    rng = np.random.default_rng(15)
    N, cap, gcap = 3, 7, 11
    a = oracle.OracleLRU(N, local_cap=cap, global_cap=gcap)
    od = {t: OrderedDict() for t in range(-1, N)}
    for step in range(40):
        n = int(rng.integers(1, 6))
        nb = rng.integers(0, 6, size=n)
        inst = rng.integers(-1, N, size=n)
        h = rng.integers(2, 40, size=int(nb.sum())).astype(np.uint64)
        ek, et = a.commit(nb, inst, h, also_global=True)
        pos = 0
        for r in range(n):
            keys = h[pos:pos + nb[r]].tolist()
            pos += int(nb[r])
            if inst[r] < 0:
                continue
            for t in (int(inst[r]), -1):
                for key in reversed(keys):  # deepest first: the least recent of the request
                    od[t].pop(key, None)
                    od[t][key] = None
        want = []
        for t, d in od.items():
            c = gcap if t < 0 else cap
            while len(d) > c:
                want.append((d.popitem(last=False)[0], t))
        assert sorted(zip(ek.tolist(), et.tolist())) == sorted(want), step
        for t in range(-1, N):
            assert set(a.stamp[t]) == set(od[t]), (step, t)


def check_index_set_semantics(L):
    """Insert/evict behave as set operations per tier (against Python sets)."""
    rng = np.random.default_rng(14)
    N = 5
    ix = oracle.OracleIndex(N, L)
    ref = {t: set() for t in range(-1, N)}
    universe = rng.integers(2, 2**62, size=300).astype(np.uint64)
    for step in range(40):
        k = rng.choice(universe, size=int(rng.integers(0, 60)))
        t = rng.integers(-1, N, size=len(k)).astype(np.int32)
        if rng.random() < 0.6:
            ix.insert(k, t)
            for a, b in zip(k.tolist(), t.tolist()):
                ref[b].add(a)
        else:
            ix.evict(k, t)
            for a, b in zip(k.tolist(), t.tolist()):
                ref[b].discard(a)
        for key in rng.choice(universe, size=30).tolist():
            for tier in range(-1, N):
                assert ix.contains(key, tier) == (key in ref[tier])


# ---------------------------------------------------------------------------
# session-centric policy (Figure 10)
# ---------------------------------------------------------------------------

def eq1_cost(n, Lp, c_lin, c_att):
    """Eq. 1 as printed: c_linear*n + c_attn*n*(L - n/2), exactly."""
    return Fraction(c_lin) * n + Fraction(c_att) * n * (Lp - Fraction(n, 2))


def _policy(ix, B, reqs, queued, turn, est_hit, c_lin=1, c_att=0, d0=1 << 60, d1=0,
            hit_num=1, hit_den=2, rr_base=0, S=1):
    from synth.traces import pack
    tokens, offsets = pack(reqs)
    return ix.route_batch_policy(B, S, 0, tokens, offsets, np.asarray(queued, np.int64),
                                 np.asarray(turn, np.int32), np.asarray(est_hit, np.int64),
                                 c_lin, c_att, d0, d1, hit_num, hit_den, rr_base)


def _held(L, ix, t, B, tier_blocks):
    h = oracle.block_hashes(t, B, 0, L)
    for tier, k in tier_blocks.items():
        if k:
            ix.insert(h[:k], tier)


def check_policy_eq1_boundary(L):
    """Balance branch: the load model is Eq. 1 plus the queue. Instance 1
    caches k blocks, instance 0 none; instance 1 wins exactly when
    q_1 - q_0 < cost(L, L) - cost(L - kB, L), ties to instance 0."""
    rng = np.random.default_rng(40)
    for B, Lp, k, c_lin, c_att in ((4, 64, 5, 3, 1), (8, 77, 3, 1, 2), (2, 31, 9, 0, 7),
                                   (16, 500, 17, 11, 3), (4, 9, 1, 5, 1)):
        t = rng.integers(0, 151936, size=Lp, dtype=np.int32)
        ix = oracle.OracleIndex(2, L)
        _held(L, ix, t, B, {1: k})
        T = eq1_cost(Lp, Lp, c_lin, c_att) - eq1_cost(Lp - k * B, Lp, c_lin, c_att)
        lo, hi = T.numerator // T.denominator, -((-T.numerator) // T.denominator)
        for D in (lo - 1, lo, hi, hi + 1):
            q0 = 1 << 30
            out = _policy(ix, B, [t], [q0, q0 + D], [0], [0], c_lin=c_lin, c_att=c_att)
            want = 1 if D < T else 0
            assert int(out["instance"][0]) == want, (B, Lp, k, D, T)
            assert int(out["stick"][0]) == 0
            assert int(out["local_hit"][0]) == (k * B if want else 0)


def check_policy_first_turn_is_cost_argmin(L):
    """First-turn requests take the balance branch; with C_ATT = 0 its load
    q_i + C_LIN*(L - B*c_i) is the argmin cost of a3-a5 with w_load = 1,
    w_miss = C_LIN and an empty global tier (one request, rotation from 0,
    so ties go to the lowest id in both)."""
    rng = np.random.default_rng(41)
    B = 2
    for trial in range(40):
        N = int(rng.integers(1, 7))
        base = rng.integers(0, 3, size=10 * B, dtype=np.int32)
        ix = oracle.OracleIndex(N, L)
        for i in range(N):
            for _ in range(int(rng.integers(0, 3))):
                ix.insert(oracle.block_hashes(_mutate(rng, base, int(rng.integers(0, 11 * B))), B, 0, L), i)
        req = _mutate(rng, base, int(rng.integers(0, 11 * B)))
        q = rng.integers(0, 30, size=N)
        c_lin = int(rng.integers(0, 4))
        a = _policy(ix, B, [req], q, [0], [0], c_lin=c_lin)
        b = _route(ix, B, 1, [req], q, w=(1, c_lin, 0))
        assert int(a["instance"][0]) == int(b["instance"][0])
        assert int(a["local_hit"][0]) == int(b["local_hit"][0]) and int(a["stick"][0]) == 0


def check_policy_sticks_to_longest_local_hit(L):
    """A follow-up with a cached session and a loose deadline sticks to
    prev = argmax_i c_i (lowest id among equals), whatever the loads."""
    rng = np.random.default_rng(42)
    B = 2
    for trial in range(40):
        N = int(rng.integers(1, 7))
        base = rng.integers(0, 3, size=10 * B, dtype=np.int32)
        stored = {i: [_mutate(rng, base, int(rng.integers(0, 11 * B)))
                      for _ in range(int(rng.integers(0, 3)))] for i in range(N)}
        ix = oracle.OracleIndex(N, L)
        for i, ps in stored.items():
            for p in ps:
                ix.insert(oracle.block_hashes(p, B, 0, L), i)
        req = _mutate(rng, base, int(rng.integers(0, 11 * B)))
        c = [brute_hit(req, stored[i], B) for i in range(N)]
        out = _policy(ix, B, [req], rng.integers(0, 1 << 20, size=N), [3], [0])
        if max(c) > 0:
            assert int(out["instance"][0]) == int(np.argmax(c)) and int(out["stick"][0]) == 1
            assert int(out["local_hit"][0]) == B * max(c)
        else:  # nothing cached: not session_cached, so balanced
            assert int(out["stick"][0]) == 0


def check_policy_session_cached_threshold(L):
    """session_cached: c[prev] > HIT_RATIO * est_hit, strictly; at equality
    the request is balanced like a first turn."""
    rng = np.random.default_rng(43)
    B, Lp, k = 4, 40, 6
    t = rng.integers(0, 151936, size=Lp, dtype=np.int32)
    ix = oracle.OracleIndex(3, L)
    _held(L, ix, t, B, {2: k})
    q = [0, 5, 1 << 40]  # instance 0 is the least loaded
    for num, den in ((1, 2), (3, 4), (9, 10), (1, 1)):
        # B*k*den == num*e exactly for e = B*k*den/num when that is an integer
        e = Fraction(B * k * den, num)
        if e.denominator != 1:
            continue
        e = int(e)
        out = _policy(ix, B, [t, t], q, [1, 1], [e, e - 1], hit_num=num, hit_den=den)
        assert int(out["stick"][0]) == 0 and int(out["instance"][0]) == 0
        assert int(out["stick"][1]) == 1 and int(out["instance"][1]) == 2


def check_policy_slo_migration(L):
    """meets_ttft: estimate_load <= SLACK*PREFILL_RATE*(b + a*L), here the
    budget d0 + d1*L in cost units. prev sticks while it meets the deadline
    (inclusive), migrates to the least-loaded instance when another one meets
    it, and sticks again when no instance meets it."""
    rng = np.random.default_rng(44)
    B, Lp, k, c_lin, c_att = 4, 64, 10, 2, 1
    t = rng.integers(0, 151936, size=Lp, dtype=np.int32)
    ix = oracle.OracleIndex(3, L)
    _held(L, ix, t, B, {1: k})
    q = [50, 4000, 20]
    est = [q[i] + eq1_cost(Lp - (k * B if i == 1 else 0), Lp, c_lin, c_att) for i in range(3)]
    assert all(e.denominator == 1 for e in est)  # n is even in every case here
    assert est[2] < est[0] < est[1]
    d1 = 3
    for d0, want, stick in ((est[1] - d1 * Lp, 1, 1),       # prev meets exactly
                            (est[1] - d1 * Lp - 1, 2, 0),   # prev misses, others meet
                            (est[2] - d1 * Lp, 2, 0),       # only the least loaded meets
                            (est[2] - d1 * Lp - 1, 1, 1)):  # no instance meets: stick
        out = _policy(ix, B, [t], q, [1], [0], c_lin=c_lin, c_att=c_att, d0=int(d0), d1=d1)
        assert (int(out["instance"][0]), int(out["stick"][0])) == (want, stick), (d0, est)


def check_policy_round_robin_ties(L):
    """rr_argmin: with nothing cached and equal queues every load ties, and
    request r of the batch goes to (rr_base + r) mod N."""
    rng = np.random.default_rng(45)
    for N in (1, 2, 5, 8):
        ix = oracle.OracleIndex(N, L)
        reqs = [rng.integers(0, 151936, size=int(rng.integers(0, 90)), dtype=np.int32) for _ in range(13)]
        for base in range(N):
            out = _policy(ix, 4, reqs, [9] * N, [0] * 13, [0] * 13, c_lin=1, c_att=1, rr_base=base)
            assert np.array_equal(out["instance"], (base + np.arange(13)) % N)


def _coloc(ix, B, reqs, queued, tpot, nreq, turn, est_hit, c_lin=1, c_att=0, d0=1 << 60, d1=0,
           hit_num=1, hit_den=2, rr_base=0, S=1):
    from synth.traces import pack
    tokens, offsets = pack(reqs)
    return ix.route_batch_coloc(B, S, 0, tokens, offsets, np.asarray(queued, np.int64),
                                np.asarray(tpot, np.int64), np.asarray(nreq, np.int64),
                                np.asarray(turn, np.int32), np.asarray(est_hit, np.int64),
                                c_lin, c_att, d0, d1, hit_num, hit_den, rr_base)


def check_coloc_reduces_to_disaggregated(L):
    """Appendix B against Figure 10: with every instance passing the TPOT
    check, one request per instance and a deadline every instance meets, the
    colocated policy decides exactly as the disaggregated one."""
    rng = np.random.default_rng(50)
    B = 2
    for trial in range(40):
        N = int(rng.integers(1, 7))
        base = rng.integers(0, 3, size=10 * B, dtype=np.int32)
        ix = oracle.OracleIndex(N, L)
        for i in range(N):
            for _ in range(int(rng.integers(0, 3))):
                ix.insert(oracle.block_hashes(_mutate(rng, base, int(rng.integers(0, 11 * B))), B, 0, L), i)
        reqs = [_mutate(rng, base, int(rng.integers(0, 11 * B))) for _ in range(5)]
        q = rng.integers(0, 50, size=N)
        kw = dict(c_lin=int(rng.integers(0, 4)), c_att=int(rng.integers(0, 3)), rr_base=int(rng.integers(0, N)))
        turn, est = rng.integers(0, 2, size=5), rng.integers(0, 30, size=5)
        a = _coloc(ix, B, reqs, q, [1 << 60] * N, [1] * N, turn, est, **kw)
        b = _policy(ix, B, reqs, q, turn, est, **kw)
        for k in ("instance", "stick", "local_hit", "global_hit"):
            assert np.array_equal(a[k], b[k]), (trial, k)


def check_coloc_tpot_filter(L):
    """An instance whose live decodes cannot absorb the prefill (2*cost_i >
    2*T_i) is not a candidate: a cached follow-up leaves prev when prev fails
    the check, the balance skips failing instances, and when none passes
    every instance is a candidate again."""
    rng = np.random.default_rng(51)
    B, Lp, k, c_lin, c_att = 4, 48, 8, 3, 1
    t = rng.integers(0, 151936, size=Lp, dtype=np.int32)
    ix = oracle.OracleIndex(3, L)
    _held(L, ix, t, B, {1: k})
    cost = [eq1_cost(Lp - (k * B if i == 1 else 0), Lp, c_lin, c_att) for i in range(3)]
    assert all(x.denominator == 1 for x in cost)
    big = 1 << 50
    q = [7, 5, 100]  # instance 0 the least loaded; queues do not count in the TPOT check
    kw = dict(c_lin=c_lin, c_att=c_att)
    out = _coloc(ix, B, [t], q, [big, int(cost[1]), big], [1, 1, 1], [1], [0], **kw)
    assert (int(out["instance"][0]), int(out["stick"][0])) == (1, 1)   # prev passes exactly
    out = _coloc(ix, B, [t], q, [big, int(cost[1]) - 1, big], [1, 1, 1], [1], [0], **kw)
    assert (int(out["instance"][0]), int(out["stick"][0])) == (0, 0)   # prev fails: balanced
    out = _coloc(ix, B, [t], q, [int(cost[0]) - 1, int(cost[1]) - 1, big], [1, 1, 1], [1], [0], **kw)
    assert (int(out["instance"][0]), int(out["stick"][0])) == (2, 0)   # only instance 2 passes
    out = _coloc(ix, B, [t], q, [0, 0, 0], [1, 1, 1], [1], [0], **kw)
    assert (int(out["instance"][0]), int(out["stick"][0])) == (1, 1)   # none passes: all are candidates


def check_coloc_lmetric_product(L):
    """The balance target minimises estimate_load * num_requests (LMetric's
    product, not a sum): it flips exactly where the products cross, an idle
    instance (no requests) scores 0, and equal products rotate."""
    rng = np.random.default_rng(52)
    B, Lp, c_lin, c_att = 4, 40, 2, 1
    t = rng.integers(0, 151936, size=Lp, dtype=np.int32)
    ix = oracle.OracleIndex(2, L)
    c = eq1_cost(Lp, Lp, c_lin, c_att)  # nothing cached: same prefill cost everywhere
    assert c.denominator == 1
    c = int(c)
    big = [1 << 60] * 2
    for q0, q1, r0, r1 in ((0, 0, 3, 2), (10, 0, 2, 3), (5 * c, c, 1, 3), (0, 10 ** 6, 7, 0)):
        e0, e1 = q0 + c, q1 + c
        want = 0 if e0 * r0 < e1 * r1 else 1 if e1 * r1 < e0 * r0 else 0  # ties: rotation from 0
        out = _coloc(ix, B, [t], [q0, q1], big, [r0, r1], [0], [0], c_lin=c_lin, c_att=c_att)
        assert int(out["instance"][0]) == want, (q0, q1, r0, r1)
    out = _coloc(ix, B, [t] * 4, [0, 0], big, [2, 2], [0] * 4, [0] * 4, c_lin=c_lin, c_att=c_att, rr_base=1)
    assert np.array_equal(out["instance"], [1, 0, 1, 0])
    # products beyond 64 bits: est2 about 2^60 times 2^20 requests
    out = _coloc(ix, B, [t], [(1 << 59) - 1, 1 << 59], big, [1 << 20, (1 << 20) - 1], [0], [0],
                 c_lin=c_lin, c_att=c_att)
    assert int(out["instance"][0]) == 1


def check_coloc_no_last_resort(L):
    """Under colocation a cached follow-up sticks only if prev meets the
    deadline; when no instance meets it the request is balanced (Figure 10
    would stick)."""
    rng = np.random.default_rng(53)
    B, Lp, k = 4, 64, 10
    t = rng.integers(0, 151936, size=Lp, dtype=np.int32)
    ix = oracle.OracleIndex(3, L)
    _held(L, ix, t, B, {1: k})
    q = [50, 4000, 20]
    big = [1 << 60] * 3
    kw = dict(c_lin=2, c_att=1, d0=0, d1=0)  # a deadline nobody meets
    a = _coloc(ix, B, [t], q, big, [1, 1, 1], [1], [0], **kw)
    b = _policy(ix, B, [t], q, [1], [0], **kw)
    assert (int(b["instance"][0]), int(b["stick"][0])) == (1, 1)
    assert int(a["stick"][0]) == 0 and int(a["instance"][0]) != 1


# ---------------------------------------------------------------------------
# session reconstruction (Appendix A)
# ---------------------------------------------------------------------------

def _link(L, B, reqs, users, turns, seed=0):
    from synth.traces import pack
    tokens, offsets = pack(reqs)
    return oracle.link_sessions(B, seed, tokens, offsets, users, turns, L)


def check_link_against_token_prefixes(L):
    """Brute force by token comparison: r follows the latest earlier p of the
    same user and turn_r - 1 whose full blocks are the first tokens of r."""
    rng = np.random.default_rng(60)
    B = 2
    for trial in range(30):
        base = rng.integers(0, 3, size=12 * B, dtype=np.int32)
        n = int(rng.integers(1, 25))
        reqs = [_mutate(rng, base, int(rng.integers(0, 12 * B))) for _ in range(n)]
        users = rng.integers(0, 3, size=n)
        turns = rng.integers(0, 4, size=n)
        parent, session = _link(L, B, reqs, users, turns)
        want_session = []
        for r in range(n):
            want = -1
            for q in range(r - 1, -1, -1):
                nq = len(reqs[q]) // B
                if users[q] != users[r] or turns[q] != turns[r] - 1 or nq > len(reqs[r]) // B:
                    continue
                if np.array_equal(reqs[q][:nq * B], reqs[r][:nq * B]):
                    want = q
                    break
            assert parent[r] == want, (trial, r)
            want_session.append(r if want < 0 else want_session[want])
            assert session[r] == want_session[r], (trial, r)


def check_link_recovers_generated_sessions(L):
    """A multi-turn trace without truncation, one user per session: every
    turn extends the previous one, so the chains are the generator's
    sessions and each session's id is its first request."""
    from synth import agent_trace
    from synth.traces import pack
    tr = agent_trace("c1_tiny", scale=0.25, seed=5)
    bs = list(tr.batches())
    reqs, sess, turns = [], [], []
    for bt in bs:
        for r in range(bt.n_requests):
            reqs.append(bt.tokens[bt.offsets[r]:bt.offsets[r + 1]])
        sess.extend(bt.sessions.tolist())
        turns.extend(bt.turns.tolist())
    sess, turns = np.array(sess), np.array(turns)
    parent, session = _link(L, tr.params.block_size, reqs, sess, turns)
    first = {}
    for r, s_ in enumerate(sess):
        first.setdefault(int(s_), r)
    assert all(int(session[r]) == first[int(s_)] for r, s_ in enumerate(sess))
    assert np.all((parent >= 0) == (turns > 0))


def check_link_special_cases(L):
    """Different users or a turn gap never link; the latest of two equal
    parents wins; a prompt shorter than a block links as the empty prefix."""
    rng = np.random.default_rng(61)
    B = 4
    a = rng.integers(0, 151936, size=8 * B, dtype=np.int32)
    ext = np.concatenate([a, rng.integers(0, 151936, size=3 * B, dtype=np.int32)])
    tiny = a[:B - 1]
    reqs = [a, a, ext, ext, tiny, a]
    users = [1, 1, 1, 2, 3, 3]
    turns = [0, 0, 1, 1, 0, 1]
    parent, session = _link(L, B, reqs, users, turns)
    assert parent.tolist() == [-1, -1, 1, -1, -1, 4]
    assert session.tolist() == [0, 1, 1, 3, 4, 4]
    parent, _ = _link(L, B, [a, ext], [1, 1], [0, 2])  # turn gap
    assert parent.tolist() == [-1, -1]
    # a chain of four turns: every request's session is the first one
    ext2 = np.concatenate([ext, rng.integers(0, 151936, size=2 * B, dtype=np.int32)])
    ext3 = np.concatenate([ext2, rng.integers(0, 151936, size=5, dtype=np.int32)])
    parent, session = _link(L, B, [a, ext, ext2, ext3], [7] * 4, [0, 1, 2, 3])
    assert parent.tolist() == [-1, 0, 1, 2] and session.tolist() == [0, 0, 0, 0]


# ---------------------------------------------------------------------------
# baseline scorers (Section 5.1)
# ---------------------------------------------------------------------------

def _baseline(ix, B, reqs, scorer, queued, batch, lam=(1, 2)):
    from synth.traces import pack
    tokens, offsets = pack(reqs)
    return ix.route_batch_baseline(B, 1, 0, tokens, offsets, scorer, np.asarray(queued, np.int64),
                                   np.asarray(batch, np.int64), *lam)


def _bailian_f(l, lmax, hit_tokens, Lp, lam):
    """Section 5.1's weighted sum, exactly: (1 - lambda) * l / max l +
    lambda * (1 - hit ratio)."""
    lh = Fraction(l, lmax) if lmax else Fraction(0)
    ch = Fraction(hit_tokens, Lp) if Lp else Fraction(0)
    return (1 - lam) * lh + lam * (1 - ch)


def check_baselines_against_their_definitions(L):
    """Bailian's normalised weighted sum and LMetric's product, evaluated in
    exact rationals from hits found by token comparison, against the
    oracle's choice (ties to the lowest id)."""
    rng = np.random.default_rng(70)
    B = 2
    for trial in range(60):
        N = int(rng.integers(1, 7))
        base = rng.integers(0, 3, size=10 * B, dtype=np.int32)
        stored = {i: [_mutate(rng, base, int(rng.integers(0, 11 * B)))
                      for _ in range(int(rng.integers(0, 3)))] for i in range(N)}
        ix = oracle.OracleIndex(N, L)
        for i, ps in stored.items():
            for p_ in ps:
                ix.insert(oracle.block_hashes(p_, B, 0, L), i)
        req = _mutate(rng, base, int(rng.integers(0, 11 * B)))
        c = [brute_hit(req, stored[i], B) for i in range(N)]
        Lp = len(req)
        batch = rng.integers(0, [1, 4, 50][trial % 3], size=N)
        q = rng.integers(0, 40, size=N)
        lam = (int(rng.integers(0, 7)), 6)
        f = [_bailian_f(int(batch[i]), int(batch.max()), B * c[i], Lp, Fraction(*lam)) for i in range(N)]
        out = _baseline(ix, B, [req], 1, q, batch, lam)
        assert int(out["instance"][0]) == min(range(N), key=lambda i: (f[i], i)), (trial, f)
        g = [(int(q[i]) + Lp - B * c[i]) * int(batch[i]) for i in range(N)]
        out = _baseline(ix, B, [req], 2, q, batch)
        assert int(out["instance"][0]) == min(range(N), key=lambda i: (g[i], i)), (trial, g)


def check_baselines_special_cases(L):
    """Bailian with lambda = 0 is join-the-shortest-batch; with lambda = 1 it
    is the longest local hit; scaling every batch size leaves it unchanged.
    LMetric sends work to an idle instance (no requests) first."""
    rng = np.random.default_rng(71)
    B = 4
    t = rng.integers(0, 151936, size=60, dtype=np.int32)
    ix = oracle.OracleIndex(4, L)
    _held(L, ix, t, B, {2: 9, 3: 4})
    batch = np.array([5, 3, 9, 3])
    assert int(_baseline(ix, B, [t], 1, [0] * 4, batch, (0, 5))["instance"][0]) == 1
    assert int(_baseline(ix, B, [t], 1, [0] * 4, batch, (5, 5))["instance"][0]) == 2
    for lam in ((1, 3), (2, 3), (7, 10)):
        a = _baseline(ix, B, [t], 1, [0] * 4, batch, lam)["instance"][0]
        b = _baseline(ix, B, [t], 1, [0] * 4, batch * 1000, lam)["instance"][0]
        assert a == b
    out = _baseline(ix, B, [t], 2, [10 ** 9, 0, 0, 0], [0, 3, 1, 2])
    assert int(out["instance"][0]) == 0


# ---------------------------------------------------------------------------
# sequential-update variant (reading 7)
# ---------------------------------------------------------------------------

def _seq(ix, B, reqs, load, w, S=1):
    from synth.traces import pack
    tokens, offsets = pack(reqs)
    return ix.route_batch_sequential(B, S, 0, tokens, offsets, np.asarray(load, np.int64), *w)


def check_sequential_matches_snapshot_without_load(L):
    """With w_load = 0 the loads never matter: the sequential decisions are
    the snapshot ones, and the final loads are the starting loads plus each
    request's work on its instance."""
    rng = np.random.default_rng(80)
    B = 2
    for trial in range(30):
        N = int(rng.integers(1, 7))
        base = rng.integers(0, 3, size=10 * B, dtype=np.int32)
        ix = oracle.OracleIndex(N, L)
        for i in range(N):
            for _ in range(int(rng.integers(0, 3))):
                ix.insert(oracle.block_hashes(_mutate(rng, base, int(rng.integers(0, 11 * B))), B, 0, L), i)
        reqs = [_mutate(rng, base, int(rng.integers(0, 11 * B))) for _ in range(12)]
        load = rng.integers(0, 100, size=N)
        a = _seq(ix, B, reqs, load, (0, 3, 1))
        b = _route(ix, B, 1, reqs, load, w=(0, 3, 1))
        for k in ("instance", "local_hit", "global_hit", "session_key"):
            assert np.array_equal(a[k], b[k]), (trial, k)
        work = np.zeros(N, np.int64)
        for r, t in enumerate(reqs):
            work[b["instance"][r]] += len(t) - int(b["local_hit"][r])
        assert np.array_equal(a["load_after"], load + work)


def check_sequential_join_shortest_queue(L):
    """Empty index, equal loads, equal prompts: each request joins the
    shortest queue and lengthens it, so request r goes to r mod N; with
    unequal prompts the choice follows the running queues exactly."""
    rng = np.random.default_rng(81)
    for N in (1, 2, 3, 7):
        ix = oracle.OracleIndex(N, L)
        reqs = [rng.integers(0, 151936, size=40, dtype=np.int32) for _ in range(15)]
        out = _seq(ix, 4, reqs, [0] * N, (1, 4, 2))
        assert np.array_equal(out["instance"], np.arange(15) % N)
        lens = rng.integers(1, 200, size=15)
        reqs = [rng.integers(0, 151936, size=int(x), dtype=np.int32) for x in lens]
        q = np.array(rng.integers(0, 300, size=N))
        want = []
        for x in lens:
            i = int(np.argmin(q))  # w_load * q + w_miss * L: only q differs
            want.append(i)
            q[i] += x
        out = _seq(ix, 4, reqs, q - np.bincount(want, weights=lens, minlength=N).astype(np.int64), (1, 4, 2))
        assert out["instance"].tolist() == want


# ---------------------------------------------------------------------------
# reuse breakdown (Section 3.1)
# ---------------------------------------------------------------------------

def check_reuse_against_token_prefixes(L):
    """Brute force by token comparison: block b of r is reused when an
    earlier request starts with r's first b+1 blocks; the prefix stops at the
    first block that is not; each reused block goes to the system prompt when
    b < sys_r, else to intra- or inter-session by the earliest such request's
    session."""
    from synth.traces import pack
    rng = np.random.default_rng(90)
    B = 2
    for trial in range(25):
        base = rng.integers(0, 3, size=12 * B, dtype=np.int32)
        n = int(rng.integers(1, 30))
        reqs = [_mutate(rng, base, int(rng.integers(0, 12 * B))) for _ in range(n)]
        sessions = rng.integers(0, 4, size=n)
        sys_b = rng.integers(0, 4, size=n)
        tokens, offsets = pack(reqs)
        out = oracle.reuse_breakdown(B, 0, tokens, offsets, sessions, sys_b, L)
        for r in range(n):
            want = dict(hit=0, sys=0, intra=0, inter=0)
            for b in range(len(reqs[r]) // B):
                pre = reqs[r][:(b + 1) * B]
                prod = next((q for q in range(r) if len(reqs[q]) >= len(pre) and
                             np.array_equal(reqs[q][:len(pre)], pre)), -1)
                if prod < 0:
                    break
                want["hit"] += 1
                key = "sys" if b < sys_b[r] else "intra" if sessions[prod] == sessions[r] else "inter"
                want[key] += 1
            for k in want:
                assert int(out[k][r]) == want[k], (trial, r, k)


def check_reuse_on_a_multi_turn_trace(L):
    """Turn t of a session resends turn t-1 whole: with one session per user
    and no truncation, every follow-up reuses at least its parent's blocks,
    first turns reuse only the shared system prompt, and the parts add up."""
    from synth import agent_trace
    from synth.traces import pack
    tr = agent_trace("c1_tiny", scale=0.25, seed=9)
    B = tr.params.block_size
    reqs, sess, turns = [], [], []
    for bt in tr.batches():
        for r in range(bt.n_requests):
            reqs.append(bt.tokens[bt.offsets[r]:bt.offsets[r + 1]])
        sess.extend(bt.sessions.tolist())
        turns.extend(bt.turns.tolist())
    tokens, offsets = pack(reqs)
    sys_b = np.full(len(reqs), tr.system_prompt_len // B, np.int32)
    out = oracle.reuse_breakdown(B, 0, tokens, offsets, sess, sys_b, L)
    assert np.array_equal(out["hit"], out["sys"] + out["intra"] + out["inter"])
    last = {}
    for r, (s_, t_) in enumerate(zip(sess, turns)):
        if t_ > 0:
            assert out["hit"][r] >= len(reqs[last[s_]]) // B
        else:
            assert out["intra"][r] == 0
        last[s_] = r
    assert out["intra"].sum() > 0 and out["sys"].sum() > 0


def _tick_loads(N, T, n_windows, inst, start, end):
    """Running requests counted tick by tick: S_i(w) = sum over the ticks t of
    window w of the requests on i with start <= t < end."""
    S = np.zeros((n_windows, N), np.int64)
    for w in range(n_windows):
        for t in range(w * T, (w + 1) * T):
            for i_, s_, e_ in zip(inst, start, end):
                if s_ <= t < e_:
                    S[w, i_] += 1
    return S


def check_imbalance_against_tick_counts(L):
    """Brute force in discrete time: every tick of a window, count each
    instance's running requests; the sums, their maximum (lowest instance on
    ties) and their total per window."""
    rng = np.random.default_rng(31)
    for trial in range(150):
        N = int(rng.integers(1, 6))
        T = int(rng.integers(1, 8))
        nw = int(rng.integers(0, 7))
        n = int(rng.integers(0, 20))
        inst = rng.integers(0, N, size=n)
        start = rng.integers(0, 45, size=n)
        end = start + rng.integers(0, 25, size=n)
        out = oracle.window_imbalance(N, T, nw, inst, start, end, L)
        S = _tick_loads(N, T, nw, inst, start, end)
        assert np.array_equal(out["sum"], S.sum(axis=1)), trial
        assert np.array_equal(out["max"], S.max(axis=1) if nw else S.sum(axis=1)), trial
        assert np.array_equal(out["argmax"], S.argmax(axis=1) if nw else np.zeros(0)), trial


def check_imbalance_special_cases(L):
    """One instance: the maximum is the total (imbalance 1). Equal requests
    dealt round-robin: every instance carries the same load (N max = sum).
    Everything on one instance: that instance, and max = sum (imbalance N).
    Conservation: the windows' totals add up to the requests' running time
    inside the covered span; windows twice as long add pairs of totals."""
    rng = np.random.default_rng(32)
    n = 200
    start = rng.integers(0, 5000, size=n)
    end = start + rng.integers(0, 3000, size=n)
    one = oracle.window_imbalance(1, 300, 20, np.zeros(n, np.int32), start, end, L)
    assert np.array_equal(one["max"], one["sum"]) and (one["argmax"] == 0).all()
    N = 8
    rr = oracle.window_imbalance(N, 100, 30, np.arange(8 * 50) % N, np.repeat(np.arange(50) * 37, 8),
                                 np.repeat(np.arange(50) * 37 + 450, 8), L)
    assert np.array_equal(N * rr["max"], rr["sum"]) and rr["sum"].any()
    assert (rr["argmax"][rr["sum"] > 0] == 0).all()
    hot = oracle.window_imbalance(N, 300, 20, np.full(n, 5, np.int32), start, end, L)
    busy = hot["sum"] > 0
    assert np.array_equal(hot["max"], hot["sum"]) and (hot["argmax"][busy] == 5).all()
    inst = rng.integers(0, N, size=n)
    a = oracle.window_imbalance(N, 250, 32, inst, start, end, L)
    covered = np.clip(end, 0, 250 * 32) - np.clip(start, 0, 250 * 32)
    assert a["sum"].sum() == covered.sum()
    b = oracle.window_imbalance(N, 500, 16, inst, start, end, L)
    assert np.array_equal(b["sum"], a["sum"][0::2] + a["sum"][1::2])
    assert (b["max"] <= a["max"][0::2] + a["max"][1::2]).all()
    # an idle window reports zeros; invalid requests are refused
    idle = oracle.window_imbalance(N, 10, 3, [1], [100], [200], L)
    assert not idle["max"].any() and not idle["sum"].any() and not idle["argmax"].any()
    for bad in (([N], [0], [1]), ([-1], [0], [1]), ([0], [-1], [1]), ([0], [5], [4])):
        try:
            oracle.window_imbalance(N, 10, 3, *bad, L)
        except ValueError:
            continue
        raise AssertionError(bad)


ALL_CHECKS = [
    check_published_vector,
    check_bijection,
    check_prefix_locality,
    check_tail_and_empty,
    check_seed_and_block_size,
    check_sentinel_remap,
    check_multiword_digest,
    check_session_key,
    check_brute_force_prefix,
    check_non_prefix_closed,
    check_jsq_when_index_empty,
    check_argmax_hit_when_load_ignored,
    check_equal_costs_pick_zero,
    check_paper_examples,
    check_hand_costs,
    check_batch_invariants,
    check_index_set_semantics,
    check_lru_recency,
    check_policy_eq1_boundary,
    check_policy_first_turn_is_cost_argmin,
    check_policy_sticks_to_longest_local_hit,
    check_policy_session_cached_threshold,
    check_policy_slo_migration,
    check_policy_round_robin_ties,
    check_coloc_reduces_to_disaggregated,
    check_coloc_tpot_filter,
    check_coloc_lmetric_product,
    check_coloc_no_last_resort,
    check_link_against_token_prefixes,
    check_link_recovers_generated_sessions,
    check_link_special_cases,
    check_baselines_against_their_definitions,
    check_baselines_special_cases,
    check_sequential_matches_snapshot_without_load,
    check_sequential_join_shortest_queue,
    check_reuse_against_token_prefixes,
    check_reuse_on_a_multi_turn_trace,
    check_imbalance_against_tick_counts,
    check_imbalance_special_cases,
]
