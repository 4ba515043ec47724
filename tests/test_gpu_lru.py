"""Slot reuse and the device-side LRU of capped tiers.

Slot reuse: a key that leaves its last tier gives its slot back, so a table
sized for the live keys takes any number of inserted and evicted ones; the
table's contents are checked against a plain dict model after every step.

Device LRU (smetric_index_set_lru + smetric_index_commit_batch): replaying
the agent traces with routing, commits, queue drains and evictions all on
the device gives, batch after batch, the routing outputs, loads and tier
contents of the oracle replayed with the host replay driver's LRU (recency
(batch, request, -block), least recent evicted first)."""

import itertools

import numpy as np
import pytest
import torch

import oracle
import paper_2607_08565_gb300 as pkg
from synth import ReplayDriver, agent_trace
from synth.traces import pack
from gpu_util import T, assert_outputs_equal, make_index, n_blocks

pytestmark = pytest.mark.gpu


def U(t):
    """A device tensor of 64-bit words as a host uint64 array."""
    return t.cpu().view(torch.int64).numpy().view(np.uint64)


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def _bits(mask_row, N):
    """Tier set of one key from its mask words: local tiers, then -1 for the global tier."""
    out = set()
    for t in range(N + 1):
        if (int(mask_row[t >> 6]) >> (t & 63)) & 1:
            out.add(t if t < N else -1)
    return out


def _check_model(ix, model, N, extra_keys=()):
    """Every key of the model (and every extra key, absent from it) has
    exactly the model's tiers on the device."""
    keys = np.array(sorted(set(model) | set(extra_keys)), dtype=np.uint64)
    if len(keys) == 0:
        return
    m = U(ix.lookup(T(keys)))
    for j, k in enumerate(keys.tolist()):
        got = _bits(m[j], N)
        want = model.get(k, set())
        assert got == want, f"key {k:#x}: device tiers {sorted(got)} model {sorted(want)}"


def _keys(rng, n):
    return rng.integers(2, 1 << 63, size=n, dtype=np.int64).astype(np.uint64)


def _apply(ix, keys, tiers, insert):
    k = T(np.asarray(keys, np.uint64))
    t = T(np.asarray(tiers, np.int32))
    (ix.insert if insert else ix.evict)(k, t)
    ix.check()


@pytest.mark.parametrize("N", [3, 100])
def test_slot_reuse_churn_ten_times_capacity(N):
    """Insert and evict 10x the table's capacity in distinct keys, each in one
    to three tiers, the tiers of one key cleared in the same call (so that the
    last bits of different mask words are cleared concurrently); then the
    table still fills to 90 % of its slots."""
    rng = np.random.default_rng(7 + N)
    ix = make_index(N, 4, 1, cap=4096, max_req=16, max_tok=1 << 12)
    slots = -(-4096 // 15) * 15
    inserted = 0
    for rnd in range(42):
        keys = _keys(rng, 1024)
        ntier = rng.integers(1, 4, size=len(keys))
        kk = np.repeat(keys, ntier)
        tt = np.concatenate([rng.choice(np.arange(-1, N), size=c, replace=False) for c in ntier]).astype(np.int32)
        _apply(ix, kk, tt, True)
        model = {}
        for k, t in zip(kk.tolist(), tt.tolist()):
            model.setdefault(k, set()).add(t)
        if rnd % 8 == 0:
            _check_model(ix, model, N)
        perm = rng.permutation(len(kk))
        _apply(ix, kk[perm], tt[perm], False)
        if rnd % 8 == 0:
            _check_model(ix, {}, N, extra_keys=keys.tolist())
        inserted += len(keys)
    assert inserted >= 10 * slots
    keys = _keys(rng, int(0.9 * slots))
    tiers = rng.integers(-1, N, size=len(keys)).astype(np.int32)
    _apply(ix, keys, tiers, True)
    _check_model(ix, {k: {t} for k, t in zip(keys.tolist(), tiers.tolist())}, N)
    ix.close()


@pytest.mark.parametrize("N,load", [(5, 0.95), (70, 0.9)])
def test_slot_reuse_random_model(N, load):
    """A random walk of inserts and evictions around a high load factor (so
    that many keys sit past full home buckets and overflow counts rise and
    fall), every step checked against a dict model, absent keys included."""
    rng = np.random.default_rng(11 + N)
    ix = make_index(N, 4, 1, cap=3000, max_req=16, max_tok=1 << 12)
    slots = -(-3000 // 15) * 15
    model = {}
    pool = []
    for step in range(30):
        live = len(model)
        n_new = max(0, int(load * slots) - live) if step % 2 == 0 else int(rng.integers(0, 200))
        n_new = min(n_new, int(load * slots) - live)
        fresh = _keys(rng, max(n_new, 0)).tolist()
        kk, tt = [], []
        for k in fresh:
            for t in rng.choice(np.arange(-1, N), size=int(rng.integers(1, 3)), replace=False).tolist():
                kk.append(k)
                tt.append(t)
        for k in rng.choice(np.array(list(model), dtype=np.uint64), size=min(len(model), 100)).tolist() \
                if model else []:
            t = int(rng.integers(-1, N))
            kk.append(k)
            tt.append(t)
        if kk:
            _apply(ix, np.array(kk, np.uint64), tt, True)
            for k, t in zip(kk, tt):
                model.setdefault(k, set()).add(t)
        # evict: some keys wholly, some in one tier, some absent pairs
        ek, et = [], []
        keys_now = list(model)
        for k in rng.choice(np.array(keys_now, dtype=np.uint64), size=len(keys_now) // 3, replace=False).tolist():
            ts = sorted(model[k])
            drop = ts if rng.random() < 0.6 else ts[:1]
            for t in drop:
                ek.append(k)
                et.append(t)
        for k in _keys(rng, 20).tolist():
            ek.append(k)
            et.append(int(rng.integers(-1, N)))
        perm = rng.permutation(len(ek))
        _apply(ix, np.array(ek, np.uint64)[perm], np.array(et, np.int32)[perm], False)
        gone = []
        for k, t in zip(ek, et):
            if k in model:
                model[k].discard(t)
                if not model[k]:
                    del model[k]
                    gone.append(k)
        pool = gone[:200]
        _check_model(ix, model, N, extra_keys=pool)
    ix.close()


# ---------------------------------------------------------------------------
# device LRU
# ---------------------------------------------------------------------------

def replay_device_lru(trace, n_batches=None, check_keys=512, seed=0, fused_every=0):
    """Route, commit (with the queue drain) and evict on the device; the
    oracle routes the same batches and takes the host driver's inserts and
    evictions. Every batch: outputs and loads equal, the LRU sizes equal the
    host driver's, the evicted keys left their tiers and `check_keys` keys
    of the batch have the host LRU's tiers. With fused_every = m, every m-th
    batch goes through the one-call route_commit_batch instead."""
    p = trace.params
    N = p.num_instances
    batches = list(itertools.islice(trace.batches(), n_batches))
    total_blocks = sum(n_blocks(b.offsets, p.block_size) for b in batches)
    local_cap = trace.local_cap or 0
    global_cap = trace.global_cap if (trace.global_policy == "lru" and trace.global_cap) else 0
    if trace.global_policy == "all":
        slots = total_blocks
    else:
        slots = min(total_blocks, N * local_cap + global_cap) if local_cap else total_blocks
    ix = make_index(N, p.block_size, p.session_blocks, cap=max(1024, int(slots / 0.6)),
                    max_req=max(b.n_requests for b in batches), max_tok=max(b.n_tokens for b in batches),
                    seed=p.hash_seed)
    ix.set_lru(local_cap, global_cap)
    ox = oracle.OracleIndex(N)
    do = ReplayDriver(N, p.block_size, local_cap=trace.local_cap, global_policy=trace.global_policy,
                      global_cap=trace.global_cap)
    w = (p.w_load, p.w_miss, p.w_glob)
    load = torch.zeros(N, dtype=torch.int64, device="cuda")
    also_global = trace.global_policy != "none"
    rng = np.random.default_rng(seed)
    stats = dict(evicted=0, local=0)
    for k, bt in enumerate(batches):
        off = T(bt.offsets)
        if fused_every and k % fused_every == fused_every - 1:
            out = ix.route_commit_batch(T(bt.tokens), off, load, w, also_global=also_global)
        else:
            out = ix.route_batch(T(bt.tokens), off, load, w, want_hashes=True)
            ix.commit_batch(off, out, also_global=also_global, load=load)
        g = {key: (U(v) if v.dtype == torch.uint64 else v.cpu().numpy()) for key, v in out.items()}
        ix.check()
        nb = n_blocks(bt.offsets, p.block_size)
        g["block_hashes"] = g["block_hashes"][:nb]
        o = ox.route_batch(p.block_size, p.session_blocks, p.hash_seed, bt.tokens, bt.offsets,
                           do.load, *w, want_hashes=True, n_threads=8)
        assert_outputs_equal(g, o, ctx=f"{trace.name} batch {k}")
        ik, it_, ek, et = do.after_batch(bt.offsets, o["instance"], o["local_hit"], o["block_hashes"])
        ox.insert(ik, it_)
        ox.evict(ek, et)
        assert np.array_equal(load.cpu().numpy(), do.load), f"{trace.name} batch {k}: loads"
        sizes = ix.lru_sizes().cpu().numpy()
        want = [len(d) if local_cap else 0 for d in do.local_lru] + [len(do.global_lru) if global_cap else 0]
        assert sizes.tolist() == want, f"{trace.name} batch {k}: LRU sizes"
        # evicted keys: gone from the tier they were evicted from (unless the
        # host LRU holds them again, which it cannot within one batch)
        if len(ek):
            m = U(ix.lookup(T(ek)))
            bit = np.where(et < 0, N, et).astype(np.int64)
            word = m[np.arange(len(ek)), bit >> 6]
            assert not np.any((word >> (bit & 63).astype(np.uint64)) & np.uint64(1)), \
                f"{trace.name} batch {k}: an evicted key still in its tier"
        # sampled keys of the batch: capped tiers as the host LRU holds them
        if nb:
            sk = np.unique(g["block_hashes"][rng.integers(0, nb, size=min(check_keys, nb))])
            m = U(ix.lookup(T(sk)))
            for j, key in enumerate(sk.tolist()):
                got = _bits(m[j], N)
                if local_cap:
                    for i in range(N):
                        assert (i in got) == (key in do.local_lru[i]), (trace.name, k, key, i)
                if global_cap:
                    assert (-1 in got) == (key in do.global_lru), (trace.name, k, key, "global")
        stats["evicted"] += len(ek)
        stats["local"] += int(o["local_hit"].sum())
    ix.close()
    ox.close()
    return stats


def test_lru_replay_config2_reduced():
    """Also through the one-call route_commit_batch on every other batch."""
    tr = agent_trace("c2_medium", scale=0.1, seed=2)
    tr.n_turns = 6
    tr.local_cap = 3000
    st = replay_device_lru(tr, fused_every=2)
    assert st["evicted"] > 0 and st["local"] > 0


def test_lru_replay_config3_reduced_both_tiers_capped():
    tr = agent_trace("c3_long", scale=0.05, seed=3)
    tr.n_turns = 6
    tr.local_cap = 400
    tr.global_cap = 3000
    st = replay_device_lru(tr)
    assert st["evicted"] > 0


def test_lru_replay_only_global_capped():
    tr = agent_trace("c3_long", scale=0.05, seed=4)
    tr.n_turns = 5
    tr.local_cap = None
    tr.global_cap = 2000
    assert replay_device_lru(tr)["evicted"] > 0


@pytest.mark.slow
def test_lru_replay_config2_full():
    """Config 2 at full size (64 batches of 256 requests, local tiers capped
    at 200k blocks, every block in the uncapped global tier), with commits,
    drains and LRU evictions on the device."""
    st = replay_device_lru(agent_trace("c2_medium"))
    assert st["local"] > 0


@pytest.mark.slow
def test_lru_replay_config3_full():
    """Config 3 at full size (128 batches of 1024 requests, local tiers
    capped at 1M blocks, the global tier at 16M), with commits, drains and
    LRU evictions on the device."""
    st = replay_device_lru(agent_trace("c3_long"))
    assert st["evicted"] > 0


def _tiny_batch(rng, n_req, B, alphabet=2, max_blocks=6):
    base = rng.integers(0, alphabet, size=max_blocks * B, dtype=np.int32)
    reqs = []
    for _ in range(n_req):
        n = int(rng.integers(0, (max_blocks + 1) * B))
        keep = int(rng.integers(0, n + 1))
        reqs.append(np.concatenate([base[:keep], rng.integers(0, alphabet, size=n - keep, dtype=np.int32)]))
    return pack(reqs)


@pytest.mark.parametrize("N,local_cap,global_cap", [(2, 3, 0), (3, 5, 7), (4, 0, 4), (70, 2, 9)])
def test_lru_tiny_batches_every_key(N, local_cap, global_cap):
    """Tiny-alphabet batches (blocks shared within and across requests, keys
    touched several times in one batch): after every commit, every key ever
    seen has exactly the tiers of the LRU oracle (and of the host replay
    driver's LRU), and the sizes match."""
    B = 4
    rng = np.random.default_rng(N * 100 + local_cap)
    ix = make_index(N, B, 1, cap=2048, max_req=64, max_tok=1 << 12)
    ix.set_lru(local_cap, global_cap)
    do = ReplayDriver(N, B, local_cap=local_cap or None, global_policy="lru" if global_cap else "all",
                      global_cap=global_cap or None)
    ol = oracle.OracleLRU(N, local_cap=local_cap, global_cap=global_cap)
    seen = set()
    seen_local = [set() for _ in range(N)]
    for step in range(25):
        tok, off = _tiny_batch(rng, int(rng.integers(1, 40)), B)
        lens = np.diff(off)
        inst = rng.integers(0, N, size=len(lens)).astype(np.int32)
        hb, _ = ix.block_hashes(T(tok), T(off))
        ix.check()
        hb_h = U(hb)[:n_blocks(off, B)]
        lh = np.zeros(len(lens), np.int32)
        out = dict(instance=T(inst), local_hit=T(lh), block_hashes=hb)
        ix.commit_batch(T(off), out, also_global=True)
        ix.check()
        do.after_batch(off, inst, lh, hb_h)
        ol.commit(np.diff(off) // B, inst, hb_h, also_global=True)
        seen.update(hb_h.tolist())
        nbr = np.diff(off) // B
        for r, i in enumerate(inst.tolist()):
            a = int(nbr[:r].sum())
            seen_local[i].update(hb_h[a:a + int(nbr[r])].tolist())
        model = {}
        for i in range(N):  # an uncapped tier holds every key committed to it
            for key in (ol.stamp[i] if local_cap else seen_local[i]):
                model.setdefault(key, set()).add(i)
        for key in (ol.stamp[-1] if global_cap else seen):
            model.setdefault(key, set()).add(-1)
        for i in range(N):  # the two host formulations agree
            assert set(ol.stamp[i]) == (set(do.local_lru[i]) if local_cap else set())
        assert set(ol.stamp[-1]) == (set(do.global_lru) if global_cap else set())
        _check_model(ix, model, N, extra_keys=seen)
        sizes = ix.lru_sizes().cpu().numpy().tolist()
        assert sizes == [ol.size(i) for i in range(N)] + [ol.size(-1)]
    ix.close()


def test_lru_cap_below_one_request_and_invalid_batch():
    """A request longer than the cap keeps only its leading blocks (the
    deepest are the least recent); an invalid batch commits and evicts
    nothing."""
    N, B = 2, 4
    ix = make_index(N, B, 1, cap=1024, max_req=8, max_tok=1 << 10)
    ix.set_lru(3, 0)
    tok = np.arange(40, dtype=np.int32)
    off = np.array([0, 40], np.int64)
    hb, _ = ix.block_hashes(T(tok), T(off))
    h = U(hb)[:10]
    out = dict(instance=T(np.array([1], np.int32)), local_hit=T(np.zeros(1, np.int32)), block_hashes=hb)
    ix.commit_batch(T(off), out)
    ix.check()
    m = U(ix.lookup(T(h)))
    assert [int(x[0]) for x in m] == [2, 2, 2] + [0] * 7
    assert ix.lru_sizes().cpu().numpy().tolist() == [0, 3, 0]
    bad = np.array([0, 50, 40], np.int64)  # decreasing offsets: an invalid batch
    out2 = dict(instance=T(np.array([0, 0], np.int32)), local_hit=T(np.zeros(2, np.int32)), block_hashes=hb)
    ix.commit_batch(T(bad), out2)
    assert ix.status() == pkg.SMETRIC_ERR_INVALID_ARG
    assert ix.lru_sizes().cpu().numpy().tolist() == [0, 3, 0]
    m = U(ix.lookup(T(h)))
    assert [int(x[0]) for x in m] == [2, 2, 2] + [0] * 7
    ix.close()


def test_lru_owns_capped_tiers_and_turns_off():
    N, B = 3, 4
    ix = make_index(N, B, 1, cap=1024, max_req=8, max_tok=1 << 10)
    ix.set_lru(5, 0)
    k = T(np.array([11, 12], np.uint64))
    ix.insert(k, T(np.array([0, -1], np.int32)))  # local tier 0 is capped: refused; global is not
    assert ix.status() == pkg.SMETRIC_ERR_INVALID_ARG
    m = U(ix.lookup(k))
    assert int(m[0, 0]) == 0 and int(m[1, 0]) == 1 << N
    ix.evict(k[1:], T(np.array([-1], np.int32)))
    ix.check()
    assert not U(ix.lookup(k)).any()
    with pytest.raises(pkg.SmetricError):
        ix.set_lru(-1, 0)
    with pytest.raises(pkg.SmetricError):
        ix.set_lru(0, 1 << 41)
    ix.set_lru(0, 0)  # off: host updates of every tier are accepted again
    ix.insert(k, T(np.array([0, 0], np.int32)))
    ix.check()
    assert ix.lru_sizes().cpu().numpy().tolist() == [0] * (N + 1)
    ix.clear()
    assert not U(ix.lookup(k)).any()
    ix.close()
