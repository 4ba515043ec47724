"""The seeded workload generators and the replay driver (no GPU)."""

import numpy as np

from synth import ReplayDriver, agent_trace, burst_trace
from synth.traces import VOCAB


def test_agent_trace_deterministic_and_append_only():
    a = list(agent_trace("c1_tiny", scale=0.25, seed=5).batches())
    b = list(agent_trace("c1_tiny", scale=0.25, seed=5).batches())
    assert len(a) == len(b) > 1
    for x, y in zip(a, b):
        assert np.array_equal(x.tokens, y.tokens) and np.array_equal(x.offsets, y.offsets)
    # turn t+1 of a session extends turn t (Section 2: each request resends the history)
    prev = {}
    for bt in a:
        for r, s in enumerate(bt.sessions.tolist()):
            t = bt.tokens[bt.offsets[r]:bt.offsets[r + 1]]
            if s in prev:
                assert len(t) > len(prev[s]) and np.array_equal(t[:len(prev[s])], prev[s])
            prev[s] = t
    assert a[0].tokens.min() >= 0 and a[0].tokens.max() < VOCAB


def test_agent_trace_config_shapes():
    c1 = agent_trace("c1_tiny")
    assert (c1.n_sessions, c1.n_turns, c1.batch_size, c1.params.num_instances,
            c1.params.block_size) == (64, 8, 64, 4, 16)
    c2 = agent_trace("c2_medium")
    assert (c2.n_sessions, c2.n_turns, c2.batch_size, c2.params.num_instances,
            c2.local_cap, c2.global_policy) == (1024, 16, 256, 16, 200_000, "all")
    c3 = agent_trace("c3_long")
    assert (c3.n_sessions, c3.n_turns, c3.batch_size, c3.params.num_instances,
            c3.params.block_size, c3.local_cap, c3.global_cap) == \
        (4096, 32, 1024, 32, 64, 1_000_000, 16_000_000)


def test_truncation_drops_a_quarter():
    tr = agent_trace("c3_long", scale=0.02, seed=1)
    hist = {}
    seen_trunc = False
    for bt in tr.batches():
        for r, s in enumerate(bt.sessions.tolist()):
            t = bt.tokens[bt.offsets[r]:bt.offsets[r + 1]]
            full = hist.get(s)
            hist[s] = t
            if full is not None and len(t) < len(full):
                seen_trunc = True
    assert seen_trunc


def test_burst_trace_structure():
    tr = burst_trace(num_instances=8, block_size=16, n_sessions=500, batch_size=256,
                     len_lo=200, len_hi=2000)
    bt = tr.batch(0)
    assert bt.n_requests == 256 and bt.load.shape == (8,)
    assert bt.load.min() >= 0 and bt.load.max() <= 2_000_000
    for r, s in enumerate(bt.sessions.tolist()):
        t = bt.tokens[bt.offsets[r]:bt.offsets[r + 1]]
        assert len(t) == tr.session_len[s]
        assert np.array_equal(t[:tr.prefix_len[s]], tr.session_prefix(s))
    # Zipf popularity: the most popular session recurs many times
    _, counts = np.unique(bt.sessions, return_counts=True)
    assert counts.max() > 10
    assert np.array_equal(tr.batch(0).tokens, bt.tokens)
    assert not np.array_equal(tr.batch(1).sessions, bt.sessions)
    tiers = tr.session_tiers(int(bt.sessions[0]))
    assert tiers[0] == -1 and all(0 <= t < 8 for t in tiers[1:])


def test_replay_driver_lru_evicts_deepest_oldest_first():
    d = ReplayDriver(2, 2, local_cap=3)
    off = np.array([0, 8, 14], dtype=np.int64)  # request 0: 4 blocks, request 1: 3 blocks
    h = np.arange(10, 17, dtype=np.uint64)
    ins_k, ins_t, ev_k, ev_t = d.after_batch(off, np.array([0, 0]), np.array([0, 0]), h)
    assert sorted(ins_k.tolist()) == list(range(10, 17)) and set(ins_t.tolist()) == {0}
    # 7 blocks in a 3-block tier: the oldest stamps are request 0's, deepest first
    assert ev_k.tolist() == [13, 12, 11, 10] and set(ev_t.tolist()) == {0}
    assert d.load.tolist() == [(8 + 6) >> 1, 0]
