"""The trace configurations end to end on the GPU against the CPU oracle.

Configs 1-3 are multi-batch replays: after every batch each side inserts the
routed blocks into its own index, evicts by LRU and drains its load, so the
two replays stay identical only if every batch's outputs are bit-exact.
Config 4 runs at full size in the launch configuration the benchmark times
(65,536 sessions, 64 instances, B = 32, batches of 8,192 requests): every
request of the four batches the benchmark rotates is compared with the
oracle, and invariants that hold at any size are checked on every request.
Configs 2 and 3 are also replayed whole (the long cases carry the slow mark).
"""

import os

import numpy as np
import pytest
import torch

import oracle
import paper_2607_08565_gb300 as pkg
from synth import agent_trace, burst_trace
from gpu_util import T, assert_outputs_equal, gpu_route, make_index, replay_both

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def test_replay_config1_full():
    st = replay_both(agent_trace("c1_tiny"))
    assert st["batches"] == 8 and st["requests"] == 512
    assert st["local"] > 0  # later turns hit the instance that served earlier ones


def test_replay_config2_reduced_with_eviction():
    tr = agent_trace("c2_medium", scale=0.1, seed=2)
    tr.n_turns = 6
    tr.local_cap = 3000  # small enough that LRU eviction runs every batch
    st = replay_both(tr)
    assert st["evicted"] > 0 and st["glob"] > 0


def test_replay_config3_reduced_with_truncation_and_eviction():
    tr = agent_trace("c3_long", scale=0.05, seed=3)
    tr.n_turns = 6
    tr.local_cap = 400
    tr.global_cap = 3000
    st = replay_both(tr)
    assert st["evicted"] > 0


@pytest.mark.slow
def test_replay_config2_full():
    """Config 2 at full size: 1024 sessions x 16 turns, 64 batches of 256
    requests, local tiers LRU-capped at 200k blocks, every block in the
    global tier; both replays compared batch by batch."""
    st = replay_both(agent_trace("c2_medium"), shared_driver=True)
    assert st["batches"] == 64 and st["requests"] == 64 * 256
    assert st["glob"] > 0 and st["local"] > 0


@pytest.mark.slow
def test_replay_config3_full():
    """Config 3 at full size: 4096 sessions x 32 turns, 128 batches of 1024
    requests with half the turns truncated, local tiers LRU-capped at 1M
    blocks and the global tier at 16M; both replays compared batch by
    batch."""
    st = replay_both(agent_trace("c3_long"), shared_driver=True)
    assert st["batches"] == 128 and st["requests"] == 128 * 1024
    assert st["evicted"] > 0


def test_replay_config3_first_batches_full_size():
    """Config 3 at full size (4096 sessions, batches of 1024): its first two
    turn waves, both replays compared batch by batch."""
    st = replay_both(agent_trace("c3_long"), n_batches=8)
    assert st["requests"] == 8 * 1024


def _populate_c4(ix, tr, chunk=4096):
    """Hash every session prefix on the GPU and insert its blocks into the
    global tier and the session's local tiers."""
    p = tr.params
    B = p.block_size
    buf = np.empty(int(tr.prefix_len.max()) * chunk, np.int32)
    for ids, tok, off in tr.prepopulation(chunk=chunk, out=buf):
        hb, _ = ix.block_hashes(T(tok), T(off))
        nb = torch.from_numpy(tr.prefix_len[ids] // B).to(hb.device)
        total = int(nb.sum())
        hb = hb[:total].view(torch.int64)  # CUDA mask indexing has no uint64 kernels
        owner = torch.repeat_interleave(torch.arange(len(ids), device=hb.device), nb)
        sess = torch.from_numpy(ids).to(hb.device)[owner]
        ix.insert(hb, -1)
        for tier_of, member in ((tr.home, tr.in_home), (tr.second, tr.in_second)):
            m = torch.from_numpy(member).to(hb.device)[sess]
            t = torch.from_numpy(tier_of).to(hb.device)[sess]
            ix.insert(hb[m].contiguous(), t[m].contiguous())
    ix.check()


def test_config4_full_size_sampled():
    tr = burst_trace()
    p = tr.params
    N, B = p.num_instances, p.block_size
    nkeys = tr.n_prefix_blocks()
    bt = tr.batch(0)
    ix = make_index(N, B, p.session_blocks, cap=int(nkeys / 0.7) + 1,
                    max_req=bt.n_requests, max_tok=bt.n_tokens)
    _populate_c4(ix, tr)
    w = (p.w_load, p.w_miss, p.w_glob)
    g = gpu_route(ix, bt.tokens, bt.offsets, bt.load, w, want_hashes=False)

    # invariants on every request
    lens = bt.lengths()
    assert np.all((g["instance"] >= 0) & (g["instance"] < N))
    assert np.all(g["local_hit"] + g["global_hit"] <= (lens // B) * B)
    assert np.all(g["local_hit"] % B == 0) and np.all(g["global_hit"] % B == 0)
    # every request of a session carries the session's cached prefix, which
    # the global tier holds in full
    reach = (g["local_hit"] + g["global_hit"]) // B
    assert np.all(reach == tr.prefix_len[bt.sessions] // B)
    # the session key is a function of the session (identical leading blocks)
    keys = {}
    for s, k in zip(bt.sessions.tolist(), g["session_key"].tolist()):
        assert keys.setdefault(s, k) == k
    assert len(set(keys.values())) == len(keys)

    # the oracle on a sample, one request at a time, with an index holding
    # the sampled sessions' prefixes
    rng = np.random.default_rng(0)
    sample = np.sort(rng.choice(bt.n_requests, size=96, replace=False))
    sessions = np.unique(bt.sessions[sample])
    ox = oracle.OracleIndex(N)
    for s in sessions.tolist():
        h = oracle.block_hashes(tr.session_prefix(s), B, p.hash_seed)
        for t in tr.session_tiers(s):
            ox.insert(h, t)
    for r in sample.tolist():
        a, b = bt.offsets[r], bt.offsets[r + 1]
        o = ox.route_batch(B, p.session_blocks, p.hash_seed, bt.tokens[a:b],
                           np.array([0, b - a], np.int64), bt.load, *w)
        one = {f: g[f][r:r + 1] for f in ("instance", "local_hit", "global_hit", "session_key")}
        assert_outputs_equal(one, o, fields=("instance", "local_hit", "global_hit", "session_key"),
                             ctx=f"config 4 request {r}")
    ix.close()


@pytest.mark.slow
def test_config4_bench_batches_every_request():
    """The four config-4 batches the benchmark rotates (65,536 sessions,
    64 instances, B = 32, 8,192 requests each), routed in the benchmark's
    launch configuration on the fully populated index: every output of every
    request, and every block hash, equals the oracle's. The oracle's index
    holds the prefixes of every session the four batches use; requests hit
    only their own session's blocks (the reach check below), so the rest of
    the GPU index does not change any decision."""
    tr = burst_trace()
    p = tr.params
    N, B = p.num_instances, p.block_size
    nkeys = tr.n_prefix_blocks()
    host = [tr.batch(k) for k in range(4)]
    ix = make_index(N, B, p.session_blocks, cap=int(nkeys / 0.7) + 1,
                    max_req=max(max(b.n_requests for b in host), 4096),
                    max_tok=max(max(b.n_tokens for b in host), 4096 * int(tr.prefix_len.max())))
    _populate_c4(ix, tr)
    ox = oracle.OracleIndex(N)
    sessions = np.unique(np.concatenate([b.sessions for b in host]))
    for s in sessions.tolist():
        h = oracle.block_hashes(tr.session_prefix(s), B, p.hash_seed)
        for t in tr.session_tiers(s):
            ox.insert(h, t)
    w = (p.w_load, p.w_miss, p.w_glob)
    for k, bt in enumerate(host):
        g = gpu_route(ix, bt.tokens, bt.offsets, bt.load, w, want_hashes=True)
        o = ox.route_batch(B, p.session_blocks, p.hash_seed, bt.tokens, bt.offsets, bt.load, *w,
                           want_hashes=True, n_threads=os.cpu_count() or 1)
        assert_outputs_equal(g, o, ctx=f"config 4 batch {k}")
        reach = (o["local_hit"] + o["global_hit"]) // B
        assert np.all(reach == tr.prefix_len[bt.sessions] // B)
    ox.close()
    ix.close()


@pytest.mark.parametrize("N,B", [(8, 64), (256, 16)])
def test_config5_corner_points_sampled(N, B):
    """Two corners of the config-5 sweep (fewest instances with the largest
    blocks; most instances with the smallest), with filler keys packing the
    table, at reduced session count."""
    tr = burst_trace("c5_sweep", num_instances=N, block_size=B, n_sessions=2048, batch_size=2048)
    p = tr.params
    nkeys = tr.n_prefix_blocks()
    n_fill = nkeys // 2
    bt = tr.batch(3)
    ix = make_index(N, B, 4, cap=int((nkeys + n_fill) / 0.7) + 1, max_req=bt.n_requests,
                    max_tok=bt.n_tokens)
    _populate_c4(ix, tr, chunk=1024)
    fk, ft = tr.filler_keys(n_fill)
    ix.insert(T(fk), T(ft))
    ix.check()
    g = gpu_route(ix, bt.tokens, bt.offsets, bt.load, (1, 4, 2), want_hashes=False)
    rng = np.random.default_rng(1)
    sample = np.sort(rng.choice(bt.n_requests, size=48, replace=False))
    ox = oracle.OracleIndex(N)
    for s in np.unique(bt.sessions[sample]).tolist():
        h = oracle.block_hashes(tr.session_prefix(s), B)
        for t in tr.session_tiers(s):
            ox.insert(h, t)
    ox.insert(fk, ft)
    tok, off = bt.tokens, bt.offsets
    sub = [tok[off[r]:off[r + 1]] for r in sample]
    from synth.traces import pack
    st, so = pack(sub)
    o = ox.route_batch(B, 4, 0, st, so, bt.load, 1, 4, 2)
    sel = {f: g[f][sample] for f in ("instance", "local_hit", "global_hit", "session_key")}
    assert_outputs_equal(sel, o, fields=("instance", "local_hit", "global_hit", "session_key"))
    ix.close()


def _config5_full_size(N, B, batch, n_sample):
    """A config-5 sweep point at the full session count, in the benchmark's
    launch configuration. Random filler keys with random tiers pad the
    table to load factor 0.7 of its capacity; the oracle recomputes
    `n_sample` requests (every request when None) and invariants are
    checked on every request."""
    tr = burst_trace("c5_sweep", num_instances=N, block_size=B, batch_size=batch)
    p = tr.params
    nkeys = tr.n_prefix_blocks()
    n_fill = nkeys // 2
    bt = tr.batch(1)
    ix = make_index(N, B, p.session_blocks, cap=int((nkeys + n_fill) / 0.7) + 1,
                    max_req=max(bt.n_requests, 4096), max_tok=bt.n_tokens)
    _populate_c4(ix, tr)
    fk, ft = tr.filler_keys(n_fill)
    ix.insert(T(fk.view(np.int64)), T(ft))
    ix.check()
    w = (p.w_load, p.w_miss, p.w_glob)
    g = gpu_route(ix, bt.tokens, bt.offsets, bt.load, w, want_hashes=n_sample is None)
    lens = bt.lengths()
    assert np.all((g["instance"] >= 0) & (g["instance"] < N))
    assert np.all(g["local_hit"] + g["global_hit"] <= (lens // B) * B)
    rng = np.random.default_rng(N + B)
    sample = np.arange(bt.n_requests) if n_sample is None else \
        np.sort(rng.choice(bt.n_requests, size=n_sample, replace=False))
    ox = oracle.OracleIndex(N)
    sample_hashes = []
    for s in np.unique(bt.sessions[sample]).tolist():
        h = oracle.block_hashes(tr.session_prefix(s), B, p.hash_seed)
        sample_hashes.append(h)
        for t in tr.session_tiers(s):
            ox.insert(h, t)
    from synth.traces import pack
    if n_sample is None:
        st, so = bt.tokens, bt.offsets
    else:
        st, so = pack([bt.tokens[bt.offsets[r]:bt.offsets[r + 1]] for r in sample])
    o = ox.route_batch(B, p.session_blocks, p.hash_seed, st, so, bt.load, *w, want_hashes=True,
                       n_threads=os.cpu_count() or 1)
    # the oracle leaves out the filler keys (tens of millions): exact as long
    # as none of them equals a block hash of the sample, which is checked
    assert not np.isin(np.concatenate(sample_hashes + [o["block_hashes"]]), fk).any()
    fields = ("instance", "local_hit", "global_hit", "session_key")
    if n_sample is None:
        assert_outputs_equal(g, o, ctx=f"config 5 N={N} B={B} batch={batch}")
    else:
        sel = {f: g[f][sample] for f in fields}
        assert_outputs_equal(sel, o, fields=fields, ctx=f"config 5 N={N} B={B} batch={batch}")
    ox.close()
    ix.close()


@pytest.mark.parametrize("N,B,batch", [(256, 16, 8192), (8, 64, 8192), (64, 32, 32768)])
def test_config5_full_size_points_sampled(N, B, batch):
    """Config-5 sweep points at the full session count: the most instances
    with the smallest blocks, the fewest with the largest, and the largest
    batch; 256 requests of each recomputed by the oracle."""
    _config5_full_size(N, B, batch, 256)


@pytest.mark.slow
def test_config5_largest_point_every_request():
    """The sweep's largest batch (32,768 requests, N = 64, B = 32) on the
    filler-padded table: every output of every request, and every block
    hash, equals the oracle's."""
    _config5_full_size(64, 32, 32768, None)


@pytest.mark.parametrize("pipeline", [True, False])
def test_route_batches_equal_one_route_per_batch(pipeline):
    """Config-4-shaped batches (2,048 sessions, 512 requests a batch) routed
    five per smetric_route_batches call, on an index with a second scratch
    set (consecutive batches overlapped on two streams) and on one without:
    every output of every batch equals that batch's own smetric_route_batch
    call, including a batch with a decreasing offset (invalid-batch outputs
    and the latched error) and an empty batch; repeated calls agree."""
    tr = burst_trace(n_sessions=2048, batch_size=512)
    p = tr.params
    chunk = 512
    host = [tr.batch(k) for k in range(3)]
    max_tok = max(max(b.n_tokens for b in host), chunk * int(tr.prefix_len.max()))
    ix = pkg.SMetricIndex(p.num_instances, p.block_size, p.session_blocks,
                          capacity_slots=int(tr.n_prefix_blocks() / 0.7) + 1, max_batch_requests=chunk,
                          max_batch_tokens=max_tok, hash_seed=p.hash_seed, pipeline=pipeline)
    _populate_c4(ix, tr, chunk=chunk)
    batches = [(T(b.tokens), T(b.offsets), T(b.load)) for b in host]
    bad_off = host[2].offsets.copy()
    bad_off[5] = bad_off[6] + 1
    empty = (T(np.zeros(0, np.int32)), T(np.zeros(1, np.int64)), T(host[0].load))
    batches = [batches[0], batches[1], (batches[2][0], T(bad_off), batches[2][2]), empty, batches[2]]
    w = (p.w_load, p.w_miss, p.w_glob)
    want, codes = [], []
    for b in batches:
        want.append({k: v.cpu().numpy() for k, v in ix.route_batch(*b, w).items()})
        codes.append(ix.status())
    assert codes == [pkg.SMETRIC_OK, pkg.SMETRIC_OK, pkg.SMETRIC_ERR_INVALID_ARG, pkg.SMETRIC_OK, pkg.SMETRIC_OK]
    for rep in range(2):
        got = ix.route_batches(batches, w)
        assert ix.status() == pkg.SMETRIC_ERR_INVALID_ARG
        assert len(got) == len(batches)
        for j, (g, o) in enumerate(zip(got, want)):
            g = {k: v.cpu().numpy() for k, v in g.items()}
            assert_outputs_equal(g, o, fields=("instance", "local_hit", "global_hit", "session_key"),
                                 ctx=f"pipeline={pipeline} call {rep} batch {j}")
    assert np.all(want[2]["instance"] == -1) and np.all(want[4]["instance"] >= 0)
    ix.close()
