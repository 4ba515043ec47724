"""Device-side index maintenance (smetric_index_commit_batch): replaying an
agent trace with the inserts and the queue drain done on the GPU gives, batch
after batch, the same routing outputs and loads as the oracle replayed with
the host driver; capped tiers take the host driver's evictions."""

import itertools

import numpy as np
import pytest
import torch

import oracle
import paper_2607_08565_gb300 as pkg
from synth import ReplayDriver, agent_trace
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


def replay_with_device_commit(trace, n_batches=None):
    p = trace.params
    batches = list(itertools.islice(trace.batches(), n_batches))
    total_blocks = sum(n_blocks(b.offsets, p.block_size) for b in batches)
    ix = make_index(p.num_instances, p.block_size, p.session_blocks, cap=max(1024, int(total_blocks / 0.5)),
                    max_req=max(b.n_requests for b in batches), max_tok=max(b.n_tokens for b in batches),
                    seed=p.hash_seed)
    ox = oracle.OracleIndex(p.num_instances)
    kw = dict(local_cap=trace.local_cap, global_policy=trace.global_policy, global_cap=trace.global_cap)
    dg = ReplayDriver(p.num_instances, p.block_size, **kw)  # GPU side: its evictions only
    do = ReplayDriver(p.num_instances, p.block_size, **kw)  # oracle side: everything on the host
    w = (p.w_load, p.w_miss, p.w_glob)
    load = torch.zeros(p.num_instances, dtype=torch.int64, device="cuda")
    also_global = trace.global_policy != "none"
    evicted = 0
    for k, bt in enumerate(batches):
        off = T(bt.offsets)
        out = ix.route_batch(T(bt.tokens), off, load, w, want_hashes=True)
        ix.commit_batch(off, out, also_global=also_global, load=load)
        ix.check()
        g = {key: (U(v) if v.dtype == torch.uint64 else v.cpu().numpy()) for key, v in out.items()}
        g["block_hashes"] = g["block_hashes"][:n_blocks(bt.offsets, p.block_size)]
        o = ox.route_batch(p.block_size, p.session_blocks, p.hash_seed, bt.tokens, bt.offsets,
                           do.load, *w, want_hashes=True, n_threads=8)
        assert_outputs_equal(g, o, ctx=f"{trace.name} batch {k}")
        _, _, ek, et = dg.after_batch(bt.offsets, g["instance"], g["local_hit"], g["block_hashes"])
        if len(ek):
            ix.evict(T(ek), T(et))
            ix.check()
        ik, it_, ek, et = do.after_batch(bt.offsets, o["instance"], o["local_hit"], o["block_hashes"])
        ox.insert(ik, it_)
        ox.evict(ek, et)
        evicted += len(ek)
        assert np.array_equal(load.cpu().numpy(), do.load), f"{trace.name} batch {k}: loads"
    ix.close()
    return evicted


def test_commit_replay_uncapped_tiers():
    """c1_tiny: local tiers uncapped, empty global tier: the whole replay step
    runs on the device."""
    replay_with_device_commit(agent_trace("c1_tiny"))


def test_commit_replay_global_tier_and_host_evictions():
    """c2_medium at a quarter scale: every block also enters the global tier
    (on the device); the capped local tiers evict on the host's orders."""
    tr = agent_trace("c2_medium", scale=0.25)
    assert replay_with_device_commit(tr, n_batches=6) >= 0


def test_commit_rejects_bad_outputs_and_skips_invalid_batches():
    N, B = 3, 4
    ix = make_index(N, B, 1)
    rng = np.random.default_rng(90)
    tok = rng.integers(0, 151936, size=400, dtype=np.int32)
    off = T(np.array([0, 100, 250, 400], np.int64))
    out = ix.route_batch(T(tok), off, T(np.zeros(N, np.int64)), (1, 4, 2), want_hashes=True)
    ix.check()
    load = T(np.array([10, 20, 30], np.int64))
    bad = dict(out, instance=T(np.array([0, 3, 1], np.int32)))
    ix.commit_batch(off, bad, load=load)
    assert ix.status() == pkg.SMETRIC_ERR_INVALID_ARG
    assert np.array_equal(load.cpu().numpy(), [10, 20, 30])  # loads left as they were
    bad = dict(out, local_hit=T(np.array([0, 151, 0], np.int32)))  # request 1 has 150 tokens
    ix.commit_batch(off, bad, load=load)
    assert ix.status() == pkg.SMETRIC_ERR_INVALID_ARG
    skipped = dict(out, instance=T(np.full(3, -1, np.int32)))  # an invalid batch commits nothing
    ix.commit_batch(off, skipped, load=load)
    assert ix.status() == pkg.SMETRIC_OK and np.array_equal(load.cpu().numpy(), [5, 10, 15])
    h = out["block_hashes"][:25]
    assert not U(ix.lookup(h)).any()
    ix.commit_batch(off, out, also_global=True, load=load)
    ix.check()
    inst = out["instance"].cpu().numpy()
    m = U(ix.lookup(h))
    lens = np.array([100, 150, 150]) // B
    r_of = np.repeat(np.arange(3), lens)
    for f in range(25):
        assert int(m[f, 0]) == (1 << int(inst[r_of[f]])) | (1 << N)
    with pytest.raises(pkg.SmetricError):
        pkg.smetric_index_commit_batch(ix.handle, off, 3, out["instance"], out["local_hit"],
                                       out["block_hashes"], 2)  # unknown flag
    ix.close()
