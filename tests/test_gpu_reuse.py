"""KV$ reuse breakdown (Section 3.1, Findings 1-3) on the CUDA path against
the CPU oracle, element by element through the C ABI: hit, system-prompt,
intra- and inter-session blocks of every request must be equal."""

import numpy as np
import pytest
import torch

import oracle
import paper_2607_08565_gb300 as pkg
from synth import agent_trace
from synth.traces import pack
from gpu_util import T, make_index

pytestmark = pytest.mark.gpu
KEYS = ("hit", "sys", "intra", "inter")


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def _gpu(ix, tok, off, sessions, sys_b, **kw):
    out = ix.reuse_breakdown(T(tok), T(off), T(np.asarray(sessions, np.int32)), T(np.asarray(sys_b, np.int32)), **kw)
    return {k: v.cpu().numpy() for k, v in out.items()}


def _both(B, seed, reqs, sessions, sys_b):
    tok, off = pack(reqs)
    ix = make_index(2, B, 1, max_req=max(len(reqs), 1), max_tok=max(len(tok), 1), seed=seed)
    g = _gpu(ix, tok, off, sessions, sys_b)
    ix.check()
    ix.close()
    return g, oracle.reuse_breakdown(B, seed, tok, off, sessions, sys_b)


def _assert_equal(g, o, ctx):
    for k in KEYS:
        bad = np.nonzero(g[k] != o[k])[0]
        assert len(bad) == 0, f"{ctx} {k}: {len(bad)} mismatches at {bad[:5]}: gpu {g[k][bad[:5]]} oracle {o[k][bad[:5]]}"


@pytest.mark.parametrize("B", [2, 4, 16])
def test_reuse_matches_oracle_tiny_alphabet(B):
    """Prompts over a three-token alphabet share prefixes in every way, so
    every attribution occurs; lengths span several 32-block rounds of a warp
    and ragged tails; some requests hold no full block."""
    rng = np.random.default_rng(100 + B)
    seen = dict.fromkeys(KEYS, 0)
    for trial in range(6):
        base = rng.integers(0, 3, size=80 * B, dtype=np.int32)
        n = int(rng.integers(1, 400)) if trial else 1
        reqs = []
        for _ in range(n):
            keep = int(rng.integers(0, 80 * B + 1))
            reqs.append(np.concatenate([base[:keep], rng.integers(0, 3, size=int(rng.integers(0, 3 * B)),
                                                                   dtype=np.int32)]))
        sessions = rng.integers(0, 5, size=n)
        sys_b = rng.integers(0, 40, size=n)
        g, o = _both(B, trial, reqs, sessions, sys_b)
        _assert_equal(g, o, f"B={B} trial={trial}")
        for k in KEYS:
            seen[k] += int(o[k].sum())
    assert all(v > 0 for v in seen.values()), seen


@pytest.mark.parametrize("name,scale", [("c1_tiny", 1.0), ("c3_long", 0.125), ("c2_medium", 0.25)])
def test_reuse_on_agent_traces(name, scale):
    """Agent traces in arrival order with the generator's sessions and its
    system-prompt span: equal to the oracle, and the parts add up."""
    tr = agent_trace(name, scale=scale, seed=7)
    reqs, sess = [], []
    for bt in tr.batches():
        for r in range(bt.n_requests):
            reqs.append(bt.tokens[bt.offsets[r]:bt.offsets[r + 1]])
        sess.extend(bt.sessions.tolist())
    B = tr.params.block_size
    sys_b = np.full(len(reqs), tr.system_prompt_len // B, np.int32)
    g, o = _both(B, 0, reqs, sess, sys_b)
    _assert_equal(g, o, name)
    assert np.array_equal(g["hit"], g["sys"] + g["intra"] + g["inter"])
    assert g["intra"].sum() > 0


def test_reuse_with_sessions_from_links():
    """The sessions that smetric_link_sessions reconstructs from hashes feed
    the breakdown directly; both stay equal to the oracle's chain."""
    tr = agent_trace("c1_tiny", scale=0.5, seed=3)
    reqs, users, turns = [], [], []
    for bt in tr.batches():
        for r in range(bt.n_requests):
            reqs.append(bt.tokens[bt.offsets[r]:bt.offsets[r + 1]])
        users.extend(bt.sessions.tolist())
        turns.extend(bt.turns.tolist())
    tok, off = pack(reqs)
    B = tr.params.block_size
    users, turns = np.array(users, np.int64), np.array(turns, np.int32)
    ix = make_index(2, B, tr.params.session_blocks, max_req=len(reqs), max_tok=len(tok))
    _, gs = ix.link_sessions(T(tok), T(off), T(users), T(turns))
    sys_b = np.full(len(reqs), tr.system_prompt_len // B, np.int32)
    out = ix.reuse_breakdown(T(tok), T(off), gs, T(sys_b))
    ix.check()
    g = {k: v.cpu().numpy() for k, v in out.items()}
    ix.close()
    _, os_ = oracle.link_sessions(B, 0, tok, off, users, turns)
    _assert_equal(g, oracle.reuse_breakdown(B, 0, tok, off, os_, sys_b), "linked")


def test_reuse_edge_cases():
    rng = np.random.default_rng(5)
    B = 4
    ix = make_index(2, B, 1, max_req=64, max_tok=1 << 12)
    # no requests: nothing launched, nothing written
    ix.reuse_breakdown(T(np.zeros(4, np.int32)), T(np.zeros(1, np.int64)), T(np.zeros(0, np.int32)),
                       T(np.zeros(0, np.int32)))
    ix.check()
    # identical prompts: each later one reuses all of its blocks, from request 0
    p = rng.integers(0, 100, size=10 * B + 3, dtype=np.int32)
    tok, off = pack([p] * 5)
    g = _gpu(ix, tok, off, [0, 0, 1, 1, 0], [2, 2, 2, 20, 0])
    ix.check()
    assert g["hit"].tolist() == [0, 10, 10, 10, 10]
    assert g["sys"].tolist() == [0, 2, 2, 10, 0]
    assert g["intra"].tolist() == [0, 8, 0, 0, 10]
    assert g["inter"].tolist() == [0, 0, 8, 0, 0]
    # empty and sub-block requests between full ones
    reqs = [p, p[:0], p[:B - 1], p, p[:3 * B]]
    tok, off = pack(reqs)
    g = _gpu(ix, tok, off, [0] * 5, [0] * 5)
    ix.check()
    _assert_equal(g, oracle.reuse_breakdown(B, 0, tok, off, [0] * 5, [0] * 5), "empty")
    assert g["hit"].tolist() == [0, 0, 0, 10, 3]
    # a negative system span latches INVALID_ARG and counts as 0
    tok, off = pack([p] * 3)
    g = _gpu(ix, tok, off, [0, 0, 0], [0, -3, 0])
    assert ix.status() == pkg.SMETRIC_ERR_INVALID_ARG
    _assert_equal(g, oracle.reuse_breakdown(B, 0, tok, off, [0] * 3, [0] * 3), "negative span")
    # decreasing offsets: every output -1
    bad_off = np.array([0, 8, 4, 12], np.int64)
    g = _gpu(ix, tok, bad_off, [0] * 3, [0] * 3)
    assert ix.status() == pkg.SMETRIC_ERR_INVALID_ARG
    assert all((g[k] == -1).all() for k in KEYS)
    # a workspace below the bound is refused before any launch
    small = torch.empty(pkg.smetric_reuse_workspace_bytes(len(tok) // B) - 16, dtype=torch.uint8, device="cuda")
    with pytest.raises(pkg.SmetricError) as e:
        _gpu(ix, tok, off, [0] * 3, [0] * 3, workspace=small)
    assert e.value.code == pkg.SMETRIC_ERR_INVALID_ARG
    ix.check()
    ix.close()


def _first_table_limit(n_blocks):
    """Distinct blocks the L2-sized first table takes before the kernels fall
    back to the full table: half its slots, a power of two >= 2 ceil(n/8)."""
    g = 64
    while g < 2 * ((n_blocks + 7) // 8):
        g <<= 1
    return g // 2


@pytest.mark.parametrize("distinct", [True, False])
def test_reuse_first_table_and_fallback(distinct):
    """All blocks distinct (the first table overflows, the full one takes
    over) and few distinct (the first table holds them): both equal to the
    oracle."""
    rng = np.random.default_rng(17)
    B, n = 4, 600
    if distinct:
        reqs = [rng.integers(0, 1 << 30, size=int(rng.integers(0, 60 * B)), dtype=np.int32) for _ in range(n)]
    else:
        pool = [rng.integers(0, 1 << 30, size=100 * B, dtype=np.int32) for _ in range(4)]
        reqs = [pool[i % 4][:int(rng.integers(0, 100 * B))] for i in range(n)]
    sessions = rng.integers(0, 3, size=n)
    sys_b = rng.integers(0, 10, size=n)
    g, o = _both(B, 1, reqs, sessions, sys_b)
    _assert_equal(g, o, f"distinct={distinct}")
    nb = np.array([len(r) // B for r in reqs])
    fresh = int((nb - o["hit"]).sum())  # blocks no earlier request holds
    limit = _first_table_limit(int(nb.sum()))
    assert (fresh > limit) == distinct, (fresh, limit)


def test_reuse_full_window_properties():
    """A whole c2_medium window (16,384 requests, 256M tokens) at once: the
    parts add up, first turns reuse no intra-session blocks, every
    follow-up reuses at least its parent turn's blocks (a turn resends the
    previous one whole), and a sample of requests agrees with a direct
    first-occurrence computation over the hashes."""
    tr = agent_trace("c2_medium", scale=1.0, seed=11)
    reqs, sess, turns = [], [], []
    for bt in tr.batches():
        for r in range(bt.n_requests):
            reqs.append(bt.tokens[bt.offsets[r]:bt.offsets[r + 1]])
        sess.extend(bt.sessions.tolist())
        turns.extend(bt.turns.tolist())
    tok, off = pack(reqs)
    del reqs
    B = tr.params.block_size
    n = len(off) - 1
    ix = make_index(2, B, tr.params.session_blocks, max_req=n, max_tok=len(tok))
    sys_b = np.full(n, tr.system_prompt_len // B, np.int32)
    dtok, doff = T(tok), T(off)
    g = _gpu(ix, tok, off, sess, sys_b)
    ix.check()
    hb, _ = ix.block_hashes(dtok, doff)
    ix.check()
    hb = hb.cpu().numpy()
    ix.close()
    assert np.array_equal(g["hit"], g["sys"] + g["intra"] + g["inter"])
    nb = np.diff(off) // B
    last = {}
    for r, (s_, t_) in enumerate(zip(sess, turns)):
        if t_ > 0 and tr.truncate_prob == 0:
            assert g["hit"][r] >= nb[last[s_]]
        if t_ == 0:
            assert g["intra"][r] == 0
        last[s_] = r
    # first occurrence of every hash, then sampled requests recomputed
    first_b = np.concatenate([[0], np.cumsum(nb)])
    req_of = np.repeat(np.arange(n), nb)
    uniq, idx = np.unique(hb[:first_b[-1]], return_index=True)
    rng = np.random.default_rng(0)
    sess = np.asarray(sess)
    for r in rng.choice(n, size=200, replace=False):
        want = dict.fromkeys(KEYS, 0)
        for b in range(nb[r]):
            p = req_of[idx[np.searchsorted(uniq, hb[first_b[r] + b])]]
            if p >= r:
                break
            want["hit"] += 1
            want["sys" if b < sys_b[r] else "intra" if sess[p] == sess[r] else "inter"] += 1
        for k in KEYS:
            assert int(g[k][r]) == want[k], (r, k)
