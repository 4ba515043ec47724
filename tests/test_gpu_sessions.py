"""Session reconstruction (Appendix A) on the CUDA path against the CPU
oracle, element by element through the C ABI: parent and session of every
request must be equal."""

import numpy as np
import pytest
import torch

import oracle
import paper_2607_08565_gb300 as pkg
from synth import agent_trace
from synth.traces import pack
from gpu_util import T, make_index

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def _both(B, S, seed, reqs, users, turns):
    tok, off = pack(reqs)
    n = len(reqs)
    ix = make_index(2, B, S, max_req=max(n, 1), max_tok=max(len(tok), 1), seed=seed)
    gp, gs = ix.link_sessions(T(tok), T(off), T(np.asarray(users, np.int64)), T(np.asarray(turns, np.int32)))
    ix.check()
    op, os_ = oracle.link_sessions(B, seed, tok, off, users, turns)
    ix.close()
    return gp.cpu().numpy(), gs.cpu().numpy(), op, os_


@pytest.mark.parametrize("B", [2, 4, 16])
def test_links_match_oracle_tiny_alphabet(B):
    """Prompts over a three-token alphabet share prefixes in every way; few
    users and turns so that many requests qualify as parents."""
    rng = np.random.default_rng(B)
    links = 0
    for trial in range(5):
        base = rng.integers(0, 3, size=12 * B, dtype=np.int32)
        n = int(rng.integers(1, 600)) if trial else 1  # one request: nothing to link
        reqs = []
        for _ in range(n):
            keep = int(rng.integers(0, 12 * B + 1))
            reqs.append(np.concatenate([base[:keep], rng.integers(0, 3, size=int(rng.integers(0, 3 * B)),
                                                                   dtype=np.int32)]))
        users = rng.integers(0, 4, size=n)
        turns = rng.integers(0, 5, size=n)
        gp, gs, op, os_ = _both(B, 1, trial, reqs, users, turns)
        assert np.array_equal(gp, op), (B, trial)
        assert np.array_equal(gs, os_), (B, trial)
        links += int((op >= 0).sum())
    assert links > 0


@pytest.mark.parametrize("name,scale", [("c1_tiny", 1.0), ("c3_long", 0.125)])
def test_links_on_agent_traces(name, scale):
    """Agent traces replayed in arrival order (turn waves), one user per
    session: equal to the oracle, and without truncation the chains are the
    generator's sessions."""
    tr = agent_trace(name, scale=scale, seed=7)
    reqs, users, turns = [], [], []
    for bt in tr.batches():
        for r in range(bt.n_requests):
            reqs.append(bt.tokens[bt.offsets[r]:bt.offsets[r + 1]])
        users.extend(bt.sessions.tolist())
        turns.extend(bt.turns.tolist())
    users, turns = np.array(users), np.array(turns)
    gp, gs, op, os_ = _both(tr.params.block_size, tr.params.session_blocks, 0, reqs, users, turns)
    assert np.array_equal(gp, op) and np.array_equal(gs, os_)
    if tr.truncate_prob == 0:
        first = {}
        for r, u in enumerate(users):
            first.setdefault(int(u), r)
        assert all(int(gs[r]) == first[int(u)] for r, u in enumerate(users))


def test_links_invalid_offsets():
    ix = make_index(2, 4, 1)
    tok = np.arange(40, dtype=np.int32)
    off = np.array([0, 20, 10, 40], np.int64)
    p, s_ = ix.link_sessions(T(tok), T(off), T(np.zeros(3, np.int64)), T(np.zeros(3, np.int32)))
    assert ix.status() == pkg.SMETRIC_ERR_INVALID_ARG
    assert np.all(p.cpu().numpy() == -1) and np.all(s_.cpu().numpy() == -1)
    ix.close()
