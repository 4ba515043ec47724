"""smetric_block_hashes_noalloc: block hashes and session keys from the fixed
scratch compiled into the library, with no index and no allocation. Its
outputs must equal those of smetric_block_hashes (an index's scratch) on the
same batches, call after call, and those of the CPU oracle; a batch beyond
the fixed scratch must be refused before anything is enqueued.

The file name sorts last so that the test also runs after every other GPU
test has used the library in the same process."""

import numpy as np
import pytest
import torch

import oracle
import paper_2607_08565_gb300 as pkg
from synth.traces import pack

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda:0")


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def _batch(rng, n, lo, hi, B):
    lens = rng.integers(lo, hi, size=n)
    lens[: min(n, 3)] = [0, B - 1, B][: min(n, 3)]  # empty, below one block, exactly one block
    reqs = [rng.integers(0, 151936, size=int(L), dtype=np.int32) for L in lens]
    return pack(reqs)


def _noalloc(tok, off, B, S, seed, status, cap=None):
    n = len(off) - 1
    nb = int(len(tok) // B)
    hb = torch.full((max(nb, 1),), 7, dtype=torch.int64, device=DEV)  # u64 words, int64 for torch ops
    sk = torch.full((max(n, 1),), 7, dtype=torch.int64, device=DEV)
    t, o = torch.from_numpy(tok).to(DEV), torch.from_numpy(off).to(DEV)
    rc = pkg.smetric_block_hashes_noalloc(t, len(tok), o, n, B, S, seed, sk, hb,
                                          nb if cap is None else cap, status)
    return rc, hb, sk


def _with_index(tok, off, B, S, seed):
    ix = pkg.SMetricIndex(4, B, S, capacity_slots=64, max_batch_requests=len(off) - 1,
                          max_batch_tokens=max(len(tok), 1), hash_seed=seed)
    hb, sk = ix.block_hashes(torch.from_numpy(tok).to(DEV), torch.from_numpy(off).to(DEV))
    ix.check()
    ix.close()
    return U(hb), U(sk)


def _oracle(tok, off, B, S, seed):
    """Block hashes (request-major) and session keys from the CPU oracle."""
    hs, keys = [], []
    for r in range(len(off) - 1):
        h = oracle.block_hashes(tok[off[r]:off[r + 1]], B, seed)
        hs.append(h)
        keys.append(int(h[min(len(h), S) - 1]) if len(h) else 0)
    return np.concatenate(hs).astype(np.uint64), np.array(keys, dtype=np.uint64)


def U(t):
    """A device tensor of 64-bit words as a host uint64 array."""
    return t.cpu().view(torch.int64).numpy().view(np.uint64)


def _used_blocks(off, B):
    return int((np.diff(off) // B).sum())


@pytest.mark.parametrize("B,S,seed", [(32, 1, 0), (16, 3, 12345), (6, 2, 2**63 + 5)])
def test_two_calls_in_a_row_equal_the_index_path(B, S, seed):
    rng = np.random.default_rng(B * 7 + S)
    batches = [_batch(rng, 300, 0, 60 * B, B), _batch(rng, 41, 0, 250 * B, B)]
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    results = []
    for tok, off in batches:  # back to back on the same stream, the scratch reused
        rc, hb, sk = _noalloc(tok, off, B, S, seed, status)
        assert rc == pkg.SMETRIC_OK
        results.append((hb, sk))
    torch.cuda.synchronize()
    assert int(status.item()) == pkg.SMETRIC_OK
    for (tok, off), (hb, sk) in zip(batches, results):
        rhb, rsk = _with_index(tok, off, B, S, seed)
        m = _used_blocks(off, B)
        assert np.array_equal(U(hb)[:m], rhb[:m])
        assert np.array_equal(U(sk)[: len(off) - 1], rsk[: len(off) - 1])
        # and the CPU oracle's own hashes and session keys, request by request
        ohb, osk = _oracle(tok, off, B, S, seed)
        assert np.array_equal(U(hb)[:m], ohb)
        assert np.array_equal(U(sk)[: len(off) - 1], osk)


def test_largest_accepted_batch_and_refusals():
    B = 32
    n_max, nb_max = pkg.SMETRIC_NOALLOC_MAX_REQUESTS, pkg.SMETRIC_NOALLOC_MAX_BLOCKS
    rng = np.random.default_rng(5)
    # exactly the limits: n_max requests holding nb_max full blocks in all
    per = np.full(n_max, nb_max // n_max * B)
    per[: nb_max - int((per // B).sum())] += B
    tok = rng.integers(0, 151936, size=int(per.sum()), dtype=np.int32)
    off = np.concatenate([[0], np.cumsum(per)]).astype(np.int64)
    assert len(off) - 1 == n_max and len(tok) // B == nb_max
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    rc, hb, sk = _noalloc(tok, off, B, 2, 9, status)
    assert rc == pkg.SMETRIC_OK
    rhb, rsk = _with_index(tok, off, B, 2, 9)
    assert np.array_equal(U(hb), rhb[:nb_max]) and np.array_equal(U(sk), rsk[:n_max])
    ohb, osk = _oracle(tok, off, B, 2, 9)
    assert np.array_equal(U(hb), ohb) and np.array_equal(U(sk), osk)
    assert int(status.item()) == 0

    # one request or one block more: refused, outputs untouched
    tok2 = np.concatenate([tok, rng.integers(0, 151936, size=B, dtype=np.int32)])
    off_blocks = off.copy()
    off_blocks[-1] += B
    off_reqs = np.concatenate([off, [off[-1]]])
    for t, o in ((tok2, off_blocks), (tok, off_reqs)):
        rc, hb, sk = _noalloc(t, o, B, 2, 9, status)
        assert rc == pkg.SMETRIC_ERR_TOO_LARGE
        torch.cuda.synchronize()
        assert np.all(U(hb) == 7) and np.all(U(sk) == 7)
    assert pkg.smetric_strerror(pkg.SMETRIC_ERR_TOO_LARGE) != "unknown error"


def test_invalid_offsets_latch_into_the_callers_status():
    B = 16
    rng = np.random.default_rng(6)
    tok, off = _batch(rng, 20, 0, 500, B)
    bad = off.copy()
    bad[5] = bad[6] + 1  # decreasing
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    rc, hb, sk = _noalloc(tok, bad, B, 1, 0, status)
    assert rc == pkg.SMETRIC_OK  # detected on the device
    torch.cuda.synchronize()
    assert int(status.item()) == pkg.SMETRIC_ERR_INVALID_ARG
    assert not U(sk).any()
    # the next call with good offsets is unaffected once the caller re-zeroes its status
    status.zero_()
    rc, hb, sk = _noalloc(tok, off, B, 1, 0, status)
    rhb, rsk = _with_index(tok, off, B, 1, 0)
    assert rc == pkg.SMETRIC_OK and int(status.item()) == 0
    m = _used_blocks(off, B)
    assert np.array_equal(U(hb)[:m], rhb[:m]) and np.array_equal(U(sk), rsk[:20])


def test_calls_leave_free_device_memory_unchanged():
    B = 32
    rng = np.random.default_rng(7)
    tok, off = _batch(rng, 500, 0, 3000, B)
    t, o = torch.from_numpy(tok).to(DEV), torch.from_numpy(off).to(DEV)
    nb = len(tok) // B
    hb = torch.empty(nb, dtype=torch.int64, device=DEV)
    sk = torch.empty(500, dtype=torch.int64, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    args = (t, len(tok), o, 500, B, 1, 0, sk, hb, nb, status)
    assert pkg.smetric_block_hashes_noalloc(*args) == pkg.SMETRIC_OK  # first call: module and symbol set up
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for _ in range(20):
        assert pkg.smetric_block_hashes_noalloc(*args) == pkg.SMETRIC_OK
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    assert int(status.item()) == 0
