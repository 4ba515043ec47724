"""CUDA path vs the CPU oracle, element by element, through the C ABI.

Every routing output is integer or 64-bit hash work, so the bar is
bit-exact equality on every element."""

import numpy as np
import pytest
import torch

import oracle
import paper_2607_08565_gb300 as pkg
from synth.traces import pack
from gpu_util import (T, assert_outputs_equal, gpu_hashes, gpu_route, make_index, n_blocks,
                      populate_both, tiny_alphabet_case)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def _edge_lengths(B, rng):
    base = [0, 1, B - 1, B, B + 1, 2 * B, 2 * B + 1, 31 * B, 32 * B, 32 * B + 1, 33 * B - 1,
            33 * B, 64 * B + 3, 65 * B - 1]
    return base + rng.integers(0, 70 * B, size=24).tolist()


# ---------------------------------------------------------------------------
# (a)-(b): block hashes and session keys
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("B", [2, 4, 6, 16, 32, 64, 126, 256])
@pytest.mark.parametrize("seed", [0, 0xDEADBEEFCAFEF00D])
def test_block_hashes_ragged(B, seed):
    rng = np.random.default_rng(B * 7 + (seed & 0xFF))
    lens = _edge_lengths(B, rng)
    rng.shuffle(lens)
    # full int32 range, so negative token values exercise the uint32 view
    reqs = [rng.integers(-2**31, 2**31, size=L, dtype=np.int64).astype(np.int32) for L in lens]
    tok, off = pack(reqs)
    for S in (1, 3, 40):
        ix = make_index(4, B, S, seed=seed, max_tok=max(len(tok), 1))
        hb, sk = gpu_hashes(ix, tok, off)
        want_h = np.concatenate([oracle.block_hashes(r, B, seed) for r in reqs])
        assert np.array_equal(hb, want_h)
        for r, t in enumerate(reqs):
            h = oracle.block_hashes(t, B, seed)
            assert sk[r] == (0 if len(h) == 0 else h[min(len(h), S) - 1]), (r, len(t))
        ix.close()


@pytest.mark.parametrize("shift", [0, 1, 2, 3])
def test_block_hashes_into_caller_buffer_of_any_32_byte_phase(shift):
    """The chain writes hashes four per 32-byte store when the caller's hash
    buffer and the digests share a 32-byte phase, one per store when not:
    every phase gives the oracle's hashes and session keys."""
    rng = np.random.default_rng(60 + shift)
    B = 32
    reqs = [rng.integers(0, 151936, size=int(L), dtype=np.int32) for L in rng.integers(0, 3000, 200)]
    tok, off = pack(reqs)
    ix = make_index(4, B, 2)
    nb = n_blocks(off, B)
    cap = len(tok) // B  # the call requires room for n_tokens / B hashes
    big = torch.zeros(cap + 4, dtype=torch.int64, device="cuda")
    hb = big[shift:shift + cap]  # shift s: 8 s bytes past a 32-byte boundary
    sk = torch.zeros(len(off) - 1, dtype=torch.int64, device="cuda")
    pkg.smetric_block_hashes(ix.handle, T(tok), len(tok), T(off), len(off) - 1, sk, hb, cap, None)
    ix.check()
    o = oracle.OracleIndex(4).route_batch(B, 2, 0, tok, off, np.zeros(4, np.int64), 1, 4, 2,
                                           want_hashes=True)
    got = hb[:nb].cpu().numpy().view(np.uint64)
    assert np.array_equal(got, o["block_hashes"])
    assert np.array_equal(sk.cpu().numpy().view(np.uint64), o["session_key"])
    ix.close()


def test_block_hashes_wide_gaps_between_blocks():
    """Many requests shorter than one block between full blocks: a 32-block
    chunk then spans far more tokens than it hashes."""
    rng = np.random.default_rng(3)
    B = 16
    lens = []
    for _ in range(40):
        lens += [B + 3] + [B - 1] * 50 + [int(rng.integers(0, 3 * B))]
    reqs = [rng.integers(0, 151936, size=L, dtype=np.int32) for L in lens]
    tok, off = pack(reqs)
    ix = make_index(2, B, 2, max_req=len(reqs), max_tok=len(tok))
    hb, _ = gpu_hashes(ix, tok, off)
    assert np.array_equal(hb, np.concatenate([oracle.block_hashes(r, B) for r in reqs]))


def test_block_hashes_end_of_buffer_odd_start():
    """The last block ends exactly at the end of the token buffer and starts on
    an odd token, so its staged words include one partial word."""
    rng = np.random.default_rng(5)
    B = 32
    for first in (1, 3, 5):
        reqs = [rng.integers(0, 151936, size=first, dtype=np.int32),
                rng.integers(0, 151936, size=40 * B, dtype=np.int32)]
        tok, off = pack(reqs)
        ix = make_index(2, B, 2, max_tok=len(tok))
        hb, _ = gpu_hashes(ix, tok, off)
        assert np.array_equal(hb, oracle.block_hashes(reqs[1], B))


def test_sentinel_chain_values():
    from pins import sentinel_tokens
    rng = np.random.default_rng(6)
    for target, want in ((0, 2), (1, 3)):
        for seed in (0, 99):
            t = np.concatenate([sentinel_tokens(target, seed),
                                rng.integers(0, 151936, size=6, dtype=np.int32)])
            tok, off = pack([t, t[:2], t[:3]])
            ix = make_index(1, 2, 1, seed=seed)
            hb, sk = gpu_hashes(ix, tok, off)
            want_h = np.concatenate([oracle.block_hashes(x, 2, seed) for x in (t, t[:2], t[:3])])
            assert hb[0] == want and np.array_equal(hb, want_h)
            assert sk[0] == want


# ---------------------------------------------------------------------------
# index: insert / evict / lookup
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("N", [5, 63, 64, 127, 191, 256])
def test_index_set_semantics(N):
    rng = np.random.default_rng(N)
    ix = make_index(N, 16, 1, cap=4096)
    W = ix.W
    assert W == (N + 1 + 63) // 64
    ref = {t: set() for t in range(-1, N)}
    universe = rng.integers(2, 2**63, size=1500, dtype=np.int64).astype(np.uint64)
    for step in range(25):
        k = rng.choice(universe, size=int(rng.integers(1, 800)))
        t = rng.integers(-1, N, size=len(k)).astype(np.int32)
        if rng.random() < 0.65:
            ix.insert(T(k), T(t))
            for a, b in zip(k.tolist(), t.tolist()):
                ref[b].add(a)
        else:
            ix.evict(T(k), T(t))
            for a, b in zip(k.tolist(), t.tolist()):
                ref[b].discard(a)
        ix.check()
        q = np.concatenate([rng.choice(universe, size=300), np.array([2, 3, 12345], np.uint64)])
        m = ix.lookup(T(q)).cpu().numpy().reshape(len(q), W)
        for j, key in enumerate(q.tolist()):
            for tier in range(-1, N):
                bit = N if tier < 0 else tier
                got = (int(m[j, bit // 64]) >> (bit % 64)) & 1
                assert got == (key in ref[tier]), (step, key, tier)
    ix.close()


def test_index_rejects_bad_keys_and_tiers():
    ix = make_index(4, 16, 1)
    for keys, tiers in (([5, 0], [0, 0]), ([5, 1], [0, 1]), ([9], [4]), ([9], [-2])):
        ix.insert(T(np.array(keys, np.uint64)), T(np.array(tiers, np.int32)))
        assert ix.status() == pkg.SMETRIC_ERR_INVALID_ARG
        assert ix.status() == pkg.SMETRIC_OK  # the latch was cleared
    m = ix.lookup(T(np.array([5, 9], np.uint64))).cpu().numpy()
    assert m[0, 0] == 1 and m[1, 0] == 0  # the one valid pair (key 5, tier 0) went in


def test_index_full_reports_and_stays_consistent():
    ix = make_index(2, 16, 1, cap=100)  # rounded up to 7 buckets of 15 slots
    keys = np.arange(1000, 1300, dtype=np.uint64) * np.uint64(0x9E3779B97F4A7C15)
    keys = np.maximum(keys, 2)
    ix.insert(T(keys), T(np.zeros(len(keys), np.int32)))
    assert ix.status() == pkg.SMETRIC_ERR_TABLE_FULL
    m = ix.lookup(T(keys)).cpu().numpy()[:, 0]
    assert int((m & 1).sum()) == 105  # exactly the slots that exist
    ix.evict(T(keys), T(np.zeros(len(keys), np.int32)))
    assert ix.status() == pkg.SMETRIC_OK
    assert int(ix.lookup(T(keys)).cpu().numpy().sum()) == 0
    # every slot was given back: the table takes as many keys again
    ix.insert(T(keys[::-1].copy()), T(np.ones(len(keys), np.int32)))
    assert ix.status() == pkg.SMETRIC_ERR_TABLE_FULL
    m = ix.lookup(T(keys)).cpu().numpy()[:, 0]
    assert int(((m >> 1) & 1).sum()) == 105 and int((m & 1).sum()) == 0


def test_create_reports_oom_and_the_device_stays_usable():
    """A table no device holds (2^40 slots of 16 bytes, 16 TiB) is refused
    with SMETRIC_ERR_OOM and no index; the next index on the device works."""
    with pytest.raises(pkg.SmetricError) as e:
        make_index(4, 16, 1, cap=1 << 40)
    assert e.value.code == pkg.SMETRIC_ERR_OOM
    ix = make_index(4, 16, 1)
    ix.insert(T(np.array([5], np.uint64)), T(np.array([2], np.int32)))
    ix.check()
    assert ix.lookup(T(np.array([5], np.uint64))).cpu().numpy()[0, 0] == 4
    ix.close()


# ---------------------------------------------------------------------------
# (c)-(d): routing
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("N,B", [(1, 2), (3, 4), (5, 16), (63, 4), (64, 2), (65, 4), (128, 16),
                                 (191, 2), (192, 4), (256, 2)])
def test_route_matches_oracle_tiny_alphabet(N, B):
    rng = np.random.default_rng(N * 1000 + B)
    for trial in range(3):
        stored, reqs = tiny_alphabet_case(rng, N, B, n_req=150)
        S = int(rng.integers(1, 6))
        ix = make_index(N, B, S, cap=4096)
        ox = oracle.OracleIndex(N)
        populate_both(ix, ox, stored, B)
        tok, off = pack(reqs)
        for load in (rng.integers(0, 5, size=N), rng.integers(0, 2**40, size=N),
                     np.zeros(N, np.int64)):
            for w in ((1, 4, 2), (0, 3, 1), (5, 1, 7), (2**20, 2**20, 2**20), (0, 0, 0)):
                g = gpu_route(ix, tok, off, load, w)
                o = ox.route_batch(B, S, 0, tok, off, load, *w, want_hashes=True)
                assert_outputs_equal(g, o, ctx=f"N={N} B={B} trial={trial} w={w}")
        ix.close()


def test_route_requests_sharing_leading_blocks():
    """Requests with equal first blocks share their leader's probes up to the
    first differing block: members that are prefixes of the leader, extend
    it, diverge at block 0, 1, in the middle or only in the partial tail, a
    hot group of hundreds of members, a leader shorter than its members,
    empty and sub-block requests, all interleaved in one batch."""
    rng = np.random.default_rng(31)
    N, B = 64, 16
    bases = [rng.integers(0, 151936, size=int(rng.integers(20, 60)) * B + 7, dtype=np.int32)
             for _ in range(6)]
    reqs = []
    for i, base in enumerate(bases):
        nb = len(base) // B
        reqs.append(base[:B * 3])                                        # shortest: the leader when first
        reqs.append(base.copy())
        for cut in (0, 1, 2, nb // 2, nb - 1, nb):
            tail = rng.integers(0, 151936, size=int(rng.integers(0, 5 * B)), dtype=np.int32)
            reqs.append(np.concatenate([base[:cut * B], tail]))
        reqs.append(np.concatenate([base, rng.integers(0, 151936, size=3 * B, dtype=np.int32)]))
        reqs.append(base[:len(base) - 3])                                # differs only in the tail
        if i == 0:
            for _ in range(300):                                          # hot group
                k = int(rng.integers(1, nb + 1))
                reqs.append(np.concatenate([base[:k * B],
                                            rng.integers(0, 151936, size=int(rng.integers(0, 40)),
                                                         dtype=np.int32)]))
    reqs += [np.zeros(0, np.int32), bases[1][:B - 1], bases[2][:B]]
    order = np.concatenate([[0, 1], 2 + rng.permutation(len(reqs) - 2)])  # a short leader stays first
    reqs = [reqs[j] for j in order]
    stored = {}
    for t in range(-1, N):
        picks = rng.choice(len(bases), size=int(rng.integers(0, 3)), replace=False)
        stored[t] = [bases[j][:int(rng.integers(0, len(bases[j]) + 1))] for j in picks]
    ix = make_index(N, B, 2, cap=1 << 15)
    ox = oracle.OracleIndex(N)
    populate_both(ix, ox, stored, B)
    tok, off = pack(reqs)
    hits = np.zeros(2, np.int64)
    for load in (rng.integers(0, 50, size=N), np.zeros(N, np.int64), rng.integers(0, 10**6, size=N)):
        g = gpu_route(ix, tok, off, load, (1, 4, 2))
        o = ox.route_batch(B, 2, 0, tok, off, load, 1, 4, 2, want_hashes=True)
        assert_outputs_equal(g, o, ctx="shared leading blocks")
        hits += [g["local_hit"].max(), g["global_hit"].max()]
    assert hits.min() > 0  # both tiers contribute somewhere
    ix.close()


@pytest.mark.parametrize("B", [16, 32, 64, 6])
def test_hash_many_short_and_few_long_requests(B):
    """Batch shapes at the edges of the digest and chain work split: many
    short requests (several per warp, some empty), a few very long ones (one
    request's chain much longer than the others), and a mix; B = 6 takes the
    digest kernel for any even block size."""
    rng = np.random.default_rng(40 + B)
    shapes = [
        rng.integers(0, 4 * B, size=20000),                     # many short (some empty)
        np.array([300000, 7, 120000, 0, 2 * B]),                # few long
        np.concatenate([rng.integers(0, 3 * B, size=3000), [250000], rng.integers(0, 60 * B, size=500)]),
    ]
    for lens in shapes:
        reqs = [rng.integers(0, 151936, size=int(L), dtype=np.int32) for L in lens]
        tok, off = pack(reqs)
        ix = make_index(8, B, 3, max_req=len(lens), max_tok=len(tok) + 16)
        hb, sk = gpu_hashes(ix, tok, off)
        o = oracle.OracleIndex(8).route_batch(B, 3, 0, tok, off, np.zeros(8, np.int64), 1, 4, 2,
                                               want_hashes=True)
        assert np.array_equal(hb, o["block_hashes"]) and np.array_equal(sk, o["session_key"])
        g = gpu_route(ix, tok, off, np.zeros(8, np.int64), (1, 4, 2))
        assert_outputs_equal(g, o, ctx=f"B={B} n={len(lens)}")
        ix.close()


def test_route_special_cases():
    rng = np.random.default_rng(21)
    N, B = 9, 8
    reqs = [rng.integers(0, 151936, size=int(L), dtype=np.int32) for L in rng.integers(0, 600, 70)]
    tok, off = pack(reqs)
    ix = make_index(N, B, 4)
    # empty index: join the shortest queue, ties to the lowest id
    load = np.array([5, 3, 9, 3, 3, 8, 7, 4, 3])
    g = gpu_route(ix, tok, off, load, (1, 4, 2))
    assert np.all(g["instance"] == 1) and not g["local_hit"].any() and not g["global_hit"].any()
    # equal costs everywhere: instance 0
    g = gpu_route(ix, tok, off, np.full(N, 11), (1, 4, 2))
    assert np.all(g["instance"] == 0)


def test_route_rejects_bad_offsets_and_loads():
    rng = np.random.default_rng(22)
    N, B = 4, 16
    ix = make_index(N, B, 2)
    tok = rng.integers(0, 151936, size=1000, dtype=np.int32)
    good = np.array([0, 100, 400, 1000], np.int64)
    cases = [
        (np.array([0, 400, 100, 1000], np.int64), np.zeros(N), pkg.SMETRIC_ERR_INVALID_ARG),
        (np.array([0, 100, 400, 1001], np.int64), np.zeros(N), pkg.SMETRIC_ERR_INVALID_ARG),
        (np.array([-16, 100, 400, 1000], np.int64), np.zeros(N), pkg.SMETRIC_ERR_INVALID_ARG),
        (good, np.array([0, 2**40 + 1, 0, 0]), pkg.SMETRIC_ERR_OVERFLOW),
        (good, np.array([0, -1, 0, 0]), pkg.SMETRIC_ERR_OVERFLOW),
    ]
    for off, load, code in cases:
        out = ix.route_batch(T(tok), T(off), T(np.asarray(load, np.int64)), (1, 4, 2))
        assert ix.status() == code
        assert np.all(out["instance"].cpu().numpy() == -1)
        assert not out["session_key"].cpu().numpy().any()
    out = ix.route_batch(T(tok), T(good), T(np.zeros(N, np.int64)), (1, 4, 2))
    assert ix.status() == pkg.SMETRIC_OK and np.all(out["instance"].cpu().numpy() == 0)
    with pytest.raises(pkg.SmetricError):  # weight above 2^20: rejected on the host
        ix.route_batch(T(tok), T(good), T(np.zeros(N, np.int64)), (1, 2**20 + 1, 2))
    with pytest.raises(pkg.SmetricError):  # unaligned token pointer
        pkg.smetric_route_batch(ix.handle, T(tok).data_ptr() + 4, 999, T(good), 3,
                                T(np.zeros(N, np.int64)), (1, 4, 2), T(np.zeros(3, np.int32)),
                                T(np.zeros(3, np.int32)), T(np.zeros(3, np.int32)),
                                T(np.zeros(3, np.uint64)))


def test_batch_of_3100_requests_parity_and_late_errors():
    """A batch of 3,100 requests (several passes of the offset scan's warps):
    outputs equal the oracle's, an invalid offset early, in the middle or at
    the end of the batch, or a bad load, is caught, and the next good batch is
    unaffected."""
    rng = np.random.default_rng(31)
    N, B, S = 5, 8, 2
    stored, reqs = tiny_alphabet_case(rng, N, B, n_req=3100, max_blocks=12)
    ix = make_index(N, B, S, cap=1 << 15, max_req=4096)
    ox = oracle.OracleIndex(N)
    populate_both(ix, ox, stored, B)
    tok, off = pack(reqs)
    load = rng.integers(0, 50, size=N)
    before = pkg.smetric_launch_count(ix.handle)
    g = gpu_route(ix, tok, off, load, (1, 4, 2))
    assert pkg.smetric_launch_count(ix.handle) - before == 5  # prep, digest, leaders, chain and probe, walk
    o = ox.route_batch(B, S, 0, tok, off, load, 1, 4, 2, want_hashes=True)
    assert_outputs_equal(g, o, ctx="3100 requests")
    for r in (0, 1500, 2600, 3099):  # ranges of the first, a middle and the last CTA
        bad = off.copy()
        bad[r + 1] = bad[r] - 1 if bad[r] > 0 else len(tok) + 1
        out = ix.route_batch(T(tok), T(bad), T(load), (1, 4, 2))
        assert ix.status() == pkg.SMETRIC_ERR_INVALID_ARG, r
        assert np.all(out["instance"].cpu().numpy() == -1)
    out = ix.route_batch(T(tok), T(off), T(np.array([0, 0, -1, 0, 0])), (1, 4, 2))
    assert ix.status() == pkg.SMETRIC_ERR_OVERFLOW
    assert np.all(out["instance"].cpu().numpy() == -1)
    g = gpu_route(ix, tok, off, load, (1, 4, 2))  # the next good batch is unaffected
    assert_outputs_equal(g, o, ctx="after errors")
    ix.close()


def test_empty_batch_and_token_free_batch():
    ix = make_index(3, 16, 1)
    out = ix.route_batch(T(np.zeros(0, np.int32)), T(np.zeros(1, np.int64)),
                         T(np.zeros(3, np.int64)), (1, 4, 2))
    assert ix.status() == pkg.SMETRIC_OK and out["instance"].numel() == 0
    off = np.array([0, 5, 10, 15], np.int64)  # every request shorter than one block
    tok = np.arange(15, dtype=np.int32)
    g = gpu_route(ix, tok, off, np.array([4, 2, 9]), (1, 4, 2))
    assert np.all(g["instance"] == 1) and not g["session_key"].any()


def test_route_host_buffers_match_device_path():
    rng = np.random.default_rng(23)
    N, B = 8, 16
    stored, reqs = tiny_alphabet_case(rng, N, B, n_req=90, alphabet=2)
    tok, off = pack(reqs)
    ix = make_index(N, B, 3, host_staging=True, max_req=200, max_tok=len(tok) + 7)
    ox = oracle.OracleIndex(N)
    populate_both(ix, ox, stored, B)
    load = rng.integers(0, 100, size=N)
    g = gpu_route(ix, tok, off, load, (1, 4, 2), want_hashes=False)
    n = len(reqs)
    h = dict(instance=np.zeros(n, np.int32), local_hit=np.zeros(n, np.int32),
             global_hit=np.zeros(n, np.int32), session_key=np.zeros(n, np.uint64))
    rc = pkg.smetric_route_batch_host(ix.handle, tok, len(tok), off, n, np.asarray(load, np.int64),
                                      (1, 4, 2), h["instance"], h["local_hit"], h["global_hit"],
                                      h["session_key"])
    assert rc == pkg.SMETRIC_OK
    assert_outputs_equal(h, g, fields=("instance", "local_hit", "global_hit", "session_key"))
    o = ox.route_batch(B, 3, 0, tok, off, load, 1, 4, 2)
    assert_outputs_equal(h, o, fields=("instance", "local_hit", "global_hit", "session_key"))


def test_route_host_buffers_large_batch():
    """A larger host batch (600 requests, 9.6M tokens): outputs equal the
    device path's, call after call, and for a sample the oracle's; offsets a
    device check refuses give every request the invalid-batch outputs."""
    rng = np.random.default_rng(29)
    N, B = 16, 32
    n = 600
    lens = rng.integers(8000, 24000, size=n)
    # requests share prefixes with a few stored prompts so that hits occur
    base = [rng.integers(0, 151936, size=24000, dtype=np.int32) for _ in range(4)]
    reqs = []
    for L in lens.tolist():
        b = base[int(rng.integers(0, 4))]
        keep = int(rng.integers(0, L + 1))
        reqs.append(np.concatenate([b[:keep], rng.integers(0, 151936, size=L - keep, dtype=np.int32)]))
    tok, off = pack(reqs)
    assert off[-1] >= 8 << 20
    ix = make_index(N, B, 2, cap=1 << 16, host_staging=True, max_req=n, max_tok=len(tok))
    ox = oracle.OracleIndex(N)
    stored = {t: [base[t % 4][: 16000 + 512 * t]] for t in range(-1, N, 3)}
    populate_both(ix, ox, stored, B)
    load = rng.integers(0, 200000, size=N)
    g = gpu_route(ix, tok, off, load, (1, 4, 2), want_hashes=False)

    def host_route(offsets):
        h = dict(instance=np.zeros(n, np.int32), local_hit=np.zeros(n, np.int32),
                 global_hit=np.zeros(n, np.int32), session_key=np.zeros(n, np.uint64))
        rc = pkg.smetric_route_batch_host(ix.handle, tok, len(tok), offsets, n, np.asarray(load, np.int64),
                                          (1, 4, 2), h["instance"], h["local_hit"], h["global_hit"],
                                          h["session_key"])
        return rc, h

    for rep in range(2):
        rc, h = host_route(off)
        assert rc == pkg.SMETRIC_OK
        assert_outputs_equal(h, g, fields=("instance", "local_hit", "global_hit", "session_key"),
                             ctx=f"host buffers, call {rep}")
    sample = np.sort(rng.choice(n, size=40, replace=False))
    st, so = pack([tok[off[r]:off[r + 1]] for r in sample])
    o = ox.route_batch(B, 2, 0, st, so, load, 1, 4, 2)
    assert_outputs_equal({k: v[sample] for k, v in h.items()}, o,
                         fields=("instance", "local_hit", "global_hit", "session_key"))
    assert np.any(h["local_hit"] > 0)
    bad = off.copy()
    bad[450] = bad[451] + 1  # decreasing, late in the batch
    rc, hb = host_route(bad)
    assert rc == pkg.SMETRIC_ERR_INVALID_ARG
    assert np.all(hb["instance"] == -1) and not hb["session_key"].any()
    ix.close()


def test_profile_and_launch_count():
    rng = np.random.default_rng(24)
    ix = make_index(4, 16, 2)
    reqs = [rng.integers(0, 151936, size=3000, dtype=np.int32) for _ in range(20)]
    tok, off = pack(reqs)
    before = pkg.smetric_launch_count(ix.handle)
    pkg.smetric_profile_enable(ix.handle, True)
    for _ in range(3):
        gpu_route(ix, tok, off, np.zeros(4), (1, 4, 2))
    prof = pkg.smetric_profile_read(ix.handle)
    assert set(prof) == {"k_prep", "k_digest", "k_chain_probe", "k_walk"}
    assert all(v[1] == 3 and v[0] > 0 for v in prof.values())
    # 5 kernels per route: prep, digest, leaders, chain with group stage and probe, walk
    assert pkg.smetric_launch_count(ix.handle) - before == 15
    pkg.smetric_profile_enable(ix.handle, False)
