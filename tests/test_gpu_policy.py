"""The session-centric policy (Figure 10) on the CUDA path against the CPU
oracle, element by element through the C ABI: instance, stick flag, local
and global hit and session key must be bit-exact."""

import numpy as np
import pytest
import torch

import oracle
import paper_2607_08565_gb300 as pkg
from synth.traces import pack
from gpu_util import T, assert_outputs_equal, make_index, populate_both, tiny_alphabet_case

pytestmark = pytest.mark.gpu

FIELDS = ("instance", "local_hit", "global_hit", "stick", "session_key")


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def _params(rng, N, tight=False):
    den = int(rng.integers(1, 1 << 20))
    return dict(c_lin=int(rng.integers(0, 1 << 20)), c_att=int(rng.integers(0, 1 << 12)),
                ttft_d0=int(rng.integers(0, 1 << 30 if tight else 1 << 60)),
                ttft_d1=int(rng.integers(0, 1 << 12 if tight else 1 << 35)),
                hit_num=int(rng.integers(0, den + 1)), hit_den=den, rr_base=int(rng.integers(0, N)))


def gpu_policy(ix, tok, off, queued, turn, est_hit, p):
    out = ix.route_batch_policy(T(tok), T(off), T(np.asarray(queued, np.int64)), T(np.asarray(turn, np.int32)),
                                T(np.asarray(est_hit, np.int64)), p)
    ix.check()
    return {k: v.cpu().numpy() for k, v in out.items()}


def oracle_policy(ox, B, S, tok, off, queued, turn, est_hit, p):
    return ox.route_batch_policy(B, S, 0, tok, off, queued, turn, est_hit, p["c_lin"], p["c_att"],
                                 p["ttft_d0"], p["ttft_d1"], p["hit_num"], p["hit_den"], p["rr_base"])


@pytest.mark.parametrize("N,B", [(1, 4), (3, 2), (8, 16), (64, 4), (130, 2), (256, 8)])
def test_policy_matches_oracle_tiny_alphabet(N, B):
    rng = np.random.default_rng(N * 131 + B)
    for trial in range(3):
        stored, reqs = tiny_alphabet_case(rng, N, B, n_req=300, max_blocks=12)
        S = int(rng.integers(1, 4))
        ix = make_index(N, B, S, cap=8192)
        ox = oracle.OracleIndex(N)
        populate_both(ix, ox, stored, B)
        tok, off = pack(reqs)
        n = len(reqs)
        L = np.diff(off)
        for case in range(6):
            p = _params(rng, N, tight=case % 2 == 0)
            if case == 4:
                p.update(c_att=0, c_lin=1)
            queued = rng.integers(0, [1 << 59, 1 << 20, 8, 1 << 40, 3, 1 << 59][case], size=N)
            turn = rng.integers(0, 3, size=n) * (case != 5)
            est_hit = np.minimum(rng.integers(0, 2 * L + 1), (1 << 31) - 1)
            g = gpu_policy(ix, tok, off, queued, turn, est_hit, p)
            o = oracle_policy(ox, B, S, tok, off, queued, turn, est_hit, p)
            assert_outputs_equal(g, o, fields=FIELDS, ctx=f"N={N} B={B} trial={trial} case={case}")
            if case == 5:
                assert not g["stick"].any()
        ix.close()


def test_policy_on_a_burst_batch():
    """A burst batch (2,048 requests over 4,096 Zipf-popular sessions with
    cached prefixes in the global, home and second tiers) under loose and
    tight deadlines: every output equal to the oracle's."""
    from synth import burst_trace
    tr = burst_trace(num_instances=16, block_size=32, n_sessions=4096, batch_size=2048,
                     len_lo=2000, len_hi=12000)
    p = tr.params
    bt = tr.batch(0)
    ix = make_index(p.num_instances, p.block_size, p.session_blocks, cap=int(tr.n_prefix_blocks() / 0.7) + 1,
                    max_req=bt.n_requests, max_tok=bt.n_tokens)
    ox = oracle.OracleIndex(p.num_instances)
    sessions = np.unique(bt.sessions)
    for ids, tok, off in tr.prepopulation(sessions):
        for j, sid in enumerate(ids):
            h = oracle.block_hashes(tok[off[j]:off[j + 1]], p.block_size)
            for t in tr.session_tiers(sid):
                ox.insert(h, t)
                ix.insert(T(h), T(np.full(len(h), t, np.int32)))
    ix.check()
    rng = np.random.default_rng(77)
    est_hit = tr.prefix_len[bt.sessions]
    turn = np.ones(bt.n_requests, np.int32)
    turn[rng.random(bt.n_requests) < 0.1] = 0
    for d0, d1 in ((1 << 60, 0), (1 << 22, 1 << 8), (0, 0)):
        pol = dict(c_lin=4, c_att=1, ttft_d0=d0, ttft_d1=d1, hit_num=9, hit_den=10, rr_base=3)
        queued = rng.integers(0, 1 << 34, size=p.num_instances)
        g = gpu_policy(ix, bt.tokens, bt.offsets, queued, turn, est_hit, pol)
        o = oracle_policy(ox, p.block_size, p.session_blocks, bt.tokens, bt.offsets, queued, turn, est_hit, pol)
        assert_outputs_equal(g, o, fields=FIELDS, ctx=f"burst d0={d0}")
        assert g["stick"].any() and not g["stick"].all()
    ix.close()


def test_policy_rejects_bad_parameters_and_inputs():
    rng = np.random.default_rng(78)
    N, B = 4, 16
    ix = make_index(N, B, 1)
    tok = rng.integers(0, 151936, size=1000, dtype=np.int32)
    off = np.array([0, 100, 400, 1000], np.int64)
    good = dict(c_lin=1, c_att=1, ttft_d0=1000, ttft_d1=1, hit_num=1, hit_den=2, rr_base=0)
    args = (T(tok), T(off), T(np.zeros(N, np.int64)), T(np.ones(3, np.int32)), T(np.zeros(3, np.int64)))
    for bad in (dict(c_lin=(1 << 20) + 1), dict(c_att=(1 << 12) + 1), dict(ttft_d0=-1),
                dict(ttft_d1=(1 << 35) + 1), dict(hit_num=3, hit_den=2), dict(hit_den=0),
                dict(rr_base=N), dict(rr_base=-1)):
        with pytest.raises(pkg.SmetricError) as e:
            ix.route_batch_policy(*args, {**good, **bad})
        assert e.value.code == pkg.SMETRIC_ERR_INVALID_ARG, bad
    # values the device checks: queued cost, expected hit
    for queued, est in ((np.array([0, (1 << 59) + 1, 0, 0]), np.zeros(3)),
                        (np.array([0, -1, 0, 0]), np.zeros(3)),
                        (np.zeros(N), np.array([0, -1, 0])),
                        (np.zeros(N), np.array([0, 0, 1 << 31]))):
        out = ix.route_batch_policy(T(tok), T(off), T(np.asarray(queued, np.int64)), T(np.ones(3, np.int32)),
                                    T(np.asarray(est, np.int64)), good)
        assert ix.status() == pkg.SMETRIC_ERR_OVERFLOW
        assert np.all(out["instance"].cpu().numpy() == -1) and not out["stick"].cpu().numpy().any()
    out = ix.route_batch_policy(*args, good)
    assert ix.status() == pkg.SMETRIC_OK and np.all(out["instance"].cpu().numpy() >= 0)
    ix.close()


def test_policy_rejects_prompts_longer_than_its_limit():
    """Eq. 1 needs L*L below 2^48 here: a prompt of 2^24 + 1 tokens latches
    OVERFLOW; 2^24 tokens route."""
    n_tok = pkg.SMETRIC_POLICY_MAX_LEN + 1
    ix = make_index(2, 64, 1, cap=1 << 16, max_req=8, max_tok=n_tok)
    tok = torch.zeros(n_tok, dtype=torch.int32, device="cuda")
    pol = dict(c_lin=1, c_att=1, ttft_d0=0, ttft_d1=0, hit_num=1, hit_den=1, rr_base=1)
    for L, code in ((n_tok, pkg.SMETRIC_ERR_OVERFLOW), (n_tok - 1, pkg.SMETRIC_OK)):
        off = torch.tensor([0, L], dtype=torch.int64, device="cuda")
        out = ix.route_batch_policy(tok, off, T(np.zeros(2, np.int64)), T(np.zeros(1, np.int32)),
                                    T(np.zeros(1, np.int64)), pol)
        assert ix.status() == code
        assert int(out["instance"].cpu()[0]) == (-1 if code else 1)  # equal loads: rotation from rr_base
    ix.close()


# ---------------------------------------------------------------------------
# PD colocation (Appendix B)
# ---------------------------------------------------------------------------

def gpu_coloc(ix, tok, off, queued, tpot, nreq, turn, est_hit, p):
    out = ix.route_batch_policy_coloc(T(tok), T(off), T(np.asarray(queued, np.int64)), T(np.asarray(tpot, np.int64)),
                                      T(np.asarray(nreq, np.int64)), T(np.asarray(turn, np.int32)),
                                      T(np.asarray(est_hit, np.int64)), p)
    ix.check()
    return {k: v.cpu().numpy() for k, v in out.items()}


def oracle_coloc(ox, B, S, tok, off, queued, tpot, nreq, turn, est_hit, p):
    return ox.route_batch_coloc(B, S, 0, tok, off, queued, tpot, nreq, turn, est_hit, p["c_lin"], p["c_att"],
                                p["ttft_d0"], p["ttft_d1"], p["hit_num"], p["hit_den"], p["rr_base"])


@pytest.mark.parametrize("N,B", [(1, 4), (3, 2), (8, 16), (64, 4), (130, 2), (256, 8)])
def test_coloc_matches_oracle_tiny_alphabet(N, B):
    rng = np.random.default_rng(N * 977 + B)
    for trial in range(3):
        stored, reqs = tiny_alphabet_case(rng, N, B, n_req=300, max_blocks=12)
        S = int(rng.integers(1, 4))
        ix = make_index(N, B, S, cap=8192)
        ox = oracle.OracleIndex(N)
        populate_both(ix, ox, stored, B)
        tok, off = pack(reqs)
        n = len(reqs)
        L = np.diff(off)
        for case in range(6):
            p = _params(rng, N, tight=case % 2 == 0)
            queued = rng.integers(0, [1 << 59, 1 << 20, 8, 1 << 40, 3, 1 << 59][case], size=N)
            # TPOT budgets around the prefill costs, some unlimited, some zero
            tpot = rng.integers(0, 1 << [60, 30, 12, 45, 8, 60][case], size=N)
            tpot[rng.random(N) < 0.2] = pkg.SMETRIC_POLICY_MAX_TPOT
            tpot[rng.random(N) < 0.1] = 0
            nreq = rng.integers(0, [1 << 20, 4, 64, 2, 1 << 20, 1000][case], size=N)
            turn = rng.integers(0, 3, size=n) * (case != 5)
            est_hit = np.minimum(rng.integers(0, 2 * L + 1), (1 << 31) - 1)
            g = gpu_coloc(ix, tok, off, queued, tpot, nreq, turn, est_hit, p)
            o = oracle_coloc(ox, B, S, tok, off, queued, tpot, nreq, turn, est_hit, p)
            assert_outputs_equal(g, o, fields=FIELDS, ctx=f"coloc N={N} B={B} trial={trial} case={case}")
        ix.close()


def test_coloc_rejects_out_of_range_inputs():
    rng = np.random.default_rng(79)
    N, B = 4, 16
    ix = make_index(N, B, 1)
    tok = rng.integers(0, 151936, size=1000, dtype=np.int32)
    off = np.array([0, 100, 400, 1000], np.int64)
    good = dict(c_lin=1, c_att=1, ttft_d0=1000, ttft_d1=1, hit_num=1, hit_den=2, rr_base=0)
    ok_t, ok_r = np.full(N, 1 << 40), np.ones(N)
    for tpot, nreq in ((np.array([0, (1 << 60) + 1, 0, 0]), ok_r), (np.array([0, -1, 0, 0]), ok_r),
                       (ok_t, np.array([0, (1 << 20) + 1, 0, 0])), (ok_t, np.array([-1, 0, 0, 0]))):
        out = ix.route_batch_policy_coloc(T(tok), T(off), T(np.zeros(N, np.int64)), T(np.asarray(tpot, np.int64)),
                                          T(np.asarray(nreq, np.int64)), T(np.ones(3, np.int32)),
                                          T(np.zeros(3, np.int64)), good)
        assert ix.status() == pkg.SMETRIC_ERR_OVERFLOW
        assert np.all(out["instance"].cpu().numpy() == -1)
    with pytest.raises(pkg.SmetricError):
        pkg.smetric_route_batch_policy_coloc(ix.handle, T(tok), 1000, T(off), 3, T(np.zeros(N, np.int64)), None,
                                             T(np.ones(N, np.int64)), T(np.ones(3, np.int32)),
                                             T(np.zeros(3, np.int64)), good, T(np.zeros(3, np.int32)),
                                             T(np.zeros(3, np.int32)), T(np.zeros(3, np.int32)),
                                             T(np.zeros(3, np.int32)), T(np.zeros(3, np.uint64)))
    out = ix.route_batch_policy_coloc(T(tok), T(off), T(np.zeros(N, np.int64)), T(ok_t.astype(np.int64)),
                                      T(ok_r.astype(np.int64)), T(np.ones(3, np.int32)), T(np.zeros(3, np.int64)),
                                      good)
    assert ix.status() == pkg.SMETRIC_OK
    ix.close()


# ---------------------------------------------------------------------------
# baseline scorers (Section 5.1)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("N,B", [(1, 4), (3, 2), (8, 16), (64, 4), (256, 8)])
def test_baselines_match_oracle_tiny_alphabet(N, B):
    rng = np.random.default_rng(N * 313 + B)
    stored, reqs = tiny_alphabet_case(rng, N, B, n_req=300, max_blocks=12)
    ix = make_index(N, B, 2, cap=8192)
    ox = oracle.OracleIndex(N)
    populate_both(ix, ox, stored, B)
    tok, off = pack(reqs)
    for case in range(8):
        scorer = pkg.SMETRIC_SCORER_BAILIAN if case % 2 == 0 else pkg.SMETRIC_SCORER_LMETRIC
        queued = rng.integers(0, [1 << 40, 100, 1, 1 << 20][case // 2], size=N)
        batch = rng.integers(0, [1 << 20, 8, 1, 300][case // 2], size=N)  # all zero in case 4-5
        den = int(rng.integers(1, 1 << 20))
        lam = (int(rng.integers(0, den + 1)), den)
        out = ix.route_batch_baseline(T(tok), T(off), scorer, T(np.asarray(queued, np.int64)),
                                      T(np.asarray(batch, np.int64)), lam)
        ix.check()
        g = {k: v.cpu().numpy() for k, v in out.items()}
        o = ox.route_batch_baseline(B, 2, 0, tok, off, scorer, queued, batch, *lam)
        assert_outputs_equal(g, o, fields=("instance", "local_hit", "global_hit", "session_key"),
                             ctx=f"N={N} B={B} case={case}")
    ix.close()


def test_baselines_refusals():
    rng = np.random.default_rng(80)
    N, B = 4, 16
    ix = make_index(N, B, 1)
    tok = rng.integers(0, 151936, size=1000, dtype=np.int32)
    off = np.array([0, 100, 400, 1000], np.int64)
    q, b = T(np.zeros(N, np.int64)), T(np.ones(N, np.int64))
    for scorer, lam in ((0, (1, 2)), (3, (1, 2)), (1, (3, 2)), (1, (0, 0)), (2, (1, (1 << 20) + 1))):
        with pytest.raises(pkg.SmetricError):
            ix.route_batch_baseline(T(tok), T(off), scorer, q, b, lam)
    for queued, batch in ((np.array([0, (1 << 40) + 1, 0, 0]), np.ones(N)),
                          (np.zeros(N), np.array([0, (1 << 20) + 1, 0, 0]))):
        out = ix.route_batch_baseline(T(tok), T(off), pkg.SMETRIC_SCORER_LMETRIC, T(np.asarray(queued, np.int64)),
                                      T(np.asarray(batch, np.int64)))
        assert ix.status() == pkg.SMETRIC_ERR_OVERFLOW
        assert np.all(out["instance"].cpu().numpy() == -1)
    ix.close()


# ---------------------------------------------------------------------------
# sequential-update variant
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("N,B", [(1, 4), (3, 2), (8, 16), (64, 4), (256, 8)])
def test_sequential_matches_oracle(N, B):
    rng = np.random.default_rng(N * 71 + B)
    stored, reqs = tiny_alphabet_case(rng, N, B, n_req=400, max_blocks=12)
    ix = make_index(N, B, 2, cap=8192)
    ox = oracle.OracleIndex(N)
    populate_both(ix, ox, stored, B)
    tok, off = pack(reqs)
    for w in ((1, 4, 2), (1, 1, 0), (5, 1, 7), (0, 3, 1), (2 ** 20, 2 ** 20, 2 ** 20)):
        load = rng.integers(0, [1 << 30, 50][w[0] > 1000], size=N)
        out = ix.route_batch_sequential(T(tok), T(off), T(np.asarray(load, np.int64)), w)
        ix.check()
        g = {k: v.cpu().numpy() for k, v in out.items()}
        o = ox.route_batch_sequential(B, 2, 0, tok, off, load, *w)
        assert_outputs_equal(g, o, fields=("instance", "local_hit", "global_hit", "session_key"),
                             ctx=f"N={N} B={B} w={w}")
        assert np.array_equal(g["load_after"], o["load_after"])
    ix.close()


def test_sequential_overflow_guard():
    N, B = 3, 4
    ix = make_index(N, B, 1)
    tok = np.zeros(64, np.int32)
    off = np.array([0, 32, 64], np.int64)
    out = ix.route_batch_sequential(T(tok), T(off), T(np.array([0, (1 << 42) - 63, 0], np.int64)))
    assert ix.status() == pkg.SMETRIC_ERR_OVERFLOW
    assert np.all(out["instance"].cpu().numpy() == -1)
    out = ix.route_batch_sequential(T(tok), T(off), T(np.array([0, (1 << 40), 0], np.int64)))
    assert ix.status() == pkg.SMETRIC_OK and out["instance"].cpu().numpy().tolist() == [0, 2]
    ix.close()
