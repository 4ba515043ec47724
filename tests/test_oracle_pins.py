"""The CPU oracle against what the paper and mathematics fix (no GPU)."""

import pytest

import oracle
from pins import ALL_CHECKS


@pytest.mark.parametrize("check", ALL_CHECKS, ids=lambda f: f.__name__)
def test_oracle_pin(check):
    check(oracle.lib())


def test_oracle_threads_do_not_change_results():
    import numpy as np
    from synth import burst_trace

    tr = burst_trace(num_instances=8, block_size=16, n_sessions=64, batch_size=48,
                     len_lo=100, len_hi=900)
    p = tr.params
    ix = oracle.OracleIndex(p.num_instances)
    for ids, tok, off in tr.prepopulation():
        for j, s in enumerate(ids):
            h = oracle.block_hashes(tok[off[j]:off[j + 1]], p.block_size)
            for t in tr.session_tiers(s):
                ix.insert(h, t)
    bt = tr.batch(0)
    a = ix.route_batch(p.block_size, 2, 0, bt.tokens, bt.offsets, bt.load, 1, 4, 2, True, 1)
    b = ix.route_batch(p.block_size, 2, 0, bt.tokens, bt.offsets, bt.load, 1, 4, 2, True, 4)
    for k in a:
        assert np.array_equal(a[k], b[k])
    assert np.any(a["local_hit"] > 0) and np.any(a["global_hit"] > 0)
