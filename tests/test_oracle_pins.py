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


def test_oracle_reproduces_the_frozen_hash_vectors():
    """tests/golden/hash_vectors.json (written by make_hash_vectors.py from
    the oracle) still holds: the hash a caller sees does not drift."""
    import json
    import os

    import numpy as np

    here = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
    with open(os.path.join(here, "hash_vectors.json")) as f:
        d = json.load(f)
    seqs = {"zeros": np.zeros(53, np.int32), "iota": np.arange(129, dtype=np.int32),
            "extremes": np.array([-1, 0, 2**31 - 1, -2**31] * 16, np.int32),
            "vocab_seed7": np.random.default_rng(7).integers(0, 151936, size=323, dtype=np.int32)}
    assert len(d["cases"]) == 32
    for c in d["cases"]:
        h = oracle.block_hashes(seqs[c["tokens"]], c["block_size"], int(c["seed"], 16))
        assert [f"{int(x):016x}" for x in h] == c["hashes"], (c["tokens"], c["block_size"], c["seed"])
