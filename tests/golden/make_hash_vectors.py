"""Writes hash_vectors.json: the block chain hashes of a few fixed token
sequences, computed by the CPU oracle alone, so that another implementation
of the same hash (a serving engine computing the same keys, say) can check
itself against them, and so that any later change to the oracle's hash shows.

    python tests/golden/make_hash_vectors.py

Token sequences: all zeros, 0..L-1, int32 extremes, and a seeded draw from
[0, 151936) (the synthetic workloads' vocabulary). Each case lists B, the
seed, the tokens (or how to rebuild them), and the hash of every full block.
"""

import json
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import oracle  # noqa: E402


def sequences():
    yield "zeros", np.zeros(3 * 16 + 5, np.int32)
    yield "iota", np.arange(4 * 32 + 1, dtype=np.int32)
    yield "extremes", np.array([-1, 0, 2**31 - 1, -2**31] * 16, np.int32)
    yield "vocab_seed7", np.random.default_rng(7).integers(0, 151936, size=5 * 64 + 3, dtype=np.int32)


def main():
    cases = []
    for name, tok in sequences():
        for B in (2, 16, 32, 64):
            for seed in (0, 0x5EED5EED5EED5EED):
                h = oracle.block_hashes(tok, B, seed)
                cases.append({"tokens": name, "block_size": B, "seed": f"{seed:#018x}",
                              "hashes": [f"{int(x):016x}" for x in h]})
    out = {
        "what": "block chain hashes h_0..h_{n-1} of each token sequence (n = floor(len / B)), "
                "written by tests/golden/make_hash_vectors.py from the CPU oracle",
        "token_sequences": {
            "zeros": "53 zeros",
            "iota": "0, 1, ..., 128",
            "extremes": "[-1, 0, 2147483647, -2147483648] repeated 16 times",
            "vocab_seed7": "numpy.random.default_rng(7).integers(0, 151936, size=323, dtype=int32)",
        },
        "cases": cases,
    }
    with open(os.path.join(HERE, "hash_vectors.json"), "w") as f:
        json.dump(out, f, indent=1)
        f.write("\n")


if __name__ == "__main__":
    main()
