"""Golden block-hash vectors (tests/golden/hash_vectors.txt, written by
tests/golden/make_golden.py from the oracle) guard the hash definition."""
import os

import numpy as np

import oracle

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "hash_vectors.txt")


def load_golden():
    rows = []
    with open(GOLDEN) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            name, toks, keys = [p.strip() for p in line.split("|")]
            t = np.array([int(v) for v in toks.split(",")], np.int32)
            k = np.array([int(v, 16) for v in keys.split()], np.uint64)
            rows.append((name, t, k))
    return rows


def test_oracle_reproduces_golden_hash_vectors():
    rows = load_golden()
    assert len(rows) == 5
    for name, t, k in rows:
        got, _ = oracle.hash_blocks(t, np.array([0, len(t)]))
        assert np.array_equal(got, k), name
        assert len(k) == len(t) // 16
