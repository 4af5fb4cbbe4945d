"""Writes tests/golden/hash_vectors.txt from the CPU oracle only.

The block-hash definition is this project's reading (the paper says only
that the gateway's prefix index may be a hash table, Sec. 2); these vectors
freeze that definition so that any later change to it is deliberate.
Run:  python tests/golden/make_golden.py
"""
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)
import oracle  # noqa: E402


def cases():
    yield "iota48", np.arange(48, dtype=np.int32)
    yield "zeros33", np.zeros(33, dtype=np.int32)
    yield "negatives32", -np.arange(1, 33, dtype=np.int32)
    yield "vocab_edge16", np.full(16, 31999, dtype=np.int32)
    yield "seeded80", np.random.default_rng(2024).integers(0, 32000, 80).astype(np.int32)


def main():
    out = os.path.join(os.path.dirname(os.path.abspath(__file__)), "hash_vectors.txt")
    with open(out, "w") as f:
        f.write("# name | tokens (int32, comma separated) | block keys (uint64 hex)\n")
        for name, t in cases():
            keys, _ = oracle.hash_blocks(t, np.array([0, len(t)]))
            f.write(f"{name} | {','.join(str(int(v)) for v in t)} | "
                    f"{' '.join(format(int(k), '016x') for k in keys)}\n")
    print("wrote", out)


if __name__ == "__main__":
    main()
