"""Host logic of bench.py that feeds its roofline numbers: the algorithmic
byte and flop counts of a routing batch against a brute-force recount on the
tiny workload, and the traffic lines' code hash (comments do not count, code
does).  No GPU needed."""
import importlib.util
import os
import sys

import numpy as np
import pytest

import oracle
from paper_2606_00946_gb300 import workload as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    argv, sys.argv = sys.argv, ["bench.py"]
    try:
        spec.loader.exec_module(mod)
    finally:
        sys.argv = argv
    return mod


def test_route_costs_against_a_recount(bench):
    wl = W.generate("tiny")
    cfg = wl.cfg
    R, N = cfg.n_req, cfg.n_inst
    ref = oracle.route(wl)
    hits = ref["hits"]
    keys, key_off = oracle.hash_blocks(wl.tok, wl.tok_off)
    lens = np.diff(wl.tok_off)
    got = bench.route_costs(cfg, R, N, hits, lens, keys, key_off)
    # tokens: every token of every prompt once
    assert got["tok_bytes"] == 4 * int(lens.sum())
    # probes: distinct keys each instance is asked about (the miss included)
    probes = 0
    for i in range(N):
        seen = set()
        for r in range(R):
            nb = lens[r] // 16
            for b in range(min(hits[r, i] + 1, nb)):
                seen.add(int(keys[key_off[r] + b]))
        probes += 8 * len(seen)
    assert probes > 0 and got["probe_bytes"] == probes
    assert got["prefix_bytes"] == got["tok_bytes"] + probes + 8 * R
    w = cfg.widths
    per_pair = 2 * 6 * w[1] + sum(2 * w[l] * w[l + 1] for l in range(1, len(w) - 1))
    assert got["score_flops"] == per_pair * R * N + 2 * N * cfg.d_inst * w[1] + 2 * R * cfg.d_req * w[1]
    assert got["score_flops_dense"] == sum(2 * w[l] * w[l + 1] for l in range(len(w) - 1)) * R * N


def test_distinct_probes_with_shared_prefixes(bench):
    # two requests share their first two blocks (keys 11, 12); instance 0
    # caches both, instance 1 only block 0, instance 2 nothing
    keys = np.array([11, 12, 13, 11, 12, 99], np.uint64)
    key_off = np.array([0, 3, 6], np.int64)
    lens = np.array([48, 50], np.int64)                 # 3 full blocks each
    hits = np.array([[2, 1, 0], [2, 1, 0]], np.int32)
    # instance 0 is asked 11, 12, 13, 99; instance 1: 11, 12; instance 2: 11
    assert bench.distinct_probes(hits, lens, keys, key_off) == 4 + 2 + 1


def test_code_digest_ignores_comments_only(bench, tmp_path, monkeypatch):
    csrc = tmp_path / "paper_2606_00946_gb300" / "csrc"
    csrc.mkdir(parents=True)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    f = csrc / "k.cu"
    f.write_text("// a kernel\n__global__ void k(int* p) { p[0] = 1; }  /* store */\n")
    d0 = bench.code_digest(["k.cu"])
    f.write_text("// the same kernel, new words\n__global__ void k(int* p) {\n  p[0] = 1;\n}\n")
    assert bench.code_digest(["k.cu"]) == d0
    f.write_text("__global__ void k(int* p) { p[0] = 2; }\n")
    assert bench.code_digest(["k.cu"]) != d0
