"""ls_prefix_hits_static (static device scratch, no allocation) against the
context path ls_route_batch and the oracle.

The file name sorts last, so in a full run these tests see a device on which
every other test has already run; they must pass alone in a fresh process
too.  Per-instance tables are built here on the host from the oracle's
instance keys (linear probing from key & (slots - 1), key 0 stored as 1).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_00946_gb300 import build as B
from paper_2606_00946_gb300 import harness as H
from paper_2606_00946_gb300 import lodestar as L
from paper_2606_00946_gb300 import workload as W


def host_tables(keys, key_off, n_inst, slots):
    """[n_inst, slots] uint64 open-addressing tables holding each instance's keys."""
    mask = np.uint64(slots - 1)
    T = np.zeros((n_inst, slots), np.uint64)
    for i in range(n_inst):
        k = np.asarray(keys[key_off[i]:key_off[i + 1]], np.uint64).copy()
        k[k == 0] = 1
        k = np.unique(k)
        assert len(k) <= slots // 2
        pos = (k & mask).astype(np.int64)
        pending = np.arange(len(k))
        tab = T[i]
        while pending.size:
            p = pos[pending]
            occ = tab[p] != 0
            pos[pending[occ]] = (p[occ] + 1) & (slots - 1)
            cand = pending[~occ]
            _, first = np.unique(pos[cand], return_index=True)
            won = cand[first]
            tab[pos[won]] = k[won]
            keep = np.ones(len(k), bool)
            keep[won] = False
            pending = pending[keep[pending]]
    return T


_cache = {}


def staged(name):
    if name not in _cache:
        B.build()
        wl = W.generate(name)
        r = H.Router.for_config(wl.cfg)
        dw = H.DeviceWorkload(wl)
        dw.load(r)
        ik, iko = oracle.instance_keys(wl)
        slots = W.table_capacity(wl.cfg.cache_blocks)
        tabs = torch.from_numpy(host_tables(ik, iko, wl.cfg.n_inst, slots).view(np.int64)).cuda()
        _cache[name] = (wl, dw, r, tabs, slots)
    return _cache[name]


def static_hits(wl, dw, tabs, slots, a, b, stream=None):
    n = b - a
    hits = torch.full((n, wl.cfg.n_inst), -7, dtype=torch.int32, device="cuda")
    n_tokens = int(wl.tok_off[b] - wl.tok_off[a])
    L.check(L.ls_prefix_hits_static(n, dw.tok, dw.tok_off[a:b + 1], n_tokens, tabs, slots,
                                    wl.cfg.n_inst, hits, stream))
    return hits


def route_hits(wl, dw, r, a, b):
    return r.route(dw.tok, dw.tok_off[a:b + 1], dw.req_feats[a:b], wl.cfg.n_inst)["hits"]


@pytest.mark.gpu
@pytest.mark.parametrize("name,a,b", [("tiny", 0, 64), ("homogeneous", 0, 192),
                                      ("homogeneous", 1000, 1500)])
def test_static_hits_match_route_two_calls_in_a_row(name, a, b):
    wl, dw, r, tabs, slots = staged(name)
    want = route_hits(wl, dw, r, a, b)
    # two calls back to back on one stream, no synchronisation between them:
    # the second must see counters reset by its own memset
    h1 = static_hits(wl, dw, tabs, slots, a, b)
    h2 = static_hits(wl, dw, tabs, slots, a, b)
    torch.cuda.synchronize()
    assert torch.equal(h1, want)
    assert torch.equal(h2, want)
    assert int(want.max()) > 0


@pytest.mark.gpu
def test_static_hits_oracle_and_different_batches_in_a_row():
    wl, dw, r, tabs, slots = staged("homogeneous")
    h1 = static_hits(wl, dw, tabs, slots, 300, 700)
    h2 = static_hits(wl, dw, tabs, slots, 2000, 2100)
    torch.cuda.synchronize()
    ik, iko = oracle.instance_keys(wl)
    for (a, b), h in (((300, 700), h1), ((2000, 2100), h2)):
        off = wl.tok_off[a:b + 1]
        rk, rko = oracle.hash_blocks(wl.tok, off)
        want = oracle.prefix_hits(rk, rko, ik, iko)
        assert np.array_equal(h.cpu().numpy(), want)


@pytest.mark.gpu
def test_static_limits_rejected_on_host():
    wl, dw, r, tabs, slots = staged("homogeneous")
    hits = torch.zeros(wl.cfg.n_req, wl.cfg.n_inst, dtype=torch.int32, device="cuda")
    n_tokens = int(wl.tok_off[-1] - wl.tok_off[0])      # ~8.4M tokens: > LS_STATIC_MAX_BLOCKS blocks
    assert n_tokens // 16 > L.LS_STATIC_MAX_BLOCKS
    rc = L.ls_prefix_hits_static(wl.cfg.n_req, dw.tok, dw.tok_off, n_tokens, tabs, slots, wl.cfg.n_inst, hits)
    assert rc == L.LS_ERR_ARG and "LS_STATIC_MAX_BLOCKS" in L.last_error()
    # a context-free call on the same device still works afterwards
    h = static_hits(wl, dw, tabs, slots, 0, 64)
    assert torch.equal(h, route_hits(wl, dw, r, 0, 64))


def test_static_arguments_rejected_before_any_device_work():
    # host checks only: the pointers below are never dereferenced
    B.build()
    fake = 1 << 20
    cases = [
        (dict(n_inst=0), "n_inst"),
        (dict(slots=24), "power of two"),
        (dict(slots=8), "power of two"),
        (dict(tables=fake + 8), "16-byte"),
        (dict(n_tokens=16 * (L.LS_STATIC_MAX_BLOCKS + 1)), "LS_STATIC_MAX_BLOCKS"),
        (dict(n_req=L.LS_STATIC_MAX_PAIRS // 4 + 1, n_inst=4), "LS_STATIC_MAX_PAIRS"),
        (dict(hits=None), "NULL"),
    ]
    for over, msg in cases:
        a = dict(n_req=4, tok=fake, tok_off=fake, n_tokens=64, tables=fake, slots=16, n_inst=2, hits=fake)
        a.update(over)
        rc = L.ls_prefix_hits_static(a["n_req"], a["tok"], a["tok_off"], a["n_tokens"], a["tables"],
                                     a["slots"], a["n_inst"], a["hits"], 0)
        assert rc == L.LS_ERR_ARG, over
        assert msg in L.last_error(), (over, L.last_error())
    assert L.ls_prefix_hits_static(0, None, None, 0, None, 16, 1, None, 0) == L.LS_OK
