"""Pins of the oracle's sequential-commit route (each decision adds one queued
request and the prompt's blocks to the chosen instance before the next
request is scored).  No GPU.

- the same route restated through the pinned batch route: per request, the
  instance rows and key sets rebuilt from the earlier decisions, then a batch
  route of that one request;
- one request is the batch route;
- a closed form: with a predictor whose output is the queue count, equal
  instances are taken in turn (the lowest index first), where the batch
  route sends every request to instance 0;
- a repeated prompt finds its whole prefix on the instance the first copy
  went to.
"""
import dataclasses

import numpy as np

import oracle
from paper_2606_00946_gb300 import workload as W


def _small(name="tiny", **kw):
    cfg = dataclasses.replace(W.CONFIGS[name], n_samples=0, **kw)
    return W.generate(cfg, with_samples=False)


def _restated(wl, queue_col=0):
    """Request by request through the batch route, with the state of the earlier decisions."""
    cfg = wl.cfg
    ik, iko = oracle.instance_keys(wl)
    sets = [list(ik[iko[i]:iko[i + 1]]) for i in range(cfg.n_inst)]
    inst = wl.inst_state.copy()
    rk, rko = oracle.hash_blocks(wl.tok, wl.tok_off)
    out_h, out_s, out_c = [], [], []
    for r in range(cfg.n_req):
        keys = np.concatenate([np.asarray(s, np.uint64) for s in sets]) if sum(map(len, sets)) else np.zeros(0, np.uint64)
        off = np.concatenate([[0], np.cumsum([len(s) for s in sets])]).astype(np.int64)
        wl_r = dataclasses.replace(wl, inst_state=inst.copy())
        ref = oracle.route(wl_r, inst_keys=(keys, off), req_idx=np.array([r]))
        c = int(ref["choice"][0])
        out_h.append(ref["hits"][0]); out_s.append(ref["scores"][0]); out_c.append(c)
        inst[c, queue_col] = np.float32(inst[c, queue_col] + np.float32(1.0))
        sets[c].extend(rk[rko[r]:rko[r + 1]].tolist())
    return np.array(out_h), np.array(out_s), np.array(out_c), inst


def test_sequential_route_equals_its_restatement_through_the_batch_route():
    for name, kw in (("tiny", dict(n_req=24)), ("paper", dict(n_req=12, cache_blocks=512))):
        wl = _small(name, **kw)
        got = oracle.route_sequential(wl)
        h, s, c, inst = _restated(wl)
        assert np.array_equal(got["hits"], h)
        assert np.array_equal(got["scores"], s)
        assert np.array_equal(got["choice"], c)
        assert np.array_equal(got["inst"], inst)
        # later requests saw earlier commits: some hit or queue differs from the batch route
        batch = oracle.route(wl)
        assert not np.array_equal(got["scores"], batch["scores"])


def test_one_request_is_the_batch_route():
    wl = _small(n_req=1)
    got = oracle.route_sequential(wl)
    ref = oracle.route(wl)
    assert np.array_equal(got["hits"], ref["hits"]) and np.array_equal(got["scores"], ref["scores"])
    assert np.array_equal(got["choice"], ref["choice"])


def test_queue_commits_take_equal_instances_in_turn():
    wl = _small(n_req=20)
    cfg = wl.cfg
    inst = wl.inst_state.copy()
    inst[:] = inst[0]                                   # identical instances
    mean = np.zeros(cfg.d, np.float32)
    std = np.ones(cfg.d, np.float32)
    params = np.zeros(W.param_count(cfg.widths), np.float32)
    w = np.asarray(cfg.widths)
    # layer 1 copies the queued-count feature (column 6) into unit 0, the
    # later layers pass unit 0 on: prediction = queued count
    params[6] = 1.0
    off = w[0] * w[1] + w[1]
    for l in range(1, len(w) - 1):
        params[off] = 1.0
        off += w[l] * w[l + 1] + w[l + 1]
    # no prefix sharing: empty caches
    wl2 = dataclasses.replace(wl, inst_state=inst, mean=mean, std=std, params=params,
                              chain_blocks=np.zeros_like(wl.chain_blocks), rand_keys=wl.rand_keys[:0],
                              inst_rand_off=np.zeros_like(wl.inst_rand_off))
    seq = oracle.route_sequential(wl2, mode="f32")
    assert seq["choice"].tolist() == [r % cfg.n_inst for r in range(cfg.n_req)]
    assert np.array_equal(seq["inst"][:, 0], inst[:, 0] + np.bincount(seq["choice"], minlength=cfg.n_inst))
    assert (oracle.route(wl2, mode="f32")["choice"] == 0).all()


def test_a_repeated_prompt_finds_its_prefix_where_the_first_copy_went():
    wl = _small(n_req=6)
    tok, off = wl.tok, wl.tok_off
    first = tok[off[1]:off[2]]
    seqs = [tok[off[r]:off[r + 1]] for r in range(6)] + [first]
    tok2 = np.concatenate(seqs)
    off2 = np.concatenate([[0], np.cumsum([len(s) for s in seqs])]).astype(np.int64)
    cfg = dataclasses.replace(wl.cfg, n_req=7)
    req = np.concatenate([wl.req_feats, wl.req_feats[1:2]])
    wl2 = dataclasses.replace(wl, cfg=cfg, tok=tok2, tok_off=off2, req_feats=req)
    got = oracle.route_sequential(wl2)
    nb = len(first) // 16
    c1 = got["choice"][1]
    assert got["hits"][6, c1] == nb
