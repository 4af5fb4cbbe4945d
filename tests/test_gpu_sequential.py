"""Sequential-commit routing on the GPU (ls_route_sequential) against the
oracle, through the C ABI.

The oracle replays the GPU's own decisions (forced choices), so every step is
checked against the definition from the same state: each request's hit
lengths bit-exact, its predictions at the parity bars (tests/parity_bars.py,
with the rounding analysis of that step's feature rows), its selection exact
on the GPU's scores and equal to the oracle's wherever the top-2 gap is
clear.  The state the call leaves (queues and caches) is then checked through
a batch route of the same requests: hits bit-exact against the oracle's final
key sets, predictions against the oracle with the final instance rows.
"""
import dataclasses
import os

import numpy as np
import pytest
import torch

import oracle
from parity_bars import assert_choices, assert_scores_close
from paper_2606_00946_gb300 import build as B
from paper_2606_00946_gb300 import harness as H
from paper_2606_00946_gb300 import lodestar as L
from paper_2606_00946_gb300 import workload as W

pytestmark = pytest.mark.gpu
THREADS = max(1, min(16, os.cpu_count() or 1))
TOL = {"f32": 1e-5, "bf16": 2e-2}


@pytest.fixture(scope="module", autouse=True)
def _built():
    B.build()


def _step_refs(wl, hits, forced, q_col):
    """Per-step oracle predictions with rounding analysis: the instance rows
    each request saw (queues raised by the earlier forced choices)."""
    cfg = wl.cfg
    R, N = cfg.n_req, cfg.n_inst
    Ls = np.diff(wl.tok_off)
    inst = wl.inst_state.copy()
    xs = []
    for r in range(R):
        xs.append(oracle.features(Ls[r:r + 1], hits[r:r + 1], inst, wl.req_feats[r:r + 1], wl.mean, wl.std))
        c = int(forced[r])
        inst[c, q_col] = np.float32(inst[c, q_col] + np.float32(1.0))
    y, eb, fl = oracle.mlp_forward_bounds(cfg.dtype, cfg.widths, wl.params, np.concatenate(xs))
    return {"scores": y.astype(np.float32).reshape(R, N), "ebound": eb.reshape(R, N),
            "flip": fl.reshape(R, N)}, inst


CASES = [
    ("tiny", dict(n_req=64)),
    ("paper", dict(n_req=96, cache_blocks=2048)),
    ("homogeneous", dict(n_req=160, cache_blocks=2048)),
]


@pytest.mark.parametrize("name,over", CASES)
def test_sequential_route_steps_and_final_state(name, over):
    cfg = dataclasses.replace(W.CONFIGS[name], n_samples=0, **over)
    wl = W.generate(cfg, with_samples=False)
    # room for the keys the batch's commits add (a full table latches LS_ERR_TABLE_FULL)
    room = cfg.cache_blocks + int(np.sum(np.diff(wl.tok_off) // 16))
    r = H.Router.for_config(cfg, max_keys_per_instance=room)
    dw = H.DeviceWorkload(wl)
    dw.load(r)
    q_col = 0
    out = r.route_sequential(dw.tok, dw.tok_off, dw.req_feats, cfg.n_inst, queue_col=q_col)
    assert r.sync() == L.LS_OK
    gc = out["choice"].cpu().numpy()
    gh = out["hits"].cpu().numpy()
    gs = out["scores"].cpu().numpy()
    ik, iko = oracle.instance_keys(wl)
    rep = oracle.route_sequential(wl, inst_keys=(ik, iko), queue_col=q_col, forced=gc)
    assert np.array_equal(gh, rep["hits"])
    ref, inst_final = _step_refs(wl, gh, gc, q_col)
    assert np.array_equal(rep["inst"], inst_final)
    assert_scores_close(gs, ref, TOL[cfg.dtype], f"sequential {name}")
    frac = assert_choices(gc, gs, ref, TOL[cfg.dtype])
    assert frac >= (0.9 if cfg.dtype == "f32" else 0.8)   # decisions the clear-gap check pins
    assert np.array_equal(out["best"].cpu().numpy(), gs[np.arange(cfg.n_req), gc])
    # commits mattered: some later request saw a hit or a queue the batch route does not see
    batch0 = oracle.route(wl, inst_keys=(ik, iko))
    assert not np.array_equal(gh, batch0["hits"]) or not np.array_equal(gs, batch0["scores"])
    # the state left behind: a batch route now sees the final caches and queues
    after = r.route(dw.tok, dw.tok_off, dw.req_feats, cfg.n_inst)
    rk, rko = oracle.hash_blocks(wl.tok, wl.tok_off)
    sets_k, sets_o = [ik], [iko]
    extra = [[] for _ in range(cfg.n_inst)]
    for q in range(cfg.n_req):
        extra[gc[q]].extend(rk[rko[q]:rko[q + 1]].tolist())
    keys = np.concatenate([np.concatenate([ik[iko[i]:iko[i + 1]], np.asarray(extra[i], np.uint64)])
                           for i in range(cfg.n_inst)])
    off = np.concatenate([[0], np.cumsum([iko[i + 1] - iko[i] + len(extra[i]) for i in range(cfg.n_inst)])])
    want_h = oracle.prefix_hits(rk, rko, keys, off.astype(np.int64))
    assert np.array_equal(after["hits"].cpu().numpy(), want_h)
    wl_f = dataclasses.replace(wl, inst_state=inst_final)
    ref_after = oracle.route(wl_f, hits=want_h, bounds=True, threads=THREADS)
    assert_scores_close(after["scores"].cpu().numpy(), ref_after, TOL[cfg.dtype], f"after sequential {name}")
    r.close()


def test_sequential_route_on_a_full_table_latches_table_full():
    cfg = dataclasses.replace(W.CONFIGS["tiny"], n_samples=0)
    wl = W.generate(cfg, with_samples=False)
    r = H.Router.for_config(cfg)                   # caches hold exactly max_keys_per_instance blocks
    dw = H.DeviceWorkload(wl)
    dw.load(r)
    r.route_sequential(dw.tok, dw.tok_off, dw.req_feats, cfg.n_inst)
    assert r.sync() == L.LS_ERR_TABLE_FULL
    r.close()


def test_sequential_route_arguments():
    cfg = dataclasses.replace(W.CONFIGS["tiny"], n_samples=0)
    wl = W.generate(cfg, with_samples=False)
    r = H.Router.for_config(cfg)
    dw = H.DeviceWorkload(wl)
    dw.load(r)
    ch = torch.empty(cfg.n_req, dtype=torch.int32, device="cuda")
    be = torch.empty(cfg.n_req, device="cuda")
    rc, _ = L.ls_route_sequential(r.h, cfg.n_req, dw.tok, dw.tok_off, dw.req_feats, cfg.d_inst, ch, be)
    assert rc == L.LS_ERR_ARG                            # queue column out of range
    rc, _ = L.ls_route_sequential(r.h, 0, dw.tok, dw.tok_off[:1], dw.req_feats, 0, ch, be)
    assert rc == L.LS_OK                                  # empty batch
    r2 = H.Router.for_config(cfg, prefix_mode="two_phase")
    dw.load(r2)
    rc, _ = L.ls_route_sequential(r2.h, cfg.n_req, dw.tok, dw.tok_off, dw.req_feats, 0, ch, be)
    assert rc == L.LS_ERR_ARG                            # needs the prefix index
    assert r.sync() == L.LS_OK
    r.close()
    r2.close()
