"""Two-pool training data (Sec. 4.3.2) on the GPU vs the CPU oracle, through
the C ABI.

Bars: which records are candidates (the pending ring's bookkeeping) and the
replay pool's contents after a round are bit-exact, the latter against the
oracle's admission rule applied to the GPU's own distances; embeddings and
distances within the predictor's tolerance of the oracle's (bf16 products
and fp32 sums on tensor cores against fp64); training on F u R and bounds
over F u R as for the FIFO alone.
"""
import dataclasses

import numpy as np
import pytest
import torch

import oracle
from paper_2606_00946_gb300 import build as B
from paper_2606_00946_gb300 import harness as H
from paper_2606_00946_gb300 import workload as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    B.build()


class Pools:
    """The oracle side's record stream: FIFO slots, pending range, replay pool."""

    def __init__(self, C, P, Rc, d):
        self.C, self.P, self.Rc = C, P, Rc
        self.x = np.zeros((0, d), np.float32)
        self.y = np.zeros(0, np.float32)
        self.adm = 0
        self.rx = np.zeros((0, d), np.float32)
        self.ry = np.zeros(0, np.float32)

    def log(self, x, y):
        self.x = np.concatenate([self.x, x])
        self.y = np.concatenate([self.y, y])

    def pending(self):
        hi = max(0, len(self.y) - self.C)
        lo = min(hi, max(self.adm, hi - self.P))
        return lo, hi

    def fifo(self):
        n = len(self.y)
        nF = min(n, self.C)
        # slot s holds the newest stream position p < n with p % C == s
        pos = [(n - 1) - ((n - 1 - s) % self.C) for s in range(nF)]
        return self.x[pos], self.y[pos]


def _setup(name, C, P, Rc, batch, **over):
    cfg = dataclasses.replace(W.CONFIGS[name], n_samples=0, **over)
    wl = W.generate(cfg, with_samples=False)
    r = H.Router.for_config(cfg, ring_capacity=C, pending_capacity=P, replay_capacity=Rc, max_train_batch=batch)
    dw = H.DeviceWorkload(wl)
    dw.load(r)
    return cfg, wl, r


def _round(cfg, wl, r, pools, rng, n_new, mode):
    x, y = W.records(rng, cfg, n_new)
    r.log(torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda())
    pools.log(x, y)
    lo, hi = pools.pending()
    assert r.info().pending_count == hi - lo
    d_gpu, n_gpu = r.replay_admit(diag=True)
    m, nk = hi - lo, len(pools.ry)
    d_gpu = d_gpu.cpu().numpy()[:m].astype(np.float64)
    n_gpu = n_gpu.cpu().numpy()[:nk].astype(np.float64)
    cx, cy = pools.x[lo:hi], pools.y[lo:hi]
    # embeddings and distances against the oracle's (fp64)
    gc = oracle.replay_embed(mode, cfg.widths, wl.params, cx, cy, wl.mean, wl.std)
    gk = oracle.replay_embed(mode, cfg.widths, wl.params, pools.rx, pools.ry, wl.mean, wl.std)
    d_or, n_or = oracle.replay_distances(gc, gk)
    scale = np.mean(np.sum(np.concatenate([gc, gk]) ** 2, axis=1)) if m + nk else 1.0
    tol = 2e-5 if mode == "f32" else 5e-2
    for g, o in ((d_gpu, d_or), (n_gpu, n_or)):
        fin = np.isfinite(o)
        assert (np.isfinite(g) == fin).all()
        assert np.all(np.abs(g[fin] - o[fin]) <= tol * (o[fin] + scale))
    # the pool after the round: the oracle's rule on the GPU's distances, exactly
    src, cnt = oracle.replay_select(d_gpu, n_gpu, pools.Rc)
    nx = np.zeros((cnt, cfg.d), np.float32)
    ny = np.zeros(cnt, np.float32)
    for s, v in enumerate(src):
        if v >= 0:
            nx[s], ny[s] = cx[v], cy[v]
        else:
            nx[s], ny[s] = pools.rx[-1 - v], pools.ry[-1 - v]
    gx, gy = r.replay()
    np.testing.assert_array_equal(gx.cpu().numpy(), nx)
    np.testing.assert_array_equal(gy.cpu().numpy(), ny)
    # the oracle's own distances admit (nearly) the same candidates: they differ
    # only where two distances are within the tolerance of each other
    src_o, cnt_o = oracle.replay_select(d_or, n_or, pools.Rc)
    assert cnt_o == cnt
    a_g, a_o = set(int(v) for v in src if v >= 0), set(int(v) for v in src_o if v >= 0)
    overlap = len(a_g & a_o) / max(1, len(a_g | a_o))
    pools.rx, pools.ry, pools.adm = nx, ny, hi
    return m, int(sum(1 for v in src[:nk] if v >= 0)), overlap


@pytest.mark.parametrize("name,C,P,Rc,batch,mode,over", [
    ("homogeneous", 256, 256, 128, 256, "bf16", {}),                        # tensor-core distances
    ("homogeneous", 5000, 5000, 5000, 4096, "bf16", {}),                    # the paper's pool sizes
    ("tiny", 64, 48, 24, 64, "f32", {}),                                    # CUDA-core distances
])
def test_replay_rounds_parity(name, C, P, Rc, batch, mode, over):
    cfg, wl, r = _setup(name, C, P, Rc, batch, **over)
    pools = Pools(C, P, Rc, cfg.d)
    rng = np.random.default_rng(7)
    m, rep, _ = _round(cfg, wl, r, pools, rng, C - 10, mode)        # nothing evicted yet
    assert m == 0 and len(pools.ry) == 0
    m, rep, _ = _round(cfg, wl, r, pools, rng, C // 2, mode)        # first evictions fill free slots
    assert m > 0 and len(pools.ry) == min(Rc, m)
    overlaps = []
    replaced = 0
    for n_new in (C // 2, C, C // 3, C):                               # full pool: replacements
        m, rep, overlap = _round(cfg, wl, r, pools, rng, n_new, mode)
        replaced += rep
        overlaps.append(overlap)
    assert replaced > 0 and min(overlaps) >= (0.999 if mode == "f32" else 0.8), overlaps
    # more evictions than the pending ring holds: only the newest wait
    for _ in range(3):
        x, y = W.records(rng, cfg, C)
        r.log(torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda())
        pools.log(x, y)
    lo, hi = pools.pending()
    assert hi - lo == P and r.info().pending_count == P
    _round(cfg, wl, r, pools, rng, 1, mode)
    assert r.info().replay_count == len(pools.ry) == Rc
    # training on F u R and bounds over F u R
    fx, fy = pools.fifo()
    ux = np.concatenate([fx, pools.rx])
    uy = np.concatenate([fy, pools.ry])
    idx = np.concatenate([np.arange(len(fy) - 20, len(fy)), len(fy) + np.arange(len(pools.ry))]).astype(np.int32)
    idx = idx[: min(len(idx), batch)]
    loss = torch.zeros(1, device="cuda")
    r.train(len(idx), torch.from_numpy(idx).cuda(), opt="sgd", lr=1e-3, loss_out=loss)
    ol = oracle.Trainer(cfg.widths, wl.params, mode).step(ux, uy, idx, wl.mean, wl.std, "sgd", 1e-3)
    assert abs(loss.item() - ol) <= (1e-5 if mode == "f32" else 2e-2) * ol
    r.refresh_bounds()
    lo_g, hi_g = r.bounds(which=0)
    lo_o, hi_o = oracle.ring_bounds(ux, len(ux))
    np.testing.assert_array_equal(lo_g.cpu().numpy(), lo_o)
    np.testing.assert_array_equal(hi_g.cpu().numpy(), hi_o)
    r.close()


def test_replay_arguments():
    cfg = W.CONFIGS["tiny"]
    with pytest.raises(RuntimeError):
        H.Router.for_config(cfg, ring_capacity=64, pending_capacity=0, replay_capacity=8)
    r = H.Router.for_config(cfg, ring_capacity=64)
    from paper_2606_00946_gb300 import lodestar as L
    assert L.ls_replay_admit(r.h) == L.LS_ERR_STATE                    # no replay pool
    r.close()
    r = H.Router.for_config(cfg, ring_capacity=64, pending_capacity=16, replay_capacity=8)
    x = torch.zeros(65, cfg.d, device="cuda")
    assert L.ls_log_samples(r.h, 65, x, torch.zeros(65, device="cuda")) == L.LS_ERR_ARG
    assert L.ls_replay_admit(r.h) == L.LS_ERR_STATE                    # no parameters yet
    r.close()
