"""The online-training configuration as a whole (Sec. 4.3.1 P2: training
runs beside routing and reaches it only through an atomic publish; Sec. 4.3.2
online learning): a ring of 2^20 logged 128-dim records, 1000 Adam steps
(batch 4096, lr 3e-4, sequential minibatches) on one stream, and every 10
steps a route of the heterogeneous-shaped batch (64 instances x 8192 prompts
of 8k-32k tokens) on a second stream and a publish on the first.

Checks, through the C ABI:
  - the loss curve stays inside an envelope of the oracle's own 1000-step run
    from the same start on the same minibatches (oracle.train_np): every
    window of 50 steps within 5% of the oracle's window mean, every step
    within 20%, and the curve falls by the same factor;
  - every route's predictions, on 8 sampled requests each, against the oracle
    run with the weights of the version that route reports (the master
    weights captured on the training stream right after each publish), at the
    parity bars of tests/parity_bars.py; hit lengths bit-exact.
"""
import os

import numpy as np
import pytest
import torch

import oracle
from oracle.train_np import NpTrainer
from parity_bars import assert_choices, assert_scores_close
from paper_2606_00946_gb300 import build as B
from paper_2606_00946_gb300 import harness as H
from paper_2606_00946_gb300 import lodestar as L
from paper_2606_00946_gb300 import workload as W

pytestmark = pytest.mark.gpu

STEPS, EVERY, PER_ROUTE = 1000, 10, 8
THREADS = max(1, min(16, os.cpu_count() or 1))


@pytest.fixture(scope="module", autouse=True)
def _built():
    B.build()


def test_online_training_schedule_loss_envelope_and_version_parity():
    wl = W.generate("training")
    cfg = wl.cfg
    R, N, Bt = cfg.n_req, cfg.n_inst, cfg.train_batch
    r = H.Router.for_config(cfg, ring_capacity=cfg.n_samples)
    dw = H.DeviceWorkload(wl)
    dw.load(r)                                              # publishes version 1 = the initial weights
    r.log(torch.from_numpy(wl.samples_x).cuda(), torch.from_numpy(wl.samples_y).cuda())
    n_routes = STEPS // EVERY
    losses = torch.zeros(STEPS, device="cuda")
    snaps = torch.zeros(n_routes + 1, r.n_params, device="cuda")
    snaps[0] = dw.params
    scores = torch.empty(n_routes, R, N, device="cuda")
    hits = torch.empty(R, N, dtype=torch.int32, device="cuda")
    choice = torch.empty(n_routes, R, dtype=torch.int32, device="cuda")
    best = torch.empty(n_routes, R, device="cuda")
    sa, sb = torch.cuda.Stream(), torch.cuda.Stream()
    torch.cuda.synchronize()
    versions = []
    for k in range(STEPS):
        r.train(Bt, None, opt="adam", lr=cfg.train_lr, loss_out=losses[k:k + 1], stream=sb)
        if k % EVERY == EVERY - 1:
            j = len(versions)
            o = r.route(dw.tok, dw.tok_off, dw.req_feats, N, stream=sa,
                        out={"choice": choice[j], "best": best[j], "scores": scores[j], "hits": hits})
            versions.append(o["version"])
            r.publish(stream=sb)
            L.check(L.ls_get_params(r.h, snaps[j + 1], sb))  # the weights of version j + 2
    torch.cuda.synchronize()
    assert r.sync() == L.LS_OK
    assert versions == list(range(1, n_routes + 1))           # each route saw the publish before it
    info = r.info()
    assert info.train_steps == STEPS and info.weight_version == n_routes + 1

    # (1) loss envelope against the oracle's own run
    tr = NpTrainer(cfg.widths, wl.params)
    count = cfg.n_samples
    want = np.array([tr.step(wl.samples_x, wl.samples_y, (k * Bt + np.arange(Bt)) % count, wl.mean, wl.std,
                             cfg.train_lr) for k in range(STEPS)])
    got = losses.cpu().numpy().astype(np.float64)
    assert np.all(np.abs(got - want) <= 0.2 * want), np.max(np.abs(got - want) / want)
    gw, ow = got.reshape(-1, 50).mean(1), want.reshape(-1, 50).mean(1)
    assert np.all(np.abs(gw - ow) <= 0.05 * ow), np.max(np.abs(gw - ow) / ow)
    assert abs(gw[-1] / gw[0] - ow[-1] / ow[0]) <= 0.05 * ow[-1] / ow[0]
    assert ow[-1] < 0.5 * ow[0]                               # the run learns

    # (2) each route against the oracle with the weights of its version
    rng = np.random.default_rng(44)
    samples = [np.sort(rng.choice(R, size=PER_ROUTE, replace=False)) for _ in range(n_routes)]
    allreq = np.unique(np.concatenate(samples))
    sub = [wl.tok[wl.tok_off[q]:wl.tok_off[q + 1]] for q in allreq]
    so = np.concatenate([[0], np.cumsum([len(t) for t in sub])]).astype(np.int64)
    rk, rko = oracle.hash_blocks(np.concatenate(sub), so)
    ik, iko = oracle.instance_keys(wl)
    oh = oracle.prefix_hits(rk, rko, ik, iko, by_marking=True, threads=THREADS)
    gh = hits.cpu().numpy()
    assert np.array_equal(gh[allreq], oh)
    row = {q: i for i, q in enumerate(allreq)}
    snaps_h = snaps.cpu().numpy()
    sc, ch = scores.cpu().numpy(), choice.cpu().numpy()
    for j, smp in enumerate(samples):
        v = versions[j]
        ref = oracle.route(wl, hits=oh[[row[q] for q in smp]], params=snaps_h[v - 1], req_idx=smp, bounds=True,
                           threads=THREADS)
        assert_scores_close(sc[j][smp], ref, 2e-2, "online training routes")
        assert_choices(ch[j][smp], sc[j][smp], ref, 2e-2)
    # the versions differ: the first and the last route's weights are not the same
    assert not np.array_equal(snaps_h[0], snaps_h[-1])
    r.close()
