"""CUDA path vs the CPU oracle on the same seeded inputs, through the C ABI.

Bars: bit-exact block keys, hit lengths and selected instances (the selector
is checked on the GPU's own scores; against the oracle's scores wherever the
oracle's top-2 gap is clear of rounding); predictions within 1e-5 (fp32) /
2e-2 (bf16) of max(|o|, 1e-3 s), rows that fp32 accumulation cannot pin to
that bar held to their rounding radius and counted (tests/parity_bars.py).
"""
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

TOL = {"f32": 1e-5, "bf16": 2e-2}
THREADS = max(1, min(16, os.cpu_count() or 1))


@pytest.fixture(scope="module", autouse=True)
def _built():
    B.build()


_cache = {}


def staged(name):
    if name not in _cache:
        wl = W.generate(name)
        r = H.Router.for_config(wl.cfg)
        dw = H.DeviceWorkload(wl)
        dw.load(r)
        _cache[name] = (wl, dw, r)
    return _cache[name]


_okeys = {}


def oracle_inst_keys(name, wl):
    if name not in _okeys:
        _okeys[name] = oracle.instance_keys(wl)
    return _okeys[name]


def u64(t):
    return t.cpu().numpy().view(np.uint64)


# ----------------------------------------------------------------------------
# hashing
# ----------------------------------------------------------------------------

def test_hash_golden_vectors():
    from test_golden import load_golden
    wl, dw, r = staged("tiny")
    for name, t, k in load_golden():
        tok = torch.from_numpy(t).cuda()
        off = torch.tensor([0, len(t)], dtype=torch.int64, device="cuda")
        keys, _ = r.hash_blocks(tok, off)
        assert np.array_equal(u64(keys), k), name


@pytest.mark.parametrize("name", ["tiny", "homogeneous", "heterogeneous"])
def test_hash_parity(name):
    wl, dw, r = staged(name)
    keys, ko = r.hash_blocks(dw.tok, dw.tok_off)
    want, wko = oracle.hash_blocks(wl.tok, wl.tok_off)
    assert np.array_equal(ko.cpu().numpy(), wko)
    assert np.array_equal(u64(keys), want)


def test_hash_unaligned_ragged_and_empty():
    wl, dw, r = staged("tiny")
    rng = np.random.default_rng(11)
    lens = [0, 1, 15, 16, 17, 31, 32, 33, 255, 256, 257, 4095, 4096, 4097, 16 * 300 + 3]
    seqs = [rng.integers(-2**31, 2**31 - 1, size=n, dtype=np.int64).astype(np.int32) for n in lens]
    tok = np.concatenate([np.array([7], np.int32)] + seqs)           # shift: odd starting offsets
    off = np.concatenate([[1], 1 + np.cumsum([len(s) for s in seqs])]).astype(np.int64)
    keys, ko = r.hash_blocks(torch.from_numpy(tok).cuda(), torch.from_numpy(off).cuda())
    want, _ = oracle.hash_blocks(tok, off)
    assert np.array_equal(u64(keys), want)


# ----------------------------------------------------------------------------
# prefix hits
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("name", ["tiny", "homogeneous", "heterogeneous"])
def test_hits_parity(name):
    wl, dw, r = staged(name)
    out = r.route(dw.tok, dw.tok_off, dw.req_feats, wl.cfg.n_inst)
    rk, rko = oracle.hash_blocks(wl.tok, wl.tok_off)
    ik, iko = oracle_inst_keys(name, wl)
    want = oracle.prefix_hits(rk, rko, ik, iko)
    got = out["hits"].cpu().numpy()
    assert np.array_equal(got, want)
    assert want.max() > 0 and (want == 0).any()


@pytest.mark.parametrize("name", ["tiny", "homogeneous", "heterogeneous"])
@pytest.mark.parametrize("mode", ["two_phase", "fused"])
def test_prefix_modes_agree(name, mode):
    # the default (prefix index over all instances) against per-instance tables
    wl, dw, r = staged(name)
    out = r.route(dw.tok, dw.tok_off, dw.req_feats, wl.cfg.n_inst)
    r2 = H.Router.for_config(wl.cfg, prefix_mode=mode)
    dw.load(r2)
    out2 = r2.route(dw.tok, dw.tok_off, dw.req_feats, wl.cfg.n_inst)
    assert torch.equal(out["hits"], out2["hits"])
    assert torch.equal(out["choice"], out2["choice"]) and torch.equal(out["scores"], out2["scores"])
    r2.close()


def test_batch_over_token_capacity_is_latched_not_faulted():
    wl, dw, r = staged("tiny")
    small = H.Router.for_config(wl.cfg, max_batch_tokens=1000, prefix_mode="two_phase")
    dw.load(small)
    small.route(dw.tok, dw.tok_off, dw.req_feats, wl.cfg.n_inst)   # ~20k tokens > 1000
    assert small.sync() == L.LS_ERR_ARG
    # a batch that fits, taken from the middle of the token buffer (slots are
    # relative to the batch's first offset)
    off = wl.tok_off
    a = 10
    b = a + 1
    while b < len(off) - 1 and off[b + 1] - off[a] <= 1000:
        b += 1
    sub = dw.tok_off[a:b + 1]
    ok = small.route(dw.tok, sub, dw.req_feats[a:b], wl.cfg.n_inst)
    assert small.sync() == L.LS_OK
    ref = r.route(dw.tok, sub, dw.req_feats[a:b], wl.cfg.n_inst)
    assert torch.equal(ok["hits"], ref["hits"]) and torch.equal(ok["scores"], ref["scores"])
    small.close()


def test_large_hits_every_request_and_scores_on_512():
    # the large cluster (256 instances x 16,384 requests, 2^20 cached blocks
    # each) routed whole in the launch shape the bench times: hit lengths of
    # every request against the oracle's marking over every instance key, then
    # predictions and selections of 512 sampled requests
    wl, dw, r = staged("large")
    out = r.route(dw.tok, dw.tok_off, dw.req_feats, wl.cfg.n_inst)
    got = out["hits"].cpu().numpy()
    rk, rko = oracle.hash_blocks(wl.tok, wl.tok_off)
    ik, iko = oracle_inst_keys("large", wl)
    want = oracle.prefix_hits(rk, rko, ik, iko, by_marking=True, threads=THREADS)
    assert np.array_equal(got, want)
    assert want.max() > 0 and (want == 0).any()
    idx = np.sort(np.random.default_rng(5).choice(wl.cfg.n_req, size=512, replace=False))
    ref = oracle.route(wl, hits=want[idx], req_idx=idx, bounds=True, threads=THREADS)
    sg = out["scores"].cpu().numpy()[idx]
    assert_scores_close(sg, ref, TOL["bf16"], "large 512 x 256")
    assert_choices(out["choice"].cpu().numpy()[idx], sg, ref, TOL["bf16"])
    c_own, _ = oracle.argmin(out["scores"].cpu().numpy())
    assert np.array_equal(out["choice"].cpu().numpy(), c_own)


# ----------------------------------------------------------------------------
# features, predictions, selection
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("name", ["tiny", "homogeneous"])
def test_features_parity(name):
    wl, dw, r = staged(name)
    out = r.route(dw.tok, dw.tok_off, dw.req_feats, wl.cfg.n_inst)
    x = r.features(dw.tok_off, out["hits"], dw.req_feats).cpu().numpy()
    want = oracle.features(np.diff(wl.tok_off), out["hits"].cpu().numpy(), wl.inst_state, wl.req_feats,
                           wl.mean, wl.std)
    ulp = np.abs(x.view(np.int32).astype(np.int64) - want.view(np.int32).astype(np.int64))
    assert ulp.max() <= 1


def _bf16_ordered(bits):
    # bf16 bit patterns to integers that order as the values do (sign-magnitude -> two's complement)
    b = bits.astype(np.int64) & 0xFFFF
    return np.where(b & 0x8000, -(b & 0x7FFF), b)


@pytest.mark.parametrize("case", ["homogeneous", "heterogeneous", "wide"])
def test_production_feature_rows(case):
    # the bf16 rows the tensor-core scorer read (feature image of the pipelined
    # scorer; pair chunks + template rows of the others), every row of the
    # batch, against the oracle's features rounded to bf16: at most one bf16
    # ulp apart (the fp32 z-score may differ by one fp32 ulp under FMA
    # contraction, which can move a bf16 rounding), almost all bit-exact
    import dataclasses
    own = case == "wide"
    if own:
        cfg = dataclasses.replace(W.CONFIGS["large"], n_req=48, cache_blocks=1024, n_samples=0)
        wl = W.generate(cfg)
        r = H.Router.for_config(cfg)
        dw = H.DeviceWorkload(wl)
        dw.load(r)
    else:
        wl, dw, r = staged(case)
    cfg = wl.cfg
    out = r.route(dw.tok, dw.tok_off, dw.req_feats, cfg.n_inst)
    rows = cfg.n_req * cfg.n_inst
    g = torch.empty(rows, cfg.d, dtype=torch.int16, device="cuda")
    L.check(L.ls_read_features(r.h, 0, rows, g))
    want = oracle.features(np.diff(wl.tok_off), out["hits"].cpu().numpy(), wl.inst_state, wl.req_feats,
                           wl.mean, wl.std)
    wb = torch.from_numpy(want).to(torch.bfloat16).view(torch.int16).numpy()
    diff = np.abs(_bf16_ordered(g.cpu().numpy()) - _bf16_ordered(wb))
    assert diff.max() <= 1, diff.max()
    assert (diff == 0).mean() > 0.999
    if own:
        r.close()


def test_route_parity_tiny_fp32():
    wl, dw, r = staged("tiny")
    out = r.route(dw.tok, dw.tok_off, dw.req_feats, wl.cfg.n_inst)
    ref = oracle.route(wl, inst_keys=oracle_inst_keys("tiny", wl), bounds=True)
    assert np.array_equal(out["hits"].cpu().numpy(), ref["hits"])
    sg = out["scores"].cpu().numpy()
    assert_scores_close(sg, ref, TOL["f32"], "tiny fp32")
    frac = assert_choices(out["choice"].cpu().numpy(), sg, ref, TOL["f32"])
    assert frac > 0.95
    assert np.array_equal(out["best"].cpu().numpy(), sg[np.arange(len(sg)), out["choice"].cpu().numpy()])


@pytest.mark.parametrize("name,n_sample", [("homogeneous", 4096), ("heterogeneous", 1024)])
def test_route_parity_bf16(name, n_sample):
    wl, dw, r = staged(name)
    out = r.route(dw.tok, dw.tok_off, dw.req_feats, wl.cfg.n_inst)
    idx = np.sort(np.random.default_rng(3).choice(wl.cfg.n_req, size=n_sample, replace=False))
    ref = oracle.route(wl, inst_keys=oracle_inst_keys(name, wl), req_idx=idx, bounds=True, threads=THREADS)
    sg = out["scores"].cpu().numpy()
    assert np.array_equal(out["hits"].cpu().numpy()[idx], ref["hits"])
    assert_scores_close(sg[idx], ref, TOL["bf16"], f"{name} {n_sample} x {wl.cfg.n_inst}")
    assert_choices(out["choice"].cpu().numpy()[idx], sg[idx], ref, TOL["bf16"])
    # the selector on every request of the batch
    c_own, b_own = oracle.argmin(sg)
    assert np.array_equal(out["choice"].cpu().numpy(), c_own)


@pytest.mark.parametrize("name", ["homogeneous", "heterogeneous", "large"])
def test_tensor_core_scorer_matches_cuda_core_scorer(name):
    wl, dw, r = staged(name)
    assert r.info().scorer == L.LS_SCORER_TENSOR_CORES
    out = r.route(dw.tok, dw.tok_off, dw.req_feats, wl.cfg.n_inst)
    r2 = H.Router.for_config(wl.cfg, scorer="cuda_cores")
    assert r2.info().scorer == L.LS_SCORER_CUDA_CORES
    dw.load(r2)
    out2 = r2.route(dw.tok, dw.tok_off, dw.req_feats, wl.cfg.n_inst)
    assert torch.equal(out["hits"], out2["hits"])
    s1, s2 = out["scores"].cpu().numpy(), out2["scores"].cpu().numpy()
    # both scorers against the oracle on sampled requests; each selector exact on its own scores
    idx = np.sort(np.random.default_rng(8).choice(wl.cfg.n_req, size=64, replace=False))
    ref = oracle.route(wl, hits=out["hits"].cpu().numpy()[idx], req_idx=idx, bounds=True, threads=THREADS)
    for sc, ch, tag in ((s1, out["choice"], "tensor cores"), (s2, out2["choice"], "CUDA cores")):
        assert_scores_close(sc[idx], ref, TOL["bf16"], f"{name} {tag}")
        assert np.array_equal(ch.cpu().numpy(), oracle.argmin(sc)[0])
    r2.close()


@pytest.mark.parametrize("n_inst", [24, 200])
def test_pipelined_scorer_with_tiles_across_requests(n_inst):
    # instance counts that do not divide the 128-row tile (tiles span request
    # boundaries), and more instances than rows in a tile
    import dataclasses
    cfg = dataclasses.replace(W.CONFIGS["homogeneous"], n_inst=n_inst, n_req=64, cache_blocks=1024,
                              n_samples=0)
    wl = W.generate(cfg)
    r = H.Router.for_config(cfg)
    dw = H.DeviceWorkload(wl)
    dw.load(r)
    assert r.info().scorer == L.LS_SCORER_TENSOR_CORES
    out = r.route(dw.tok, dw.tok_off, dw.req_feats, n_inst)
    ref = oracle.route(wl, bounds=True)
    assert np.array_equal(out["hits"].cpu().numpy(), ref["hits"])
    sg = out["scores"].cpu().numpy()
    assert_scores_close(sg, ref, TOL["bf16"], f"tiles across requests, {n_inst} instances")
    assert_choices(out["choice"].cpu().numpy(), sg, ref, TOL["bf16"])
    r.close()


@pytest.mark.parametrize("hidden,n_inst,wide_dims,n_req,kernel", [
    ((512, 512), 24, False, 96, "pair"), ((256, 512), 256, True, 48, "pair"), ((512, 512), 256, True, 48, "pair"),
    ((512, 512), 24, True, 100, "pair"), ((512, 256), 24, True, 5, "pair"), ((256, 256), 24, True, 100, "pair"),
    ((512, 128), 200, False, 48, "wide"), ((128, 512), 7, False, 96, "wide"), ((256, 128), 24, True, 100, "wide"),
    ((512, 512), 24, True, 100, "wide"), ((256, 512), 256, True, 48, "wide"),
    ((256, 256, 256), 24, True, 100, "pair"), ((256, 256, 256), 64, False, 37, "pair"),
    ((256, 256, 256), 7, True, 5, "pair"), ((256, 256, 256), 24, True, 100, "generic")])
def test_wide_scorer_shapes(hidden, n_inst, wide_dims, n_req, kernel, monkeypatch):
    # the streamed-weight tensor-core scorers against the oracle: the pair
    # kernel (CTA pairs of 2-SM products, hidden widths multiples of 256) and
    # the one-CTA wide kernel (multiples of 128; pair shapes too when planned
    # with LS_TC_PAIR=0): tiles across request boundaries, one to four
    # layer-1 jobs, 64- and 128-column feature tiles, an odd number of tiles
    # (19: the last pair's second tile is past the batch) and a batch of one
    # tile; three hidden layers of 256 on the pair kernel (its second layer a
    # compaction job reading the first's activations in tensor memory) and on
    # the generic one-tile kernel
    import dataclasses
    if kernel in ("wide", "generic"):
        monkeypatch.setenv("LS_TC_PAIR", "0")
    base = W.CONFIGS["large" if wide_dims else "homogeneous"]
    cfg = dataclasses.replace(base, hidden=hidden, n_inst=n_inst, n_req=n_req, cache_blocks=1024, n_samples=0)
    wl = W.generate(cfg)
    r = H.Router.for_config(cfg)
    dw = H.DeviceWorkload(wl)
    dw.load(r)
    assert r.info().scorer == L.LS_SCORER_TENSOR_CORES
    assert r.info().tc_kernel == {"wide": L.LS_TC_WIDE, "pair": L.LS_TC_PAIR, "generic": L.LS_TC_GENERIC}[kernel]
    out = r.route(dw.tok, dw.tok_off, dw.req_feats, n_inst)
    ref = oracle.route(wl, bounds=True, threads=THREADS)
    assert np.array_equal(out["hits"].cpu().numpy(), ref["hits"])
    sg = out["scores"].cpu().numpy()
    assert_scores_close(sg, ref, TOL["bf16"], f"wide scorer {hidden} x {n_inst}")
    assert_choices(out["choice"].cpu().numpy(), sg, ref, TOL["bf16"])
    # a second route of the same batch gives the same bits (no state carried between launches)
    again = r.route(dw.tok, dw.tok_off, dw.req_feats, n_inst)
    assert torch.equal(again["scores"], out["scores"])
    assert r.sync() == L.LS_OK
    r.close()


def test_optional_outputs_do_not_change_the_result():
    wl, dw, r = staged("homogeneous")
    full = r.route(dw.tok, dw.tok_off, dw.req_feats, wl.cfg.n_inst)
    bare = r.route(dw.tok, dw.tok_off, dw.req_feats, wl.cfg.n_inst, want_scores=False, want_hits=False)
    assert torch.equal(full["choice"], bare["choice"]) and torch.equal(full["best"], bare["best"])


def test_instance_permutation_and_count_independence():
    # Sec. 4.1: one shared model, instance identity is never an input.
    wl, dw, r = staged("tiny")
    base = r.route(dw.tok, dw.tok_off, dw.req_feats, wl.cfg.n_inst)
    N = wl.cfg.n_inst
    perm = np.random.default_rng(4).permutation(N)
    ko = dw.inst_key_off.cpu().numpy()
    keys = [dw.inst_keys[ko[i]:ko[i + 1]] for i in range(N)]
    pk = torch.cat([keys[i] for i in perm])
    pko = torch.tensor(np.concatenate([[0], np.cumsum([len(keys[i]) for i in perm])]), device="cuda")
    r2 = H.Router.for_config(wl.cfg)
    r2.set_normalizer(dw.mean, dw.std)
    r2.snapshot(N, dw.inst_state[torch.from_numpy(perm).cuda()].contiguous(), pk, pko)
    r2.set_params(dw.params)
    r2.publish()
    out = r2.route(dw.tok, dw.tok_off, dw.req_feats, N)
    assert torch.equal(out["scores"], base["scores"][:, torch.from_numpy(perm).cuda()])
    assert torch.equal(out["hits"], base["hits"][:, torch.from_numpy(perm).cuda()])
    # fewer instances: the remaining instances' scores are unchanged
    keep = 3
    r2.snapshot(keep, dw.inst_state[:keep].contiguous(), torch.cat(keys[:keep]),
                torch.tensor(np.concatenate([[0], np.cumsum([len(k) for k in keys[:keep]])]), device="cuda"))
    out3 = r2.route(dw.tok, dw.tok_off, dw.req_feats, keep)
    assert torch.equal(out3["scores"], base["scores"][:, :keep])
    r2.close()


def test_edge_cases_empty_short_single_and_nan():
    wl, dw, r = staged("tiny")
    # empty batch
    out = r.route(dw.tok, dw.tok_off[:1], dw.req_feats[:0], wl.cfg.n_inst)
    assert out["choice"].numel() == 0
    # empty prompt, prompt shorter than a block, one request
    tok = torch.tensor([5, 6, 7], dtype=torch.int32, device="cuda")
    off = torch.tensor([0, 0, 3], dtype=torch.int64, device="cuda")
    out = r.route(tok, off, dw.req_feats[:2], wl.cfg.n_inst)
    assert (out["hits"] == 0).all()
    ref = oracle.features(np.array([0, 3]), np.zeros((2, wl.cfg.n_inst), np.int32), wl.inst_state,
                          wl.req_feats[:2], wl.mean, wl.std)
    y, eb, fl = oracle.mlp_forward_bounds("f32", wl.cfg.widths, wl.params, ref)
    assert_scores_close(out["scores"].cpu().numpy(),
                        {"scores": y.reshape(2, -1), "ebound": eb.reshape(2, -1), "flip": fl.reshape(2, -1)},
                        TOL["f32"], "empty and short prompts")
    # NaN predictions: every score NaN -> choice 0, best NaN
    p = dw.params.clone()
    p[-1] = float("nan")
    r.set_params(p)
    r.publish()
    out = r.route(dw.tok, dw.tok_off, dw.req_feats, wl.cfg.n_inst)
    assert (out["choice"] == 0).all() and torch.isnan(out["best"]).all()
    r.set_params(dw.params)
    r.publish()


def test_publish_versions_and_isolation():
    wl = W.generate("tiny")
    r = H.Router.for_config(wl.cfg)
    dw = H.DeviceWorkload(wl)
    dw.load(r, publish=False)
    rc, _ = L.ls_route_batch(r.h, 1, dw.tok, dw.tok_off, dw.req_feats,
                             torch.empty(1, dtype=torch.int32, device="cuda"),
                             torch.empty(1, device="cuda"))
    assert rc == L.LS_ERR_STATE
    r.publish()
    a = r.route(dw.tok, dw.tok_off, dw.req_feats, wl.cfg.n_inst)
    assert a["version"] == 1
    # new master weights are invisible until published
    p2 = dw.params * 0.5
    r.set_params(p2)
    b = r.route(dw.tok, dw.tok_off, dw.req_feats, wl.cfg.n_inst)
    assert b["version"] == 1 and torch.equal(a["scores"], b["scores"])
    r.publish()
    c = r.route(dw.tok, dw.tok_off, dw.req_feats, wl.cfg.n_inst)
    assert c["version"] == 2
    ref = oracle.route(wl, hits=c["hits"].cpu().numpy(), params=p2.cpu().numpy(), bounds=True)
    assert_scores_close(c["scores"].cpu().numpy(), ref, TOL["f32"], "after a publish")
    assert r.info().weight_version == 2
    r.close()


# ----------------------------------------------------------------------------
# training
# ----------------------------------------------------------------------------

def _weights_close(g, o, before, tol):
    """Post-step weights, and the step itself (w' - w) in norm."""
    g, o, before = (np.asarray(a, np.float64) for a in (g, o, before))
    assert np.all(np.abs(g - o) <= 1e-5 * np.maximum(np.abs(o), 1e-3) + np.abs(o - before) * tol * 4)
    dg, do = g - before, o - before
    assert np.linalg.norm(dg - do) <= tol * np.linalg.norm(do)


def test_train_sgd_tiny_fp32():
    wl, dw, r = staged("tiny")
    r.set_params(dw.params)
    x = torch.from_numpy(wl.samples_x).cuda()
    y = torch.from_numpy(wl.samples_y).cuda()
    r.log(x, y)
    loss = torch.zeros(1, device="cuda")
    n = wl.cfg.n_samples
    idx = torch.arange(n, dtype=torch.int32, device="cuda")
    r.train(n, idx, opt="sgd", lr=1e-3, loss_out=loss)
    got = r.get_params().cpu().numpy()
    tr = oracle.Trainer(wl.cfg.widths, wl.params, "f32")
    oloss = tr.step(wl.samples_x, wl.samples_y, np.arange(n, dtype=np.int32), wl.mean, wl.std, "sgd", 1e-3)
    assert abs(loss.item() - oloss) <= 1e-5 * oloss
    _weights_close(got, tr.params, wl.params, 1e-3)
    assert r.sync() == L.LS_OK
    r.set_params(dw.params)
    r.publish()


def _train_router(cfg, ring):
    return H.Router(cfg.widths, cfg.d_inst, cfg.d_req, cfg.dtype, max_instances=4, max_requests=16,
                    max_keys_per_instance=64, ring_capacity=ring, max_train_batch=4096)


@pytest.mark.parametrize("steps,batch", [(1, 4096), (10, 300)])
def test_train_adam_bf16(steps, batch):
    # Every step is compared from the GPU's own starting state (weights, Adam
    # moments, step count), so bf16 drift between the trajectories cannot hide
    # or fake a difference in the step itself.
    cfg = W.CONFIGS["training"]
    rng = np.random.default_rng(12)
    n = 20000
    x, y = W.records(rng, cfg, n)
    mean, std = W.normaliser(np.random.default_rng(13), cfg)
    params = W.xavier_params(cfg.widths, 0)
    r = _train_router(cfg, n)
    r.set_normalizer(torch.from_numpy(mean).cuda(), torch.from_numpy(std).cuda())
    r.set_params(torch.from_numpy(params).cuda())
    r.log(torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda())
    loss = torch.zeros(1, device="cuda")
    lr = 3e-4
    for k in range(steps):
        idx = W.minibatch_indices(4, k, n, batch)
        before = r.get_params().cpu().numpy()
        m0, v0, t0 = r.get_opt_state()
        r.train(batch, torch.from_numpy(idx).cuda(), opt="adam", lr=lr, loss_out=loss)
        after = r.get_params().cpu().numpy()
        m1, v1, t1 = r.get_opt_state()
        assert t1 == t0 + 1 == k + 1
        tr = oracle.Trainer(cfg.widths, before, "bf16")
        tr.m, tr.v, tr.t = m0.cpu().numpy().astype(np.float64), v0.cpu().numpy().astype(np.float64), t0
        g = oracle.Trainer(cfg.widths, before, "bf16").step(x, y, idx, mean, std, "sgd", 0.0,
                                                           want_grad=True)[1]
        ol = tr.step(x, y, idx, mean, std, "adam", lr)
        assert abs(loss.item() - ol) <= 2e-2 * ol
        dg, do = after - before.astype(np.float64), tr.params - before.astype(np.float64)
        # coordinates whose gradient is clear of bf16 noise and whose first
        # moment does not cancel (|m| at least a tenth of its new term)
        clear = (np.abs(g) > 0.05 * np.sqrt(np.mean(g ** 2))) & (np.abs(tr.m) > 0.01 * np.abs(g))
        assert clear.mean() > 0.5
        assert np.all(np.abs(dg - do)[clear] <= 0.1 * np.abs(do)[clear] + 0.05 * lr)
        assert np.mean(np.abs(dg - do)[clear] <= 0.02 * np.abs(do)[clear] + 0.01 * lr) > 0.99
        assert np.mean(np.sign(dg) == np.sign(do)) > 0.99
        # first moment: m1 - m0 = (1 - beta1) g, so it carries the gradient's tolerance
        mg, mo = m1.cpu().numpy().astype(np.float64), tr.m
        assert np.linalg.norm(mg - mo) <= 0.1 * 2e-2 * np.linalg.norm(g) + 1e-6 * np.linalg.norm(mo)
        assert np.abs(after - tr.params).max() <= 2.5 * lr
    assert r.sync() == L.LS_OK
    r.close()


@pytest.mark.parametrize("cfg_name,dropout", [("training", 0.0), ("homogeneous", 0.2)])
def test_persistent_train_step_same_bits(cfg_name, dropout):
    # The one-launch step (phases met at a grid barrier, the output layer's
    # 256 columns in one CTA) against one launch per phase: parameters, Adam
    # moments and loss equal bit for bit after several steps.
    cfg = W.CONFIGS[cfg_name]
    rng = np.random.default_rng(31)
    n = 9000
    x, y = W.records(rng, cfg, n)
    mean, std = W.normaliser(np.random.default_rng(32), cfg)
    params = W.xavier_params(cfg.widths, 5)
    out = []
    for tc in (-1, 24):
        r = H.Router(cfg.widths, cfg.d_inst, cfg.d_req, cfg.dtype, max_instances=4, max_requests=16,
                     max_keys_per_instance=64, ring_capacity=n, max_train_batch=4096, dropout=dropout,
                     dropout_seed=77, train_ctas=tc)
        r.set_normalizer(torch.from_numpy(mean).cuda(), torch.from_numpy(std).cuda())
        r.set_params(torch.from_numpy(params).cuda())
        r.log(torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda())
        loss = torch.zeros(1, device="cuda")
        losses = []
        for k, batch in enumerate((4096, 1000, 300)):
            idx = W.minibatch_indices(6, k, n, batch)
            r.train(batch, torch.from_numpy(idx).cuda(), opt="adam", lr=1e-3, loss_out=loss)
            losses.append(loss.item())
        r.train(2048, None, opt="adam", lr=1e-3, loss_out=loss)  # sequential slots
        losses.append(loss.item())
        m, v, t = r.get_opt_state()
        out.append((r.get_params().cpu(), m.cpu(), v.cpu(), t, losses))
        assert r.sync() == L.LS_OK
        r.close()
    (p0, m0, v0, t0, l0), (p1, m1, v1, t1, l1) = out
    assert t0 == t1 == 4 and l0 == l1
    assert torch.equal(p0, p1) and torch.equal(m0, m1) and torch.equal(v0, v1)


@pytest.mark.parametrize("cfg_name", ["tiny", "training"])
def test_train_on_empty_buffer_is_a_state_error(cfg_name):
    # Nothing logged yet: the call is refused with LS_ERR_STATE (tensor-core
    # path for the bf16 config, plain path for the fp32 one).  A step that
    # still finds the buffer empty on the device (records logged on another,
    # unordered stream) latches the same error and reads no record.
    cfg = W.CONFIGS[cfg_name]
    params = W.xavier_params(cfg.widths, 1)
    mean, std = W.normaliser(np.random.default_rng(2), cfg)
    r = _train_router(cfg, 1024)
    r.set_normalizer(torch.from_numpy(mean).cuda(), torch.from_numpy(std).cuda())
    r.set_params(torch.from_numpy(params).cuda())
    with pytest.raises(L.LodestarError) as e:
        r.train(256, None, opt="adam", lr=1e-3)
    assert e.value.code == L.LS_ERR_STATE
    assert r.sync() == L.LS_OK
    r.close()


def _train_state(r):
    m, v, t = r.get_opt_state()
    return r.get_params().cpu(), m.cpu(), v.cpu(), t


@pytest.mark.parametrize("cfg_name,train_ctas", [("tiny", 0), ("training", 0), ("training", 24)])
def test_step_that_finds_no_record_changes_nothing(cfg_name, train_ctas):
    # Records logged on a stream the training step is not ordered after: the
    # log waits behind a ~0.2 s spin on its own stream, so the step runs first
    # and finds the buffer empty on the device.  It latches LS_ERR_STATE, its
    # loss is NaN, and parameters, Adam moments and the step count are left as
    # they were (bit for bit); the next, ordered step then trains normally.
    cfg = W.CONFIGS[cfg_name]
    rng = np.random.default_rng(21)
    x, y = W.records(rng, cfg, 512)
    params = W.xavier_params(cfg.widths, 1)
    mean, std = W.normaliser(np.random.default_rng(2), cfg)
    r = H.Router(cfg.widths, cfg.d_inst, cfg.d_req, cfg.dtype, max_instances=4, max_requests=16,
                 max_keys_per_instance=64, ring_capacity=1024, max_train_batch=4096, train_ctas=train_ctas)
    r.set_normalizer(torch.from_numpy(mean).cuda(), torch.from_numpy(std).cuda())
    r.set_params(torch.from_numpy(params).cuda())
    xs, ys = torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda()
    # one Adam step on a second context's state would differ; take this one's
    # state after a first, ordered step so that the moments are nonzero
    r.log(xs[:256], ys[:256])
    loss = torch.zeros(1, device="cuda")
    r.train(256, None, opt="adam", lr=1e-3, loss_out=loss)
    assert r.sync() == L.LS_OK
    before = _train_state(r)
    r2 = H.Router(cfg.widths, cfg.d_inst, cfg.d_req, cfg.dtype, max_instances=4, max_requests=16,
                  max_keys_per_instance=64, ring_capacity=1024, max_train_batch=4096, train_ctas=train_ctas)
    r2.set_normalizer(torch.from_numpy(mean).cuda(), torch.from_numpy(std).cuda())
    r2.set_params(before[0].cuda())
    r2.set_opt_state(before[1].cuda(), before[2].cuda(), before[3])
    b2 = _train_state(r2)
    torch.cuda.synchronize()
    side, main = torch.cuda.Stream(), torch.cuda.Stream()
    with torch.cuda.stream(side):
        torch.cuda._sleep(400_000_000)          # ~0.2 s at 2 GHz, bounded
        r2.log(xs[256:], ys[256:], stream=side)
    r2.train(256, None, opt="adam", lr=1e-3, loss_out=loss, stream=main)
    main.synchronize()
    assert np.isnan(loss.item())
    assert r2.sync() == L.LS_ERR_STATE
    after = _train_state(r2)
    assert torch.equal(after[0], b2[0]) and torch.equal(after[1], b2[1]) and torch.equal(after[2], b2[2])
    assert after[3] == b2[3]
    # ordered now: the step trains and counts
    r2.train(256, None, opt="adam", lr=1e-3, loss_out=loss)
    assert np.isfinite(loss.item()) and r2.sync() == L.LS_OK
    assert _train_state(r2)[3] == b2[3] + 1 and not torch.equal(_train_state(r2)[0], b2[0])
    r.close()
    r2.close()


@pytest.mark.parametrize("cfg_name", ["tiny", "training"])
def test_step_with_bad_slot_changes_nothing(cfg_name):
    # A minibatch slot outside the filled buffer latches LS_ERR_ARG and the
    # step changes nothing (parameters, moments, step count; loss NaN).
    cfg = W.CONFIGS[cfg_name]
    x, y = W.records(np.random.default_rng(22), cfg, 300)
    mean, std = W.normaliser(np.random.default_rng(2), cfg)
    r = _train_router(cfg, 1024)
    r.set_normalizer(torch.from_numpy(mean).cuda(), torch.from_numpy(std).cuda())
    r.set_params(torch.from_numpy(W.xavier_params(cfg.widths, 3)).cuda())
    r.log(torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda())
    loss = torch.zeros(1, device="cuda")
    r.train(128, None, opt="adam", lr=1e-3, loss_out=loss)
    assert r.sync() == L.LS_OK
    before = _train_state(r)
    idx = np.arange(128, dtype=np.int32)
    idx[77] = 300                                   # one past the filled part
    r.train(128, torch.from_numpy(idx).cuda(), opt="adam", lr=1e-3, loss_out=loss)
    assert np.isnan(loss.item())
    assert r.sync() == L.LS_ERR_ARG
    after = _train_state(r)
    assert all(torch.equal(a, b) for a, b in zip(after[:3], before[:3])) and after[3] == before[3]
    r.close()


def test_train_gradient_bf16_via_sgd():
    # SGD with lr 0.1 exposes the bf16 gradient as (w - w') / 0.1.
    cfg = W.CONFIGS["training"]
    rng = np.random.default_rng(14)
    n = 4096
    x, y = W.records(rng, cfg, n)
    mean, std = W.normaliser(np.random.default_rng(15), cfg)
    params = W.xavier_params(cfg.widths, 0)
    r = _train_router(cfg, n)
    r.set_normalizer(torch.from_numpy(mean).cuda(), torch.from_numpy(std).cuda())
    r.set_params(torch.from_numpy(params).cuda())
    r.log(torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda())
    idx = W.minibatch_indices(4, 0, n, 4096)
    r.train(4096, torch.from_numpy(idx).cuda(), opt="sgd", lr=0.1)
    g_gpu = (params.astype(np.float64) - r.get_params().cpu().numpy()) / 0.1
    _, g_or = oracle.Trainer(cfg.widths, params, "bf16").step(x, y, idx, mean, std, "sgd", 0.0,
                                                              want_grad=True)
    assert np.linalg.norm(g_gpu - g_or) <= 2e-2 * np.linalg.norm(g_or)
    r.close()


def test_ring_wraparound_then_train():
    cfg = W.CONFIGS["tiny"]
    rng = np.random.default_rng(16)
    x, y = W.records(rng, cfg, 700)
    r = _train_router(cfg, 256)
    mean, std = W.normaliser(np.random.default_rng(17), cfg)
    params = W.xavier_params(cfg.widths, 0)
    r.set_normalizer(torch.from_numpy(mean).cuda(), torch.from_numpy(std).cuda())
    r.set_params(torch.from_numpy(params).cuda())
    ox, oy, count = np.zeros((256, cfg.d), np.float32), np.zeros(256, np.float32), 0
    for a, b in ((0, 100), (100, 350), (350, 700)):   # the last batch is longer than the ring
        r.log(torch.from_numpy(x[a:b]).cuda(), torch.from_numpy(y[a:b]).cuda())
        count = oracle.ring_append(ox, oy, count, x[a:b], y[a:b])
    assert r.info().ring_count == 700
    idx = np.arange(256, dtype=np.int32)
    loss = torch.zeros(1, device="cuda")
    r.train(256, torch.from_numpy(idx).cuda(), opt="sgd", lr=1e-3, loss_out=loss)
    tr = oracle.Trainer(cfg.widths, params, "f32")
    ol = tr.step(ox, oy, idx, mean, std, "sgd", 1e-3)
    assert abs(loss.item() - ol) <= 1e-5 * ol
    # sequential minibatch (idx = NULL): slots (k*B + j) mod count
    r.train(100, None, opt="sgd", lr=1e-3, loss_out=loss)
    ol2 = tr.step(ox, oy, (1 * 100 + np.arange(100)) % 256, mean, std, "sgd", 1e-3)
    assert abs(loss.item() - ol2) <= 1e-5 * ol2
    r.close()


# ----------------------------------------------------------------------------
# device-latched errors (no GPU fault involved)
# ----------------------------------------------------------------------------

def test_table_full_and_bad_slot_are_latched():
    cfg = W.CONFIGS["tiny"]
    r = H.Router(cfg.widths, cfg.d_inst, cfg.d_req, "f32", max_instances=2, max_requests=4,
                 max_keys_per_instance=100, ring_capacity=16, max_train_batch=16)
    keys = torch.arange(1, 151, dtype=torch.int64, device="cuda")
    off = torch.tensor([0, 150, 150], dtype=torch.int64, device="cuda")
    state = torch.zeros(2, cfg.d_inst, device="cuda")
    r.snapshot(2, state, keys, off)
    assert r.sync() == L.LS_ERR_TABLE_FULL
    assert r.sync() == L.LS_OK                       # cleared after reporting
    r.snapshot(2, state, keys[:100], torch.tensor([0, 100, 100], dtype=torch.int64, device="cuda"))
    assert r.sync() == L.LS_OK
    mean = torch.zeros(cfg.d, device="cuda")
    r.set_normalizer(mean, torch.ones(cfg.d, device="cuda"))
    r.set_params(torch.from_numpy(W.xavier_params(cfg.widths, 0)).cuda())
    r.log(torch.zeros(4, cfg.d, device="cuda"), torch.ones(4, device="cuda"))
    r.train(2, torch.tensor([1, 9], dtype=torch.int32, device="cuda"), opt="sgd", lr=0.0)
    assert r.sync() == L.LS_ERR_ARG
    r.close()


# ----------------------------------------------------------------------------
# a whole step captured in a CUDA graph; tracing
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("branches", [1, 2])
def test_graph_replay_matches_eager_steps(branches):
    # Two contexts fed the same inputs: one issues snapshot/route/log/train/
    # publish eagerly every step, the other replays one captured graph.  The
    # device counters make each replay a new step, so routes, losses, weights
    # and counters agree bit for bit.
    wl = W.generate("homogeneous")
    cfg = wl.cfg
    Bt = 512
    ctxs = []
    for _ in range(2):
        r = H.Router.for_config(cfg, ring_capacity=8 * Bt, max_train_batch=Bt)
        dw = H.DeviceWorkload(wl)
        dw.load(r)
        ctxs.append((r, dw))
    R, N = cfg.n_req, cfg.n_inst
    sx = torch.from_numpy(wl.samples_x[: 6 * Bt]).cuda()
    sy = torch.from_numpy(wl.samples_y[: 6 * Bt]).cuda()
    states = [ctxs[0][1].inst_state,
              torch.from_numpy(W.instance_state(np.random.default_rng(99), cfg)).cuda()]

    def make(r, dw):
        bufs = dict(state=torch.empty_like(states[0]), x=torch.empty(Bt, cfg.d, device="cuda"),
                    y=torch.empty(Bt, device="cuda"), loss=torch.zeros(1, device="cuda"),
                    out={"choice": torch.empty(R, dtype=torch.int32, device="cuda"),
                         "best": torch.empty(R, device="cuda"),
                         "scores": torch.empty(R, N, device="cuda"), "hits": None})

        def feed(k):
            bufs["state"].copy_(states[k & 1])
            a = (k * Bt) % len(sy)
            bufs["x"].copy_(sx[a:a + Bt])
            bufs["y"].copy_(sy[a:a + Bt])

        side = torch.cuda.Stream()

        def body():
            # branches == 2: log + train on a second stream beside the route,
            # joined before the publish
            main = torch.cuda.current_stream()
            side.wait_stream(main)
            r.snapshot(N, bufs["state"])
            r.route(dw.tok, dw.tok_off, dw.req_feats, N, out=bufs["out"])
            with torch.cuda.stream(side if branches == 2 else main):
                r.log(bufs["x"], bufs["y"])
                r.train(Bt, None, opt="adam", lr=1e-3, loss_out=bufs["loss"])
            main.wait_stream(side)
            r.publish()
        return bufs, feed, body

    (ra, dwa), (rb, dwb) = ctxs
    A, feed_a, body_a = make(ra, dwa)
    Bb, feed_b, body_b = make(rb, dwb)
    feed_a(0); body_a()
    feed_b(0); body_b()                     # eager warm-up step on both
    g = H.StepGraph(body_b)                 # recording runs nothing
    prev = ra.get_params().cpu().numpy()    # published at the end of step 0
    sample = np.arange(0, R, R // 8)
    for k in range(1, 6):
        feed_a(k); body_a()
        feed_b(k); g.replay()
        torch.cuda.synchronize()
        assert torch.equal(A["out"]["choice"], Bb["out"]["choice"])
        assert torch.equal(A["out"]["scores"], Bb["out"]["scores"])
        assert torch.equal(A["loss"], Bb["loss"])
        if k % 2 == 0:
            # step k routed with the weights published by step k - 1 and the
            # workload's own instance state
            ref = oracle.route(wl, params=prev, req_idx=sample, inst_keys=oracle_inst_keys("homogeneous", wl),
                               bounds=True)
            assert_scores_close(Bb["out"]["scores"].cpu().numpy()[sample], ref, TOL["bf16"], "graph replay")
        prev = ra.get_params().cpu().numpy()
    assert torch.equal(ra.get_params(), rb.get_params())
    ia, ib = ra.info(), rb.info()
    assert (ia.ring_count, ia.train_steps, ia.weight_version) == (6 * Bt, 6, 7)
    assert (ib.ring_count, ib.train_steps, ib.weight_version) == (6 * Bt, 6, 7)
    assert ra.sync() == L.LS_OK and rb.sync() == L.LS_OK
    ra.close(); rb.close()


def test_trace_counts_and_times_launches():
    wl, dw, r = staged("tiny")
    L.check(L.ls_trace_enable(r.h, True))
    L.ls_trace_read(r.h)
    for _ in range(3):
        r.route(dw.tok, dw.tok_off, dw.req_feats, wl.cfg.n_inst)
    rc, tr = L.ls_trace_read(r.h)
    L.check(L.ls_trace_enable(r.h, False))
    assert rc == L.LS_OK and tr
    for name, (launches, ms, timed) in tr.items():
        assert launches == timed == 3, (name, launches, timed)
        assert ms > 0.0
