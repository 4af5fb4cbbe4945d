"""Algorithm 4 guards on the GPU vs the CPU oracle, through the C ABI.

Bars: feature bounds bit-exact (as values: -0 == +0); statuses, choices and
best scores bit-exact against the oracle's guarded selection applied to the
GPU's own scores and hits (hits themselves are bit-exact against the oracle
in the prefix tests); cold-start and out-of-range statuses do not depend on
the predictor, so they also equal the oracle's from its own hits.
"""
import dataclasses

import numpy as np
import pytest
import torch

import oracle
from paper_2606_00946_gb300 import build as B
from paper_2606_00946_gb300 import harness as H
from paper_2606_00946_gb300 import lodestar as L
from paper_2606_00946_gb300 import workload as W

pytestmark = pytest.mark.gpu

KV_COL = 4          # instance-state column of KV-cache utilisation (workload layout)


@pytest.fixture(scope="module", autouse=True)
def _built():
    B.build()


def _cfg(name, **kw):
    return dataclasses.replace(W.CONFIGS[name], **kw) if kw else W.CONFIGS[name]


def _staged(cfg, ring):
    wl = W.generate(cfg, with_samples=False)
    r = H.Router.for_config(cfg, ring_capacity=ring)
    dw = H.DeviceWorkload(wl)
    dw.load(r)
    return wl, dw, r


def _log(r, ox, oy, count, x, y):
    r.log(torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda())
    return oracle.ring_append(ox, oy, count, x, y)


def _oracle_guards(wl, out, lo, hi, n, g):
    return oracle.guards(np.diff(wl.tok_off), oracle.group_keys(wl.tok, wl.tok_off),
                         out["hits"].cpu().numpy(), wl.inst_state, wl.req_feats,
                         out["scores"].cpu().numpy(), lo, hi, n, n_min=g["n_min"], ood=g["ood"],
                         k=g["k"], kv_col=g["kv_col"], tau_sat=g["tau_sat"], tau_ben=g["tau_ben"])


def _assert_same(out, want):
    ch, best, st = want
    np.testing.assert_array_equal(out["status"].cpu().numpy(), st)
    np.testing.assert_array_equal(out["choice"].cpu().numpy(), ch)
    np.testing.assert_array_equal(out["best"].cpu().numpy(), best)   # NaN == NaN here


# ----------------------------------------------------------------------------
# feature bounds of the sample ring
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("name,d_req,cap,batches", [
    ("tiny", 0, 256, [100, 250, 400]),       # d = 16, the last batch longer than the ring
    ("tiny", 5, 300, [7, 120]),              # d = 21: 12 rows per pass, 4 threads idle
    ("tiny", 300, 200, [150, 90]),           # d = 316 > 256: columns strided by the block
    ("homogeneous", 24, 65536, [65536, 4096]),
])
def test_ring_bounds_parity(name, d_req, cap, batches):
    cfg = _cfg(name, d_req=d_req, n_samples=0)
    wl, dw, r = _staged(cfg, cap)
    lo0, hi0 = r.bounds(which=0)                       # nothing logged: the empty range
    assert torch.isinf(lo0).all() and (lo0 > 0).all() and torch.isinf(hi0).all() and (hi0 < 0).all()
    rng = np.random.default_rng(cap + d_req)
    ox, oy, count = np.zeros((cap, cfg.d), np.float32), np.zeros(cap, np.float32), 0
    for n in batches:
        x, y = W.records(rng, cfg, n)
        x[rng.random(x.shape) < 0.01] = np.nan
        x[rng.random(x.shape) < 0.01] *= -0.0           # signed zeros
        count = _log(r, ox, oy, count, x, y)
        r.refresh_bounds()
        lo, hi = r.bounds(which=0)
        wlo, whi = oracle.ring_bounds(ox, count)
        np.testing.assert_array_equal(lo.cpu().numpy(), wlo)
        np.testing.assert_array_equal(hi.cpu().numpy(), whi)
    # the publish carries the staged bounds to routing
    r.publish()
    plo, phi = r.bounds(which=1)
    assert torch.equal(plo, lo) and torch.equal(phi, hi)
    r.close()


# ----------------------------------------------------------------------------
# guarded route
# ----------------------------------------------------------------------------

def _guard_case(cfg, n_records, g, seed=21, bad_req=()):
    wl, dw, r = _staged(cfg, max(n_records, 1024))
    if bad_req and cfg.d_req:       # request extras far outside anything logged
        wl.req_feats[list(bad_req), 0] = 1e6
        dw.req_feats.copy_(torch.from_numpy(wl.req_feats))
    ox = np.zeros((max(n_records, 1024), cfg.d), np.float32)
    oy = np.zeros(len(ox), np.float32)
    x, y = W.records(np.random.default_rng(seed), cfg, n_records)
    # the buffer holds records of the current instance states (requests routed
    # to them earlier), so the snapshot itself lies inside the bounds
    x[:cfg.n_inst, 6:6 + cfg.d_inst] = wl.inst_state
    count = _log(r, ox, oy, 0, x, y)
    r.refresh_bounds()
    r.publish()
    lo, hi = oracle.ring_bounds(ox, count)
    r.set_guards(**g)
    out = r.route_guarded(dw.tok, dw.tok_off, dw.req_feats, cfg.n_inst)
    return wl, dw, r, out, lo, hi, count


CASES = [
    # name, overrides, records
    ("tiny", {}, 256),
    ("homogeneous", {}, 65536),
    ("homogeneous", {"n_inst": 24, "n_req": 512, "cache_blocks": 1024}, 8192),
    ("homogeneous", {"n_inst": 40, "n_req": 512, "cache_blocks": 1024}, 8192),
    ("homogeneous", {"n_inst": 7, "n_req": 300, "cache_blocks": 1024}, 8192),
]


@pytest.mark.parametrize("name,over,n_rec", CASES)
def test_guarded_route_parity(name, over, n_rec):
    cfg = _cfg(name, n_samples=0, **over)
    g = dict(n_min=1, ood=True, k=2, kv_col=KV_COL, tau_sat=0.3, tau_ben=0.0)
    wl, dw, r, out, lo, hi, count = _guard_case(cfg, n_rec, g, bad_req=(1, 5))
    want = _oracle_guards(wl, out, lo, hi, count, g)
    _assert_same(out, want)
    st = want[2]
    assert (st == L.LS_ROUTE_KFILTER).any()
    if cfg.d_req:
        assert st[1] == st[5] == L.LS_ROUTE_OOD
    # the filter moved some choices away from the plain argmin
    plain, _ = oracle.argmin(out["scores"].cpu().numpy())
    ok = st == L.LS_ROUTE_KFILTER
    if cfg.n_inst > 2:
        assert (out["choice"].cpu().numpy()[ok] != plain[ok]).any()
    # cold-start and out-of-range statuses equal the oracle's from its own hits
    rk, rko = oracle.hash_blocks(wl.tok, wl.tok_off)
    ohits = oracle.prefix_hits(rk, rko, *oracle.instance_keys(wl))
    assert np.array_equal(out["hits"].cpu().numpy(), ohits)
    # one instance value outside the bounds puts every request out of range
    st2 = wl.inst_state.copy()
    st2[cfg.n_inst - 1, cfg.d_inst - 1] = -1e6
    r.snapshot(cfg.n_inst, torch.from_numpy(st2).cuda())
    out2 = r.route_guarded(dw.tok, dw.tok_off, dw.req_feats, cfg.n_inst)
    wl2 = dataclasses.replace(wl, inst_state=st2)
    _assert_same(out2, _oracle_guards(wl2, out2, lo, hi, count, g))
    assert (out2["status"] == L.LS_ROUTE_OOD).all()
    r.close()


def test_guard_thresholds_and_cold_start():
    cfg = _cfg("homogeneous", n_samples=0, n_inst=32, n_req=512, cache_blocks=1024)
    g = dict(n_min=0, ood=False, k=2, kv_col=KV_COL, tau_sat=0.3, tau_ben=0.0)
    wl, dw, r, out, lo, hi, count = _guard_case(cfg, 4096, g)
    hits = out["hits"].cpu().numpy()
    # tau_ben at the median hit-token count: about half the requests filtered
    hmax16 = 16.0 * hits.max(axis=1)
    for tau_ben in (float(np.median(hmax16)), -1.0, 1e9):
        g2 = dict(g, tau_ben=tau_ben)
        r.set_guards(**g2)
        out = r.route_guarded(dw.tok, dw.tok_off, dw.req_feats, cfg.n_inst)
        _assert_same(out, _oracle_guards(wl, out, lo, hi, count, g2))
    # the gpu_kv mean exactly at tau_sat does not filter (strict >)
    kv = wl.inst_state[:, KV_COL].astype(np.float64)
    mean = np.float32(kv.sum() / len(kv))
    for ts in (float(mean), float(np.nextafter(mean, np.float32(-1))), 0.8):
        g2 = dict(g, tau_sat=ts)
        r.set_guards(**g2)
        out = r.route_guarded(dw.tok, dw.tok_off, dw.req_feats, cfg.n_inst)
        _assert_same(out, _oracle_guards(wl, out, lo, hi, count, g2))
    # cold start: the device count when the route runs decides
    g2 = dict(g, n_min=count + 10)
    r.set_guards(**g2)
    out = r.route_guarded(dw.tok, dw.tok_off, dw.req_feats, cfg.n_inst)
    st = out["status"].cpu().numpy()
    assert (st == L.LS_ROUTE_COLD_START).all() and (out["choice"].cpu().numpy() == -1).all()
    assert torch.isnan(out["best"]).all()
    x, y = W.records(np.random.default_rng(3), cfg, 10)
    r.log(torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda())
    out = r.route_guarded(dw.tok, dw.tok_off, dw.req_feats, cfg.n_inst)
    assert (out["status"].cpu().numpy() != L.LS_ROUTE_COLD_START).all()
    r.close()


def test_guards_off_equal_the_plain_route():
    cfg = _cfg("homogeneous", n_samples=0)
    wl, dw, r, out, lo, hi, count = _guard_case(cfg, 2048, dict(n_min=0, ood=False, k=0, kv_col=0,
                                                                 tau_sat=0.8, tau_ben=0.0))
    plain = r.route(dw.tok, dw.tok_off, dw.req_feats, cfg.n_inst)       # fused selector path
    assert (out["status"] == 0).all()
    assert torch.equal(out["choice"], plain["choice"]) and torch.equal(out["best"], plain["best"])
    assert torch.equal(out["scores"], plain["scores"]) and torch.equal(out["hits"], plain["hits"])
    r.close()


def test_out_of_range_empty_bounds_and_edge_prompts():
    cfg = _cfg("tiny", n_samples=0)
    wl, dw, r = _staged(cfg, 1024)
    # no refresh yet: the published bounds are the empty range -> all out of range
    r.set_guards(n_min=0, ood=True, k=2, kv_col=KV_COL, tau_sat=-1.0, tau_ben=-1.0)
    out = r.route_guarded(dw.tok, dw.tok_off, dw.req_feats, cfg.n_inst)
    assert (out["status"] == L.LS_ROUTE_OOD).all()
    # guards without the range check on empty, short and single-block prompts:
    # the filter needs a full block (a prefix group key)
    r.set_guards(n_min=0, ood=False, k=2, kv_col=KV_COL, tau_sat=-1.0, tau_ben=-1.0)
    tok = torch.tensor(list(range(40)), dtype=torch.int32, device="cuda")
    off = torch.tensor([0, 0, 3, 19, 40], dtype=torch.int64, device="cuda")
    rf = dw.req_feats[:4].contiguous()
    out = r.route_guarded(tok, off, rf, cfg.n_inst)
    wl2 = dataclasses.replace(wl, tok=tok.cpu().numpy(), tok_off=off.cpu().numpy(),
                              req_feats=rf.cpu().numpy())
    lo, hi = oracle.ring_bounds(np.zeros((1, cfg.d), np.float32), 0)
    g = dict(n_min=0, ood=False, k=2, kv_col=KV_COL, tau_sat=-1.0, tau_ben=-1.0)
    _assert_same(out, _oracle_guards(wl2, out, lo, hi, 0, g))
    st = out["status"].cpu().numpy()
    assert st[0] == st[1] == 0 and st[2] == st[3] == L.LS_ROUTE_KFILTER
    # empty batch
    e = r.route_guarded(dw.tok, dw.tok_off[:1], dw.req_feats[:0], cfg.n_inst)
    assert e["status"].numel() == 0
    r.close()


def test_set_guards_rejects_bad_arguments():
    cfg = _cfg("tiny", n_samples=0)
    r = H.Router.for_config(cfg)
    assert L.ls_set_guards(r.h, k=-1) == L.LS_ERR_ARG
    assert L.ls_set_guards(r.h, k=cfg.n_inst + 1) == L.LS_ERR_ARG
    assert L.ls_set_guards(r.h, k=2, kv_col=cfg.d_inst) == L.LS_ERR_ARG
    assert L.ls_set_guards(r.h, k=2, kv_col=KV_COL) == L.LS_OK
    r.close()


# ----------------------------------------------------------------------------
# fallback heuristics (Algorithms 1 and 2, pre-computed as Algorithm 3 does)
# ----------------------------------------------------------------------------

HEUR_CASES = [
    ("tiny", {}),
    ("homogeneous", {}),
    ("homogeneous", {"n_inst": 24, "n_req": 512, "cache_blocks": 1024}),
    ("homogeneous", {"n_inst": 40, "n_req": 512, "cache_blocks": 1024}),
    ("homogeneous", {"n_inst": 7, "n_req": 300, "cache_blocks": 1024}),
]


@pytest.mark.parametrize("name,over", HEUR_CASES)
def test_fallback_heuristic_parity(name, over):
    cfg = _cfg(name, n_samples=0, **over)
    g = dict(n_min=1, ood=True, k=2, kv_col=KV_COL, tau_sat=0.3, tau_ben=0.0)
    wl, dw, r, out, lo, hi, count = _guard_case(cfg, 4096, g)
    L_ = np.diff(wl.tok_off)
    c = wl.inst_state[:, 0] + wl.inst_state[:, 1]
    spread = float(c.max() - c.min())
    settings = [
        dict(heuristic=1, count_cols=(0, 1), theta_imbal=spread + 1.0, k_overload=1.0),   # balanced
        dict(heuristic=1, count_cols=(0, 1), theta_imbal=spread + 1.0, k_overload=-0.5),
        dict(heuristic=1, count_cols=(0, 1), theta_imbal=spread - 0.5, k_overload=1.0),   # imbalanced
        dict(heuristic=1, count_cols=(1, -1), theta_imbal=1e9, k_overload=0.0),
        dict(heuristic=2, count_cols=(0, 1), tau_prefix=0.5),
        dict(heuristic=2, count_cols=(0, -1), tau_prefix=0.05),
    ]
    picks = set()
    for hs in settings:
        r.set_guards(**g, **hs)
        got = r.route_guarded(dw.tok, dw.tok_off, dw.req_feats, cfg.n_inst)
        want = oracle.heuristic(L_, got["hits"].cpu().numpy(), wl.inst_state, mode=hs["heuristic"],
                                count_cols=hs["count_cols"], theta_imbal=hs.get("theta_imbal", 8.0),
                                k=hs.get("k_overload", 1.0), tau=hs.get("tau_prefix", 0.5))
        np.testing.assert_array_equal(got["fallback"].cpu().numpy(), want)
        # the guarded selection itself is unchanged by the heuristic
        _assert_same(got, _oracle_guards(wl, got, lo, hi, count, g))
        picks.add(len(np.unique(want)))
    assert max(picks) > 1                              # some setting spreads the requests
    # cold batch: the heuristic is still formed for every request
    r.set_guards(**dict(g, n_min=count + 1), **settings[0])
    got = r.route_guarded(dw.tok, dw.tok_off, dw.req_feats, cfg.n_inst)
    assert (got["status"] == L.LS_ROUTE_COLD_START).all()
    want = oracle.heuristic(L_, got["hits"].cpu().numpy(), wl.inst_state, mode=1, count_cols=(0, 1),
                            theta_imbal=spread + 1.0, k=1.0)
    np.testing.assert_array_equal(got["fallback"].cpu().numpy(), want)
    r.close()


def test_fallback_heuristic_nan_counts_and_bad_arguments():
    cfg = _cfg("tiny", n_samples=0)
    wl, dw, r = _staged(cfg, 1024)
    st = wl.inst_state.copy()
    st[0, 0] = np.nan                                  # NaN count: never least loaded, never eligible
    st[3, 0] = st[5, 0] = 0.0
    st[3, 1] = st[5, 1] = 0.0
    r.snapshot(cfg.n_inst, torch.from_numpy(st).cuda())
    L_ = np.diff(wl.tok_off)
    for hs in (dict(heuristic=1, theta_imbal=1e9, k_overload=1.0), dict(heuristic=1, theta_imbal=0.0),
               dict(heuristic=2, tau_prefix=0.99)):
        r.set_guards(**hs)
        got = r.route_guarded(dw.tok, dw.tok_off, dw.req_feats, cfg.n_inst)
        want = oracle.heuristic(L_, got["hits"].cpu().numpy(), st, mode=hs["heuristic"],
                                theta_imbal=hs.get("theta_imbal", 8.0), k=hs.get("k_overload", 1.0),
                                tau=hs.get("tau_prefix", 0.5))
        np.testing.assert_array_equal(got["fallback"].cpu().numpy(), want)
    assert L.ls_set_guards(r.h, heuristic=3) == L.LS_ERR_ARG
    assert L.ls_set_guards(r.h, heuristic=1, count_cols=(cfg.d_inst, -1)) == L.LS_ERR_ARG
    assert L.ls_set_guards(r.h, heuristic=1, count_cols=(0, -2)) == L.LS_ERR_ARG
    r.close()


def test_fp64_decisions_at_their_bounds():
    # Decisions the fp64 reading takes differently from fp32 arithmetic: the
    # kernel's fp32 statistics find these within their error bound and take
    # the fp64 path, so every status and fallback equals the oracle's.
    cfg = _cfg("tiny", n_samples=0)
    wl, dw, r = _staged(cfg, 1024)
    N, L_ = cfg.n_inst, np.diff(wl.tok_off)
    g = dict(n_min=0, ood=False, k=2, kv_col=KV_COL, tau_ben=-1.0)
    base = wl.inst_state.copy()

    def run(st, **hs):
        r.snapshot(N, torch.from_numpy(st).cuda())
        r.set_guards(**g, **hs)
        out = r.route_guarded(dw.tok, dw.tok_off, dw.req_feats, N)
        want = oracle.guards(L_, oracle.group_keys(wl.tok, wl.tok_off), out["hits"].cpu().numpy(), st,
                             wl.req_feats, out["scores"].cpu().numpy(), np.full(cfg.d, -np.inf, np.float32),
                             np.full(cfg.d, np.inf, np.float32), 0, n_min=0, ood=False, k=2, kv_col=KV_COL,
                             tau_sat=hs["tau_sat"], tau_ben=-1.0)
        _assert_same(out, want)
        fb = out["fallback"].cpu().numpy()
        if hs.get("heuristic", 0):
            np.testing.assert_array_equal(fb, oracle.heuristic(
                L_, out["hits"].cpu().numpy(), st, mode=hs["heuristic"], count_cols=hs["count_cols"],
                theta_imbal=hs["theta_imbal"], k=hs["k_overload"]))
        return out["status"].cpu().numpy(), fb

    # K-filter: mean of kv = 0.5 + 2^-27 > 0.5 in fp64 (an fp32 sum gives 0.5)
    st = base.copy()
    st[:, KV_COL] = 0.5
    st[1, KV_COL] = 0.5 + 2.0 ** -24
    status, _ = run(st, tau_sat=0.5)
    has_block = L_ >= 16
    assert (status[has_block] == L.LS_ROUTE_KFILTER).all()
    st[1, KV_COL] = 0.5
    status, _ = run(st, tau_sat=0.5)
    assert (status == 0).all()
    # Algorithm 1: mu + k sigma = 3 exactly (k = 1) and 3 - 2^-24 (k one fp32 ulp below 1)
    st = base.copy()
    st[:, 0] = [1, 1, 3, 3, 1, 1, 3, 3]
    st[:, 1] = 0
    for k in (1.0, float(np.nextafter(np.float32(1.0), np.float32(0)))):
        _, fb = run(st, tau_sat=2.0, heuristic=1, count_cols=(0, 1), theta_imbal=99.0, k_overload=k)
        if k < 1.0:
            assert np.isin(fb, [0, 1, 4, 5]).all()       # the count-3 instances are overloaded
    # counts 2^24 + delta, distinct only in fp64; spread 3 against theta 2.5 / 3.5
    st[:, 0] = 2.0 ** 24
    st[:, 1] = [1, 0, 3, 2, 1, 0, 2, 3]
    for theta, k in ((2.5, 9.0), (3.5, 9.0), (3.5, -9.0), (3.5, 0.0)):
        run(st, tau_sat=2.0, heuristic=1, count_cols=(0, 1), theta_imbal=theta, k_overload=k)
    _, fb = run(st, tau_sat=2.0, heuristic=1, count_cols=(0, 1), theta_imbal=2.5, k_overload=9.0)
    assert (fb == 1).all()                               # imbalanced: the least loaded, lowest index
    r.close()
