"""Pins of the oracle's Algorithm 4 guards (cold start, out-of-range
features, consistent-hashing K-filter) against facts that do not come from
the oracle: numpy's NaN-aware reductions, exhaustive enumeration over the
candidates, exact threshold boundaries, and the defining properties of
consistent hashing (exactly K distinct candidates, nesting in K, stability
when an instance leaves, balance over keys).  No GPU needed.
"""
import warnings

import numpy as np
import pytest

import oracle

BLOCK = 16


def _raw_rows(L, hits, inst, req):
    """Raw feature rows of every (r, i) pair written out from the feature
    list of Sec. 4.1: L, h, 16h, 16h/L, L-16h, ceil(L/16)-h, then the
    instance row and the request extras (fp32, as the router forms them)."""
    R, N = hits.shape
    rows = np.zeros((R, N, 6 + inst.shape[1] + req.shape[1]), np.float32)
    for r in range(R):
        for i in range(N):
            h = int(hits[r, i])
            Lf = np.float32(L[r])
            ht = np.float32(BLOCK * h)
            rows[r, i, 0] = Lf
            rows[r, i, 1] = np.float32(h)
            rows[r, i, 2] = ht
            rows[r, i, 3] = ht / Lf if L[r] > 0 else np.float32(0)
            rows[r, i, 4] = np.float32(L[r] - BLOCK * h)
            rows[r, i, 5] = np.float32(-(-L[r] // BLOCK) - h)
            rows[r, i, 6:6 + inst.shape[1]] = inst[i]
            rows[r, i, 6 + inst.shape[1]:] = req[r]
    return rows


def _setting(seed=0, R=6, N=5, d_inst=3, d_req=2):
    rng = np.random.default_rng(seed)
    L = rng.integers(20, 200, size=R).astype(np.int64)
    hits = np.stack([rng.integers(0, L[r] // BLOCK + 1, size=N) for r in range(R)]).astype(np.int32)
    inst = rng.standard_normal((N, d_inst)).astype(np.float32)
    req = rng.standard_normal((R, d_req)).astype(np.float32)
    scores = rng.standard_normal((R, N)).astype(np.float32)
    gkey = rng.integers(1, 2**63, size=R, dtype=np.int64).astype(np.uint64)
    return L, gkey, hits, inst, req, scores


def _first_argmin(row):
    # numpy's argmin returns the first index of the minimum
    return int(np.argmin(row))


# ----------------------------------------------------------------------------
# feature bounds of the training buffer
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("count", [0, 1, 13, 50, 123])
def test_ring_bounds_are_nan_skipping_min_max_of_held_rows(count):
    cap, d = 50, 7
    rng = np.random.default_rng(count)
    ring = rng.standard_normal((cap, d)).astype(np.float32) * 10
    ring[rng.random((cap, d)) < 0.1] = np.nan
    ring[:, 6] = np.nan                       # a column with no number at all
    held = min(count, cap)
    if held < cap:                            # slots not yet written must not count
        ring[held:, :6] = 1e30
    lo, hi = oracle.ring_bounds(ring, count)
    with warnings.catch_warnings():
        warnings.simplefilter("ignore", RuntimeWarning)      # the all-NaN column
        want_lo = np.nanmin(ring[:held], axis=0) if held else np.full(d, np.inf, np.float32)
        want_hi = np.nanmax(ring[:held], axis=0) if held else np.full(d, -np.inf, np.float32)
    want_lo = np.where(np.isnan(want_lo), np.inf, want_lo)
    want_hi = np.where(np.isnan(want_hi), -np.inf, want_hi)
    np.testing.assert_array_equal(lo, want_lo.astype(np.float32))
    np.testing.assert_array_equal(hi, want_hi.astype(np.float32))


# ----------------------------------------------------------------------------
# cold start and out-of-range guards
# ----------------------------------------------------------------------------

def _wide(d):
    return np.full(d, -np.inf, np.float32), np.full(d, np.inf, np.float32)


def test_without_guards_the_choice_is_the_plain_argmin():
    L, g, hits, inst, req, scores = _setting(1)
    scores[2, 3] = scores[2, 1] = scores[2].min() - 1   # tie: lowest index wins
    lo, hi = _wide(11)
    ch, best, st = oracle.guards(L, g, hits, inst, req, scores, lo, hi, n=0)
    assert (st == 0).all()
    assert ch.tolist() == [_first_argmin(s) for s in scores]
    np.testing.assert_array_equal(best, scores[np.arange(len(ch)), ch])


def test_cold_start_is_n_strictly_below_n_min():
    L, g, hits, inst, req, scores = _setting(2)
    lo, hi = _wide(11)
    ch, best, st = oracle.guards(L, g, hits, inst, req, scores, lo, hi, n=99, n_min=100)
    assert (st == oracle.ROUTE_COLD_START).all() and (ch == -1).all() and np.isnan(best).all()
    ch, best, st = oracle.guards(L, g, hits, inst, req, scores, lo, hi, n=100, n_min=100)
    assert (st == 0).all() and ch.tolist() == [_first_argmin(s) for s in scores]


def test_out_of_range_checks_every_column_with_inclusive_bounds():
    L, g, hits, inst, req, scores = _setting(3)
    rows = _raw_rows(L, hits, inst, req)               # [R, N, d]
    lo, hi = rows.min(axis=(0, 1)), rows.max(axis=(0, 1))
    ch, best, st = oracle.guards(L, g, hits, inst, req, scores, lo, hi, n=1, ood=True)
    assert (st == 0).all()                             # the observed extremes are inside
    d = rows.shape[2]
    for j in range(d):
        for side in ("lo", "hi"):
            l2, h2 = lo.copy(), hi.copy()
            if side == "lo":
                l2[j] = np.nextafter(lo[j], np.float32(np.inf))
                bad = (rows[:, :, j] < l2[j]).any(axis=1)
            else:
                h2[j] = np.nextafter(hi[j], np.float32(-np.inf))
                bad = (rows[:, :, j] > h2[j]).any(axis=1)
            ch, best, st = oracle.guards(L, g, hits, inst, req, scores, l2, h2, n=1, ood=True)
            assert bad.any()
            assert (st == np.where(bad, oracle.ROUTE_OOD, 0)).all(), (j, side)
            assert (ch[bad] == -1).all() and np.isnan(best[bad]).all()
            assert ch[~bad].tolist() == [_first_argmin(s) for s in scores[~bad]]


def test_out_of_range_nan_feature_and_empty_bounds():
    L, g, hits, inst, req, scores = _setting(4)
    lo, hi = _wide(11)
    req = req.copy()
    req[3, 1] = np.nan
    _, _, st = oracle.guards(L, g, hits, inst, req, scores, lo, hi, n=1, ood=True)
    assert st.tolist() == [0, 0, 0, 2, 0, 0]
    elo, ehi = oracle.ring_bounds(np.zeros((4, 11), np.float32), 0)   # empty buffer
    _, _, st = oracle.guards(L, g, hits, inst, req, scores, elo, ehi, n=1, ood=True)
    assert (st == oracle.ROUTE_OOD).all()


def test_cold_start_is_tested_before_out_of_range():
    L, g, hits, inst, req, scores = _setting(5)
    elo, ehi = np.full(11, np.inf, np.float32), np.full(11, -np.inf, np.float32)
    _, _, st = oracle.guards(L, g, hits, inst, req, scores, elo, ehi, n=0, n_min=1, ood=True)
    assert (st == oracle.ROUTE_COLD_START).all()


# ----------------------------------------------------------------------------
# consistent hashing (rendezvous) candidates
# ----------------------------------------------------------------------------

def test_hrw_gives_min_k_n_distinct_instances_nested_in_k():
    rng = np.random.default_rng(6)
    for _ in range(200):
        g = int(rng.integers(0, 2**63)) * 2 + int(rng.integers(0, 2))
        N = int(rng.integers(1, 40))
        prev = []
        for K in range(0, N + 3):
            c = oracle.hrw_candidates(g, N, K).tolist()
            assert len(c) == min(K, N) and len(set(c)) == len(c)
            assert all(0 <= i < N for i in c)
            assert c[:len(prev)] == prev               # C_K is a prefix of C_{K+1}
            prev = c


def test_hrw_is_stable_when_an_instance_leaves():
    # consistent hashing: removing an instance moves only the keys it held
    rng = np.random.default_rng(7)
    N, K = 16, 2
    moved = 0
    for _ in range(2000):
        g = int(rng.integers(0, 2**63))
        full = oracle.hrw_candidates(g, N, K).tolist()
        less = oracle.hrw_candidates(g, N - 1, K).tolist()
        if N - 1 not in full:
            assert less == full
        else:
            moved += 1
            kept = [i for i in full if i != N - 1]
            assert less[:len(kept)] == kept and len(less) == K
    assert 2000 * K / N * 0.7 < moved < 2000 * K / N * 1.3


def test_hrw_spreads_keys_evenly():
    rng = np.random.default_rng(8)
    N, K, n = 16, 2, 20000
    cnt = np.zeros(N)
    for _ in range(n):
        for i in oracle.hrw_candidates(int(rng.integers(0, 2**63)), N, K):
            cnt[i] += 1
    exp = n * K / N
    assert np.abs(cnt - exp).max() < 0.1 * exp         # ~5 binomial sigmas


def test_group_key_is_the_first_block_key():
    rng = np.random.default_rng(9)
    head = rng.integers(0, 32000, 16).astype(np.int32)
    a = np.concatenate([head, rng.integers(0, 32000, 40).astype(np.int32)])
    b = np.concatenate([head, rng.integers(0, 32000, 7).astype(np.int32)])
    c = rng.integers(0, 32000, 30).astype(np.int32)
    short = rng.integers(0, 32000, 15).astype(np.int32)
    seqs = [a, b, c, short]
    off = np.zeros(5, np.int64)
    off[1:] = np.cumsum([len(s) for s in seqs])
    gk = oracle.group_keys(np.concatenate(seqs), off)
    keys, ko = oracle.hash_blocks(head, np.array([0, 16]))
    assert gk[0] == gk[1] == keys[0] and gk[2] != gk[0] and gk[3] == 0


# ----------------------------------------------------------------------------
# K-filter
# ----------------------------------------------------------------------------

def _kv_setting(seed, R=40, N=12, kv=0.9):
    rng = np.random.default_rng(seed)
    L = rng.integers(16, 300, size=R).astype(np.int64)
    hits = np.stack([rng.integers(0, L[r] // BLOCK + 1, size=N) for r in range(R)]).astype(np.int32)
    inst = rng.standard_normal((N, 6)).astype(np.float32)
    inst[:, 4] = kv
    req = np.zeros((R, 0), np.float32)
    scores = rng.standard_normal((R, N)).astype(np.float32)
    g = rng.integers(1, 2**63, size=R, dtype=np.int64).astype(np.uint64)
    return L, g, hits, inst, req, scores


def test_kfilter_moves_the_choice_into_the_candidates():
    L, g, hits, inst, req, scores = _kv_setting(10)
    hits[:, 0] = np.maximum(hits[:, 0], 1)              # every prompt has a hit
    lo, hi = _wide(12)
    ch, best, st = oracle.guards(L, g, hits, inst, req, scores, lo, hi, n=1, k=2, kv_col=4,
                                 tau_sat=0.8, tau_ben=0.0)
    changed = 0
    for r in range(len(L)):
        cand = oracle.hrw_candidates(int(g[r]), scores.shape[1], 2).tolist()
        top = _first_argmin(scores[r])
        assert st[r] == oracle.ROUTE_KFILTER
        if top in cand:
            assert ch[r] == top
        else:
            # exhaustive: the smallest score among the candidates, lowest index on ties
            want = min(cand, key=lambda i: (scores[r, i], i))
            assert ch[r] == want
            changed += 1
        assert best[r] == scores[r, ch[r]]
    assert changed > len(L) // 2


def test_kfilter_thresholds_are_strict():
    L, g, hits, inst, req, scores = _kv_setting(11, N=4)
    inst[:, 4] = [0.5, 1.0, 0.75, 0.75]                 # mean exactly 0.75
    hits[:] = 0
    hits[:, 2] = 3                                      # max hit tokens = 48
    L[:] = 100
    lo, hi = _wide(12)
    plain = [_first_argmin(s) for s in scores]

    def run(ts, tb):
        return oracle.guards(L, g, hits, inst, req, scores, lo, hi, n=1, k=1, kv_col=4,
                             tau_sat=ts, tau_ben=tb)

    ch, _, st = run(0.75, 0.0)
    assert (st == 0).all() and ch.tolist() == plain
    ch, _, st = run(np.nextafter(np.float32(0.75), np.float32(0)), 0.0)
    assert (st == oracle.ROUTE_KFILTER).all()
    assert ch.tolist() == [int(oracle.hrw_candidates(int(x), 4, 1)[0]) for x in g]
    ch, _, st = run(0.5, 48.0)
    assert (st == 0).all() and ch.tolist() == plain
    ch, _, st = run(0.5, 47.99)
    assert (st == oracle.ROUTE_KFILTER).all()


def test_kfilter_mean_is_taken_in_fp64():
    # kv = [0.5, 0.5 + 2^-24, 0.5, 0.5]: the mean is 0.5 + 2^-26 > 0.5 in fp64
    # (an fp32 running sum rounds 1 + 2^-24 to 1 and ends at exactly 2.0)
    L, g, hits, inst, req, scores = _kv_setting(14, N=4)
    inst[:, 4] = [0.5, 0.5 + 2.0 ** -24, 0.5, 0.5]
    lo, hi = _wide(12)
    _, _, st = oracle.guards(L, g, hits, inst, req, scores, lo, hi, n=1, k=1, kv_col=4,
                             tau_sat=0.5, tau_ben=-1.0)
    assert (st == oracle.ROUTE_KFILTER).all()
    inst[1, 4] = 0.5
    _, _, st = oracle.guards(L, g, hits, inst, req, scores, lo, hi, n=1, k=1, kv_col=4,
                             tau_sat=0.5, tau_ben=-1.0)
    assert (st == 0).all()


def test_kfilter_reads_the_kv_column_and_needs_a_full_block():
    L, g, hits, inst, req, scores = _kv_setting(12)
    lo, hi = _wide(12)
    inst[:, 3] = 0.1                                    # another column, below threshold
    _, _, st = oracle.guards(L, g, hits, inst, req, scores, lo, hi, n=1, k=2, kv_col=3,
                             tau_sat=0.8, tau_ben=-1.0)
    assert (st == 0).all()
    L2 = np.full_like(L, 15)                            # no full block: no prefix group
    _, _, st = oracle.guards(L2, g, np.zeros_like(hits), inst, req, scores, lo, hi, n=1, k=2,
                             kv_col=4, tau_sat=0.8, tau_ben=-1.0)
    assert (st == 0).all()


def test_kfilter_with_k_at_least_n_keeps_the_argmin():
    L, g, hits, inst, req, scores = _kv_setting(13, N=5)
    lo, hi = _wide(12)
    ch, _, st = oracle.guards(L, g, hits, inst, req, scores, lo, hi, n=1, k=5, kv_col=4,
                              tau_sat=0.0, tau_ben=-1.0)
    assert (st == oracle.ROUTE_KFILTER).all()
    assert ch.tolist() == [_first_argmin(s) for s in scores]
