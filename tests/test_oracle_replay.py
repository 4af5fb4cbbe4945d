"""Pins of the oracle's two-pool training-data selection (Sec. 4.3.2): the
gradient embedding against torch autograd, distances against scipy's cdist,
the admission round against hand-worked examples and set properties checked
by brute force.  No GPU needed.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_00946_gb300 import workload as W


def test_embedding_is_the_output_layer_gradient():
    # g = (yhat - y) * a_last is d/dW_out of (yhat - y)^2 / 2: compare with autograd in fp64
    cfg = W.CONFIGS["tiny"]
    rng = np.random.default_rng(0)
    params = W.xavier_params(cfg.widths, 3)
    x, y = W.records(rng, cfg, 40)
    mean, std = W.normaliser(np.random.default_rng(1), cfg, 4096)
    g = oracle.replay_embed("f64", cfg.widths, params, x, y, mean, std)
    w = cfg.widths
    xs = torch.from_numpy(((x - mean) / np.where(std < 1e-12, 1, std)).astype(np.float32).astype(np.float64))
    Ws, bs, off = [], [], 0
    for l in range(len(w) - 1):
        Ws.append(torch.tensor(params[off:off + w[l + 1] * w[l]].reshape(w[l + 1], w[l]), dtype=torch.float64,
                               requires_grad=(l == len(w) - 2)))
        off += w[l + 1] * w[l]
        bs.append(torch.tensor(params[off:off + w[l + 1]], dtype=torch.float64))
        off += w[l + 1]
    for s in range(len(y)):
        a = xs[s]
        for l in range(len(w) - 1):
            z = Ws[l] @ a + bs[l]
            a = torch.relu(z) if l + 1 < len(w) - 1 else z
        loss = 0.5 * (a[0] - float(y[s])) ** 2
        (grad,) = torch.autograd.grad(loss, Ws[-1])
        np.testing.assert_allclose(g[s], grad.numpy()[0], rtol=1e-10, atol=1e-12)


def test_distances_match_scipy_cdist():
    from scipy.spatial.distance import cdist
    rng = np.random.default_rng(2)
    gc = rng.standard_normal((17, 9))
    gk = rng.standard_normal((23, 9))
    gk[5] = gk[11]                                    # a duplicate kept pair: nearest other at 0
    d, n = oracle.replay_distances(gc, gk)
    np.testing.assert_allclose(d, cdist(gc, gk, "sqeuclidean").min(axis=1), rtol=1e-12)
    kk = cdist(gk, gk, "sqeuclidean")
    np.fill_diagonal(kk, np.inf)
    np.testing.assert_allclose(n, kk.min(axis=1), rtol=1e-12, atol=1e-300)
    assert n[5] == 0 and n[11] == 0
    d0, n1 = oracle.replay_distances(gc, gk[:0])       # nothing kept: infinitely far
    assert np.isinf(d0).all()
    _, n1 = oracle.replay_distances(gc, gk[:1])        # one kept: no other
    assert np.isinf(n1).all()


def test_select_worked_examples():
    # candidates d = [5, 1, 3] rank 0, 2, 1; kept n = [2, 0.5, 4] rank 1, 0, 2
    # full pool (cap 3): cand 0 (5) > kept 1 (0.5) replaces slot 1; cand 2 (3) > kept 0 (2)
    # replaces slot 0; cand 1 (1) <= kept 2 (4) stops
    src, cnt = oracle.replay_select([5.0, 1.0, 3.0], [2.0, 0.5, 4.0], 3)
    assert cnt == 3 and src.tolist() == [2, 0, -3]
    # one free slot (cap 4): cand 0 fills slot 3; cand 2 (3) > kept 1 (0.5) replaces slot 1;
    # cand 1 (1) <= kept 0 (2) stops
    src, cnt = oracle.replay_select([5.0, 1.0, 3.0], [2.0, 0.5, 4.0], 4)
    assert cnt == 4 and src.tolist() == [-1, 2, -3, 0]
    # empty pool: the most diverse first, equal diversity by eviction order
    src, cnt = oracle.replay_select([np.inf, np.inf, np.inf], [], 2)
    assert cnt == 2 and src.tolist() == [0, 1]
    # NaN diversity ranks last and is never admitted over a number
    src, cnt = oracle.replay_select([np.nan, 2.0], [1.0], 1)
    assert cnt == 1 and src.tolist() == [1]


@pytest.mark.parametrize("seed", range(12))
def test_select_properties_by_brute_force(seed):
    rng = np.random.default_rng(seed)
    nk = int(rng.integers(0, 30))
    mc = int(rng.integers(0, 30))
    cap = nk + int(rng.integers(0, 10))
    d = np.round(rng.random(mc) * 8, 1)               # repeated values: ties by index
    n = np.round(rng.random(nk) * 8, 1)
    if mc:
        d[rng.random(mc) < 0.1] = np.nan
    src, cnt = oracle.replay_select(d, n, cap)
    free = cap - nk
    assert cnt == nk + min(free, mc)
    cand_rank = sorted(range(mc), key=lambda e: (-(d[e] if not np.isnan(d[e]) else -np.inf), e))
    kept_rank = sorted(range(nk), key=lambda j: (n[j], j))
    admitted = [s for s in src if s >= 0]
    r = len(admitted) - min(free, mc)                  # replacements made
    assert sorted(admitted) == sorted(cand_rank[:min(free, mc) + r])   # a prefix of the ranking
    replaced = [j for j in range(nk) if src[j] >= 0]
    assert sorted(replaced) == sorted(kept_rank[:r])
    for q in range(r):                                 # every pairing made improves diversity
        c, j = cand_rank[min(free, mc) + q], kept_rank[q]
        assert src[j] == c and d[c] > n[j]
    q = r                                              # and the next pairing would not
    if min(free, mc) + q < mc and q < nk:
        c, j = cand_rank[min(free, mc) + q], kept_rank[q]
        assert not (d[c] > n[j])
    for j in range(nk):
        if src[j] < 0:
            assert src[j] == -1 - j                    # kept samples stay in their slots
