"""Pins of the oracle's dropout between hidden layers (Sec. 4.1 Model
architecture; training only): the keep rate of the counter-based generator,
and the gradient of a training step against torch autograd with the same
masks applied by torch.  No GPU needed.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_00946_gb300 import workload as W


@pytest.mark.parametrize("p", [0.1, 0.5])
def test_keep_rate_and_streams(p):
    n = 0
    keep = 0
    pats = set()
    for t in (1, 2):
        for h in (1, 2):
            pat = []
            for j in range(40):
                for o in range(50):
                    k = oracle.drop_keep(12345, p, t, h, j, o)
                    keep += k
                    n += 1
                    pat.append(k)
            pats.add(tuple(pat))
    sd = np.sqrt(n * p * (1 - p))
    assert abs(keep - n * (1 - p)) < 5 * sd
    assert len(pats) == 4                              # steps and layers draw different masks
    assert all(oracle.drop_keep(1, 0.0, 3, 1, j, 0) for j in range(200))


def _torch_grad(widths, params, x, y, idx, mean, std, p, seed, t):
    w = widths
    L = len(w) - 1
    Ws, bs, off = [], [], 0
    for l in range(L):
        Ws.append(torch.tensor(params[off:off + w[l + 1] * w[l]].reshape(w[l + 1], w[l]), dtype=torch.float64,
                               requires_grad=True))
        off += w[l + 1] * w[l]
        bs.append(torch.tensor(params[off:off + w[l + 1]], dtype=torch.float64, requires_grad=True))
        off += w[l + 1]
    xs = torch.from_numpy(((x[idx] - mean) / np.where(std < 1e-12, 1, std)).astype(np.float32).astype(np.float64))
    B = len(idx)
    a = xs
    for l in range(L):
        z = a @ Ws[l].T + bs[l]
        if l + 1 < L:
            a = torch.relu(z)
            if l + 2 < L:                                  # between hidden layers only
                m = torch.tensor([[oracle.drop_keep(seed, p, t, l + 1, j, o) for o in range(w[l + 1])]
                                  for j in range(B)], dtype=torch.float64)
                a = a * m / (1.0 - p)
        else:
            a = z
    loss = ((a[:, 0] - torch.from_numpy(y[idx].astype(np.float64))) ** 2).mean()
    loss.backward()
    g = []
    for l in range(L):
        g.append(Ws[l].grad.numpy().ravel())
        g.append(bs[l].grad.numpy())
    return float(loss.detach()), np.concatenate(g)


@pytest.mark.parametrize("widths", [(16, 32, 32, 32, 1), (16, 24, 24, 1)])
def test_training_gradient_with_dropout_matches_autograd(widths):
    cfg = W.CONFIGS["tiny"]
    rng = np.random.default_rng(4)
    params = W.xavier_params(widths, 2)
    x, y = W.records(rng, cfg, 64)
    mean, std = W.normaliser(np.random.default_rng(5), cfg, 4096)
    idx = np.arange(0, 64, 2, dtype=np.int32)
    tr = oracle.Trainer(widths, params, "f64", dropout=0.25, dropout_seed=99)
    loss, g = tr.step(x, y, idx, mean, std, "sgd", 0.0, want_grad=True)   # t = 1
    tl, tg = _torch_grad(widths, params, x, y, idx, mean, std, 0.25, 99, 1)
    assert abs(loss - tl) <= 1e-12 * max(1.0, tl)
    np.testing.assert_allclose(g, tg, rtol=1e-9, atol=1e-12)
    # dropout 0 is the plain step
    plain = oracle.Trainer(widths, params, "f64")
    _, g0 = plain.step(x, y, idx, mean, std, "sgd", 0.0, want_grad=True)
    tl0, tg0 = _torch_grad(widths, params, x, y, idx, mean, std, 0.0, 99, 1)
    np.testing.assert_allclose(g0, tg0, rtol=1e-9, atol=1e-12)
    assert not np.allclose(g, g0)
