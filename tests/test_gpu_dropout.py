"""Dropout between hidden layers (Sec. 4.1 Model architecture) in the GPU
training step vs the CPU oracle, through the C ABI.

The gradient of one SGD step (lr 0.1 exposes it as (w - w') / 0.1) must be
within the bf16 tolerance of the oracle's gradient under the same dropout
stream, and far from the gradient without dropout; the second step checks
that the stream follows the device's step counter.
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


@pytest.fixture(scope="module", autouse=True)
def _built():
    B.build()


@pytest.mark.parametrize("hidden", [(128, 128, 128), (256, 256)])
def test_train_step_with_dropout(hidden):
    cfg = dataclasses.replace(W.CONFIGS["training"], hidden=hidden)
    rng = np.random.default_rng(21)
    n = 4096
    x, y = W.records(rng, cfg, n)
    mean, std = W.normaliser(np.random.default_rng(22), cfg)
    params = W.xavier_params(cfg.widths, 0)
    r = H.Router(cfg.widths, cfg.d_inst, cfg.d_req, cfg.dtype, max_instances=4, max_requests=16,
                 max_keys_per_instance=64, ring_capacity=n, max_train_batch=4096, dropout=0.1, dropout_seed=7)
    r.set_normalizer(torch.from_numpy(mean).cuda(), torch.from_numpy(std).cuda())
    r.set_params(torch.from_numpy(params).cuda())
    r.log(torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda())
    for step in (1, 2):
        idx = W.minibatch_indices(4, step, n, 4096)
        before = r.get_params().cpu().numpy()
        r.train(4096, torch.from_numpy(idx).cuda(), opt="sgd", lr=0.1)
        g_gpu = (before.astype(np.float64) - r.get_params().cpu().numpy()) / 0.1
        tr = oracle.Trainer(cfg.widths, before, "bf16", dropout=0.1, dropout_seed=7)
        tr.t = step - 1                                 # the oracle's step number becomes `step`
        _, g_or = tr.step(x, y, idx, mean, std, "sgd", 0.0, want_grad=True)
        _, g_plain = oracle.Trainer(cfg.widths, before, "bf16").step(x, y, idx, mean, std, "sgd", 0.0,
                                                                      want_grad=True)
        err = np.linalg.norm(g_gpu - g_or)
        assert err <= 2e-2 * np.linalg.norm(g_or), (step, err / np.linalg.norm(g_or))
        assert np.linalg.norm(g_gpu - g_plain) > 5 * err
        if step == 2:                                   # another step draws other masks
            tr1 = oracle.Trainer(cfg.widths, before, "bf16", dropout=0.1, dropout_seed=7)
            _, g_t1 = tr1.step(x, y, idx, mean, std, "sgd", 0.0, want_grad=True)
            assert np.linalg.norm(g_gpu - g_t1) > 5 * err
    assert r.sync() == L.LS_OK
    r.close()


def test_dropout_needs_the_tensor_core_training_path():
    cfg = W.CONFIGS["tiny"]                             # fp32 predictor: CUDA-core training
    with pytest.raises(RuntimeError):
        H.Router.for_config(cfg, dropout=0.1)
    with pytest.raises(RuntimeError):
        H.Router.for_config(W.CONFIGS["homogeneous"], dropout=1.0)
