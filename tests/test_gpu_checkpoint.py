"""Checkpoint and resume of the online learner (master weights, Adam moments
and step count, normaliser) through the C ABI: a run saved after some steps
and restored into a fresh context continues bit for bit like the run that
never stopped, on the plain fp32 path and on the tensor-core bf16 path.
"""
import numpy as np
import pytest
import torch

from paper_2606_00946_gb300 import build as B
from paper_2606_00946_gb300 import harness as H
from paper_2606_00946_gb300 import lodestar as L
from paper_2606_00946_gb300 import workload as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    B.build()


@pytest.mark.parametrize("cfg_name,opt", [("tiny", "adam"), ("homogeneous", "adam"), ("homogeneous", "sgd")])
def test_resume_continues_bit_exact(cfg_name, opt, tmp_path):
    cfg = W.CONFIGS[cfg_name]
    n = 3000
    x, y = W.records(np.random.default_rng(41), cfg, n)
    mean, std = W.normaliser(np.random.default_rng(42), cfg)
    params = W.xavier_params(cfg.widths, 3)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()

    def fresh():
        r = H.Router(cfg.widths, cfg.d_inst, cfg.d_req, cfg.dtype, max_instances=4, max_requests=16,
                     max_keys_per_instance=64, ring_capacity=n, max_train_batch=512)
        r.log(t(x), t(y))
        return r

    def step(r, k):
        r.train(256, t(W.minibatch_indices(8, k, n, 256)), opt=opt, lr=1e-3)

    a = fresh()
    a.set_normalizer(t(mean), t(std))
    a.set_params(t(params))
    for k in range(3):
        step(a, k)
    path = tmp_path / "learner.npz"
    a.save_checkpoint(path)
    b = fresh()
    b.load_checkpoint(path)
    for k in range(3, 6):
        step(a, k)
        step(b, k)
    ma, va, sa = a.get_opt_state()
    mb, vb, sb = b.get_opt_state()
    assert sa == sb == 6
    assert torch.equal(a.get_params(), b.get_params())
    assert torch.equal(ma, mb) and torch.equal(va, vb)
    assert a.sync() == L.LS_OK and b.sync() == L.LS_OK
    a.close()
    b.close()
