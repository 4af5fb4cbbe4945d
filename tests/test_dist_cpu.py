"""Multi-rank harness logic of bench.py on CPU (gloo, world size 2): each rank
routes its own batch (replicas, no collective on the data path); the timing
is the max over ranks and the reported value is all ranks' requests over it."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    w, r, local = bench.dist_setup(world)
    assert (w, r, local) == (world, rank, rank)
    bench.barrier(w)
    ms = bench.max_over_ranks(w, 1.0 + rank)       # rank 1 is the slow one
    out[rank] = ms
    dist.destroy_process_group()


def test_max_over_ranks_gloo_world2():
    ctx = mp.get_context("spawn")
    manager = ctx.Manager()
    out = manager.dict()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    assert out[0] == out[1] == 2.0


def test_reference_arm_prints_only_on_rank0(monkeypatch, capsys):
    import bench
    monkeypatch.setattr(bench, "oracle_work", lambda wl, ik, n, rng: 0.01)

    class A:
        steps, warmup, gpus = 2, 1, 2
    assert bench.run_reference(A, 2, 1) == 0          # rank 1: no output, exit 0
    assert capsys.readouterr().out == ""
