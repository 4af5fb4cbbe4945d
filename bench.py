"""Benchmark of the Lodestar routing hot path on GB300.

One step = one pass of the whole path over one batch of the large-cluster
workload (256 instances x 16,384 pending requests, prompts 128-16k tokens with
Zipf-shared prefixes over 4096 templates, 2^20 cached blocks per instance,
128-dim features, bf16 MLP 128->512->512->1):
  ls_snapshot_update (instance state rows) -> ls_route_batch (hash, probe,
  features, MLP, argmin for 4,194,304 pairs) -> ls_log_samples (4096 records)
  -> ls_train_step (Adam, batch 4096) -> ls_publish.
Metric: routing decisions per second (requests routed per second of whole
steps).  Inputs resident in HBM and larger than L2 (541 MB of prompt tokens
per batch); CUDA events on the launching stream; W untimed warm-up steps.
Beside the headline, the line carries every configuration's own figures
(tiny latency, homogeneous and heterogeneous route rates, the online-training
configuration's samples/s, the large configuration's route rate), each with
its roofline, and the measured ceilings (random 8-byte gathers, fp32 FMA, L2
reads) the memory- and ALU-bound kernels are judged against.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Under torchrun each rank routes its own batch on its own GPU (replicas, weak
scaling, no collective on the data path); rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import json
import os
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

WORKLOAD = "large"
DESC = {
    "tiny": "tiny: 8 instances x 64 requests, prompts 32-512 tokens (+128-token system prompt, p 0.5), "
            "2048 cached blocks/instance, fp32 MLP 16-64-64-1",
    "homogeneous": "homogeneous: 32 instances x 4096 requests, prompts 64-4096 tokens with Zipf(1.1) prefixes over "
                   "256 templates, 16384 cached blocks/instance, bf16 MLP 64-256-256-1",
    "heterogeneous": "heterogeneous: 64 instances (3 GPU types) x 8192 requests, prompts 8k-32k tokens log-uniform, "
                     "65536 cached blocks/instance, bf16 MLP 128-256-256-256-1",
    "large": "large: 256 instances x 16384 requests/step, prompts 128-16384 tokens with Zipf(1.1) prefixes over 4096 "
             "templates, 2^20 cached blocks/instance (open addressing, load 0.5), bf16 MLP 128-512-512-1, "
             "Adam batch 4096",
}
INPUT_SETS_SMALL = 6   # device copies of a batch smaller than L2 that timed routes rotate over
METRIC = "routing decisions/sec (requests routed per second of whole route+log+train+publish steps)"
UNIT = "decisions/s"


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=200)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-configs", action="store_true", help="skip the other configurations' measurements")
    p.add_argument("--no-guards", action="store_true", help="skip the guarded-route measurement")
    p.add_argument("--no-replay", action="store_true", help="skip the replay-pool admission measurement")
    p.add_argument("--no-paper-point", action="store_true", help="skip the paper operating-point measurement")
    p.add_argument("--no-training-config", action="store_true",
                   help="skip the online-training throughput configuration")
    p.add_argument("--no-probes", action="store_true", help="skip the ceiling microbenchmarks")
    p.add_argument("--paper-point-only", action="store_true", help="only the paper operating-point measurement")
    p.add_argument("--replay-only", action="store_true",
                   help="only the replay-pool admission measurement (for kernel profiling)")
    p.add_argument("--guards-only", action="store_true",
                   help="only the guarded-route measurement (--steps routes; for kernel profiling)")
    p.add_argument("--train-only", action="store_true",
                   help="only Adam steps of the training configuration, alone (for kernel profiling: the first "
                        "two timed steps are inside the profiler range)")
    p.add_argument("--route-only", default=None, choices=["tiny", "homogeneous", "heterogeneous", "large"],
                   help="only --steps routes of one configuration (for kernel profiling)")
    p.add_argument("--small", action="store_true",
                   help="with --route-only: the configuration's shapes at 2048 requests and 4096 cached blocks per "
                        "instance (a few hundred MB on the device, for ncu captures)")
    p.add_argument("--cpu-seconds", type=float, default=12.0, help="target oracle work for cpu_baseline")
    return p.parse_args()


def measure_guards(L, r, dw, N, R, d, ring_rows, d_req, flush, stream, peaks, n=60):
    """Guarded route of Algorithm 4 (cold start, out-of-range bounds, K-filter
    with K = 2) with the fallback heuristic of Algorithm 1 pre-computed (as
    Algorithm 3 does) on the bench batch, beside the plain route: event-timed route
    calls (call by call, L2 flushed before each) and per-launch times of the
    guard kernel and of the ring-bounds reduction."""
    import torch
    dev = dw.tok.device
    o_plain = {"choice": torch.empty(R, dtype=torch.int32, device=dev),
               "best": torch.empty(R, dtype=torch.float32, device=dev), "scores": None, "hits": None}
    o_g = dict(o_plain, status=torch.empty(R, dtype=torch.int32, device=dev),
               fallback=torch.empty(R, dtype=torch.int32, device=dev))
    r.refresh_bounds()
    r.publish()
    # tau_sat = 0 keeps the K-filter on for every request with a hit (the
    # paper's 0.8 would switch it off on this snapshot: mean KV use ~0.5)
    r.set_guards(n_min=1, ood=True, k=2, kv_col=4, tau_sat=0.0, tau_ben=0.0, heuristic=1, count_cols=(0, 1),
                 theta_imbal=128.0, k_overload=1.0)

    def timed(fn):
        ts = []
        for k in range(n):
            flush.fill_(k & 0xFF)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fn()
            e1.record(stream)
            e1.synchronize()
            ts.append(e0.elapsed_time(e1))
        return float(np.mean(ts[3:]))

    plain_ms = timed(lambda: r.route(dw.tok, dw.tok_off, dw.req_feats, N, out=o_plain))
    guarded_ms = timed(lambda: r.route_guarded(dw.tok, dw.tok_off, dw.req_feats, N, out=o_g))
    L.ls_trace_enable(r.h, True)
    L.ls_trace_read(r.h)
    for k in range(n):
        flush.fill_(k & 0xFF)
        r.route_guarded(dw.tok, dw.tok_off, dw.req_feats, N, out=o_g)
        flush.fill_(k & 0xFF)
        r.refresh_bounds()
    torch.cuda.synchronize()
    rc, trace = L.ls_trace_read(r.h)
    L.ls_trace_enable(r.h, False)
    r.set_guards()                                   # all guards off again
    st = o_g["status"].cpu().numpy()
    agree = bool(torch.equal(o_g["choice"][st == 0], o_plain["choice"][torch.from_numpy(st == 0).to(dev)]))
    per = {k: v[1] / max(v[2], 1) for k, v in trace.items()}
    g_bytes = R * N * 8 + R * (16 + 64 + 4 * d_req + 12)
    b_bytes = ring_rows * d * 4
    hbm = peaks["hbm_gbs"]
    g_gbs = g_bytes / 1e9 / (per["guards"] / 1e3)
    b_gbs = b_bytes / 1e9 / (per["ring_bounds"] / 1e3)
    return {
        "route_plain_ms": plain_ms, "route_guarded_ms": guarded_ms,
        "guards_kernel": {"avg_launch_ms": per["guards"], "bytes_per_launch": g_bytes, "achieved": g_gbs,
                          "peak": hbm, "unit": "GB/s", "frac": g_gbs / hbm, "bound": "hbm"},
        "ring_bounds_kernel": {"avg_launch_ms": per["ring_bounds"], "bytes_per_launch": b_bytes,
                               "achieved": b_gbs, "peak": hbm, "unit": "GB/s", "frac": b_gbs / hbm,
                               "bound": "hbm", "rows": ring_rows},
        "status_counts": {"ok": int((st == 0).sum()), "k_filtered": int((st == 4).sum()),
                          "cold_start": int((st == 1).sum()), "out_of_range": int((st == 2).sum())},
        "unfiltered_choices_equal_plain_route": agree,
        "fallback_distinct_instances": int(torch.unique(o_g["fallback"]).numel()),
        "settings": "n_min 1, out-of-range check on, K 2, kv column 4, tau_sat 0, tau_ben 0; fallback "
                    "heuristic of Algorithm 1 (counts = queued + running, theta_imbal 128 so that the per-request "
                    "order decides, k 1)",
    }


def measure_replay(L, H, W, wl, dev, flush, stream, peaks, n=20):
    """Two-pool training data (Sec. 4.3.2) at the paper's sizes: FIFO 5000,
    replay pool 5000, pending ring 5000, records logged in flushes of 100.
    Each timed round logs one flush (100 evictions) and runs one admission
    round; a second series logs 4096 records per round."""
    import torch
    cfg = wl.cfg
    r = H.Router.for_config(cfg, ring_capacity=5000, pending_capacity=5000, replay_capacity=5000,
                            max_train_batch=4096)
    dw = H.DeviceWorkload(wl, device=dev)
    dw.load(r)
    rng = np.random.default_rng(11)
    x, y = W.records(rng, cfg, 20000)
    xs, ys = torch.from_numpy(x).to(dev), torch.from_numpy(y).to(dev)
    pos = 0

    def log(k):
        nonlocal pos
        for a in range(0, k, 100):
            b = min(k, a + 100)
            i = pos % (len(ys) - 100)
            r.log(xs[i:i + b - a], ys[i:i + b - a])
            pos += b - a

    log(10000)                                   # FIFO full, 5000 evicted and pending
    r.replay_admit()                             # fills the replay pool
    out = {"fifo": 5000, "replay": 5000, "pending": 5000, "hidden": cfg.widths[-2]}
    for label, k in (("flush_100", 100), ("batch_4096", 4096)):
        ts = []
        for it in range(n + 3):
            log(k)
            flush.fill_(it & 0xFF)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            r.replay_admit()
            e1.record(stream)
            e1.synchronize()
            ts.append(e0.elapsed_time(e1))
        ms = float(np.mean(ts[3:]))
        Hd, nR = cfg.widths[-2], 5000
        flops = 2.0 * k * nR * Hd + 2.0 * nR * nR * Hd      # useful distance products
        out[label] = {"ms_per_round": ms, "candidates": k, "useful_distance_gflop": flops / 1e9,
                      "achieved_tflops": flops / 1e12 / (ms / 1e3),
                      "frac_of_bf16_peak": flops / 1e12 / (ms / 1e3) / peaks["bf16_tflops"]}
    info = r.info()
    out["replay_count"] = int(info.replay_count)
    r.close()
    return out


def measure_paper_point(L, H, W, dev, stream, n=400):
    """The paper's operating point (Sec. 4.3.1 P1, Sec. 5.4 overhead): one
    request routed over 16 instances by the 3 x 128 predictor, and its
    training recipe (FIFO 5000 + replay 5000, dropout 0.1, Adam).  Latency of
    a single-request route: host wall clock of the call through the C ABI
    until its result is on the host, device time of the call (events), and
    one replay of the route captured in a CUDA graph."""
    import time
    import torch
    wl = W.generate("paper")
    cfg = wl.cfg
    r = H.Router.for_config(cfg, max_requests=1, ring_capacity=5000, pending_capacity=5000, replay_capacity=5000,
                            max_train_batch=4096, dropout=0.1, dropout_seed=1)
    dw = H.DeviceWorkload(wl, device=dev)
    dw.load(r)
    N = cfg.n_inst
    out = {"choice": torch.empty(1, dtype=torch.int32, device=dev), "best": torch.empty(1, device=dev),
           "scores": None, "hits": None}
    h_choice = torch.empty(1, dtype=torch.int32).pin_memory()
    offs = [dw.tok_off[i:i + 2] for i in range(cfg.n_req)]
    reqs = [dw.req_feats[i:i + 1] for i in range(cfg.n_req)]
    wall, dev_ms = [], []
    for k in range(n + 20):
        i = k % cfg.n_req
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        e0.record(stream)
        r.route(dw.tok, offs[i], reqs[i], N, out=out)
        e1.record(stream)
        h_choice.copy_(out["choice"], non_blocking=True)
        stream.synchronize()
        t1 = time.perf_counter()
        if k >= 20:
            wall.append(1e6 * (t1 - t0))
            dev_ms.append(1e3 * e0.elapsed_time(e1))
    g_off, g_req = offs[0].clone(), reqs[0].clone()
    graph = H.StepGraph(lambda: r.route(dw.tok, g_off, g_req, N, out=out))
    gt = []
    for k in range(n + 20):
        i = k % cfg.n_req
        g_off.copy_(offs[i])
        g_req.copy_(reqs[i])
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        graph.replay()
        e1.record(stream)
        e1.synchronize()
        if k >= 20:
            gt.append(1e3 * e0.elapsed_time(e1))
    # training recipe: a round over F u R in minibatches of 4096 (Adam, dropout 0.1)
    x, y = W.records(np.random.default_rng(3), cfg, 15000)
    r.log(torch.from_numpy(x[:5000]).to(dev), torch.from_numpy(y[:5000]).to(dev))
    r.log(torch.from_numpy(x[5000:10000]).to(dev), torch.from_numpy(y[5000:10000]).to(dev))
    r.replay_admit()
    r.log(torch.from_numpy(x[10000:]).to(dev), torch.from_numpy(y[10000:]).to(dev))
    r.replay_admit()
    info = r.info()
    buf = min(info.ring_count, 5000) + info.replay_count
    ts = []
    for k in range(23):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        r.train(4096, None, opt="adam", lr=3e-4)
        e1.record(stream)
        e1.synchronize()
        if k >= 3:
            ts.append(e0.elapsed_time(e1))
    r.close()
    pct = lambda v, q: float(np.percentile(v, q))
    return {"instances": N, "predictor": "x".join(str(w) for w in cfg.widths),
            "route_host_us": {"p50": pct(wall, 50), "p99": pct(wall, 99)},
            "route_device_us": {"p50": pct(dev_ms, 50), "p99": pct(dev_ms, 99)},
            "route_graph_replay_us": {"p50": pct(gt, 50), "p99": pct(gt, 99)},
            "train_buffer_records": int(buf), "train_step_ms_batch_4096": float(np.mean(ts)),
            "train_samples_per_s": 4096 / (float(np.mean(ts)) / 1e3),
            "note": "the paper reports a few milliseconds of router overhead per request (Fig. overhead); "
                    "host time here is the C-ABI call from Python until the choice is in pinned host memory"}


def measure_sequential(L, H, W, dev, stream, name, n_req, calls=4):
    """Sequential-commit routing (Sec. 4.2 snapshot manager; Sec. 4.3.1 P1):
    one call routes n_req requests in order, committing each decision (queue
    + 1, prompt blocks cached on the chosen instance) before the next request;
    device time per call and per request (CUDA events)."""
    import dataclasses
    import torch
    cfg = dataclasses.replace(W.CONFIGS[name], n_req=n_req, n_samples=0)
    wl = W.generate(cfg, with_samples=False)
    room = cfg.cache_blocks + (calls + 2) * int(np.sum(np.diff(wl.tok_off) // 16))
    r = H.Router.for_config(cfg, max_keys_per_instance=room)
    dw = H.DeviceWorkload(wl, device=dev)
    dw.load(r)
    r.route_sequential(dw.tok, dw.tok_off, dw.req_feats, cfg.n_inst)       # warm-up call
    ts = []
    for _ in range(calls):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        r.route_sequential(dw.tok, dw.tok_off, dw.req_feats, cfg.n_inst)
        e1.record(stream)
        e1.synchronize()
        ts.append(e0.elapsed_time(e1))
    status = r.sync()
    r.close()
    ms = float(np.median(ts))
    return {"instances": cfg.n_inst, "predictor": "x".join(str(w) for w in cfg.widths), "requests_per_call": n_req,
            "ms_per_call": ms, "us_per_request": 1e3 * ms / n_req, "decisions_per_s": n_req / (ms / 1e3),
            "status": int(status)}


def measure_training_config(L, H, W, dev, steps=1000):
    """The online-training throughput configuration: a ring of 2^20 logged
    128-dim records, Adam (lr 3e-4, batch 4096) on the 128-256-256-256-1
    predictor, on its own stream, with a route of the heterogeneous batch
    (64 instances x 8192 long prompts) and a publish every 10 training steps
    on another stream (Sec. 4.3.1 P2: training beside routing)."""
    import torch
    wl = W.generate("training")
    cfg = wl.cfg
    r = H.Router.for_config(cfg, ring_capacity=cfg.n_samples)
    dw = H.DeviceWorkload(wl, device=dev)
    dw.load(r)
    r.log(torch.from_numpy(wl.samples_x).to(dev), torch.from_numpy(wl.samples_y).to(dev))
    out = {"choice": torch.empty(cfg.n_req, dtype=torch.int32, device=dev),
           "best": torch.empty(cfg.n_req, device=dev), "scores": None, "hits": None}
    sa, sb = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    loss = torch.zeros(1, device=dev)
    torch.cuda.synchronize()  # the two streams start after the setup above (snapshot, log)

    def run(n):
        for k in range(n):
            r.train(cfg.train_batch, None, opt="adam", lr=cfg.train_lr, loss_out=loss, stream=sb)
            if k % 10 == 9:
                r.route(dw.tok, dw.tok_off, dw.req_feats, cfg.n_inst, out=out, stream=sa)
                r.publish(stream=sb)

    run(20)
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(sb)
    sa.wait_stream(sb)
    run(steps)
    sb.wait_stream(sa)
    e1.record(sb)
    e1.synchronize()
    ms = e0.elapsed_time(e1)
    # training steps alone, issued back to back on one stream
    alone = timed_back_to_back(lambda k: r.train(cfg.train_batch, None, opt="adam", lr=cfg.train_lr, loss_out=loss,
                                                 stream=sb), 200, sb)
    ms_alone = float(np.mean(alone[10:]))
    r.close()
    # roofline of one step: its flops on the tensor cores plus its bytes
    # (minibatch rows and targets read; Adam reads w, g, m, v and writes w, m,
    # v and the bf16 image: 30 B per parameter) at the measured HBM rate
    peaks = measured_peaks()[0]
    B_ = cfg.train_batch
    flops = train_flops(cfg.widths, B_)
    n_params = sum(cfg.widths[l] * cfg.widths[l + 1] + cfg.widths[l + 1] for l in range(len(cfg.widths) - 1))
    bytes_ = B_ * (cfg.d + 1) * 4 + 30 * n_params
    t_roof = flops / (peaks["bf16_tflops"] * 1e12) + bytes_ / (peaks["hbm_gbs"] * 1e9)
    rate_alone = B_ / (ms_alone / 1e3)
    return {"config": "training: ring 2^20 x 128 fp32, Adam lr 3e-4, batch 4096, 128-256-256-256-1 bf16",
            "train_steps": steps, "route_calls": steps // 10, "ms": ms,
            "train_samples_per_s": steps * cfg.train_batch / (ms / 1e3),
            "routes_per_s_beside_training": (steps // 10) * cfg.n_req / (ms / 1e3),
            "train_step_alone_ms": ms_alone, "train_samples_per_s_alone": rate_alone,
            "roofline": {"step_us": 1e6 * t_roof, "samples_per_s": B_ / t_roof, "flops": flops, "bytes": bytes_,
                         "frac_alone": rate_alone / (B_ / t_roof),
                         "frac_beside_routes": steps * B_ / (ms / 1e3) / (B_ / t_roof)}}


def measure_training_only(L, H, W, dev, steps, warmup):
    """Adam steps of the training configuration alone on one stream: the
    first two after `warmup` inside cudaProfilerStart/Stop (a target for
    `ncu --profile-from-start off`), then `steps` back to back, timed."""
    import torch
    wl = W.generate("training")
    cfg = wl.cfg
    r = H.Router.for_config(cfg, ring_capacity=cfg.n_samples)
    dw = H.DeviceWorkload(wl, device=dev)
    dw.load(r)
    r.log(torch.from_numpy(wl.samples_x).to(dev), torch.from_numpy(wl.samples_y).to(dev))
    loss = torch.zeros(1, device=dev)
    s = torch.cuda.current_stream(dev)

    def step(k=0):
        r.train(cfg.train_batch, None, opt="adam", lr=cfg.train_lr, loss_out=loss, stream=s)

    for _ in range(max(warmup, 3)):
        step()
    torch.cuda.synchronize()
    torch.cuda.cudart().cudaProfilerStart()
    step()
    step()
    torch.cuda.synchronize()
    torch.cuda.cudart().cudaProfilerStop()
    times = timed_back_to_back(step, max(steps, 10), s)
    ms = float(np.mean(times))
    out = {"config": "training: ring 2^20 x 128 fp32, Adam lr 3e-4, batch 4096, 128-256-256-256-1 bf16",
           "train_step_alone_ms": ms, "train_samples_per_s_alone": cfg.train_batch / (ms / 1e3),
           "loss": float(loss.item()), "status": int(r.sync())}
    r.close()
    return out


def dist_setup(n_gpus):
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        dist.init_process_group(backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(world, value, device=None):
    if world == 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ----------------------------------------------------------------------------
# algorithmic cost of each kernel (per launch), for the roofline object
# ----------------------------------------------------------------------------

def mlp_flops_per_score(widths):
    """Layer-1 factorised: only the 6 pair columns are per-(request, instance)
    work; instance and request columns are done once per instance / request."""
    f = 2 * 6 * widths[1]
    for l in range(1, len(widths) - 1):
        f += 2 * widths[l] * widths[l + 1]
    return f


def distinct_probes(hits, lens, keys, key_off):
    """Sum over instances of the distinct block keys the prefix walk asks that
    instance about: block b of request r is asked of instance i when blocks
    0..b-1 are all cached there (h[r, i] >= b), the miss included.  A key
    stands for its whole prefix (chained hash), so every request holding key k
    at depth b gives instance i the same answer to h >= b: k counts once per
    instance with h[r(k), i] >= b(k), r(k) any request holding it."""
    R, N = hits.shape
    nb = (np.asarray(lens) // 16).astype(np.int64)
    if len(keys) == 0:
        return 0
    depth = np.arange(len(keys), dtype=np.int64) - np.repeat(np.asarray(key_off[:-1], np.int64), nb)
    req = np.repeat(np.arange(R, dtype=np.int64), nb)
    _, first = np.unique(np.asarray(keys).view(np.uint64), return_index=True)
    r_k, b_k = req[first], depth[first]
    big = int(max(hits.max(initial=0), nb.max(initial=0))) + 2
    sh = np.sort((np.arange(R, dtype=np.int64)[:, None] * big + hits.astype(np.int64)).ravel())
    cnt = (r_k + 1) * N - np.searchsorted(sh, r_k * big + b_k, side="left")
    return int(cnt.sum())


def route_costs(cfg, R, N, hits, lens, keys, key_off):
    """Algorithmic flops and bytes of one routing batch: the scorer's
    layer-1-factorised flops (and the dense count), and the prefix matcher's
    compulsory bytes -- every prompt token read once (4 B), 8 B per distinct
    probed (instance, key), 8 B of outputs per request."""
    w = cfg.widths
    flops = (mlp_flops_per_score(w) * R * N + 2 * N * cfg.d_inst * w[1] + 2 * R * cfg.d_req * w[1])
    dense = sum(2 * w[l] * w[l + 1] for l in range(len(w) - 1)) * R * N
    tok_bytes = 4 * int(np.sum(lens))
    probe_bytes = 8 * distinct_probes(hits, lens, keys, key_off)
    out_bytes = 8 * R
    return dict(score_flops=float(flops), score_flops_dense=float(dense),
                prefix_bytes=float(tok_bytes + probe_bytes + out_bytes),
                tok_bytes=tok_bytes, probe_bytes=probe_bytes, out_bytes=out_bytes)


def route_roofline(costs, R, N, peaks):
    """Sum over the dependent phases of max(bytes / BW, flops / peak): the prefix
    phase is bytes-bound, the scoring phase flops-bound."""
    t = costs["prefix_bytes"] / (peaks["hbm_gbs"] * 1e9) + costs["score_flops"] / (peaks["bf16_tflops"] * 1e12)
    return {"roofline_ms": 1e3 * t, "decisions_per_s": R / t, "scores_per_s": R * N / t}


def train_flops(widths, B):
    fwd = sum(2 * B * widths[l] * widths[l + 1] for l in range(len(widths) - 1))
    bwd = sum(2 * B * widths[l] * widths[l + 1] for l in range(len(widths) - 1))        # dW
    bwd += sum(2 * B * widths[l] * widths[l + 1] for l in range(1, len(widths) - 1))    # dX (l >= 1)
    return fwd + bwd


# ----------------------------------------------------------------------------
# clocks during the timed region
# ----------------------------------------------------------------------------

class ClockSampler:
    """Polls nvidia-smi (one query per poll) from a thread while the timed
    region runs; reports the median SM clock, the max clock and every
    throttle reason seen active."""
    FIELDS = ("uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, uuid):
        self.uuid = (uuid or "").lower().replace("gpu-", "")
        self.rows = []
        self.error = None
        self._stop = None
        self._t = None

    def _poll(self):
        while not self._stop.is_set():
            try:
                out = subprocess.run(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits"],
                                     capture_output=True, text=True, timeout=10)
                if out.returncode != 0:
                    self.error = (out.stderr or out.stdout).strip()[:200]
                    return
                lines = [[x.strip() for x in ln.split(",")] for ln in out.stdout.splitlines()]
                lines = [p for p in lines if len(p) >= 9]
                mine = [p for p in lines if self.uuid and self.uuid in p[0].lower()]
                self.rows.extend(mine if mine else (lines if len(lines) == 1 else []))
            except Exception as e:  # no nvidia-smi: report it
                self.error = str(e)[:200]
                return
            self._stop.wait(0.02)

    def start(self):
        import threading
        self._stop = threading.Event()
        self._t = threading.Thread(target=self._poll, daemon=True)
        self._t.start()

    def stop(self):
        if self._t is None:
            return None
        self._stop.set()
        self._t.join(timeout=15)
        if not self.rows:
            return {"error": self.error or "no samples"}

        def num(x):
            try:
                return float(x)
            except ValueError:
                return float("nan")
        sm = np.array([num(r[1]) for r in self.rows])
        reasons = [n for k, n in zip(range(5, 9), self.NAMES) if any(r[k].lower() == "active" for r in self.rows)]
        return {"sm_mhz": float(np.nanmedian(sm)), "sm_max_mhz": float(np.nanmax([num(r[2]) for r in self.rows])),
                "reasons": reasons, "samples": len(self.rows),
                "power_w_max": float(np.nanmax([num(r[3]) for r in self.rows]))}


KERNEL_SOURCES = {"score_tc": ("k_score_tc.cu", "sm100.cuh"),
                  "prefix_index": ("k_prefix_index.cu", "blockhash.cuh")}


def code_digest(files):
    """Hash of the code of the given sources (comments and whitespace removed,
    so that an edit of a comment keeps a capture of the same code valid)."""
    import hashlib
    import re
    src = os.path.join(ROOT, "paper_2606_00946_gb300", "csrc")
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(src, f)) as fh:
            text = fh.read()
        text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
        text = re.sub(r"//[^\n]*", " ", text)
        h.update(" ".join(text.split()).encode())
    return h.hexdigest()[:16]


def profiled_traffic(kernel, workload):
    """DRAM bytes per launch of `kernel` on `workload` from the committed ncu
    summaries, if the summary was taken on the kernel's current source (else
    None).  A capture on a smaller case of the same kernel is scaled to the
    workload's launch when the summary says so (scale=...)."""
    import glob
    if kernel not in KERNEL_SOURCES:
        return None
    sha = code_digest(KERNEL_SOURCES[kernel])
    for path in glob.glob(os.path.join(ROOT, "profiles", "*.md")):
        for line in open(path):
            if line.startswith("roofline-traffic:"):
                kv = dict(p.split("=", 1) for p in line.split()[1:])
                if kv.get("kernel") == kernel and kv.get("code_sha256") == sha and kv.get("workload") == workload:
                    return float(kv["bytes_per_launch"]) * float(kv.get("scale", "1"))
    return None


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


# ----------------------------------------------------------------------------
# CPU oracle (cpu_baseline and --impl reference)
# ----------------------------------------------------------------------------

def cpu_model():
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.split(":")[0].strip() in ("Model name", "Model"):
                v = line.split(":", 1)[1].strip()
                if v and not v.isdigit():
                    return v
    except Exception:
        pass
    return None


def oracle_setup(wl):
    """The oracle's snapshot: each instance's key set hashed by the oracle and
    sorted once (as the router's tables are built once), plus logged records
    for its training step."""
    import oracle
    inst_sorted = oracle.sorted_instance_keys(oracle.instance_keys(wl))
    if wl.samples_x is not None:
        rx, ry = wl.samples_x, wl.samples_y
    else:
        from paper_2606_00946_gb300 import workload as W
        rx, ry = W.records(np.random.default_rng(wl.cfg.seed + 5000), wl.cfg, 4096)
    return inst_sorted, rx, ry


def oracle_work(wl, orc, n_req, rng, threads):
    """Oracle pass over a sample: route n_req requests (hash, hits against the
    sorted key sets, features, fp64-accumulated MLP, argmin) with the requests
    split over `threads` host threads (the C routines release the interpreter
    lock), then one Adam step on n_req logged records on one thread."""
    import oracle
    inst_sorted, rx, ry = orc
    idx = np.sort(rng.choice(len(wl.tok_off) - 1, size=n_req, replace=False))
    t0 = time.perf_counter()
    oracle.route(wl, req_idx=idx, inst_sorted=inst_sorted, threads=threads)
    tr = oracle.Trainer(wl.cfg.widths, wl.params, wl.cfg.dtype)
    bidx = rng.integers(0, len(ry), size=n_req).astype(np.int32)
    tr.step(rx, ry, bidx, wl.mean, wl.std, "adam", 3e-4)
    return time.perf_counter() - t0


def cpu_baseline(wl, orc, target_s, name):
    """The oracle on the host's cores (requests over all cores), beside its
    single-thread figure.  The large configuration is sampled at 1/64 of its
    requests; the others at about target_s of work."""
    rng = np.random.default_rng(0)
    cores = os.cpu_count() or 1
    R = len(wl.tok_off) - 1
    t_cal = oracle_work(wl, orc, 2, rng, 1) / 2
    n1 = int(np.clip(0.3 * target_s / max(t_cal, 1e-4), 2, R))
    t1 = oracle_work(wl, orc, n1, rng, 1)
    if name == "large":
        n = R // 64
    else:
        n = int(min(R, max(16, n1 * cores)))
    t = oracle_work(wl, orc, n, rng, cores)
    return {"value": n / t, "unit": UNIT, "cores": cores, "kind": "oracle", "cpu_model": cpu_model(),
            "single_thread_value": n1 / t1,
            "sample": f"{n} of {R} requests of the {name} batch{' (1/64)' if name == 'large' else ''} routed by "
                      f"the C oracle (hash, hits against each instance's sorted key set, features, "
                      f"fp64-accumulated bf16 MLP, argmin) over {cores} host threads, plus one Adam step on {n} "
                      f"logged records on one thread; {t:.1f} s (one thread: {n1} requests in {t1:.1f} s)"}


def run_reference(args, world, rank):
    from paper_2606_00946_gb300 import workload as W
    if rank != 0:
        return 0
    wl = W.generate(WORKLOAD)
    orc = oracle_setup(wl)
    rng = np.random.default_rng(1)
    cores = os.cpu_count() or 1
    n = cores                                   # one request per host thread: about a second per step
    for _ in range(args.warmup):
        oracle_work(wl, orc, n, rng, cores)
    times = [oracle_work(wl, orc, n, rng, cores) for _ in range(args.steps)]
    ms = 1e3 * float(np.mean(times))
    value = n / (ms / 1e3)
    cfg = wl.cfg
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded generator shaped like the paper's prefix-sharing workloads)",
            "config": {"workload": DESC[WORKLOAD], "pairs_per_step": cfg.n_req * cfg.n_inst,
                       "train_samples_per_step": cfg.train_batch, "parallelism": "replicas",
                       "sample_requests_per_step": n},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "cpu_model": cpu_model(),
                             "sample": f"{n} requests of the {WORKLOAD} batch over {cores} host threads + one Adam "
                                       f"step on {n} records per step"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


# ----------------------------------------------------------------------------
# GPU arm
# ----------------------------------------------------------------------------

def timed_back_to_back(fn, n, stream):
    """n calls issued back to back, an event on the stream between consecutive
    ones: the host stays ahead of the GPU, so each interval is one call's
    device time.  Returns the intervals in ms."""
    import torch
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(n + 1)]
    ev[0].record(stream)
    for k in range(n):
        fn(k)
        ev[k + 1].record(stream)
    ev[n].synchronize()
    return [ev[k].elapsed_time(ev[k + 1]) for k in range(n)]


def traced(L, r, fn, n):
    """n calls issued one by one with every kernel launch of the context
    bracketed by CUDA events on its launching stream (the library's tracer),
    each call behind a ~150 us GPU spin so no interval holds host time.
    Returns ({kernel: (launches, total_ms, timed)}, launches per call)."""
    import torch
    L.ls_trace_enable(r.h, True)
    L.ls_trace_read(r.h)
    torch.cuda.synchronize()
    for k in range(n):
        torch.cuda._sleep(300000)
        fn(k)
    torch.cuda.synchronize()
    rc, trace = L.ls_trace_read(r.h)
    L.ls_trace_enable(r.h, False)
    return trace


def kernel_rooflines(trace, n_calls, costs, cfg, R, N, Bt, peaks, peak_src, workload):
    """Each traced kernel's achieved rate against its bound: the prefix walk
    (compulsory bytes, HBM), the feature image (bytes written), the scorers
    (factorised flops, bf16 tensor), the training products (their flops)."""
    per = {k: v[1] / max(v[2], 1) for k, v in trace.items()}
    n_per = {k: v[0] / n_calls for k, v in trace.items()}
    out = {}
    for k in per:
        d_pad = 64 * ((cfg.d + 63) // 64)
        if k in ("prefix_index", "prefix_match"):
            alg, peak, unit, bound = costs["prefix_bytes"] / 1e9, peaks["hbm_gbs"], "GB/s", "hbm"
        elif k == "features":
            # hit lengths and prompt offsets read; written: the whole bf16
            # feature image (pipelined scorer), else each row's 16-byte pair
            # chunk plus the instance and request template rows
            if costs.get("tc_kernel") == 2:
                written = R * N * 2 * d_pad
            else:
                written = R * N * 16 + (R + N) * 2 * d_pad
            alg = (R * N * 4 + R * 8 + written) / 1e9
            peak, unit, bound = peaks["hbm_gbs"], "GB/s", "hbm"
        elif k in ("score_tc", "score_simt"):
            alg, peak, unit, bound = costs["score_flops"] / 1e12, peaks["bf16_tflops"], "TFLOP/s", "tensor"
        elif k in ("gemm_tc_fwd", "gemm_tc_dx", "gemm_tc_dw"):
            w = cfg.widths
            nh = len(w) - 2
            per_kind = {"gemm_tc_fwd": sum(2 * Bt * w[l] * w[l + 1] for l in range(nh + 1)) + 2 * Bt * w[nh],
                        "gemm_tc_dx": sum(4 * Bt * w[l] * w[l + 1] for l in range(1, nh)),
                        "gemm_tc_dw": 2 * Bt * w[0] * w[1]}
            alg = per_kind[k] / max(n_per[k], 1e-9) / 1e12
            peak, unit, bound = peaks["bf16_tflops"], "TFLOP/s", "tensor"
        else:
            continue
        achieved = alg / (per[k] / 1e3)
        out[k] = {"kernel": k, "bound": bound, "achieved": achieved, "peak": peak, "unit": unit,
                  "frac": achieved / peak, "traffic": profiled_traffic(k, workload),
                  "peak_source": f"{peak_src} (burst)",
                  "avg_launch_ms": per[k],
                  "timing": "CUDA events around each launch on its stream (library tracer), calls issued one by one"}
    return out


def setup_config(name, H, W, dev, ring=65536, small=False, **caps):
    import dataclasses
    import torch
    wl = W.generate(dataclasses.replace(W.CONFIGS[name], n_req=2048, cache_blocks=4096, n_samples=0)
                    if small else name)
    cfg = wl.cfg
    r = H.Router.for_config(cfg, ring_capacity=max(ring, 4 * cfg.train_batch), **caps)
    dw = H.DeviceWorkload(wl, device=dev)
    dw.load(r)
    if wl.samples_x is not None:
        rx, ry = wl.samples_x, wl.samples_y
    else:
        rx, ry = W.records(np.random.default_rng(cfg.seed + 5000), cfg, ring)
    sx, sy = torch.from_numpy(rx).to(dev), torch.from_numpy(ry).to(dev)
    r.log(sx, sy)                                      # fill the ring once
    return wl, cfg, r, dw, sx, sy


def input_sets(dw, small_sets):
    """Device copies of the batch: one when it is larger than L2, else enough
    rotating copies that consecutive calls read their prompts from HBM."""
    bytes_ = sum(t.numel() * t.element_size() for t in (dw.tok, dw.tok_off, dw.req_feats))
    n = 1 if bytes_ > 300e6 else small_sets
    return [(dw.tok, dw.tok_off, dw.req_feats)] + [
        (dw.tok.clone(), dw.tok_off.clone(), dw.req_feats.clone()) for _ in range(n - 1)], bytes_


def batch_costs(r, wl, cfg, dw):
    chk = r.route(dw.tok, dw.tok_off, dw.req_feats, cfg.n_inst)
    hits = chk["hits"].cpu().numpy()
    keys, ko = r.hash_blocks(dw.tok, dw.tok_off)
    costs = route_costs(cfg, cfg.n_req, cfg.n_inst, hits, np.diff(wl.tok_off), keys.cpu().numpy(), ko.cpu().numpy())
    costs["tc_kernel"] = int(r.info().tc_kernel)
    return costs


def measure_route(name, L, H, W, dev, stream, peaks, peak_src, steps, warmup, ctx=None, small=False):
    """Route calls of one configuration alone (graph replays back to back):
    decisions/s, scores/s, per-kernel rooflines and the route-level roofline."""
    import torch
    own = ctx is None
    if own:
        ctx = setup_config(name, H, W, dev, small=small)
    wl, cfg, r, dw = ctx[:4]
    R, N = cfg.n_req, cfg.n_inst
    sets, set_bytes = input_sets(dw, INPUT_SETS_SMALL)
    out = {"choice": torch.empty(R, dtype=torch.int32, device=dev),
           "best": torch.empty(R, dtype=torch.float32, device=dev), "scores": None, "hits": None}

    def call(k):
        tok, off, req = sets[k % len(sets)]
        r.route(tok, off, req, N, out=out)

    for k in range(max(warmup, 2)):
        call(k)
    torch.cuda.synchronize()
    graphs = [H.StepGraph(lambda k=k: call(k)) for k in range(len(sets))]
    for k in range(warmup):
        graphs[k % len(graphs)].replay()
    torch.cuda.synchronize()
    times = timed_back_to_back(lambda k: graphs[k % len(graphs)].replay(), steps, stream)
    ms = float(np.mean(times))
    n_tr = min(steps, 30)
    trace = traced(L, r, call, n_tr)
    costs = batch_costs(r, wl, cfg, dw)
    rl = kernel_rooflines(trace, n_tr, costs, cfg, R, N, cfg.train_batch, peaks, peak_src, name)
    per_call = {k: v[1] / max(v[2], 1) * v[0] / n_tr for k, v in trace.items()}
    roof = route_roofline(costs, R, N, peaks)
    dom = max(rl, key=lambda k: per_call.get(k, 0.0)) if rl else None
    res = {"workload": DESC[name] + (" (reduced: 2048 requests, 4096 cached blocks per instance)" if small else ""),
           "ms_per_route": ms, "decisions_per_s": R / (ms / 1e3),
           "scores_per_s": R * N / (ms / 1e3), "route_roofline": roof,
           "frac_of_route_roofline": (R / (ms / 1e3)) / roof["decisions_per_s"],
           "dominant_kernel": dom, "roofline": rl.get(dom) if dom else None, "kernel_rooflines": rl,
           "kernels_ms_per_route": per_call, "algorithmic": costs,
           "l2": f"{len(sets)} device cop{'y' if len(sets) == 1 else 'ies'} of the batch "
                 f"({len(sets) * set_bytes / 1e6:.0f} MB, L2 129 MB); no flush"}
    if own:
        r.close()
    return res


def measure_tiny(L, H, W, dev, stream, n=200):
    """The tiny configuration is latency-bound: the device time of one route
    call and of one replay of it captured in a graph."""
    import torch
    wl, cfg, r, dw = setup_config("tiny", H, W, dev)[:4]
    out = {"choice": torch.empty(cfg.n_req, dtype=torch.int32, device=dev),
           "best": torch.empty(cfg.n_req, device=dev), "scores": None, "hits": None}
    call = lambda: r.route(dw.tok, dw.tok_off, dw.req_feats, cfg.n_inst, out=out)
    for _ in range(5):
        call()
    torch.cuda.synchronize()
    g = H.StepGraph(call)

    def lat(fn):
        ts = []
        for _ in range(n):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fn()
            e1.record(stream)
            e1.synchronize()
            ts.append(1e3 * e0.elapsed_time(e1))
        return {"p50": float(np.percentile(ts, 50)), "p99": float(np.percentile(ts, 99))}
    res = {"workload": DESC["tiny"], "route_device_us": lat(call), "route_graph_replay_us": lat(g.replay),
           "roofline": "n/a: latency-bound (512 scores, 5.3 MFLOP: under a microsecond at any ceiling)"}
    r.close()
    return res


def measure_probes(L, dev, stream, peaks, sms):
    """Ceilings on this GPU: random 8-byte gathers from a table in L2 (32 MB) and
    in HBM (4 GB), fp32 FMA issue (with the SM count x 128 lanes x 2 x clock
    figure beside it) and streaming L2 reads (64 MB buffer)."""
    import torch

    def timed(fn, reps=10):
        fn()
        torch.cuda.synchronize()
        ts = []
        for _ in range(reps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fn()
            e1.record(stream)
            e1.synchronize()
            ts.append(e0.elapsed_time(e1))
        return float(np.median(ts))

    res = {}
    blocks = 8 * sms
    out = torch.empty(blocks * 256, dtype=torch.int64, device=dev)
    for label, nbytes in (("l2", 32 << 20), ("hbm", 4 << 30)):
        table = torch.randint(0, 2 ** 62, (nbytes // 8,), dtype=torch.int64, device=dev)
        per = 64
        ms = timed(lambda: L.check(L.ls_probe_gather(table, table.numel(), blocks, per, 7, out, stream)))
        n = blocks * 256 * per
        res[f"gather8_{label}"] = {"table_bytes": nbytes, "lookups_per_s": n / (ms / 1e3),
                                   "GB_per_s": 8 * n / (ms / 1e3) / 1e9, "ms": ms}
        del table
    f = torch.empty(4 * sms * 256, dtype=torch.float32, device=dev)
    iters = 20000
    ms = timed(lambda: L.check(L.ls_probe_fma(4 * sms, iters, f, stream)))
    flops = 2 * 8 * iters * 4 * sms * 256
    res["fp32_fma"] = {"tflops": flops / (ms / 1e3) / 1e12,
                       "theory_tflops_at_max_clock": sms * 128 * 2 * peaks.get("sm_max_mhz", 2070.0) * 1e6 / 1e12}
    buf = torch.empty(64 << 20, dtype=torch.uint8, device=dev)
    o = torch.empty(blocks * 256 * 4, dtype=torch.int32, device=dev)
    passes = 8
    ms = timed(lambda: L.check(L.ls_probe_read(buf, buf.numel() // 16, passes, blocks, o, stream)))
    res["l2_read"] = {"buffer_bytes": buf.numel(), "GB_per_s": buf.numel() * passes / (ms / 1e3) / 1e9}
    return res


def measure_step(name, L, H, W, dev, stream, peaks, peak_src, args, ctx, clocks=None):
    """The whole step (snapshot state + route on one graph branch, log + train
    on a second, joined before the publish), captured once per device copy of
    the batch and replayed back to back; then the same steps issued call by
    call, and a traced pass for per-kernel times."""
    import torch
    wl, cfg, r, dw, sx, sy = ctx
    R, N, Bt = cfg.n_req, cfg.n_inst, cfg.train_batch
    states = [dw.inst_state, torch.from_numpy(W.instance_state(np.random.default_rng(99), cfg)).to(dev)]
    out = {"choice": torch.empty(R, dtype=torch.int32, device=dev),
           "best": torch.empty(R, dtype=torch.float32, device=dev), "scores": None, "hits": None}
    loss = torch.zeros(1, device=dev)
    stage_state = torch.empty_like(states[0])
    stage_x = torch.empty(Bt, cfg.d, device=dev)
    stage_y = torch.empty(Bt, device=dev)
    sets, set_bytes = input_sets(dw, INPUT_SETS_SMALL)

    def feed(k):
        stage_state.copy_(states[k & 1], non_blocking=True)
        a = (k * Bt) % (len(sy) - Bt + 1)
        stage_x.copy_(sx[a:a + Bt], non_blocking=True)
        stage_y.copy_(sy[a:a + Bt], non_blocking=True)

    side = torch.cuda.Stream(dev)  # training runs beside routing (Sec. 4.3.1: off the routing path)

    def body(ks=0, overlap=True):
        tok, tok_off, req = sets[ks]
        main = torch.cuda.current_stream(dev)
        if not overlap:                             # the same calls, one after another on one stream
            r.snapshot(N, stage_state)
            r.route(tok, tok_off, req, N, out=out)
            r.log(stage_x, stage_y)
            r.train(Bt, None, opt="adam", lr=cfg.train_lr, loss_out=loss)
            r.publish()
            return
        side.wait_stream(main)                      # the step's inputs are in place
        r.snapshot(N, stage_state)
        r.route(tok, tok_off, req, N, out=out)
        with torch.cuda.stream(side):
            r.log(stage_x, stage_y)
            r.train(Bt, None, opt="adam", lr=cfg.train_lr, loss_out=loss)
        main.wait_stream(side)                      # both branches done, then one publish
        r.publish()

    def eager_step(k):
        feed(k)
        body(k % len(sets))

    for k in range(args.warmup):
        eager_step(k)
    torch.cuda.synchronize()
    graphs = [H.StepGraph(lambda ks=ks: body(ks)) for ks in range(len(sets))]

    def step(k):
        feed(k)
        graphs[k % len(sets)].replay()

    for k in range(args.warmup):
        step(args.warmup + k)
    torch.cuda.synchronize()
    if clocks is not None:
        clocks.start()
    cudart = torch.cuda.cudart()
    cudart.cudaProfilerStart()                      # brackets the region for ncu --profile-from-start off
    times = timed_back_to_back(lambda k: step(2 * args.warmup + k), args.steps, stream)
    cudart.cudaProfilerStop()
    torch.cuda.synchronize()
    clk = clocks.stop() if clocks is not None else None
    eager_times = timed_back_to_back(lambda k: eager_step(2 * args.warmup + args.steps + k),
                                     min(args.steps, 100), stream)
    # per-kernel times from steps whose two branches run one after the other:
    # a kernel of the training branch timed while the scorer holds every SM
    # would count its wait for an SM as its own time
    n_traced = min(args.steps, 60)

    def serial_step(k):
        feed(k)
        body(k % len(sets), overlap=False)

    trace = traced(L, r, serial_step, n_traced)
    costs = batch_costs(r, wl, cfg, dw)
    rl = kernel_rooflines(trace, n_traced, costs, cfg, R, N, Bt, peaks, peak_src, name)
    per_step = {k: v[1] / max(v[2], 1) * v[0] / n_traced for k, v in trace.items()}
    launches = sum(v[0] for v in trace.values()) / n_traced
    return {"times": times, "eager_times": eager_times, "clocks": clk, "costs": costs, "rooflines": rl,
            "kernels_ms_per_step": per_step, "launches_per_step": launches, "sets": sets, "set_bytes": set_bytes,
            "body": body, "states": states, "out": out, "loss": loss, "side": side}


def measure_e2e(L, H, dev, stream, args, ctx, st, world):
    """End to end through the C ABI with host buffers: every step copies its
    inputs from pinned host memory and reads its results back.  The copies of
    step k+1 run on a copy stream while step k computes; device input sets
    rotate, each with its own captured graph of the step's ABI calls."""
    import torch
    wl, cfg, r, dw, sx, sy = ctx
    R, N, Bt = cfg.n_req, cfg.n_inst, cfg.train_batch
    out, loss, side = st["out"], st["loss"], st["side"]
    h_tok = torch.from_numpy(wl.tok).pin_memory()
    h_off = torch.from_numpy(wl.tok_off).pin_memory()
    h_req = torch.from_numpy(wl.req_feats).pin_memory()
    h_st = [s_.cpu().pin_memory() for s_ in st["states"]]
    h_x = sx[:8 * Bt].cpu().pin_memory()
    h_y = sy[:8 * Bt].cpu().pin_memory()
    NB = 3 if h_tok.numel() * 4 > 300e6 else 4
    sets = [{"tok": torch.empty_like(dw.tok), "off": torch.empty_like(dw.tok_off),
             "req": torch.empty_like(dw.req_feats), "st": torch.empty_like(st["states"][0]),
             "x": torch.empty(Bt, cfg.d, device=dev), "y": torch.empty(Bt, device=dev)} for _ in range(NB)]
    h_choice = torch.empty(R, dtype=torch.int32).pin_memory()
    h_best = torch.empty(R, dtype=torch.float32).pin_memory()
    h_loss = torch.empty(1).pin_memory()
    d0 = sets[0]
    h2d = sum(d0[k].numel() * d0[k].element_size() for k in ("tok", "off", "req", "st", "x", "y"))
    d2h = R * 4 + R * 4 + 4
    cs = torch.cuda.Stream(dev)

    def e2e_body(ds):
        main = torch.cuda.current_stream(dev)
        side.wait_stream(main)
        r.snapshot(N, ds["st"])
        r.route(ds["tok"], ds["off"], ds["req"], N, out=out)
        with torch.cuda.stream(side):
            r.log(ds["x"], ds["y"])
            r.train(Bt, None, opt="adam", lr=cfg.train_lr, loss_out=loss)
        main.wait_stream(side)
        r.publish()

    def copy_in(k, ds):
        a = (k * Bt) % (7 * Bt)
        ds["tok"].copy_(h_tok, non_blocking=True)
        ds["off"].copy_(h_off, non_blocking=True)
        ds["req"].copy_(h_req, non_blocking=True)
        ds["st"].copy_(h_st[k & 1], non_blocking=True)
        ds["x"].copy_(h_x[a:a + Bt], non_blocking=True)
        ds["y"].copy_(h_y[a:a + Bt], non_blocking=True)

    def copy_out():
        h_choice.copy_(out["choice"], non_blocking=True)
        h_best.copy_(out["best"], non_blocking=True)
        h_loss.copy_(loss, non_blocking=True)

    for k in range(max(args.warmup, NB)):
        copy_in(k, sets[k % NB])
        e2e_body(sets[k % NB])
        copy_out()
    torch.cuda.synchronize()
    graphs = [H.StepGraph(lambda ds=ds: e2e_body(ds)) for ds in sets]
    copied = [torch.cuda.Event() for _ in range(NB)]
    free = [torch.cuda.Event() for _ in range(NB)]

    def run_pipelined(k0, K):
        main = torch.cuda.current_stream(dev)
        for b in range(NB):
            free[b].record(main)
        for k in range(k0, k0 + K):
            b = k % NB
            cs.wait_event(free[b])            # the graph that last read this input set is done
            with torch.cuda.stream(cs):
                copy_in(k, sets[b])
                copied[b].record(cs)
            main.wait_event(copied[b])
            graphs[b].replay()
            free[b].record(main)
            copy_out()

    run_pipelined(0, 2 * NB)                 # warm the pipeline and the graphs
    torch.cuda.synchronize()
    K = min(args.steps, 100)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    cs.wait_stream(stream)
    e0.record(stream)
    run_pipelined(2 * NB, K)
    e1.record(stream)
    e1.synchronize()
    ems = max_over_ranks(world, e0.elapsed_time(e1) / K, None)
    return {"value": world * R / (ems / 1e3), "unit": UNIT, "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h), "ms_per_step": ems, "steps": K,
            # the host link's rate over the step (one GPU's copies); a pinned
            # host-to-device copy alone moves about 210 GB/s on a GB300 host
            "h2d_GB_per_s": h2d / (ems / 1e3) / 1e9,
            "pipelined": f"inputs of step k+1 copied on a copy stream while step k computes; {NB} device input sets "
                         f"with a captured graph each; choices, best scores and loss read back every step"}


def main():
    args = parse()
    world, rank, local = dist_setup(args.gpus)
    if args.impl == "reference":
        return run_reference(args, world, rank)

    import torch
    from paper_2606_00946_gb300 import build as B
    from paper_2606_00946_gb300 import harness as H
    from paper_2606_00946_gb300 import lodestar as L
    from paper_2606_00946_gb300 import workload as W

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    B.build()
    stream = torch.cuda.current_stream(dev)
    peaks, peak_src = measured_peaks()
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    flush = torch.empty(512 << 20, dtype=torch.uint8, device=dev)

    if args.route_only:
        res = measure_route(args.route_only, L, H, W, dev, stream, peaks, peak_src, args.steps, args.warmup,
                            small=args.small)
        if rank == 0:
            print(json.dumps({"route_only": args.route_only, **res}))
        return 0
    if args.train_only:
        res = measure_training_only(L, H, W, dev, args.steps, args.warmup)
        if rank == 0:
            print(json.dumps({"train_only": True, **res}))
        return 0
    if args.paper_point_only or args.replay_only or args.guards_only:
        wl, cfg, r, dw = setup_config("homogeneous", H, W, dev)[:4]
        if args.paper_point_only:
            res = {"paper_point": measure_paper_point(L, H, W, dev, stream)}
        elif args.replay_only:
            res = {"workload": "homogeneous",
                   "replay_admission": measure_replay(L, H, W, wl, dev, flush, stream, peaks, n=max(args.steps, 4))}
        else:
            res = {"workload": "homogeneous", "guarded_route": measure_guards(
                L, r, dw, cfg.n_inst, cfg.n_req, cfg.d, int(min(65536, r.info().ring_count)), cfg.d_req, flush,
                stream, peaks, n=max(args.steps, 4))}
        if rank == 0:
            print(json.dumps(res))
        r.close()
        return 0

    # ---- the headline: whole steps of the large configuration -------------
    ctx = setup_config(WORKLOAD, H, W, dev)
    wl, cfg, r = ctx[0], ctx[1], ctx[2]
    R, N, Bt = cfg.n_req, cfg.n_inst, cfg.train_batch
    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        pass
    barrier(world)
    torch.cuda.synchronize()
    st = measure_step(WORKLOAD, L, H, W, dev, stream, peaks, peak_src, args, ctx, clocks=ClockSampler(uuid))
    barrier(world)
    ms = max_over_ranks(world, float(np.mean(st["times"])),
                        dev if world > 1 and torch.distributed.get_backend() == "nccl" else None)
    value = world * R / (ms / 1e3)
    rl = st["rooflines"]
    route_k = [k for k in rl if k in ("prefix_index", "prefix_match", "features", "score_tc", "score_simt")]
    dom = max(route_k, key=lambda k: st["kernels_ms_per_step"][k])
    roofline = dict(rl[dom], branch="route (the step's critical branch)")
    train_k = [k for k in rl if k.startswith("gemm_tc")]
    train_roofline = (dict(rl[max(train_k, key=lambda k: st["kernels_ms_per_step"][k])], branch="train")
                      if train_k else None)
    roof = route_roofline(st["costs"], R, N, peaks)
    kms = st["kernels_ms_per_step"]
    launches_per_step = st["launches_per_step"]
    clk = st["clocks"]
    costs = st["costs"]
    eager_ms = float(np.mean(st["eager_times"]))

    e2e = None
    if not args.no_e2e:
        e2e = measure_e2e(L, H, dev, stream, args, ctx, st, world)
    large_route = measure_route(WORKLOAD, L, H, W, dev, stream, peaks, peak_src, min(args.steps, 50),
                                args.warmup, ctx=ctx)
    status = r.sync()
    if status != L.LS_OK:
        print(json.dumps({"error": f"device status {status}"}), file=sys.stderr)
    del st
    r.close()
    torch.cuda.empty_cache()

    # ---- every other configuration, each with its own roofline ------------
    configs = {"large": {"route_only": large_route}}
    probes = None
    if not args.no_probes:
        probes = measure_probes(L, dev, stream, peaks, sms)
    if not args.no_configs:
        configs["tiny"] = measure_tiny(L, H, W, dev, stream)
        hctx = setup_config("homogeneous", H, W, dev)
        hst = measure_step("homogeneous", L, H, W, dev, stream, peaks, peak_src, args, hctx)
        configs["homogeneous"] = {
            "route_only": measure_route("homogeneous", L, H, W, dev, stream, peaks, peak_src, args.steps,
                                        args.warmup, ctx=hctx),
            "step": {"ms_per_step": float(np.mean(hst["times"])),
                     "decisions_per_s": hctx[1].n_req / (float(np.mean(hst["times"])) / 1e3),
                     "kernels_ms_per_step": hst["kernels_ms_per_step"],
                     "what": "snapshot + route beside log + train (Adam, batch 4096), then publish, graph replays"}}
        del hst
        if not args.no_guards:
            hw, hc, hr, hd = hctx[:4]
            configs["homogeneous"]["guarded_route"] = measure_guards(
                L, hr, hd, hc.n_inst, hc.n_req, hc.d, int(min(65536, hr.info().ring_count)), hc.d_req, flush,
                stream, peaks)
        if not args.no_replay:
            configs["homogeneous"]["replay_admission"] = measure_replay(L, H, W, hctx[0], dev, flush, stream, peaks)
        hctx[2].close()
        configs["heterogeneous"] = {"route_only": measure_route("heterogeneous", L, H, W, dev, stream, peaks,
                                                                peak_src, min(args.steps, 100), args.warmup)}
        if not args.no_training_config:
            configs["training"] = measure_training_config(L, H, W, dev)
        if not args.no_paper_point:
            configs["paper_point"] = measure_paper_point(L, H, W, dev, stream)
            configs["sequential_commit"] = {
                "paper": measure_sequential(L, H, W, dev, stream, "paper", 256),
                "homogeneous": measure_sequential(L, H, W, dev, stream, "homogeneous", 512)}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(wl, oracle_setup(wl), args.cpu_seconds, WORKLOAD)

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (seeded generator shaped like the paper's prefix-sharing workloads)",
            "config": {"workload": DESC[WORKLOAD], "pairs_per_step": R * N, "train_samples_per_step": Bt,
                       "l2": "inputs larger than L2: 541 MB of prompt tokens per batch (L2 129 MB); no flush",
                       "parallelism": "replicas"},
            "scores_per_s": world * R * N / (ms / 1e3),
            "train_samples_per_s": world * Bt / (ms / 1e3),
            "roofline": roofline,
            "route_roofline": dict(roof, frac_of_rate=value / world / roof["decisions_per_s"],
                                   what="sum over phases of max(bytes / measured HBM, factorised flops / measured "
                                        "bf16): the step's decisions/s against the route's roofline rate"),
            "train_roofline": train_roofline,
            "kernel_rooflines": rl,
            "kernels_ms_per_step": {k: v for k, v in sorted(kms.items(), key=lambda kv: -kv[1])},
            "kernels_timing": "CUDA events around each launch (library tracer) over steps issued call by call with "
                              "the routing and training calls one after the other on one stream",
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": int(round(launches_per_step * args.steps)),
            "gpu_launches_per_step": launches_per_step,
            "launch": "each step: the new instance state and records copied into the step's buffers, then one "
                      "replay of a CUDA graph of the step's ABI calls: snapshot + route on one branch, log + train "
                      "on a second, joined before the publish; kernels of each chain launched with programmatic "
                      "dependent launch",
            "ms_per_step_eager": eager_ms,
            "clocks": clk,
            "algorithmic": costs,
            "ceilings": probes,
            "configs": configs,
        }
        print(json.dumps(line))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
