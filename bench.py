"""Benchmark of the Lodestar routing hot path on GB300.

One step = one pass of the whole path over one batch of the homogeneous
workload (32 instances x 4096 pending requests, prompts 64-4096 tokens with
Zipf-shared prefixes, 64-dim features, bf16 MLP 64->256->256->1):
  ls_snapshot_update (instance state rows)  -> ls_route_batch (hash, probe,
  features, MLP, argmin for 131,072 pairs) -> ls_log_samples (4096 records)
  -> ls_train_step (Adam, batch 4096) -> ls_publish.
Metric: routing decisions per second (requests routed per second of whole
steps).  Inputs resident in HBM and larger than L2 (consecutive timed steps
read different device copies of the batch, 205 MB together); CUDA events on
the launching stream; W untimed warm-up steps.

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

WORKLOAD = "homogeneous"
WORKLOAD_DESC = (f"{WORKLOAD}: 32 instances x 4096 requests/step, prompts 64-4096 tokens with Zipf(1.1) "
                 "prefixes over 256 templates, 16384 cached blocks/instance, bf16 MLP 64-256-256-1, "
                 "Adam batch 4096")
INPUT_SETS = 6   # device copies of the batch the timed steps rotate over (> L2 together)
METRIC = "routing decisions/sec (requests routed per second of whole route+log+train+publish steps)"
UNIT = "decisions/s"


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=2000)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-guards", action="store_true", help="skip the guarded-route measurement")
    p.add_argument("--no-replay", action="store_true", help="skip the replay-pool admission measurement")
    p.add_argument("--no-paper-point", action="store_true", help="skip the paper operating-point measurement")
    p.add_argument("--no-training-config", action="store_true",
                   help="skip the online-training throughput configuration")
    p.add_argument("--paper-point-only", action="store_true", help="only the paper operating-point measurement")
    p.add_argument("--replay-only", action="store_true",
                   help="only the replay-pool admission measurement (for kernel profiling)")
    p.add_argument("--guards-only", action="store_true",
                   help="only the guarded-route measurement (--steps routes; for kernel profiling)")
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
    r.close()
    return {"config": "training: ring 2^20 x 128 fp32, Adam lr 3e-4, batch 4096, 128-256-256-256-1 bf16",
            "train_steps": steps, "route_calls": steps // 10, "ms": ms,
            "train_samples_per_s": steps * cfg.train_batch / (ms / 1e3),
            "routes_per_s_beside_training": (steps // 10) * cfg.n_req / (ms / 1e3)}


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


def route_costs(cfg, R, N, hits, lens, keys, key_off):
    """flops of the scorer and bytes of the prefix matcher for one batch."""
    w = cfg.widths
    flops = (mlp_flops_per_score(w) * R * N + 2 * N * cfg.d_inst * w[1] + 2 * R * cfg.d_req * w[1])
    nb = lens // 16
    need_blocks = np.minimum(nb, hits.max(axis=1) + 1)                 # blocks that must be hashed
    tok_bytes = 4 * int(np.sum(np.minimum(lens, 16 * need_blocks)))
    # distinct (instance, probed key): blocks 0..h (the miss included when h < n_r)
    pr = []
    for i in range(N):
        upto = np.minimum(hits[:, i] + 1, nb).astype(np.int64)
        tot = int(upto.sum())
        base = np.repeat(key_off[:-1], upto)
        within = np.arange(tot) - np.repeat(np.cumsum(upto) - upto, upto)
        pr.append(np.unique(keys[base + within]).size if tot else 0)
    probe_bytes = 8 * int(np.sum(pr))
    out_bytes = 4 * R * N + 8 * R
    return dict(score_flops=float(flops), prefix_bytes=float(tok_bytes + probe_bytes + out_bytes),
                tok_bytes=tok_bytes, probe_bytes=probe_bytes)


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


def profiled_traffic(kernel):
    """DRAM bytes per launch of `kernel` from the committed ncu summaries, if the
    summary was taken on the kernel's current source (else None)."""
    import glob
    if kernel not in KERNEL_SOURCES:
        return None
    sha = code_digest(KERNEL_SOURCES[kernel])
    for path in glob.glob(os.path.join(ROOT, "profiles", "*.md")):
        for line in open(path):
            if line.startswith("roofline-traffic:"):
                kv = dict(p.split("=", 1) for p in line.split()[1:])
                if kv.get("kernel") == kernel and kv.get("code_sha256") == sha:
                    return float(kv["bytes_per_launch"])
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

def oracle_work(wl, inst_keys, n_req, rng):
    """Oracle pass over a sample: route n_req requests (hash, hits, features,
    bf16 MLP, argmin) and one training step on n_req logged records."""
    import oracle
    idx = np.sort(rng.choice(len(wl.tok_off) - 1, size=n_req, replace=False))
    t0 = time.perf_counter()
    oracle.route(wl, inst_keys=inst_keys, req_idx=idx)
    tr = oracle.Trainer(wl.cfg.widths, wl.params, wl.cfg.dtype)
    bidx = rng.integers(0, len(wl.samples_y), size=n_req).astype(np.int32)
    tr.step(wl.samples_x, wl.samples_y, bidx, wl.mean, wl.std, "adam", 3e-4)
    return time.perf_counter() - t0


def oracle_work_threads(wl, inst_keys, n_req, rng, threads):
    """oracle_work with the requests split over `threads` host threads (the
    oracle's C routines release the interpreter lock, so the threads run on
    separate cores); the training step stays on one thread."""
    import concurrent.futures as cf
    import oracle
    idx = np.sort(rng.choice(len(wl.tok_off) - 1, size=n_req, replace=False))
    parts = [p for p in np.array_split(idx, threads) if len(p)]
    t0 = time.perf_counter()
    with cf.ThreadPoolExecutor(max_workers=threads) as ex:
        list(ex.map(lambda p: oracle.route(wl, inst_keys=inst_keys, req_idx=p), parts))
    tr = oracle.Trainer(wl.cfg.widths, wl.params, wl.cfg.dtype)
    bidx = rng.integers(0, len(wl.samples_y), size=n_req).astype(np.int32)
    tr.step(wl.samples_x, wl.samples_y, bidx, wl.mean, wl.std, "adam", 3e-4)
    return time.perf_counter() - t0


def cpu_baseline(wl, inst_keys, target_s):
    """The oracle on the host's cores (requests over all cores), beside its
    single-thread figure."""
    rng = np.random.default_rng(0)
    cores = os.cpu_count() or 1
    t_cal = oracle_work(wl, inst_keys, 16, rng)
    n1 = int(np.clip(16 * 0.5 * target_s / max(t_cal, 1e-3), 16, len(wl.tok_off) - 1))
    t1 = oracle_work(wl, inst_keys, n1, rng)
    n = int(min(len(wl.tok_off) - 1, max(16, n1 * cores)))   # about the same wall time if the cores scale
    t = oracle_work_threads(wl, inst_keys, n, rng, cores)
    return {"value": n / t, "unit": UNIT, "cores": cores, "kind": "oracle",
            "single_thread_value": n1 / t1,
            "sample": f"{n} of {len(wl.tok_off) - 1} requests of the {WORKLOAD} batch routed by the C oracle "
                      f"(hash, hits, features, fp64-accumulated bf16 MLP, argmin) over {cores} host threads, "
                      f"plus one Adam step on {n} logged records on one thread; {t:.1f} s (one thread: "
                      f"{n1} requests in {t1:.1f} s)"}


def run_reference(args, world, rank):
    from paper_2606_00946_gb300 import workload as W
    import oracle
    if rank != 0:
        return 0
    wl = W.generate(WORKLOAD)
    inst_keys = oracle.instance_keys(wl)
    rng = np.random.default_rng(1)
    cores = os.cpu_count() or 1
    n = 48 * max(1, cores // 4)
    for _ in range(args.warmup):
        oracle_work_threads(wl, inst_keys, n, rng, cores)
    times = [oracle_work_threads(wl, inst_keys, n, rng, cores) for _ in range(args.steps)]
    ms = 1e3 * float(np.mean(times))
    value = n / (ms / 1e3)
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded generator shaped like the paper's prefix-sharing workloads)",
            "config": {"workload": WORKLOAD_DESC, "pairs_per_step": 32 * 4096, "train_samples_per_step": 4096,
                       "parallelism": "replicas", "sample_requests_per_step": n},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": f"{n} requests over {cores} host threads + one Adam step on {n} records "
                                       f"per step"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


# ----------------------------------------------------------------------------
# GPU arm
# ----------------------------------------------------------------------------

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
    wl = W.generate(WORKLOAD)
    cfg = wl.cfg
    R, N, Bt = cfg.n_req, cfg.n_inst, cfg.train_batch
    ring = max(cfg.n_samples, 4 * Bt)
    r = H.Router.for_config(cfg, ring_capacity=ring)
    dw = H.DeviceWorkload(wl, device=dev)
    dw.load(r)
    sx = torch.from_numpy(wl.samples_x).to(dev)
    sy = torch.from_numpy(wl.samples_y).to(dev)
    r.log(sx, sy)                                   # fill the ring once
    states = [dw.inst_state, torch.from_numpy(W.instance_state(np.random.default_rng(99), cfg)).to(dev)]
    out = {"choice": torch.empty(R, dtype=torch.int32, device=dev),
           "best": torch.empty(R, dtype=torch.float32, device=dev), "scores": None, "hits": None}
    loss = torch.zeros(1, device=dev)
    flush = torch.empty(512 << 20, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)
    if args.paper_point_only:
        pp = measure_paper_point(L, H, W, dev, stream)
        if rank == 0:
            print(json.dumps({"paper_point": pp}))
        r.close()
        return 0
    if args.replay_only:
        rp = measure_replay(L, H, W, wl, dev, flush, stream, measured_peaks()[0], n=max(args.steps, 4))
        if rank == 0:
            print(json.dumps({"workload": WORKLOAD, "replay_admission": rp}))
        r.close()
        return 0
    if args.guards_only:
        g = measure_guards(L, r, dw, N, R, cfg.d, min(ring, int(r.info().ring_count)), cfg.d_req, flush, stream,
                           measured_peaks()[0], n=max(args.steps, 4))
        if rank == 0:
            print(json.dumps({"workload": WORKLOAD, "guarded_route": g}))
        r.close()
        return 0
    # the step's inputs arrive in fixed buffers (new instance state, new logged records)
    stage_state = torch.empty_like(states[0])
    stage_x = torch.empty(Bt, cfg.d, device=dev)
    stage_y = torch.empty(Bt, device=dev)

    def feed(k):
        stage_state.copy_(states[k & 1], non_blocking=True)
        a = (k * Bt) % len(wl.samples_y)
        stage_x.copy_(sx[a:a + Bt], non_blocking=True)
        stage_y.copy_(sy[a:a + Bt], non_blocking=True)

    side = torch.cuda.Stream(dev)  # training runs beside routing (Sec. 4.3.1: off the routing path)
    # device copies of the batch, larger than L2 together: consecutive steps
    # read their prompts from different copies, so every step's inputs come
    # from HBM (no L2 flush needed between steps)
    n_sets = INPUT_SETS
    sets = [(dw.tok, dw.tok_off, dw.req_feats)] + [
        (dw.tok.clone(), dw.tok_off.clone(), dw.req_feats.clone()) for _ in range(n_sets - 1)]
    set_bytes = sum(t.numel() * t.element_size() for t in sets[0])

    def body(ks=0):
        tok, tok_off, req = sets[ks]
        main = torch.cuda.current_stream(dev)
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
        body(k % n_sets)

    for k in range(args.warmup):
        eager_step(k)
    torch.cuda.synchronize()
    graphs = [H.StepGraph(lambda ks=ks: body(ks)) for ks in range(n_sets)]  # the step's ABI calls, recorded once

    def step(k):
        feed(k)
        graphs[k % n_sets].replay()

    for k in range(args.warmup):
        step(args.warmup + k)
    torch.cuda.synchronize()
    # per-pair hits of this batch (for the algorithmic byte count; not timed)
    chk = r.route(dw.tok, dw.tok_off, dw.req_feats, N)
    hits = chk["hits"].cpu().numpy()
    keys, ko = r.hash_blocks(dw.tok, dw.tok_off)
    costs = route_costs(cfg, R, N, hits, np.diff(wl.tok_off), keys.cpu().numpy(), ko.cpu().numpy())

    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        pass
    clocks = ClockSampler(uuid)
    cudart = torch.cuda.cudart()

    def timed_pass(fn, k0, n=None):
        # steps issued back to back, an event between consecutive steps: the
        # host stays ahead of the GPU, so each interval is one step's device time
        n = args.steps if n is None else n
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(n + 1)]
        ev[0].record(stream)
        for k in range(n):
            fn(k0 + k)
            ev[k + 1].record(stream)
        ev[n].synchronize()
        return [ev[k].elapsed_time(ev[k + 1]) for k in range(n)]

    # timed region: K whole steps (graph replays), no per-kernel instrumentation
    barrier(world)
    torch.cuda.synchronize()
    clocks.start()
    cudart.cudaProfilerStart()                      # brackets the region for ncu --profile-from-start off
    times = timed_pass(step, 2 * args.warmup)
    cudart.cudaProfilerStop()
    torch.cuda.synchronize()
    clk = clocks.stop()
    # the same K steps issued call by call (no graph), for comparison
    eager_times = timed_pass(eager_step, 2 * args.warmup + args.steps)
    # and steps issued call by call with every kernel launch bracketed by CUDA
    # events on its launching stream: per-kernel device time for the roofline
    L.ls_trace_enable(r.h, True)
    L.ls_trace_read(r.h)
    torch.cuda.synchronize()
    n_traced = min(args.steps, 120)                 # every launch gets events from the tracer's pool

    # each traced step behind a ~150 us spin on the GPU, so that the host has
    # queued the whole step before it starts and no kernel interval includes
    # host time; the step's interval excludes the spin
    tev = []
    for k in range(n_traced):
        torch.cuda._sleep(300000)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        eager_step(2 * args.warmup + 2 * args.steps + k)
        e1.record(stream)
        tev.append((e0, e1))
    torch.cuda.synchronize()
    traced_times = [a.elapsed_time(b) for a, b in tev]
    torch.cuda.synchronize()
    rc, trace = L.ls_trace_read(r.h)
    L.ls_trace_enable(r.h, False)
    barrier(world)
    ms = max_over_ranks(world, float(np.mean(times)), dev if world > 1 and torch.distributed.get_backend() == "nccl" else None)
    value = world * R / (ms / 1e3)

    # roofline of the dominant kernel: the largest device time per step on the
    # step's critical branch (snapshot + route runs beside log + train, and is
    # the longer branch); the training branch's largest kernel is reported too
    peaks, peak_src = measured_peaks()
    per = {k: v[1] / max(v[2], 1) for k, v in trace.items()}          # ms per timed launch
    per_step = {k: per[k] * v[0] / n_traced for k, v in trace.items()}  # ms per step
    n_per_step = {k: v[0] / n_traced for k, v in trace.items()}         # launches per step
    launches = int(round(sum(v[0] for v in trace.values()) * args.steps / n_traced))
    timing = ("kernel durations from CUDA events around each launch over steps issued call by call "
              "(instrumented); value and ms_per_step from the K graph replays")

    def kernel_roofline(k):
        d_pad = 64 * ((cfg.d + 63) // 64)
        if k in ("prefix_index", "prefix_match"):
            alg, peak, unit, bound = costs["prefix_bytes"] / 1e9, peaks["hbm_gbs"], "GB/s", "hbm"
        elif k == "features":     # feature image written + hits and offsets read
            alg = (R * N * (2 * d_pad + 4) + R * 8) / 1e9
            peak, unit, bound = peaks["hbm_gbs"], "GB/s", "hbm"
        elif k in ("score_simt", "score_tc"):
            alg, peak, unit, bound = costs["score_flops"] / 1e12, peaks["bf16_tflops"], "TFLOP/s", "tensor"
        else:                      # training products: the kind's flops per step over its launches per step
            # forward launches: every layer's product plus the output layer's dW
            # (in the last hidden layer's epilogue); dW + dX launches for hidden
            # layers l >= 1; the dW-only launch for layer 0
            w, Bk = cfg.widths, Bt
            nh = len(w) - 2
            per_kind = {"gemm_tc_fwd": sum(2 * Bk * w[l] * w[l + 1] for l in range(nh + 1)) + 2 * Bk * w[nh],
                        "gemm_tc_dx": sum(4 * Bk * w[l] * w[l + 1] for l in range(1, nh)),
                        "gemm_tc_dw": 2 * Bk * w[0] * w[1]}
            alg = per_kind.get(k, 0.0) / max(n_per_step[k], 1e-9) / 1e12
            peak, unit, bound = peaks["bf16_tflops"], "TFLOP/s", "tensor"
        achieved = alg / (per[k] / 1e3)
        return {"kernel": k, "bound": bound, "achieved": achieved, "peak": peak, "unit": unit,
                "frac": achieved / peak, "traffic": profiled_traffic(k),
                "peak_source": f"{peak_src} (burst)", "avg_launch_ms": per[k], "timing": timing}

    route_kernels = [k for k in per_step if k in ("prefix_index", "prefix_match", "hash_screen", "probe_walk",
                                                  "features", "score_tc", "score_simt", "argmin")]
    dom = max(route_kernels, key=lambda k: per_step[k])
    roofline = dict(kernel_roofline(dom), branch="route (the step's critical branch)")
    route_rooflines = {k: kernel_roofline(k) for k in route_kernels}
    train_kernels = [k for k in per_step if k in ("gemm_tc_fwd", "gemm_tc_dw", "gemm_tc_dx")]
    train_roofline = (dict(kernel_roofline(max(train_kernels, key=lambda k: per_step[k])), branch="train")
                      if train_kernels else None)

    training_config = None
    if not args.no_training_config:
        training_config = measure_training_config(L, H, W, dev)
    paper_point = None
    if not args.no_paper_point:
        paper_point = measure_paper_point(L, H, W, dev, stream)
    replay = None
    if not args.no_replay:
        replay = measure_replay(L, H, W, wl, dev, flush, stream, peaks)
    guards = None
    if not args.no_guards:
        guards = measure_guards(L, r, dw, N, R, cfg.d, min(ring, int(r.info().ring_count)), cfg.d_req, flush,
                                stream, peaks)

    # end to end through the C ABI with host buffers: every step copies its
    # inputs from pinned host memory and reads its results back.  The copies
    # of step k+1 run on a copy stream while step k computes (the host link,
    # ~205 GB/s, is the limit: 35 MB of prompt tokens per step); four device
    # input sets (140 MB, larger than L2) rotate, each with its own captured
    # graph of the step's ABI calls.
    e2e = None
    if not args.no_e2e:
        h_tok = torch.from_numpy(wl.tok).pin_memory()
        h_off = torch.from_numpy(wl.tok_off).pin_memory()
        h_req = torch.from_numpy(wl.req_feats).pin_memory()
        h_st = [s.cpu().pin_memory() for s in states]
        h_x = torch.from_numpy(wl.samples_x).pin_memory()
        h_y = torch.from_numpy(wl.samples_y).pin_memory()
        NB = 4
        sets = [{"tok": torch.empty_like(dw.tok), "off": torch.empty_like(dw.tok_off),
                 "req": torch.empty_like(dw.req_feats), "st": torch.empty_like(states[0]),
                 "x": torch.empty(Bt, cfg.d, device=dev), "y": torch.empty(Bt, device=dev)} for _ in range(NB)]
        h_choice = torch.empty(R, dtype=torch.int32).pin_memory()
        h_best = torch.empty(R, dtype=torch.float32).pin_memory()
        h_loss = torch.empty(1).pin_memory()
        d0 = sets[0]
        h2d = d0["tok"].numel() * 4 + d0["off"].numel() * 8 + d0["req"].numel() * 4 + d0["st"].numel() * 4 + \
            d0["x"].numel() * 4 + d0["y"].numel() * 4
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
            a = (k * Bt) % len(wl.samples_y)
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

        for k in range(args.warmup):
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
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        cs.wait_stream(stream)
        e0.record(stream)
        run_pipelined(2 * NB, args.steps)
        e1.record(stream)
        e1.synchronize()
        ems_pipe = e0.elapsed_time(e1) / args.steps
        # the same steps one at a time (copy in, step, copy out; L2 flushed between)
        et = []
        for k in range(min(args.steps, 200)):
            flush.fill_(k & 0xFF)
            b = k % NB
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            copy_in(k, sets[b])
            graphs[b].replay()
            copy_out()
            e1.record(stream)
            e1.synchronize()
            et.append(e0.elapsed_time(e1))
        ems = max_over_ranks(world, ems_pipe, None)
        e2e = {"value": world * R / (ems / 1e3), "unit": UNIT, "h2d_bytes_per_step": int(h2d),
               "d2h_bytes_per_step": int(d2h), "ms_per_step": ems,
               "pipelined": "inputs of step k+1 copied on a copy stream while step k computes; 4 device "
                            "input sets with a captured graph each; results read back every step",
               "ms_per_step_one_at_a_time": float(np.mean(et))}

    status = r.sync()
    if status != L.LS_OK:
        print(json.dumps({"error": f"device status {status}"}), file=sys.stderr)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        cpu = cpu_baseline(wl, oracle.instance_keys(wl), args.cpu_seconds)

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (seeded generator shaped like the paper's prefix-sharing workloads)",
            "config": {"workload": WORKLOAD_DESC,
                       "pairs_per_step": R * N, "train_samples_per_step": Bt,
                       "l2": f"inputs larger than L2: consecutive steps read {n_sets} rotating device copies of "
                             f"the batch ({n_sets * set_bytes / 1e6:.0f} MB in all, L2 129 MB); no flush",
                       "parallelism": "replicas"},
            "train_samples_per_s": world * Bt / (ms / 1e3),
            "scores_per_s": world * R * N / (ms / 1e3),
            "roofline": roofline,
            "train_roofline": train_roofline,
            "kernels_ms_per_step": {k: per_step[k] for k in sorted(per_step, key=lambda k: -per_step[k])},
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": launches,
            "launch": "each step: the new instance state and records copied into the step's buffers, then "
                      "one replay of a CUDA graph of the step's ABI calls recorded once per device copy of the "
                      "batch (steps rotate over the copies): snapshot + route on one branch, log + train on a "
                      "second, joined before the publish; kernels of each chain launched with programmatic "
                      "dependent launch",
            "ms_per_step_eager": float(np.mean(eager_times)),
            "ms_per_step_instrumented": float(np.mean(traced_times)),
            "instrumented_steps": n_traced,
            "gpu_launches_per_step": launches / args.steps,
            "clocks": clk,
            "algorithmic": costs,
            "guarded_route": guards,
            "replay_admission": replay,
            "route_rooflines": route_rooflines,
            "paper_point": paper_point,
            "training_config": training_config,
        }
        print(json.dumps(line))
    r.close()
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
