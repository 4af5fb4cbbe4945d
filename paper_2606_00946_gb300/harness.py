"""Device staging of seeded workloads and a small object wrapper over the ABI.

`Router` owns one library context and raises LodestarError on a failing
status.  `DeviceWorkload` copies a `workload.Workload` to the GPU and builds
each instance's key list with the library's own block hash (ls_hash_blocks),
so the CUDA path never sees a key computed elsewhere.
"""
from __future__ import annotations

import numpy as np
import torch

from . import lodestar as L
from .workload import BLOCK, Workload


def key_offsets(tok_off: torch.Tensor) -> torch.Tensor:
    """CSR offsets of block keys (floor(L/16) per sequence), int64 on tok_off's device."""
    lens = tok_off[1:] - tok_off[:-1]
    ko = torch.zeros_like(tok_off)
    ko[1:] = torch.cumsum(lens // BLOCK, 0)
    return ko


class Router:
    """One library context.  Methods mirror the ABI and raise on error."""

    def __init__(self, widths, d_inst, d_req, dtype="bf16", **caps):
        self.cfg = L.make_config(widths, d_inst, d_req, dtype, **caps)
        rc, h = L.ls_create(self.cfg)
        L.check(rc)
        self.h = h
        self._norm = None
        self.widths = list(widths)
        self.dtype = dtype
        self.n_params = L.ls_param_count(self.cfg)

    @classmethod
    def for_config(cls, cfg, **caps):
        base = dict(max_instances=cfg.n_inst, max_requests=cfg.n_req,
                    max_keys_per_instance=cfg.cache_blocks, max_load=0.5,
                    ring_capacity=max(cfg.n_samples, 1024), max_train_batch=cfg.train_batch,
                    max_batch_tokens=cfg.n_req * cfg.max_len)
        base.update(caps)
        return cls(cfg.widths, cfg.d_inst, cfg.d_req, cfg.dtype, **base)

    def close(self):
        if getattr(self, "h", None):
            L.ls_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # --- ABI -----------------------------------------------------------------
    def sync(self):
        return L.ls_sync_status(self.h)

    def info(self):
        rc, info = L.ls_get_info(self.h)
        L.check(rc)
        return info

    def set_params(self, params: torch.Tensor, stream=None):
        L.check(L.ls_set_params(self.h, params, stream))

    def get_params(self, stream=None) -> torch.Tensor:
        out = torch.empty(self.n_params, dtype=torch.float32, device="cuda")
        L.check(L.ls_get_params(self.h, out, stream))
        return out

    def get_opt_state(self, stream=None):
        m = torch.empty(self.n_params, dtype=torch.float32, device="cuda")
        v = torch.empty(self.n_params, dtype=torch.float32, device="cuda")
        rc, step = L.ls_get_opt_state(self.h, m, v, stream)
        L.check(rc)
        return m, v, step

    def set_opt_state(self, m, v, step, stream=None):
        L.check(L.ls_set_opt_state(self.h, m, v, int(step), stream))

    def set_normalizer(self, mean, std, stream=None):
        L.check(L.ls_set_normalizer(self.h, mean, std, stream))
        self._norm = (mean.detach().clone(), std.detach().clone())

    def save_checkpoint(self, path):
        """Master weights, Adam moments, step count and normaliser to an .npz."""
        if self._norm is None:
            raise ValueError("set_normalizer has not been called")
        m, v, step = self.get_opt_state()
        mean, std = self._norm
        np.savez(path, params=self.get_params().cpu().numpy(), m=m.cpu().numpy(), v=v.cpu().numpy(),
                 step=np.int64(step), mean=mean.cpu().numpy(), std=std.cpu().numpy())

    def load_checkpoint(self, path, publish=True):
        """Restore what save_checkpoint wrote; the next training step continues
        the saved run (same bits, given the same records and minibatch)."""
        z = np.load(path)
        t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
        self.set_normalizer(t(z["mean"]), t(z["std"]))
        self.set_params(t(z["params"]))
        self.set_opt_state(t(z["m"]), t(z["v"]), int(z["step"]))
        if publish:
            self.publish()

    def snapshot(self, n_inst, inst_state, keys=None, key_off=None, mode=L.LS_REPLACE, stream=None):
        n_keys = int(keys.numel()) if keys is not None else 0
        L.check(L.ls_snapshot_update(self.h, n_inst, inst_state, keys, key_off, n_keys, mode, stream))

    def hash_blocks(self, tok: torch.Tensor, tok_off: torch.Tensor, stream=None):
        ko = key_offsets(tok_off)
        keys = torch.zeros(max(int(ko[-1].item()), 1), dtype=torch.int64, device=tok.device)
        L.check(L.ls_hash_blocks(self.h, tok_off.numel() - 1, tok, tok_off, keys, ko, stream))
        return keys[: int(ko[-1].item())], ko

    def features(self, tok_off, hits, req_feats, stream=None):
        n_req, n_inst = hits.shape
        x = torch.empty(n_req * n_inst, self.widths[0], dtype=torch.float32, device="cuda")
        L.check(L.ls_assemble_features(self.h, n_req, tok_off, hits, req_feats, x, stream))
        return x

    def route(self, tok, tok_off, req_feats, n_inst, want_scores=True, want_hits=True, stream=None,
              out=None):
        n_req = tok_off.numel() - 1
        o = out or {}
        choice = o.get("choice", torch.empty(n_req, dtype=torch.int32, device="cuda"))
        best = o.get("best", torch.empty(n_req, dtype=torch.float32, device="cuda"))
        scores = o.get("scores") if "scores" in o else (
            torch.empty(n_req, n_inst, dtype=torch.float32, device="cuda") if want_scores else None)
        hits = o.get("hits") if "hits" in o else (
            torch.empty(n_req, n_inst, dtype=torch.int32, device="cuda") if want_hits else None)
        rc, ver = L.ls_route_batch(self.h, n_req, tok, tok_off, req_feats, choice, best, scores, hits,
                                   stream)
        L.check(rc)
        return dict(choice=choice, best=best, scores=scores, hits=hits, version=ver)

    def route_guarded(self, tok, tok_off, req_feats, n_inst, want_scores=True, want_hits=True, stream=None,
                      out=None):
        """Guarded route (Algorithm 4): adds a per-request status."""
        n_req = tok_off.numel() - 1
        o = out or {}
        choice = o.get("choice", torch.empty(n_req, dtype=torch.int32, device="cuda"))
        best = o.get("best", torch.empty(n_req, dtype=torch.float32, device="cuda"))
        status = o.get("status", torch.empty(n_req, dtype=torch.int32, device="cuda"))
        fallback = o.get("fallback", torch.empty(n_req, dtype=torch.int32, device="cuda"))
        scores = o.get("scores") if "scores" in o else (
            torch.empty(n_req, n_inst, dtype=torch.float32, device="cuda") if want_scores else None)
        hits = o.get("hits") if "hits" in o else (
            torch.empty(n_req, n_inst, dtype=torch.int32, device="cuda") if want_hits else None)
        rc, ver = L.ls_route_batch_guarded(self.h, n_req, tok, tok_off, req_feats, choice, best, status,
                                           fallback, scores, hits, stream)
        L.check(rc)
        return dict(choice=choice, best=best, status=status, fallback=fallback, scores=scores, hits=hits,
                    version=ver)

    def route_sequential(self, tok, tok_off, req_feats, n_inst, queue_col=0, stream=None):
        """Sequential-commit route: each decision updates the chosen instance's
        queue and cache before the next request is scored."""
        n_req = tok_off.numel() - 1
        choice = torch.empty(n_req, dtype=torch.int32, device="cuda")
        best = torch.empty(n_req, dtype=torch.float32, device="cuda")
        scores = torch.empty(n_req, n_inst, dtype=torch.float32, device="cuda")
        hits = torch.empty(n_req, n_inst, dtype=torch.int32, device="cuda")
        rc, ver = L.ls_route_sequential(self.h, n_req, tok, tok_off, req_feats, queue_col, choice, best, scores,
                                        hits, stream)
        L.check(rc)
        return dict(choice=choice, best=best, scores=scores, hits=hits, version=ver)

    def replay_admit(self, diag=False, stream=None):
        """One admission round of the replay pool; with diag, returns (d, n)
        per candidate / kept slot (device tensors of the pools' capacities)."""
        d = n = None
        if diag:
            d = torch.empty(max(int(self.cfg.pending_capacity), 1), dtype=torch.float32, device="cuda")
            n = torch.empty(max(int(self.cfg.replay_capacity), 1), dtype=torch.float32, device="cuda")
        L.check(L.ls_replay_admit(self.h, d, n, stream))
        return (d, n) if diag else None

    def replay(self):
        """Records in the replay pool: (x [n, d], y [n])."""
        cap = max(int(self.cfg.replay_capacity), 1)
        x = torch.empty(cap, self.widths[0], dtype=torch.float32, device="cuda")
        y = torch.empty(cap, dtype=torch.float32, device="cuda")
        rc, n = L.ls_get_replay(self.h, x, y)
        L.check(rc)
        return x[:n], y[:n]

    def set_guards(self, **kw):
        L.check(L.ls_set_guards(self.h, **kw))

    def refresh_bounds(self, stream=None):
        L.check(L.ls_refresh_bounds(self.h, stream))

    def bounds(self, which=1):
        lo = torch.empty(self.widths[0], dtype=torch.float32, device="cuda")
        hi = torch.empty_like(lo)
        L.check(L.ls_get_bounds(self.h, which, lo, hi))
        return lo, hi

    def log(self, feats, ttft, stream=None):
        L.check(L.ls_log_samples(self.h, ttft.numel(), feats, ttft, stream))

    def train(self, batch, idx=None, opt="adam", lr=3e-4, loss_out=None, stream=None):
        L.check(L.ls_train_step(self.h, batch, idx, L.LS_ADAM if opt == "adam" else L.LS_SGD, lr,
                                loss_out, stream))

    def publish(self, stream=None):
        L.check(L.ls_publish(self.h, stream))


class StepGraph:
    """ABI calls of one step recorded once by stream capture, then replayed.

    `body` issues the calls (on the current stream, which is the capture stream
    while recording); every pointer it passes is baked into the graph, so new
    inputs of a step are copied into the same buffers before `replay()`.  The
    library keeps its per-step counters on the device, so a replay behaves
    like issuing the calls again.  Run `body` eagerly at least once first
    (kernel loading and shared-memory attributes happen outside capture).
    """

    def __init__(self, body, stream=None):
        self.graph = torch.cuda.CUDAGraph()
        s = stream if stream is not None else torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.graph(self.graph, stream=s):
            body()
        torch.cuda.current_stream().wait_stream(s)

    def replay(self):
        self.graph.replay()


class DeviceWorkload:
    """A workload's arrays resident in HBM, plus each instance's key CSR."""

    def __init__(self, wl: Workload, device="cuda"):
        self.wl = wl
        self.device = device
        t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(device)
        self.tok = t(wl.tok)
        self.tok_off = t(wl.tok_off)
        self.req_feats = t(wl.req_feats)
        self.inst_state = t(wl.inst_state)
        self.mean = t(wl.mean)
        self.std = t(wl.std)
        self.params = t(wl.params)
        self.n_inst = wl.cfg.n_inst
        self.inst_keys = None
        self.inst_key_off = None

    def build_instance_keys(self, router: Router):
        """Instance i's keys: the first k block keys of each cached sequence it
        holds (hashed by the library), then its random stand-in keys."""
        wl = self.wl
        seq_tok = torch.from_numpy(wl.seq_tok).to(self.device)
        seq_off = torch.from_numpy(wl.seq_off).to(self.device)
        seq_keys, sko = router.hash_blocks(seq_tok, seq_off)
        del seq_tok
        chain_seq = torch.from_numpy(wl.chain_seq.astype(np.int64)).to(self.device)
        chain_k = torch.from_numpy(wl.chain_blocks.astype(np.int64)).to(self.device)
        starts = sko[chain_seq]
        total = int(chain_k.sum().item())
        excl = torch.cumsum(chain_k, 0) - chain_k
        within = torch.arange(total, device=self.device) - torch.repeat_interleave(excl, chain_k)
        chain_keys = seq_keys[torch.repeat_interleave(starts, chain_k) + within]
        del seq_keys, within
        ck_off = torch.zeros(len(chain_k) + 1, dtype=torch.int64, device=self.device)
        ck_off[1:] = torch.cumsum(chain_k, 0)
        ck_off_h = ck_off.cpu().numpy()
        rand = torch.from_numpy(wl.rand_keys.view(np.int64)).to(self.device)
        parts, off = [], [0]
        for i in range(wl.cfg.n_inst):
            a, b = ck_off_h[wl.inst_chain_off[i]], ck_off_h[wl.inst_chain_off[i + 1]]
            ra, rb = wl.inst_rand_off[i], wl.inst_rand_off[i + 1]
            parts.append(chain_keys[a:b])
            parts.append(rand[ra:rb])
            off.append(off[-1] + (b - a) + (rb - ra))
        self.inst_keys = torch.cat(parts) if parts else torch.zeros(0, dtype=torch.int64,
                                                                    device=self.device)
        self.inst_key_off = torch.tensor(off, dtype=torch.int64, device=self.device)
        return self.inst_keys, self.inst_key_off

    def load(self, router: Router, publish=True):
        """Normaliser, snapshot (state + keys), weights; publish once."""
        router.set_normalizer(self.mean, self.std)
        if self.inst_keys is None:
            self.build_instance_keys(router)
        router.snapshot(self.n_inst, self.inst_state, self.inst_keys, self.inst_key_off)
        router.set_params(self.params)
        if publish:
            router.publish()
        return router
