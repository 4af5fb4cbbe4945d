"""Plain CPU oracle of the Lodestar routing hot path -- test infrastructure.

Only the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The CUDA library never does, and this
package imports nothing from it.

The arithmetic lives in ``lodestar_oracle.c`` (scalar loops, fp64
accumulation); this module compiles it with gcc on first use and wraps each
function for numpy arrays.  Paper sections each function follows are cited in
the C source.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "lodestar_oracle.c")
_OUT = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT, "liboracle.so")
_lock = threading.Lock()
_lib = None

F64, F32, BF16 = 0, 1, 2
SGD, ADAM = 0, 1
BLOCK = 16
MODES = {"f64": F64, "f32": F32, "bf16": BF16}


def build(force: bool = False) -> str:
    """Compile the oracle (gcc, no FMA contraction, no fast-math)."""
    os.makedirs(_OUT, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-std=c11", "-O2", "-fPIC", "-shared", "-ffp-contract=off",
           "-fno-fast-math", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def lib():
    global _lib
    with _lock:
        if _lib is None:
            L = C.CDLL(build())
            P = C.c_void_p
            i64, i32, dbl = C.c_int64, C.c_int32, C.c_double
            L.or_mix64.restype = C.c_uint64
            L.or_mix64.argtypes = [C.c_uint64]
            L.or_block_content.restype = C.c_uint64
            L.or_block_content.argtypes = [P]
            L.or_hash_blocks.argtypes = [i64, P, P, P, P]
            L.or_prefix_hits.argtypes = [i64, P, P, i32, P, P, P]
            L.or_prefix_hits_by_marking.argtypes = [i64, P, P, i32, P, P, P]
            L.or_prefix_hits_sorted.argtypes = [i64, P, P, i32, P, P, P]
            L.or_raw_features_row.argtypes = [i64, i32, P, C.c_int, P, C.c_int, P]
            L.or_raw_features_row.restype = None
            L.or_features.argtypes = [i64, i32, P, P, P, C.c_int, P, C.c_int, P, P, P]
            L.or_bf16.restype = C.c_float
            L.or_bf16.argtypes = [C.c_float]
            L.or_param_count.restype = i64
            L.or_param_count.argtypes = [C.c_int, P]
            L.or_mlp_forward.argtypes = [C.c_int, C.c_int, P, P, i64, P, P]
            L.or_mlp_forward_bounds.argtypes = [C.c_int, C.c_int, P, P, i64, P, P, P, P]
            L.or_argmin.argtypes = [i64, i32, P, P, P]
            L.or_ring_append.argtypes = [i64, C.c_int, P, P, i64, i64, P, P]
            L.or_train_step.argtypes = [C.c_int, C.c_int, P, P, P, P, i64, C.c_int, dbl,
                                        C.c_int, P, P, P, P, P, P, P, C.c_float, C.c_uint64]
            L.or_drop_keep.restype = C.c_int
            L.or_drop_keep.argtypes = [C.c_uint64, C.c_float, i64, C.c_int, i64, C.c_int]
            L.or_loss.argtypes = [C.c_int, C.c_int, P, P, C.c_int, P, P, P, P, P, P]
            L.or_ring_bounds.argtypes = [i64, C.c_int, P, i64, P, P]
            L.or_hrw_candidates.restype = i32
            L.or_hrw_candidates.argtypes = [C.c_uint64, i32, i32, P]
            L.or_replay_embed.argtypes = [C.c_int, C.c_int, P, P, i64, P, P, P, P, P]
            L.or_replay_distances.argtypes = [i64, P, i64, P, C.c_int, P, P]
            L.or_replay_select.argtypes = [i64, P, i64, P, i64, P, P]
            L.or_route_sequential.argtypes = [C.c_int, C.c_int, P, P, i64, P, P, P, i32, P, P, P, C.c_int, P,
                                              C.c_int, P, P, i32, P, P, P, P]
            L.or_heuristic.argtypes = [i64, i32, P, P, P, C.c_int, C.c_int, C.c_int, C.c_int, C.c_float,
                                       C.c_float, C.c_float, P]
            L.or_guards.argtypes = [i64, i32, P, P, P, P, C.c_int, P, C.c_int, P, P, P, i64, i64,
                                    C.c_int, i32, i32, C.c_float, C.c_float, P, P, P]
            _lib = L
    return _lib


def _p(a: np.ndarray):
    return a.ctypes.data_as(C.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def _check(rc, what):
    if rc != 0:
        raise RuntimeError(f"oracle {what} failed ({rc})")


# --------------------------------------------------------------------------
# hashing and prefix hits
# --------------------------------------------------------------------------

def mix64(z: int) -> int:
    return int(lib().or_mix64(C.c_uint64(z & (2**64 - 1))))


def block_content(tokens16) -> int:
    t = _c(tokens16, np.int32)
    assert t.size == BLOCK
    return int(lib().or_block_content(_p(t)))


def key_offsets(tok_off) -> np.ndarray:
    """CSR offsets of block keys: floor(L/16) keys per sequence."""
    L = np.diff(np.asarray(tok_off, np.int64))
    off = np.zeros(len(L) + 1, np.int64)
    off[1:] = np.cumsum(L // BLOCK)
    return off


def hash_blocks(tok, tok_off):
    """Returns (keys uint64 [sum floor(L/16)], key_off int64 [n+1])."""
    tok = _c(tok, np.int32)
    tok_off = _c(tok_off, np.int64)
    koff = key_offsets(tok_off)
    keys = np.zeros(max(int(koff[-1]), 1), np.uint64)
    _check(lib().or_hash_blocks(len(tok_off) - 1, _p(tok), _p(tok_off), _p(keys), _p(koff)), "hash")
    return keys[: koff[-1]], koff


def prefix_hits(req_keys, req_key_off, inst_keys, inst_key_off, by_marking: bool = False, threads: int = 1):
    """h[r, i]; threads > 1 splits the instances over host threads (each a
    separate call on its own instances; the result does not depend on it)."""
    rk = _c(req_keys, np.uint64) if len(req_keys) else np.zeros(1, np.uint64)
    rko = _c(req_key_off, np.int64)
    ik = _c(inst_keys, np.uint64) if len(inst_keys) else np.zeros(1, np.uint64)
    iko = _c(inst_key_off, np.int64)
    R, N = len(rko) - 1, len(iko) - 1
    fn = lib().or_prefix_hits_by_marking if by_marking else lib().or_prefix_hits
    if threads > 1 and N > 1:
        import concurrent.futures as cf
        groups = [g for g in np.array_split(np.arange(N), threads) if len(g)]

        def part(g):
            a, b = int(g[0]), int(g[-1]) + 1
            sub_off = _c(iko[a:b + 1] - iko[a], np.int64)
            sub = _c(ik[iko[a]:iko[b]], np.uint64) if iko[b] > iko[a] else np.zeros(1, np.uint64)
            h = np.zeros((R, b - a), np.int32)
            _check(fn(R, _p(rk), _p(rko), b - a, _p(sub), _p(sub_off), _p(h)), "prefix_hits")
            return h

        with cf.ThreadPoolExecutor(max_workers=len(groups)) as ex:
            return np.concatenate(list(ex.map(part, groups)), axis=1)
    hits = np.zeros((R, N), np.int32)
    _check(fn(R, _p(rk), _p(rko), N, _p(ik), _p(iko), _p(hits)), "prefix_hits")
    return hits


def sorted_instance_keys(inst_keys):
    """Each instance's key set sorted ascending (CSR), built once like the
    router's snapshot tables; route() then probes it without re-sorting."""
    ik, iko = inst_keys
    out = np.empty_like(ik)
    for i in range(len(iko) - 1):
        out[iko[i]:iko[i + 1]] = np.sort(ik[iko[i]:iko[i + 1]])
    return out, iko


def prefix_hits_sorted(req_keys, req_key_off, sorted_keys):
    rk = _c(req_keys, np.uint64) if len(req_keys) else np.zeros(1, np.uint64)
    rko = _c(req_key_off, np.int64)
    sk, sko = sorted_keys
    sk = _c(sk, np.uint64) if len(sk) else np.zeros(1, np.uint64)
    sko = _c(sko, np.int64)
    R, N = len(rko) - 1, len(sko) - 1
    hits = np.zeros((R, N), np.int32)
    _check(lib().or_prefix_hits_sorted(R, _p(rk), _p(rko), N, _p(sk), _p(sko), _p(hits)), "prefix_hits_sorted")
    return hits


def instance_keys(wl, seq_keys=None, seq_key_off=None):
    """Key multiset of every instance of a workload: the oracle's own hash of
    the cached chains (first k blocks of a cached sequence) plus the
    workload's random stand-in keys.  Returns (keys, off) CSR."""
    if seq_keys is None:
        seq_keys, seq_key_off = hash_blocks(wl.seq_tok, wl.seq_off)
    parts, off = [], [0]
    N = len(wl.inst_chain_off) - 1
    for i in range(N):
        ks = []
        for c in range(int(wl.inst_chain_off[i]), int(wl.inst_chain_off[i + 1])):
            s, k = int(wl.chain_seq[c]), int(wl.chain_blocks[c])
            ks.append(seq_keys[seq_key_off[s]: seq_key_off[s] + k])
        ks.append(wl.rand_keys[wl.inst_rand_off[i]: wl.inst_rand_off[i + 1]])
        kk = np.concatenate(ks) if ks else np.zeros(0, np.uint64)
        parts.append(kk)
        off.append(off[-1] + len(kk))
    return (np.concatenate(parts).astype(np.uint64) if parts else np.zeros(0, np.uint64),
            np.asarray(off, np.int64))


# --------------------------------------------------------------------------
# features, predictor, selection
# --------------------------------------------------------------------------

def raw_features_row(L: int, h: int, inst, req) -> np.ndarray:
    """Raw (un-normalised) feature row of one (request, instance) pair."""
    inst = _c(inst, np.float32).ravel()
    req = _c(req, np.float32).ravel()
    x = np.zeros(6 + inst.size + req.size, np.float32)
    one = np.zeros(1, np.float32)
    lib().or_raw_features_row(int(L), int(h), _p(inst if inst.size else one), inst.size,
                              _p(req if req.size else one), req.size, _p(x))
    return x


def features(L, hits, inst_state, req_feats, mean, std):
    """Normalised features [R*N, d] (row r*N + i)."""
    L = _c(L, np.int64)
    hits = _c(hits, np.int32)
    inst = _c(inst_state, np.float32)
    req = _c(req_feats, np.float32)
    R, N = hits.shape
    d_inst, d_req = inst.shape[1], (req.shape[1] if req.ndim == 2 else 0)
    d = 6 + d_inst + d_req
    out = np.zeros((R * N, d), np.float32)
    reqp = req if req.size else np.zeros(1, np.float32)
    _check(lib().or_features(R, N, _p(L), _p(hits), _p(inst), d_inst, _p(reqp), d_req,
                             _p(_c(mean, np.float32)), _p(_c(std, np.float32)), _p(out)),
           "features")
    return out


def bf16(x) -> np.ndarray:
    f = np.vectorize(lambda v: lib().or_bf16(float(v)), otypes=[np.float32])
    return f(np.asarray(x, np.float32))


def param_count(widths) -> int:
    w = _c(widths, np.int32)
    return int(lib().or_param_count(len(w) - 1, _p(w)))


def mlp_forward(mode, widths, params, x) -> np.ndarray:
    mode = MODES.get(mode, mode)
    w = _c(widths, np.int32)
    p = _c(params, np.float64)
    x = _c(x, np.float64).reshape(-1, w[0])
    y = np.zeros(x.shape[0], np.float64)
    _check(lib().or_mlp_forward(mode, len(w) - 1, _p(w), _p(p), x.shape[0], _p(x), _p(y)), "mlp")
    return y


def mlp_forward_bounds(mode, widths, params, x):
    """Forward pass plus, per row, the fp32-accumulation error bound and the
    bf16 rounding-flip sensitivity (or_mlp_forward_bounds).  Returns (y, ebound, flip)."""
    mode = MODES.get(mode, mode)
    w = _c(widths, np.int32)
    p = _c(params, np.float64)
    x = _c(x, np.float64).reshape(-1, w[0])
    y = np.zeros(x.shape[0], np.float64)
    eb = np.zeros(x.shape[0], np.float64)
    fl = np.zeros(x.shape[0], np.float64)
    _check(lib().or_mlp_forward_bounds(mode, len(w) - 1, _p(w), _p(p), x.shape[0], _p(x), _p(y), _p(eb), _p(fl)),
           "mlp bounds")
    return y, eb, fl


def argmin(scores):
    s = _c(scores, np.float32)
    R, N = s.shape
    choice = np.zeros(R, np.int32)
    best = np.zeros(R, np.float32)
    _check(lib().or_argmin(R, N, _p(s), _p(choice), _p(best)), "argmin")
    return choice, best


def route(wl, hits=None, inst_keys=None, params=None, mode=None, req_idx=None, bounds=False, threads=1,
          inst_sorted=None):
    """Full oracle route of (a subset of) a workload's requests.
    Returns dict(hits, scores, choice, best); with bounds, also the per-score
    rounding analysis of mlp_forward_bounds (ebound, flip).  threads > 1 splits
    the requests over host threads (the C routines release the interpreter
    lock); the result does not depend on it."""
    if threads > 1:
        import concurrent.futures as cf
        R_all = len(wl.tok_off) - 1
        idx = np.arange(R_all) if req_idx is None else np.asarray(req_idx)
        if inst_keys is None and inst_sorted is None and hits is None:
            inst_keys = instance_keys(wl)
        parts = [p for p in np.array_split(np.arange(len(idx)), threads) if len(p)]
        with cf.ThreadPoolExecutor(max_workers=len(parts)) as ex:
            res = list(ex.map(lambda p: route(wl, None if hits is None else hits[p], inst_keys, params, mode,
                                              idx[p], bounds, 1, inst_sorted), parts))
        out = {k: np.concatenate([r[k] for r in res]) for k in res[0]}
        out["choice"], out["best"] = argmin(out["scores"])
        return out
    cfg = wl.cfg
    mode = mode or cfg.dtype
    R_all = len(wl.tok_off) - 1
    idx = np.arange(R_all) if req_idx is None else np.asarray(req_idx)
    if hits is None:
        tok_off = wl.tok_off
        seqs = [wl.tok[tok_off[r]: tok_off[r + 1]] for r in idx]
        sub_off = np.zeros(len(idx) + 1, np.int64)
        sub_off[1:] = np.cumsum([len(s) for s in seqs])
        sub_tok = np.concatenate(seqs) if seqs else np.zeros(0, np.int32)
        rk, rko = hash_blocks(sub_tok, sub_off)
        if inst_sorted is not None:
            hits = prefix_hits_sorted(rk, rko, inst_sorted)
        else:
            if inst_keys is None:
                inst_keys = instance_keys(wl)
            ik, iko = inst_keys
            hits = prefix_hits(rk, rko, ik, iko, by_marking=len(idx) * 64 < len(ik))
    L = np.diff(wl.tok_off)[idx]
    x = features(L, hits, wl.inst_state, wl.req_feats[idx], wl.mean, wl.std)
    p = wl.params if params is None else params
    if bounds:
        y, eb, fl = mlp_forward_bounds(mode, cfg.widths, p, x)
    else:
        y = mlp_forward(mode, cfg.widths, p, x)
    scores = y.astype(np.float32).reshape(len(idx), -1)
    choice, best = argmin(scores)
    out = dict(hits=hits, scores=scores, choice=choice, best=best)
    if bounds:
        out["ebound"] = eb.reshape(len(idx), -1)
        out["flip"] = fl.reshape(len(idx), -1)
    return out


def route_sequential(wl, params=None, mode=None, inst_keys=None, queue_col=0, forced=None):
    """Sequential-commit route of all of a workload's requests
    (or_route_sequential).  Returns dict(hits, scores, choice, inst) with inst
    the instance rows after the last commit."""
    cfg = wl.cfg
    mode = MODES.get(mode or cfg.dtype, mode or cfg.dtype)
    w = _c(cfg.widths, np.int32)
    p = _c(wl.params if params is None else params, np.float64)
    rk, rko = hash_blocks(wl.tok, wl.tok_off)
    rk = _c(rk, np.uint64) if len(rk) else np.zeros(1, np.uint64)
    ik, iko = instance_keys(wl) if inst_keys is None else inst_keys
    ik = _c(ik, np.uint64) if len(ik) else np.zeros(1, np.uint64)
    R, N = len(wl.tok_off) - 1, cfg.n_inst
    L = _c(np.diff(wl.tok_off), np.int64)
    inst = np.array(wl.inst_state, np.float32, copy=True)
    req = _c(wl.req_feats, np.float32) if cfg.d_req else np.zeros(1, np.float32)
    hits = np.zeros((R, N), np.int32)
    scores = np.zeros((R, N), np.float32)
    choice = np.zeros(R, np.int32)
    fc = _c(forced, np.int32) if forced is not None else None
    _check(lib().or_route_sequential(mode, len(w) - 1, _p(w), _p(p), R, _p(L), _p(rk), _p(_c(rko, np.int64)), N,
                                     _p(ik), _p(_c(iko, np.int64)), _p(inst), cfg.d_inst, _p(req), cfg.d_req,
                                     _p(_c(wl.mean, np.float32)), _p(_c(wl.std, np.float32)), int(queue_col),
                                     _p(fc) if fc is not None else None, _p(hits), _p(scores), _p(choice)),
           "route_sequential")
    return dict(hits=hits, scores=scores, choice=choice, inst=inst)


# --------------------------------------------------------------------------
# sample ring and training
# --------------------------------------------------------------------------

def ring_append(ring_x, ring_y, count, x, y):
    C_, d = ring_x.shape
    x = _c(x, np.float32)
    y = _c(y, np.float32)
    _check(lib().or_ring_append(C_, d, _p(ring_x), _p(ring_y), int(count), len(y), _p(x), _p(y)), "ring")
    return count + len(y)


class Trainer:
    """Oracle optimiser state: fp32-valued params, Adam moments, step count."""

    def __init__(self, widths, params, mode="f32", dropout=0.0, dropout_seed=0):
        self.dropout, self.dropout_seed = float(dropout), int(dropout_seed)
        self.w = _c(widths, np.int32)
        self.mode = MODES.get(mode, mode)
        self.params = _c(params, np.float64).copy()
        self.m = np.zeros_like(self.params)
        self.v = np.zeros_like(self.params)
        self.t = 0

    def step(self, ring_x, ring_y, idx, mean, std, opt="adam", lr=3e-4, want_grad=False):
        self.t += 1
        loss = np.zeros(1, np.float64)
        g = np.zeros_like(self.params) if want_grad else None
        idx = _c(idx, np.int32)
        rc = lib().or_train_step(self.mode, len(self.w) - 1, _p(self.w), _p(self.params),
                                 _p(self.m), _p(self.v), self.t, ADAM if opt == "adam" else SGD,
                                 float(lr), len(idx), _p(_c(ring_x, np.float32)),
                                 _p(_c(ring_y, np.float32)), _p(idx), _p(_c(mean, np.float32)),
                                 _p(_c(std, np.float32)), _p(loss),
                                 _p(g) if g is not None else None, self.dropout,
                                 C.c_uint64(self.dropout_seed & (2**64 - 1)))
        _check(rc, "train_step")
        return (float(loss[0]), g) if want_grad else float(loss[0])


def loss(mode, widths, params, ring_x, ring_y, idx, mean, std) -> float:
    w = _c(widths, np.int32)
    out = np.zeros(1, np.float64)
    idx = _c(idx, np.int32)
    _check(lib().or_loss(MODES.get(mode, mode), len(w) - 1, _p(w), _p(_c(params, np.float64)),
                         len(idx), _p(_c(ring_x, np.float32)), _p(_c(ring_y, np.float32)),
                         _p(idx), _p(_c(mean, np.float32)), _p(_c(std, np.float32)), _p(out)),
           "loss")
    return float(out[0])


# --------------------------------------------------------------------------
# Algorithm 4 guards
# --------------------------------------------------------------------------

ROUTE_OK, ROUTE_COLD_START, ROUTE_OOD, ROUTE_KFILTER = 0, 1, 2, 4


def ring_bounds(ring_x, count):
    """Per-feature [lo, hi] over the records the ring holds (NaN skipped)."""
    rx = _c(ring_x, np.float32)
    cap, d = rx.shape
    lo = np.zeros(d, np.float32)
    hi = np.zeros(d, np.float32)
    _check(lib().or_ring_bounds(cap, d, _p(rx), int(count), _p(lo), _p(hi)), "ring_bounds")
    return lo, hi


def hrw_candidates(gkey: int, n_inst: int, K: int) -> np.ndarray:
    """ConsistentHash_K of one prefix-group key, in rank order."""
    out = np.zeros(max(K, 1), np.int32)
    m = lib().or_hrw_candidates(C.c_uint64(gkey & (2**64 - 1)), n_inst, K, _p(out))
    return out[:m]


def group_keys(tok, tok_off) -> np.ndarray:
    """Prefix-group key of every prompt: the key of its first full block
    (0 where the prompt has none)."""
    keys, ko = hash_blocks(tok, tok_off)
    L = np.diff(np.asarray(tok_off, np.int64))
    g = np.zeros(len(L), np.uint64)
    has = L >= BLOCK
    g[has] = keys[ko[:-1][has]]
    return g


def guards(L, gkey, hits, inst_state, req_feats, scores, lo, hi, n, *, n_min=0, ood=False,
           k=0, kv_col=4, tau_sat=0.8, tau_ben=0.0):
    """Guarded selection of Algorithm 4 over given scores.
    Returns (choice int32 [R], best f32 [R], status int32 [R])."""
    L = _c(L, np.int64)
    gkey = _c(gkey, np.uint64)
    hits = _c(hits, np.int32)
    s = _c(scores, np.float32)
    inst = _c(inst_state, np.float32)
    req = _c(req_feats, np.float32)
    R, N = s.shape
    d_inst, d_req = inst.shape[1], (req.shape[1] if req.ndim == 2 else 0)
    choice = np.zeros(R, np.int32)
    best = np.zeros(R, np.float32)
    status = np.zeros(R, np.int32)
    one = np.zeros(1, np.float32)
    _check(lib().or_guards(R, N, _p(L), _p(gkey), _p(hits), _p(inst if inst.size else one), d_inst,
                           _p(req if req.size else one), d_req, _p(s), _p(_c(lo, np.float32)),
                           _p(_c(hi, np.float32)), int(n), int(n_min), int(bool(ood)), int(k),
                           int(kv_col), float(tau_sat), float(tau_ben), _p(choice), _p(best),
                           _p(status)), "guards")
    return choice, best, status


def heuristic(L, hits, inst_state, *, mode=1, count_cols=(0, 1), theta_imbal=8.0, k=1.0, tau=0.5):
    """Fallback heuristic choice per request (Algorithm 1: mode 1; Algorithm 2: mode 2)."""
    L = _c(L, np.int64)
    hits = _c(hits, np.int32)
    inst = _c(inst_state, np.float32)
    R, N = hits.shape
    out = np.zeros(R, np.int32)
    c1 = count_cols[1] if len(count_cols) > 1 else -1
    _check(lib().or_heuristic(R, N, _p(L), _p(hits), _p(inst), inst.shape[1], int(mode), int(count_cols[0]),
                              int(c1), float(theta_imbal), float(k), float(tau), _p(out)), "heuristic")
    return out


# --------------------------------------------------------------------------
# two-pool training data (FIFO + replay pool)
# --------------------------------------------------------------------------

def replay_embed(mode, widths, params, x, y, mean, std) -> np.ndarray:
    """Gradient embeddings g = (yhat - y) * last hidden activation, [M, H] fp64."""
    mode = MODES.get(mode, mode)
    w = _c(widths, np.int32)
    x = _c(x, np.float32)
    y = _c(y, np.float32)
    M = len(y)
    H = int(w[-2])
    g = np.zeros((max(M, 1), H), np.float64)
    _check(lib().or_replay_embed(mode, len(w) - 1, _p(w), _p(_c(params, np.float64)), M,
                                 _p(x if M else np.zeros(1, np.float32)), _p(y if M else np.zeros(1, np.float32)),
                                 _p(_c(mean, np.float32)), _p(_c(std, np.float32)), _p(g)), "replay_embed")
    return g[:M]


def replay_distances(gc, gk):
    """(d per candidate, n per kept): nearest kept squared distance, nearest other kept."""
    gc = _c(gc, np.float64).reshape(len(gc), -1) if len(gc) else np.zeros((0, 1))
    gk = _c(gk, np.float64).reshape(len(gk), -1) if len(gk) else np.zeros((0, 1))
    H = gc.shape[1] if len(gc) else gk.shape[1]
    d = np.zeros(max(len(gc), 1))
    n = np.zeros(max(len(gk), 1))
    one = np.zeros(1)
    _check(lib().or_replay_distances(len(gc), _p(gc if len(gc) else one), len(gk), _p(gk if len(gk) else one),
                                     int(H), _p(d), _p(n)), "replay_distances")
    return d[:len(gc)], n[:len(gk)]


def replay_select(d, n, cap):
    """Admission round: (src per slot of the new pool, new count); src >= 0 is a
    candidate index, -1 - j keeps kept sample j."""
    d = _c(d, np.float64)
    n = _c(n, np.float64)
    src = np.zeros(max(int(cap), 1), np.int64)
    cnt = np.zeros(1, np.int64)
    _check(lib().or_replay_select(len(d), _p(d if len(d) else np.zeros(1)), len(n),
                                  _p(n if len(n) else np.zeros(1)), int(cap), _p(src), _p(cnt)), "replay_select")
    return src[:int(cnt[0])], int(cnt[0])


def drop_keep(seed, p, t, h, j, o) -> bool:
    """Dropout keep decision of unit o of hidden activation h, minibatch row j, step t."""
    return bool(lib().or_drop_keep(C.c_uint64(seed & (2**64 - 1)), float(p), int(t), int(h), int(j), int(o)))
