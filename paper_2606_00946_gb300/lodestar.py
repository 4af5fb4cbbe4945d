"""Thin ctypes binding of the C ABI in include/lodestar.h.

The functions below have the ABI's names and only marshal arguments: torch
tensors become device pointers, streams become cudaStream_t handles, and the
integer status is returned unchanged.  All computation happens in the CUDA
library (_build/liblodestar.so); if it is missing the import of `lib()` fails
loudly -- there is no other implementation to fall back on.
"""
from __future__ import annotations

import ctypes as C
import os

from . import build as _build

LS_MAX_LAYERS = 8
LS_OK, LS_ERR_ARG, LS_ERR_CUDA, LS_ERR_OOM = 0, -1, -2, -3
LS_ERR_TABLE_FULL, LS_ERR_TIMEOUT, LS_ERR_STATE = -4, -5, -6
LS_F32, LS_BF16 = 0, 1
LS_REPLACE, LS_INSERT = 0, 1
LS_SGD, LS_ADAM = 0, 1
LS_SCORER_AUTO, LS_SCORER_CUDA_CORES, LS_SCORER_TENSOR_CORES = 0, 1, 2
LS_TC_NONE, LS_TC_GENERIC, LS_TC_PIPELINED, LS_TC_WIDE, LS_TC_PAIR = 0, 1, 2, 3, 4
SCORERS = {"auto": 0, "cuda_cores": 1, "tensor_cores": 2}
LS_STATIC_MAX_BLOCKS, LS_STATIC_MAX_PAIRS = 262144, 262144
LS_PREFIX_AUTO, LS_PREFIX_TWO_PHASE, LS_PREFIX_FUSED, LS_PREFIX_INDEX = 0, 1, 2, 3
PREFIX_MODES = {"auto": 0, "two_phase": 1, "fused": 2, "index": 3}
LS_ROUTE_OK, LS_ROUTE_COLD_START, LS_ROUTE_OOD, LS_ROUTE_KFILTER = 0, 1, 2, 4
LS_HEUR_NONE, LS_HEUR_PREFIX_LOAD, LS_HEUR_PREFIX = 0, 1, 2


class ls_config(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("widths", C.c_int32 * (LS_MAX_LAYERS + 1)),
                ("d_inst", C.c_int32), ("d_req", C.c_int32), ("dtype", C.c_int32),
                ("max_instances", C.c_int32), ("max_requests", C.c_int32),
                ("max_keys_per_instance", C.c_int64), ("max_load", C.c_float),
                ("ring_capacity", C.c_int64), ("max_train_batch", C.c_int32),
                ("max_batch_tokens", C.c_int64), ("prefix_mode", C.c_int32), ("scorer", C.c_int32),
                ("replay_capacity", C.c_int64), ("pending_capacity", C.c_int64), ("dropout", C.c_float),
                ("dropout_seed", C.c_uint64), ("train_ctas", C.c_int32)]


class ls_info(C.Structure):
    _fields_ = [("n_inst", C.c_int32), ("d", C.c_int32), ("n_params", C.c_int64),
                ("table_slots", C.c_int64), ("ring_count", C.c_int64),
                ("train_steps", C.c_int64), ("weight_version", C.c_uint64), ("scorer", C.c_int32),
                ("replay_count", C.c_int64), ("pending_count", C.c_int64), ("tc_kernel", C.c_int32)]


class ls_guards(C.Structure):
    _fields_ = [("n_min", C.c_int64), ("ood", C.c_int32), ("k", C.c_int32), ("kv_col", C.c_int32),
                ("tau_sat", C.c_float), ("tau_ben", C.c_float), ("heuristic", C.c_int32),
                ("count_col", C.c_int32 * 2), ("theta_imbal", C.c_float), ("k_overload", C.c_float),
                ("tau_prefix", C.c_float)]


class ls_trace_entry(C.Structure):
    _fields_ = [("name", C.c_char * 32), ("launches", C.c_int64), ("total_ms", C.c_double),
                ("timed_launches", C.c_int64)]


_P, _i32, _i64 = C.c_void_p, C.c_int32, C.c_int64
_SIGS = {
    "ls_param_count": (_i64, [C.POINTER(ls_config)]),
    "ls_create": (C.c_int, [C.POINTER(ls_config), C.POINTER(_P)]),
    "ls_destroy": (None, [_P]),
    "ls_last_error": (C.c_char_p, []),
    "ls_sync_status": (C.c_int, [_P]),
    "ls_get_info": (C.c_int, [_P, C.POINTER(ls_info)]),
    "ls_set_params": (C.c_int, [_P, _P, _P]),
    "ls_get_params": (C.c_int, [_P, _P, _P]),
    "ls_get_opt_state": (C.c_int, [_P, _P, _P, C.POINTER(_i64), _P]),
    "ls_set_opt_state": (C.c_int, [_P, _P, _P, _i64, _P]),
    "ls_set_normalizer": (C.c_int, [_P, _P, _P, _P]),
    "ls_snapshot_update": (C.c_int, [_P, _i32, _P, _P, _P, _i64, _i32, _P]),
    "ls_hash_blocks": (C.c_int, [_P, _i32, _P, _P, _P, _P, _P]),
    "ls_assemble_features": (C.c_int, [_P, _i32, _P, _P, _P, _P, _P]),
    "ls_route_batch": (C.c_int, [_P, _i32, _P, _P, _P, _P, _P, _P, _P, C.POINTER(C.c_uint64), _P]),
    "ls_log_samples": (C.c_int, [_P, _i32, _P, _P, _P]),
    "ls_train_step": (C.c_int, [_P, _i32, _P, _i32, C.c_float, _P, _P]),
    "ls_publish": (C.c_int, [_P, _P]),
    "ls_set_guards": (C.c_int, [_P, C.POINTER(ls_guards)]),
    "ls_replay_admit": (C.c_int, [_P, _P, _P, _P]),
    "ls_get_replay": (C.c_int, [_P, _P, _P, C.POINTER(_i64), _P]),
    "ls_refresh_bounds": (C.c_int, [_P, _P]),
    "ls_get_bounds": (C.c_int, [_P, _i32, _P, _P, _P]),
    "ls_route_batch_guarded": (C.c_int, [_P, _i32, _P, _P, _P, _P, _P, _P, _P, _P, _P,
                                         C.POINTER(C.c_uint64), _P]),
    "ls_read_features": (C.c_int, [_P, _i64, _i64, _P, _P]),
    "ls_route_sequential": (C.c_int, [_P, _i32, _P, _P, _P, _i32, _P, _P, _P, _P, C.POINTER(C.c_uint64), _P]),
    "ls_trace_enable": (C.c_int, [_P, _i32]),
    "ls_trace_read": (C.c_int, [_P, C.POINTER(ls_trace_entry), _i32, C.POINTER(_i32)]),
    "ls_prefix_hits_static": (C.c_int, [_i32, _P, _P, _i64, _P, _i64, _i32, _P, _P]),
    # measurement kernels of include/lodestar_probe.h
    "ls_probe_gather": (C.c_int, [_P, _i64, _i32, _i32, C.c_uint64, _P, _P]),
    "ls_probe_fma": (C.c_int, [_i32, _i64, _P, _P]),
    "ls_probe_read": (C.c_int, [_P, _i64, _i32, _i32, _P, _P]),
}

_lib = None


def lib_path() -> str:
    return _build.LIB


def lib():
    """Load the CUDA library (build it first with build.build())."""
    global _lib
    if _lib is None:
        path = lib_path()
        if not os.path.exists(path):
            raise RuntimeError(f"{path} is missing: build the CUDA library first "
                               "(__graft_entry__.build() or paper_2606_00946_gb300.build.build())")
        L = C.CDLL(path)
        for name, (res, args) in _SIGS.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def ptr(t):
    """Device pointer of a tensor (None -> NULL)."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def stream_handle(s=None):
    if s is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(s, int):
        return s
    return s.cuda_stream


class LodestarError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"lodestar status {code}: {msg}")
        self.code = code


def last_error() -> str:
    m = lib().ls_last_error()
    return m.decode() if m else ""


def check(rc: int) -> int:
    if rc != LS_OK:
        raise LodestarError(rc, last_error())
    return rc


def make_config(widths, d_inst, d_req, dtype="bf16", max_instances=64, max_requests=4096,
                max_keys_per_instance=16384, max_load=0.5, ring_capacity=65536,
                max_train_batch=4096, scorer="auto", max_batch_tokens=1 << 24,
                prefix_mode="auto", replay_capacity=0, pending_capacity=0, dropout=0.0,
                dropout_seed=0, train_ctas=0) -> ls_config:
    c = ls_config()
    c.n_layers = len(widths) - 1
    for i, w in enumerate(widths):
        c.widths[i] = int(w)
    c.d_inst, c.d_req = int(d_inst), int(d_req)
    c.dtype = LS_BF16 if dtype in ("bf16", LS_BF16) else LS_F32
    c.max_instances, c.max_requests = int(max_instances), int(max_requests)
    c.max_keys_per_instance, c.max_load = int(max_keys_per_instance), float(max_load)
    c.ring_capacity, c.max_train_batch = int(ring_capacity), int(max_train_batch)
    c.scorer = SCORERS.get(scorer, scorer)
    c.max_batch_tokens = int(max_batch_tokens)
    c.prefix_mode = PREFIX_MODES.get(prefix_mode, prefix_mode)
    c.replay_capacity, c.pending_capacity = int(replay_capacity), int(pending_capacity)
    c.dropout, c.dropout_seed = float(dropout), int(dropout_seed) & (2**64 - 1)
    c.train_ctas = int(train_ctas)
    return c


# ---------------------------------------------------------------------------
# ABI functions, same names, status returned as is
# ---------------------------------------------------------------------------

def ls_param_count(cfg: ls_config) -> int:
    return lib().ls_param_count(C.byref(cfg))


def ls_create(cfg: ls_config):
    """Returns (status, handle)."""
    h = _P()
    rc = lib().ls_create(C.byref(cfg), C.byref(h))
    return rc, h


def ls_destroy(ctx):
    lib().ls_destroy(ctx)


def ls_last_error() -> str:
    return last_error()


def ls_sync_status(ctx) -> int:
    return lib().ls_sync_status(ctx)


def ls_get_info(ctx):
    info = ls_info()
    rc = lib().ls_get_info(ctx, C.byref(info))
    return rc, info


def ls_set_params(ctx, params, stream=None) -> int:
    return lib().ls_set_params(ctx, ptr(params), stream_handle(stream))


def ls_get_params(ctx, out, stream=None) -> int:
    return lib().ls_get_params(ctx, ptr(out), stream_handle(stream))


def ls_get_opt_state(ctx, m_out, v_out, stream=None):
    step = _i64()
    rc = lib().ls_get_opt_state(ctx, ptr(m_out), ptr(v_out), C.byref(step), stream_handle(stream))
    return rc, step.value


def ls_set_opt_state(ctx, m, v, step, stream=None) -> int:
    return lib().ls_set_opt_state(ctx, ptr(m), ptr(v), int(step), stream_handle(stream))


def ls_set_normalizer(ctx, mean, std, stream=None) -> int:
    return lib().ls_set_normalizer(ctx, ptr(mean), ptr(std), stream_handle(stream))


def ls_snapshot_update(ctx, n_inst, inst_state, keys, key_off, n_keys, mode=LS_REPLACE,
                       stream=None) -> int:
    return lib().ls_snapshot_update(ctx, int(n_inst), ptr(inst_state), ptr(keys), ptr(key_off),
                                    int(n_keys), int(mode), stream_handle(stream))


def ls_hash_blocks(ctx, n_seq, tok, tok_off, keys_out, key_off, stream=None) -> int:
    return lib().ls_hash_blocks(ctx, int(n_seq), ptr(tok), ptr(tok_off), ptr(keys_out),
                                ptr(key_off), stream_handle(stream))


def ls_assemble_features(ctx, n_req, tok_off, hits, req_feats, x_out, stream=None) -> int:
    return lib().ls_assemble_features(ctx, int(n_req), ptr(tok_off), ptr(hits), ptr(req_feats),
                                      ptr(x_out), stream_handle(stream))


def ls_route_batch(ctx, n_req, tok, tok_off, req_feats, choice, best, scores_opt=None,
                   hits_opt=None, stream=None):
    """Returns (status, weight_version)."""
    v = C.c_uint64(0)
    rc = lib().ls_route_batch(ctx, int(n_req), ptr(tok), ptr(tok_off), ptr(req_feats), ptr(choice),
                              ptr(best), ptr(scores_opt), ptr(hits_opt), C.byref(v),
                              stream_handle(stream))
    return rc, v.value


def ls_log_samples(ctx, n, feats, ttft, stream=None) -> int:
    return lib().ls_log_samples(ctx, int(n), ptr(feats), ptr(ttft), stream_handle(stream))


def ls_train_step(ctx, batch, idx, opt, lr, loss_out=None, stream=None) -> int:
    return lib().ls_train_step(ctx, int(batch), ptr(idx), int(opt), float(lr), ptr(loss_out),
                               stream_handle(stream))


def ls_publish(ctx, stream=None) -> int:
    return lib().ls_publish(ctx, stream_handle(stream))


def ls_set_guards(ctx, n_min=0, ood=False, k=0, kv_col=0, tau_sat=0.8, tau_ben=0.0, heuristic=0,
                  count_cols=(0, 1), theta_imbal=8.0, k_overload=1.0, tau_prefix=0.5) -> int:
    g = ls_guards(int(n_min), 1 if ood else 0, int(k), int(kv_col), float(tau_sat), float(tau_ben),
                  int(heuristic), (C.c_int32 * 2)(int(count_cols[0]), int(count_cols[1])), float(theta_imbal),
                  float(k_overload), float(tau_prefix))
    return lib().ls_set_guards(ctx, C.byref(g))


def ls_replay_admit(ctx, d_out=None, n_out=None, stream=None) -> int:
    return lib().ls_replay_admit(ctx, ptr(d_out), ptr(n_out), stream_handle(stream))


def ls_get_replay(ctx, x_out, y_out, stream=None):
    """Returns (status, records in the replay pool)."""
    n = _i64(0)
    rc = lib().ls_get_replay(ctx, ptr(x_out), ptr(y_out), C.byref(n), stream_handle(stream))
    return rc, n.value


def ls_refresh_bounds(ctx, stream=None) -> int:
    return lib().ls_refresh_bounds(ctx, stream_handle(stream))


def ls_get_bounds(ctx, which, lo_out, hi_out, stream=None) -> int:
    return lib().ls_get_bounds(ctx, int(which), ptr(lo_out), ptr(hi_out), stream_handle(stream))


def ls_route_batch_guarded(ctx, n_req, tok, tok_off, req_feats, choice, best, status, fallback_opt=None,
                           scores_opt=None, hits_opt=None, stream=None):
    """Returns (status code of the call, weight_version)."""
    v = C.c_uint64(0)
    rc = lib().ls_route_batch_guarded(ctx, int(n_req), ptr(tok), ptr(tok_off), ptr(req_feats), ptr(choice),
                                      ptr(best), ptr(status), ptr(fallback_opt), ptr(scores_opt), ptr(hits_opt),
                                      C.byref(v), stream_handle(stream))
    return rc, v.value


def ls_read_features(ctx, row0, n_rows, out, stream=None) -> int:
    return lib().ls_read_features(ctx, int(row0), int(n_rows), ptr(out), stream_handle(stream))


def ls_route_sequential(ctx, n_req, tok, tok_off, req_feats, queue_col, choice, best, scores_opt=None,
                        hits_opt=None, stream=None):
    ver = C.c_uint64(0)
    rc = lib().ls_route_sequential(ctx, int(n_req), ptr(tok), ptr(tok_off), ptr(req_feats), int(queue_col),
                                   ptr(choice), ptr(best), ptr(scores_opt), ptr(hits_opt), C.byref(ver),
                                   stream_handle(stream))
    return rc, ver.value


def ls_trace_enable(ctx, on=True) -> int:
    return lib().ls_trace_enable(ctx, 1 if on else 0)


def ls_trace_read(ctx, max_entries=64):
    """Returns (status, {name: (launches, total_ms, timed_launches)})."""
    arr = (ls_trace_entry * max_entries)()
    n = _i32(0)
    rc = lib().ls_trace_read(ctx, arr, max_entries, C.byref(n))
    return rc, {arr[i].name.decode(): (arr[i].launches, arr[i].total_ms, arr[i].timed_launches)
                for i in range(n.value)}


def ls_prefix_hits_static(n_req, tok, tok_off, n_tokens, tables, slots_per_instance, n_inst, hits_out,
                          stream=None) -> int:
    return lib().ls_prefix_hits_static(int(n_req), ptr(tok), ptr(tok_off), int(n_tokens), ptr(tables),
                                       int(slots_per_instance), int(n_inst), ptr(hits_out),
                                       stream_handle(stream))


def ls_probe_gather(table, n_slots, blocks, per_thread, seed, out, stream=None) -> int:
    return lib().ls_probe_gather(ptr(table), int(n_slots), int(blocks), int(per_thread), int(seed), ptr(out),
                                 stream_handle(stream))


def ls_probe_fma(blocks, iters, out, stream=None) -> int:
    return lib().ls_probe_fma(int(blocks), int(iters), ptr(out), stream_handle(stream))


def ls_probe_read(buf, n16, passes, blocks, out, stream=None) -> int:
    return lib().ls_probe_read(ptr(buf), int(n16), int(passes), int(blocks), ptr(out), stream_handle(stream))
