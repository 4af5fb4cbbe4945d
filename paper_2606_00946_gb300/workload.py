"""Seeded synthetic workloads for the Lodestar routing hot path.

The paper evaluates on Mooncake traces and on synthetic prefix-sharing
workloads (Sec. 5.1, "Workloads": 10/30/50/70 % and mixed prefix-sharing
ratios, prefix groups, Poisson arrivals).  Neither the traces nor the paper's
released routing dataset are available here, so every input is drawn from a
seeded generator with the shapes of those workloads.

This module holds none of the routing method's arithmetic: it never hashes a
token, never assembles a feature, never evaluates the predictor.  Instance
caches are returned as *token sequences* (which the consumer hashes with its
own implementation) plus random 64-bit stand-in keys for unshared blocks.
Both the CPU oracle and the CUDA path consume exactly these arrays.

All draws use ``numpy.random.default_rng``; each config has its own seed and
the cache-history stream uses ``seed + 1000``.
"""
from __future__ import annotations

from dataclasses import dataclass, field
import numpy as np

BLOCK = 16          # tokens per KV block
PAIR_DIMS = 6       # pair features: L, h, 16h, kappa, L-16h, ceil(L/16)-h
INST_BASE_DIMS = 10 # queued, running, prefill tok, decode tok, KV util,
                    # free KV blocks, GPU-type one-hot (3), speed scalar
VOCAB = 32000
TYPE_SPEEDS = (1.0, 1.7, 3.1)


@dataclass(frozen=True)
class Config:
    name: str
    seed: int
    n_inst: int
    n_req: int
    length: tuple           # ("sys", lo, hi) | ("uniform", lo, hi) | ("loguniform", lo, hi)
    n_templates: int        # templates for Zipf-shared prefixes (0: system-prompt scheme)
    zipf_s: float
    cache_blocks: int       # per-instance cache budget in blocks
    d_inst: int
    d_req: int
    hidden: tuple
    dtype: str              # "f32" | "bf16"
    n_types: int
    train_batch: int = 4096
    train_opt: str = "adam"
    train_lr: float = 3e-4
    n_samples: int = 0      # logged (feature, TTFT) records to generate
    ttft_model: str = "quadratic"   # "linear" (tiny) | "quadratic"

    @property
    def d(self) -> int:
        return PAIR_DIMS + self.d_inst + self.d_req

    @property
    def widths(self) -> tuple:
        return (self.d,) + tuple(self.hidden) + (1,)

    @property
    def max_len(self) -> int:
        return self.length[2] + (128 if self.length[0] == "sys" else 0)


CONFIGS = {
    # 8 instances x 64 requests, fp32 16->64->64->1, one SGD step on 256 samples
    "tiny": Config("tiny", 1, 8, 64, ("sys", 32, 512), 0, 1.1, 2048, 10, 0,
                   (64, 64), "f32", 1, train_batch=256, train_opt="sgd",
                   train_lr=1e-3, n_samples=256, ttft_model="linear"),
    # 32 instances x 4096 requests, bf16 64->256->256->1
    "homogeneous": Config("homogeneous", 2, 32, 4096, ("uniform", 64, 4096), 256,
                          1.1, 16384, 34, 24, (256, 256), "bf16", 1,
                          n_samples=65536),
    # 64 instances (3 GPU types) x 8192 long-context requests, bf16 128->256^3->1
    "heterogeneous": Config("heterogeneous", 3, 64, 8192, ("loguniform", 8192, 32768),
                            256, 1.1, 65536, 66, 56, (256, 256, 256), "bf16", 3),
    # online training: 1M logged 128-dim records, Adam lr 3e-4, batch 4096
    "training": Config("training", 4, 64, 8192, ("loguniform", 8192, 32768), 256,
                       1.1, 65536, 66, 56, (256, 256, 256), "bf16", 3,
                       n_samples=1 << 20),
    # the paper's operating point: one request at a time over 16 instances, its
    # predictor size (3 hidden layers of 128, Sec. 4.1), a pool of 256 requests
    "paper": Config("paper", 6, 16, 256, ("uniform", 64, 4096), 256, 1.1, 16384, 34, 24,
                    (128, 128, 128), "bf16", 1, n_samples=10000),
    # 256 instances x 16384 requests, 1M cached blocks each, bf16 128->512->512->1
    "large": Config("large", 5, 256, 16384, ("uniform", 128, 16384), 4096, 1.1,
                    1 << 20, 66, 56, (512, 512), "bf16", 3),
}


def table_capacity(max_keys: int, max_load: float = 0.5) -> int:
    """Open-addressing slots for `max_keys` keys at load <= max_load (power of two)."""
    need = int(np.ceil(max_keys / max_load))
    return 1 << max(int(need - 1).bit_length(), 4)


@dataclass
class Workload:
    cfg: Config
    tok: np.ndarray            # int32 [sum L]  prompt tokens, CSR
    tok_off: np.ndarray        # int64 [R+1]
    req_feats: np.ndarray      # f32 [R, d_req]  request-level extras
    inst_state: np.ndarray     # f32 [N, d_inst] instance snapshot rows
    # instance caches: token sequences to hash (prefix-closed: first n blocks)
    seq_tok: np.ndarray        # int32, CSR of cached sequences (templates or earlier prompts)
    seq_off: np.ndarray        # int64 [S+1]
    chain_seq: np.ndarray      # int32 [C]   which sequence a cached chain comes from
    chain_blocks: np.ndarray   # int32 [C]   how many leading blocks of it are cached
    inst_chain_off: np.ndarray # int64 [N+1] CSR of chains per instance
    rand_keys: np.ndarray      # uint64 [K]  stand-in keys of unshared blocks
    inst_rand_off: np.ndarray  # int64 [N+1]
    mean: np.ndarray           # f32 [d] normaliser mean
    std: np.ndarray            # f32 [d] normaliser std (may hold 0 for constant columns)
    params: np.ndarray         # f32 flat W1,b1,W2,b2,... (row-major [out,in])
    samples_x: np.ndarray = field(default=None)   # f32 [S, d] raw logged features
    samples_y: np.ndarray = field(default=None)   # f32 [S] observed TTFT (s)

    @property
    def lengths(self) -> np.ndarray:
        return np.diff(self.tok_off)

    def max_keys_per_instance(self) -> int:
        return int(self.cfg.cache_blocks)


# ----------------------------------------------------------------------------
# elementary draws
# ----------------------------------------------------------------------------

def _zipf_probs(n: int, s: float) -> np.ndarray:
    p = np.arange(1, n + 1, dtype=np.float64) ** (-s)
    return p / p.sum()


def _draw_lengths(rng, kind, lo, hi, n) -> np.ndarray:
    if kind in ("uniform", "sys"):
        return rng.integers(lo, hi + 1, size=n).astype(np.int64)
    if kind == "loguniform":
        return np.floor(np.exp(rng.uniform(np.log(lo), np.log(hi), size=n))).astype(np.int64)
    raise ValueError(kind)


def xavier_params(widths, seed: int = 0) -> np.ndarray:
    """Xavier-uniform weights U(-a, a), a = sqrt(6/(fan_in+fan_out)), drawn in
    order W1, W2, ... row-major from default_rng(seed); biases zero."""
    rng = np.random.default_rng(seed)
    parts = []
    for l in range(len(widths) - 1):
        fi, fo = widths[l], widths[l + 1]
        a = np.sqrt(6.0 / (fi + fo))
        parts.append(rng.uniform(-a, a, size=(fo, fi)).astype(np.float32).ravel())
        parts.append(np.zeros(fo, np.float32))
    return np.concatenate(parts)


def param_count(widths) -> int:
    return int(sum(widths[l] * widths[l + 1] + widths[l + 1] for l in range(len(widths) - 1)))


def instance_state(rng, cfg: Config, n: int | None = None) -> np.ndarray:
    """Snapshot rows: queued ~ Poisson(4), running ~ U{0..64}, inflight prefill =
    running*U[0,4096], inflight decode = running*U[0,1024], KV util ~ Beta(2,2),
    free KV blocks = (1-util)*budget, GPU type one-hot, speed scalar, then
    N(0,1) 'other metrics'."""
    n = cfg.n_inst if n is None else n
    st = np.zeros((n, cfg.d_inst), np.float64)
    running = rng.integers(0, 65, size=n)
    util = rng.beta(2.0, 2.0, size=n)
    st[:, 0] = rng.poisson(4.0, size=n)
    st[:, 1] = running
    st[:, 2] = running * rng.uniform(0, 4096, size=n)
    st[:, 3] = running * rng.uniform(0, 1024, size=n)
    st[:, 4] = util
    st[:, 5] = np.floor((1.0 - util) * cfg.cache_blocks)
    types = np.arange(n) % cfg.n_types
    st[np.arange(n), 6 + types] = 1.0
    st[:, 9] = np.asarray(TYPE_SPEEDS)[types]
    if cfg.d_inst > INST_BASE_DIMS:
        st[:, INST_BASE_DIMS:] = rng.standard_normal((n, cfg.d_inst - INST_BASE_DIMS))
    return st.astype(np.float32)


def records(rng, cfg: Config, n: int):
    """Synthetic logged (raw feature row, observed TTFT) records.

    Pair columns are those of a routed pair (Sec. 4.1 Features): f0 = prompt
    length L, f1 = hit blocks h ~ U{0..floor(L/16)}, f2 = 16h, f3 = 16h/L
    (fp32), f4 = L - 16h, f5 = ceil(L/16) - h; instance columns follow
    instance_state(); request extras are N(0,1).
    TTFT models (seconds):
      linear    : y = sum_k w_k * (x_k - m_k)/s_k + 0.05 N(0,1), w_k ~ N(0, 0.1^2),
                  m, s = column mean / std of the drawn rows (constant columns skipped)
      quadratic : y = max(1e-3, 0.02 + 5e-5 L + 1e-9 L^2 + 0.03 Q - 4e-5 H
                          + 0.05 exp(0.3 N(0,1))), Q = queued, H = f2 (hit tokens).
    """
    kind, lo, hi = cfg.length
    L = _draw_lengths(rng, kind, lo, hi, n)
    if kind == "sys":
        L = L + 128 * (rng.random(n) < 0.5)
    nb = L // BLOCK
    x = np.zeros((n, cfg.d), np.float64)
    x[:, 0] = L
    h = np.floor(rng.random(n) * (nb + 1))
    x[:, 1] = h
    x[:, 2] = BLOCK * h
    x[:, 3] = (BLOCK * h).astype(np.float32) / L.astype(np.float32)
    x[:, 4] = L - BLOCK * h
    x[:, 5] = -(-L // BLOCK) - h
    x[:, PAIR_DIMS:PAIR_DIMS + cfg.d_inst] = instance_state(rng, cfg, n)
    if cfg.d_req:
        x[:, PAIR_DIMS + cfg.d_inst:] = rng.standard_normal((n, cfg.d_req))
    if cfg.ttft_model == "linear":
        m, s = x.mean(0), x.std(0)
        keep = s > 0
        w = rng.normal(0.0, 0.1, size=cfg.d)
        z = np.zeros_like(x)
        z[:, keep] = (x[:, keep] - m[keep]) / s[keep]
        y = z @ w + 0.05 * rng.standard_normal(n)
    else:
        Q = x[:, PAIR_DIMS + 0]
        y = (0.02 + 5e-5 * L + 1e-9 * L.astype(np.float64) ** 2 + 0.03 * Q
             - 4e-5 * x[:, 2] + 0.05 * np.exp(0.3 * rng.standard_normal(n)))
        y = np.maximum(y, 1e-3)
    return x.astype(np.float32), y.astype(np.float32)


def normaliser(rng, cfg: Config, n: int = 65536):
    """Per-feature mean/std (fp64 statistics of drawn records, rounded to fp32).
    Constant columns keep std = 0; the method substitutes 1 for them."""
    x, _ = records(rng, cfg, n)
    x = x.astype(np.float64)
    return x.mean(0).astype(np.float32), x.std(0).astype(np.float32)


# ----------------------------------------------------------------------------
# prompts and caches
# ----------------------------------------------------------------------------

def _sys_prompts(rng, n=4, length=128):
    return rng.integers(0, VOCAB, size=(n, length)).astype(np.int32)


def _sys_prompt_batch(rng, sysp, n, lo, hi):
    """Body U{lo..hi} random tokens; with p = 0.5 one of the system prompts is prepended."""
    seqs = []
    for _ in range(n):
        body = rng.integers(0, VOCAB, size=int(rng.integers(lo, hi + 1))).astype(np.int32)
        if rng.random() < 0.5:
            body = np.concatenate([sysp[int(rng.integers(0, len(sysp)))], body])
        seqs.append(body)
    return seqs


def _csr(seqs):
    off = np.zeros(len(seqs) + 1, np.int64)
    off[1:] = np.cumsum([len(s) for s in seqs])
    tok = np.concatenate(seqs).astype(np.int32) if seqs else np.zeros(0, np.int32)
    return tok, off


def _tiny_caches(cfg: Config, rng_hist, sysp):
    """Earlier prompts (same generator, history stream) are assigned to instances
    uniformly; each one's full blocks are cached prefix-closed until the instance
    holds `cache_blocks` distinct blocks.  Distinctness is decided on token
    content (a trie of block tuples), never on hashes."""
    N, budget = cfg.n_inst, cfg.cache_blocks
    history = []
    chains = [[] for _ in range(N)]
    tries = [dict() for _ in range(N)]
    counts = np.zeros(N, np.int64)
    while counts.min() < budget:
        seq = _sys_prompt_batch(rng_hist, sysp, 1, cfg.length[1], cfg.length[2])[0]
        i = int(rng_hist.integers(0, N))
        if counts[i] >= budget:
            continue
        trie, node, nb_new, nb = tries[i], 0, 0, len(seq) // BLOCK
        take = 0
        for b in range(nb):
            keyb = (node, seq[b * BLOCK:(b + 1) * BLOCK].tobytes())
            if keyb not in trie:
                if counts[i] + nb_new >= budget:
                    break
                trie[keyb] = len(trie) + 1
                nb_new += 1
            node = trie[keyb]
            take = b + 1
        if take == 0:
            continue
        counts[i] += nb_new
        chains[i].append((len(history), take))
        history.append(seq)
    return history, chains


def _template_caches(cfg: Config, rng_hist, n_tblocks):
    """Each instance draws templates ~ Zipf (with replacement, deduplicated) and
    caches the chain of the first k ~ U{1..n_tblocks} blocks of each, until half
    its budget is used; the other half is random nonzero 64-bit keys standing in
    for unshared suffix blocks (they never match a request)."""
    probs = _zipf_probs(cfg.n_templates, cfg.zipf_s)
    half = cfg.cache_blocks // 2
    chains, rand = [], []
    for _ in range(cfg.n_inst):
        used, seen, ch = 0, set(), []
        while used < half:
            ts = rng_hist.choice(cfg.n_templates, size=64, p=probs)
            ks = rng_hist.integers(1, n_tblocks + 1, size=64)
            for t, k in zip(ts.tolist(), ks.tolist()):
                if t in seen:
                    continue
                seen.add(t)
                k = min(k, half - used)
                ch.append((t, k))
                used += k
                if used >= half:
                    break
        chains.append(ch)
        nr = cfg.cache_blocks - used
        keys = rng_hist.integers(1, np.iinfo(np.int64).max, size=nr, dtype=np.int64).astype(np.uint64)
        keys ^= rng_hist.integers(0, 2, size=nr, dtype=np.uint64) << np.uint64(63)
        rand.append(keys)
    return chains, rand


def generate(name_or_cfg, n_req: int | None = None, with_samples: bool | None = None) -> Workload:
    """Build the seeded workload for one config.  `n_req` overrides the request
    count (same distributions, same seed) for reduced-size cases."""
    cfg = CONFIGS[name_or_cfg] if isinstance(name_or_cfg, str) else name_or_cfg
    R = cfg.n_req if n_req is None else int(n_req)
    rng = np.random.default_rng(cfg.seed)
    rng_hist = np.random.default_rng(cfg.seed + 1000)
    kind, lo, hi = cfg.length

    if kind == "sys":
        sysp = _sys_prompts(np.random.default_rng(cfg.seed + 2000))
        history, chains = _tiny_caches(cfg, rng_hist, sysp)
        # requests: fresh prompts; a quarter continue an earlier (cached) prompt
        seqs = []
        for _ in range(R):
            if rng.random() < 0.25:
                base = history[int(rng.integers(0, len(history)))]
                cut = int(rng.integers(1, len(base) + 1))
                extra = rng.integers(0, VOCAB, size=int(rng.integers(0, 256))).astype(np.int32)
                seqs.append(np.concatenate([base[:cut], extra])[: hi + 128])
            else:
                seqs.append(_sys_prompt_batch(rng, sysp, 1, lo, hi)[0])
        for s in range(len(seqs)):
            if len(seqs[s]) == 0:
                seqs[s] = rng.integers(0, VOCAB, size=1).astype(np.int32)
        tok, tok_off = _csr(seqs)
        seq_tok, seq_off = _csr(history)
        rand = [np.zeros(0, np.uint64) for _ in range(cfg.n_inst)]
    else:
        n_tblocks = cfg.max_len // BLOCK
        templates = np.random.default_rng(cfg.seed + 3000).integers(
            0, VOCAB, size=(cfg.n_templates, cfg.max_len)).astype(np.int32)
        chains, rand = _template_caches(cfg, rng_hist, n_tblocks)
        L = _draw_lengths(rng, kind, lo, hi, R)
        t = rng.choice(cfg.n_templates, size=R, p=_zipf_probs(cfg.n_templates, cfg.zipf_s))
        rho = rng.choice(np.array([0.1, 0.3, 0.5, 0.7]), size=R)
        tok_off = np.zeros(R + 1, np.int64)
        tok_off[1:] = np.cumsum(L)
        tok = rng.integers(0, VOCAB, size=int(tok_off[-1])).astype(np.int32)
        shared = np.floor(rho * L).astype(np.int64)
        for r in range(R):
            s0 = int(tok_off[r])
            tok[s0:s0 + shared[r]] = templates[t[r], :shared[r]]
        seq_tok = templates.ravel()
        seq_off = np.arange(cfg.n_templates + 1, dtype=np.int64) * cfg.max_len

    inst_chain_off = np.zeros(cfg.n_inst + 1, np.int64)
    inst_chain_off[1:] = np.cumsum([len(c) for c in chains])
    flat = [c for ch in chains for c in ch]
    chain_seq = np.array([c[0] for c in flat], np.int32)
    chain_blocks = np.array([c[1] for c in flat], np.int32)
    inst_rand_off = np.zeros(cfg.n_inst + 1, np.int64)
    inst_rand_off[1:] = np.cumsum([len(k) for k in rand])
    rand_keys = np.concatenate(rand) if rand else np.zeros(0, np.uint64)

    inst_state = instance_state(rng, cfg)
    req_feats = rng.standard_normal((R, cfg.d_req)).astype(np.float32)
    mean, std = normaliser(np.random.default_rng(cfg.seed + 4000), cfg)
    params = xavier_params(cfg.widths, 0)

    want = cfg.n_samples > 0 if with_samples is None else with_samples
    sx = sy = None
    if want and cfg.n_samples > 0:
        sx, sy = records(np.random.default_rng(cfg.seed + 5000), cfg, cfg.n_samples)

    return Workload(cfg, tok, tok_off, req_feats, inst_state, seq_tok, seq_off,
                    chain_seq, chain_blocks, inst_chain_off, rand_keys, inst_rand_off,
                    mean, std, params, sx, sy)


def minibatch_indices(seed: int, step: int, count: int, batch: int) -> np.ndarray:
    """Ring slots of minibatch `step`: default_rng((seed, step)).integers(0, count, batch)."""
    return np.random.default_rng((seed, step)).integers(0, count, size=batch).astype(np.int32)
