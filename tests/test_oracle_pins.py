"""Pins of the CPU oracle against facts that do not come from the oracle.

Each test checks one part of the oracle against mathematics, a closed form,
brute force, exhaustive enumeration or an independent library routine, so that
a dropped term, a wrong sign or index, or a transposed operand in the oracle
fails at least one of them.  No GPU needed.
"""
import dataclasses
import os
import shutil
import subprocess

import numpy as np
import pytest

import oracle
from paper_2606_00946_gb300 import workload as W

M64 = 2**64 - 1
G = 0x9E3779B97F4A7C15


# ----------------------------------------------------------------------------
# block hash
# ----------------------------------------------------------------------------

def test_mix64_splitmix64_reference_outputs():
    # The SplitMix64 generator (state += G, output = finaliser(state)) seeded
    # with 1234567 has the published first outputs below (Vigna's public-domain
    # splitmix64.c reference sequence).  Pins both multipliers and all shifts.
    s, out = 1234567, []
    for _ in range(5):
        s = (s + G) & M64
        out.append(oracle.mix64(s))
    assert out == [6457827717110365317, 3203168211198807973, 9817491932198370423,
                   4593380528125082431, 16408922859458223821]


def _unxorshift(y, s):
    x = y
    for _ in range(64 // s + 1):
        x = y ^ (x >> s)
    return x


def test_mix64_is_the_invertible_finaliser():
    # The finaliser is a bijection; invert it with modular inverses of the two
    # multipliers and by undoing the xor-shifts, then round-trip random words.
    c1, c2 = 0xBF58476D1CE4E5B9, 0x94D049BB133111EB
    i1, i2 = pow(c1, -1, 2**64), pow(c2, -1, 2**64)

    def inv(z):
        z = _unxorshift(z, 31)
        z = (z * i2) & M64
        z = _unxorshift(z, 27)
        z = (z * i1) & M64
        return _unxorshift(z, 30)

    rng = np.random.default_rng(7)
    for v in rng.integers(0, 2**63, size=200, dtype=np.uint64).tolist() + [0, 1, M64]:
        assert inv(oracle.mix64(v)) == v


def test_mix64_matches_pybind11_header_implementation(tmp_path):
    # An independent third-party implementation of the same mixer ships in the
    # pybind11 headers; compile a tiny caller against it when available.
    pb = pytest.importorskip("pybind11")
    inc = pb.get_include()
    import sysconfig
    pyinc = sysconfig.get_paths()["include"]
    if not shutil.which("g++") or not os.path.exists(os.path.join(pyinc, "Python.h")):
        pytest.skip("no C++ compiler or Python headers")
    src = tmp_path / "m.cpp"
    src.write_text('#include <pybind11/detail/internals.h>\n#include <cstdio>\n#include <cstdlib>\n'
                   'int main(int c,char**v){for(int i=1;i<c;++i)printf("%llu\\n",'
                   '(unsigned long long)pybind11::detail::mix64(strtoull(v[i],0,10)));}\n')
    exe = tmp_path / "m"
    libdir = sysconfig.get_config_var("LIBDIR")
    ver = sysconfig.get_config_var("LDVERSION")
    r = subprocess.run(["g++", "-std=c++17", "-w", f"-I{inc}", f"-I{pyinc}", str(src), "-o", str(exe),
                        f"-L{libdir}", f"-lpython{ver}"], capture_output=True)
    if r.returncode != 0:
        pytest.skip("pybind11 header does not compile here")
    vals = [1, 2, 3, 12345678901234, 2**63 + 5, M64]
    out = subprocess.run([str(exe)] + [str(v) for v in vals], capture_output=True, text=True, check=True)
    assert [int(x) for x in out.stdout.split()] == [oracle.mix64(v) for v in vals]


def _rand_tokens(rng, n):
    return rng.integers(0, 32000, size=n).astype(np.int32)


def test_hash_chain_closed_form():
    # The prefix state recurrence s_b = s_{b-1} G + c_b, s_{-1} = G has the
    # closed form s_b = G^(b+2) + sum_j c_j G^(b-j) (mod 2^64); key_b = mix64(s_b).
    rng = np.random.default_rng(1)
    t = _rand_tokens(rng, 16 * 9 + 5)
    keys, koff = oracle.hash_blocks(t, np.array([0, len(t)]))
    assert len(keys) == 9
    c = [oracle.block_content(t[16 * b:16 * b + 16]) for b in range(9)]
    for b in range(9):
        s = pow(G, b + 2, 2**64)
        for j in range(b + 1):
            s = (s + c[j] * pow(G, b - j, 2**64)) % 2**64
        k = oracle.mix64(s)
        assert int(keys[b]) == (k if k else 1)


def test_hash_prefix_and_locality_properties():
    rng = np.random.default_rng(2)
    t = _rand_tokens(rng, 16 * 12)
    base, _ = oracle.hash_blocks(t, np.array([0, len(t)]))
    # keys of a prefix are a prefix of the keys; a partial tail block adds none
    for cut in (0, 15, 16, 17, 100, 16 * 12 - 1):
        k, _ = oracle.hash_blocks(t[:cut], np.array([0, cut]))
        assert len(k) == cut // 16
        assert np.array_equal(k, base[: cut // 16])
    # changing one token of block j changes keys j.. and leaves keys ..j-1
    for pos in (0, 5, 16 * 3 + 15, 16 * 7 + 2, 16 * 12 - 1):
        t2 = t.copy()
        t2[pos] ^= 1
        k2, _ = oracle.hash_blocks(t2, np.array([0, len(t2)]))
        j = pos // 16
        assert np.array_equal(k2[:j], base[:j])
        assert np.all(k2[j:] != base[j:])
    # every one of the 16 tokens of a block matters, and block order matters
    for p in range(16):
        t3 = t.copy()
        t3[p] += 1
        assert oracle.block_content(t3[:16]) != oracle.block_content(t[:16])
    swapped = np.concatenate([t[16:32], t[:16]])
    ks, _ = oracle.hash_blocks(swapped, np.array([0, 32]))
    assert ks[1] != base[1]
    # CSR of several sequences = hashing each alone
    offs = np.array([0, 40, 40, 97, len(t)])
    kk, ko = oracle.hash_blocks(t, offs)
    for s in range(4):
        alone, _ = oracle.hash_blocks(t[offs[s]:offs[s + 1]], np.array([0, offs[s + 1] - offs[s]]))
        assert np.array_equal(kk[ko[s]:ko[s + 1]], alone)
    assert np.all(kk != 0)


def test_hash_no_collisions_on_tiny_workload():
    # Distinct block prefixes (decided on token content) must get distinct keys.
    wl = W.generate("tiny")
    seqs = [wl.tok[wl.tok_off[r]:wl.tok_off[r + 1]] for r in range(len(wl.tok_off) - 1)]
    seqs += [wl.seq_tok[wl.seq_off[s]:wl.seq_off[s + 1]] for s in range(len(wl.seq_off) - 1)]
    by_prefix = {}
    for s in seqs:
        k, _ = oracle.hash_blocks(s, np.array([0, len(s)]))
        for b in range(len(k)):
            by_prefix.setdefault(s[:16 * (b + 1)].tobytes(), set()).add(int(k[b]))
    assert all(len(v) == 1 for v in by_prefix.values())
    keys = [next(iter(v)) for v in by_prefix.values()]
    assert len(set(keys)) == len(keys)


# ----------------------------------------------------------------------------
# prefix hits: brute force on token content
# ----------------------------------------------------------------------------

def _brute_hits(req_seqs, inst_cached_prefixes):
    """h = number of leading full blocks b whose whole token prefix
    r[:16(b+1)] is cached on the instance, stopping at the first that is not."""
    out = np.zeros((len(req_seqs), len(inst_cached_prefixes)), np.int32)
    for r, s in enumerate(req_seqs):
        for i, cached in enumerate(inst_cached_prefixes):
            b = 0
            while b < len(s) // 16 and s[:16 * (b + 1)].tobytes() in cached:
                b += 1
            out[r, i] = b
    return out


def _inst_keys_from_blocks(inst_blocks):
    """inst_blocks[i] = list of (token sequence, set of block indices cached)."""
    parts, off = [], [0]
    for lst in inst_blocks:
        ks = []
        for seq, bs in lst:
            k, _ = oracle.hash_blocks(seq, np.array([0, len(seq)]))
            ks += [int(k[b]) for b in sorted(bs)]
        parts.append(np.array(ks, np.uint64))
        off.append(off[-1] + len(ks))
    return np.concatenate(parts) if parts else np.zeros(0, np.uint64), np.array(off, np.int64)


def _cached_prefix_sets(inst_blocks):
    return [{seq[:16 * (b + 1)].tobytes() for seq, bs in lst for b in bs} for lst in inst_blocks]


@pytest.mark.parametrize("seed", [0, 1, 2, 3])
def test_prefix_hits_brute_force_with_holes(seed):
    rng = np.random.default_rng(100 + seed)
    base = [_rand_tokens(rng, int(rng.integers(16, 300))) for _ in range(6)]
    reqs = []
    for _ in range(20):
        b = base[int(rng.integers(0, len(base)))]
        cut = int(rng.integers(0, len(b) + 1))
        tail = _rand_tokens(rng, int(rng.integers(0, 60)))
        reqs.append(np.concatenate([b[:cut], tail]).astype(np.int32))
    reqs.append(np.zeros(0, np.int32))           # empty prompt
    reqs.append(_rand_tokens(rng, 15))           # shorter than a block
    inst_blocks = []
    for i in range(5):
        lst = []
        for s in base:
            nb = len(s) // 16
            if nb == 0 or rng.random() < 0.3:
                continue
            if i == 4:                       # an instance with holes (not prefix-closed)
                bs = {b for b in range(nb) if rng.random() < 0.7}
            else:                            # prefix-closed chains
                bs = set(range(int(rng.integers(1, nb + 1))))
            lst.append((s, bs))
        inst_blocks.append(lst)
    inst_blocks.append([])                   # an empty instance
    inst_blocks.append([(s, set(range(len(s) // 16))) for s in base])   # everything cached
    ik, iko = _inst_keys_from_blocks(inst_blocks)
    off = np.zeros(len(reqs) + 1, np.int64)
    off[1:] = np.cumsum([len(s) for s in reqs])
    rk, rko = oracle.hash_blocks(np.concatenate(reqs), off)
    want = _brute_hits(reqs, _cached_prefix_sets(inst_blocks))
    got = oracle.prefix_hits(rk, rko, ik, iko)
    got2 = oracle.prefix_hits(rk, rko, ik, iko, by_marking=True)
    assert np.array_equal(got, want)
    assert np.array_equal(got2, want)
    assert np.all(got[-2:] == 0) and np.all(got[:, -2] == 0)
    # fully cached instance: every request that is a prefix of a base sequence
    # (tail of length 0) matches all of its full blocks
    # monotonicity: adding keys never lowers a hit
    extra = rng.integers(1, 2**63, size=50, dtype=np.uint64)
    ik2 = np.concatenate([ik[:iko[1]], extra, ik[iko[1]:]])
    iko2 = iko.copy()
    iko2[1:] += len(extra)
    got3 = oracle.prefix_hits(rk, rko, ik2, iko2)
    assert np.all(got3 >= got)


def test_prefix_hits_tiny_workload_brute_force():
    wl = W.generate("tiny")
    reqs = [wl.tok[wl.tok_off[r]:wl.tok_off[r + 1]] for r in range(len(wl.tok_off) - 1)]
    inst_blocks = []
    for i in range(wl.cfg.n_inst):
        lst = []
        for c in range(wl.inst_chain_off[i], wl.inst_chain_off[i + 1]):
            s = wl.seq_tok[wl.seq_off[wl.chain_seq[c]]:wl.seq_off[wl.chain_seq[c] + 1]]
            lst.append((s, set(range(int(wl.chain_blocks[c])))))
        inst_blocks.append(lst)
    want = _brute_hits(reqs, _cached_prefix_sets(inst_blocks))
    ik, iko = oracle.instance_keys(wl)
    rk, rko = oracle.hash_blocks(wl.tok, wl.tok_off)
    got = oracle.prefix_hits(rk, rko, ik, iko)
    assert np.array_equal(got, want)
    assert want.max() > 8 and (want == 0).any()      # the workload exercises long and zero hits
    # distinct blocks per instance equal the configured budget
    for i in range(wl.cfg.n_inst):
        assert len(np.unique(ik[iko[i]:iko[i + 1]])) == wl.cfg.cache_blocks


# ----------------------------------------------------------------------------
# features
# ----------------------------------------------------------------------------

def test_raw_features_worked_examples():
    inst = np.arange(10, dtype=np.float32) + 0.5
    req = np.array([-1.25, 2.0], np.float32)
    x = oracle.raw_features_row(100, 3, inst, req)
    assert x.tolist()[:6] == [100.0, 3.0, 48.0, np.float32(0.48), 52.0, 4.0]
    assert x[6:16].tolist() == inst.tolist() and x[16:].tolist() == req.tolist()
    # whole blocks only: L = 64, h = 4 -> nothing left to prefill or allocate
    assert oracle.raw_features_row(64, 4, inst, []).tolist()[:6] == [64.0, 4.0, 64.0, 1.0, 0.0, 0.0]
    # L = 0 (reading: kappa = 0), L < 16
    assert oracle.raw_features_row(0, 0, inst, []).tolist()[:6] == [0.0, 0.0, 0.0, 0.0, 0.0, 0.0]
    assert oracle.raw_features_row(15, 0, inst, []).tolist()[:6] == [15.0, 0.0, 0.0, 0.0, 15.0, 1.0]


def test_features_zscore_worked_example():
    L = np.array([100, 32])
    hits = np.array([[3, 0], [2, 1]], np.int32)
    inst = np.array([[1.0], [3.0]], np.float32)
    req = np.zeros((2, 0), np.float32)
    mean = np.array([50, 1, 16, 0.5, 30, 2, 2.0], np.float32)
    std = np.array([25, 2, 8, 0.25, 0, 1, 1.0], np.float32)   # std 0 -> divide by 1
    x = oracle.features(L, hits, inst, req, mean, std)
    assert x.shape == (4, 7)
    np.testing.assert_array_equal(x[0], np.array([2.0, 1.0, 4.0, (np.float32(0.48) - np.float32(0.5)) / np.float32(0.25),
                                                  22.0, 2.0, -1.0], np.float32))
    np.testing.assert_array_equal(x[3], np.array([-0.72, 0.0, 0.0, 0.0, 16.0 - 30.0, -1.0, 1.0],
                                                 np.float32))


# ----------------------------------------------------------------------------
# bf16 rounding and the predictor
# ----------------------------------------------------------------------------

def test_bf16_matches_torch_rounding():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(3)
    v = np.concatenate([rng.standard_normal(2000).astype(np.float32) * 10.0 ** rng.integers(-30, 30, 2000),
                        np.array([1 + 2**-8, 1 + 3 * 2**-8, -(1 + 2**-8), 3.3895314e38, 1e-40,
                                  -1e-42, 0.0, -0.0, np.inf, -np.inf], np.float32)]).astype(np.float32)
    want = torch.from_numpy(v).to(torch.bfloat16).to(torch.float32).numpy()
    got = oracle.bf16(v)
    np.testing.assert_array_equal(got.view(np.uint32), want.view(np.uint32))


def _random_net(rng, widths, positive=False):
    p = []
    for l in range(len(widths) - 1):
        Wl = rng.standard_normal((widths[l + 1], widths[l])) / np.sqrt(widths[l])
        b = rng.standard_normal(widths[l + 1]) * 0.1
        if positive:
            Wl, b = np.abs(Wl), np.abs(b)
        p += [Wl.astype(np.float32).ravel(), b.astype(np.float32)]
    return np.concatenate(p).astype(np.float64)


def _unpack(p, widths):
    out, o = [], 0
    for l in range(len(widths) - 1):
        n = widths[l + 1] * widths[l]
        out.append((p[o:o + n].reshape(widths[l + 1], widths[l]), p[o + n:o + n + widths[l + 1]]))
        o += n + widths[l + 1]
    return out


def test_mlp_affine_closed_form():
    # All weights, biases and inputs positive => every pre-activation positive,
    # the ReLU network is affine: y = (W3 W2 W1) x + (W3 W2 b1 + W3 b2 + b3).
    rng = np.random.default_rng(4)
    widths = [16, 64, 64, 1]
    p = _random_net(rng, widths, positive=True)
    x = np.abs(rng.standard_normal((50, 16)))
    (W1, b1), (W2, b2), (W3, b3) = _unpack(p, widths)
    Wt = W3 @ (W2 @ W1)
    c = W3 @ (W2 @ b1) + W3 @ b2 + b3
    want = x @ Wt.T + c
    got = oracle.mlp_forward("f64", widths, p, x)
    np.testing.assert_allclose(got, want.ravel(), rtol=1e-12)


def test_mlp_matches_torch_modules():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(5)
    widths = [20, 32, 48, 16, 1]
    p = _random_net(rng, widths)
    x = rng.standard_normal((64, 20)).astype(np.float32)
    layers = []
    for l, (Wl, b) in enumerate(_unpack(p, widths)):
        lin = torch.nn.Linear(widths[l], widths[l + 1]).double()
        with torch.no_grad():
            lin.weight.copy_(torch.from_numpy(Wl))
            lin.bias.copy_(torch.from_numpy(b))
        layers.append(lin)
        if l + 2 < len(widths):
            layers.append(torch.nn.ReLU())
    net = torch.nn.Sequential(*layers)
    want = net(torch.from_numpy(x.astype(np.float64))).detach().numpy().ravel()
    np.testing.assert_allclose(oracle.mlp_forward("f64", widths, p, x), want, rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(oracle.mlp_forward("f32", widths, p, x), want, rtol=1e-5, atol=1e-6)
    # bf16 rounding points, built from torch's own bf16 conversion and matmul
    bf = lambda t: t.to(torch.bfloat16).to(torch.float64)
    a = bf(torch.from_numpy(x).double())
    for l, (Wl, b) in enumerate(_unpack(p, widths)):
        z = (a @ bf(torch.from_numpy(Wl).float()).T + torch.from_numpy(b)).float().double()
        a = bf(torch.relu(z).float()) if l + 2 < len(widths) else z
    np.testing.assert_allclose(oracle.mlp_forward("bf16", widths, p, x), a.numpy().ravel(),
                               rtol=1e-6, atol=1e-7)


# ----------------------------------------------------------------------------
# argmin
# ----------------------------------------------------------------------------

def _enumerate_argmin(row):
    def key(i):
        v = float(row[i])
        return (np.isnan(v), 0.0 if np.isnan(v) else v, i)
    return min(range(len(row)), key=key)


def test_argmin_exhaustive():
    rng = np.random.default_rng(6)
    vals = np.array([0.5, -0.0, 0.0, 1.0, np.nan, -2.0, np.inf, -np.inf], np.float32)
    rows = [rng.choice(vals, size=n) for n in (1, 2, 3, 5, 8, 33) for _ in range(200)]
    rows += [np.full(4, np.nan, np.float32), np.array([0.0, -0.0], np.float32),
             np.array([-0.0, 0.0], np.float32)]
    for row in rows:
        c, b = oracle.argmin(row.reshape(1, -1).astype(np.float32))
        want = _enumerate_argmin(row)
        assert c[0] == want
        assert (np.isnan(b[0]) and np.isnan(row[want])) or b[0] == row[want]
    # every choice of a 3-element row over a small value set, exhaustively
    small = np.array([1.0, 2.0, np.nan, -0.0, 0.0], np.float32)
    import itertools
    for trip in itertools.product(small, repeat=3):
        row = np.array(trip, np.float32)
        c, _ = oracle.argmin(row.reshape(1, 3))
        assert c[0] == _enumerate_argmin(row)


# ----------------------------------------------------------------------------
# sample ring
# ----------------------------------------------------------------------------

def test_ring_wraps_oldest_first():
    rx = np.zeros((5, 2), np.float32)
    ry = np.zeros(5, np.float32)
    n = 0
    for batch in ([1, 2, 3], [4, 5, 6], [7]):
        x = np.array([[v, -v] for v in batch], np.float32)
        n = oracle.ring_append(rx, ry, n, x, np.array(batch, np.float32))
    assert n == 7
    assert ry.tolist() == [6.0, 7.0, 3.0, 4.0, 5.0]
    assert rx[:, 1].tolist() == [-6.0, -7.0, -3.0, -4.0, -5.0]


# ----------------------------------------------------------------------------
# loss, gradients, optimisers
# ----------------------------------------------------------------------------

def _train_setup(seed=8, widths=(16, 64, 64, 1), n=96):
    rng = np.random.default_rng(seed)
    d = widths[0]
    x = (rng.standard_normal((n, d)) * 3 + 1).astype(np.float32)
    y = rng.standard_normal(n).astype(np.float32)
    mean = x.mean(0).astype(np.float32)
    std = x.std(0).astype(np.float32)
    p = _random_net(rng, list(widths))
    idx = rng.integers(0, n, size=48).astype(np.int32)
    return list(widths), p, x, y, mean, std, idx


def test_loss_worked_example():
    widths = [2, 1]
    p = np.array([1.0, -1.0, 0.5])          # y = x0 - x1 + 0.5
    x = np.array([[1, 2], [3, 1]], np.float32)
    y = np.array([0.0, 2.0], np.float32)
    mean, std = np.zeros(2, np.float32), np.ones(2, np.float32)
    # predictions -0.5 and 2.5 -> errors -0.5, 0.5 -> MSE 0.25
    assert oracle.loss("f64", widths, p, x, y, np.array([0, 1], np.int32), mean, std) == 0.25


def test_gradient_finite_differences():
    widths, p, x, y, mean, std, idx = _train_setup()
    tr = oracle.Trainer(widths, p, "f64")
    _, g = tr.step(x, y, idx, mean, std, opt="sgd", lr=0.0, want_grad=True)
    rng = np.random.default_rng(9)
    coords = rng.choice(len(p), size=120, replace=False)
    for c in coords:
        h = 1e-6 * max(1.0, abs(p[c]))
        pp, pm = p.copy(), p.copy()
        pp[c] += h
        pm[c] -= h
        fd = (oracle.loss("f64", widths, pp, x, y, idx, mean, std)
              - oracle.loss("f64", widths, pm, x, y, idx, mean, std)) / (2 * h)
        assert abs(fd - g[c]) <= 1e-6 * max(1.0, np.abs(g).max()), (c, fd, g[c])


def _torch_net_grad(torch, widths, p, xn, yb):
    params = [torch.tensor(a, dtype=torch.float64, requires_grad=True)
              for Wl, b in _unpack(p, widths) for a in (Wl, b)]
    a = torch.from_numpy(xn.astype(np.float64))
    for l in range(len(widths) - 1):
        a = a @ params[2 * l].T + params[2 * l + 1]
        if l + 2 < len(widths):
            a = torch.relu(a)
    loss = ((a.ravel() - torch.from_numpy(yb.astype(np.float64))) ** 2).mean()
    loss.backward()
    return loss.item(), np.concatenate([q.grad.numpy().ravel() for q in params])


def test_gradient_matches_torch_autograd():
    torch = pytest.importorskip("torch")
    widths, p, x, y, mean, std, idx = _train_setup(widths=(12, 40, 24, 16, 1))
    xz = np.stack([(x[i] - mean) / np.where(std < 1e-12, 1, std) for i in idx]).astype(np.float32)
    want_loss, want_g = _torch_net_grad(torch, widths, p, xz, y[idx])
    tr = oracle.Trainer(widths, p, "f64")
    got_loss, g = tr.step(x, y, idx, mean, std, opt="sgd", lr=0.0, want_grad=True)
    assert abs(got_loss - want_loss) <= 1e-12 * max(1.0, want_loss)
    np.testing.assert_allclose(g, want_g, rtol=1e-10, atol=1e-12)
    # fp32 mode approximates the same gradient
    _, gm = oracle.Trainer(widths, p, "f32").step(x, y, idx, mean, std, opt="sgd", lr=0.0,
                                                 want_grad=True)
    assert np.linalg.norm(gm - want_g) <= 1e-5 * np.linalg.norm(want_g)


def test_bf16_gradient_matches_vectorised_emulation():
    # The bf16 reading (operands of every product rounded with torch's bf16
    # conversion, sums formed in fp64 then rounded to fp32, db from unrounded
    # dZ) rebuilt with whole-matrix numpy products.
    torch = pytest.importorskip("torch")
    widths, p, x, y, mean, std, idx = _train_setup(widths=(12, 40, 24, 16, 1))
    xz = np.stack([(x[i] - mean) / np.where(std < 1e-12, 1, std) for i in idx]).astype(np.float32)
    bf = lambda a: torch.from_numpy(np.asarray(a, np.float32)).to(torch.bfloat16).double().numpy()
    f32 = lambda a: np.asarray(a, np.float32).astype(np.float64)
    layers = _unpack(p, widths)
    A, Z, a = [bf(xz)], [], bf(xz)
    for l, (Wl, b) in enumerate(layers):
        z = f32(a @ bf(Wl).T + b)
        Z.append(z)
        a = z if l + 1 == len(layers) else bf(np.maximum(z, 0))
        if l + 1 < len(layers):
            A.append(a)
    dz = f32((2 * (a.ravel() - y[idx]) / len(idx))[:, None])
    grads = []
    for l in range(len(layers) - 1, -1, -1):
        Wl, _ = layers[l]
        grads.append((f32(bf(dz).T @ A[l]), f32(dz.sum(0))))
        if l > 0:
            dz = f32(bf(dz) @ bf(Wl)) * (Z[l - 1] > 0)
    want = np.concatenate([np.concatenate([gW.ravel(), gb]) for gW, gb in grads[::-1]])
    _, got = oracle.Trainer(widths, p, "bf16").step(x, y, idx, mean, std, opt="sgd", lr=0.0,
                                                   want_grad=True)
    assert np.linalg.norm(got - want) <= 1e-6 * np.linalg.norm(want)


def test_sgd_closed_form():
    widths, p, x, y, mean, std, idx = _train_setup()
    tr = oracle.Trainer(widths, p, "f64")
    _, g = tr.step(x, y, idx, mean, std, opt="sgd", lr=0.0, want_grad=True)
    tr2 = oracle.Trainer(widths, p, "f64")
    tr2.step(x, y, idx, mean, std, opt="sgd", lr=1e-3)
    np.testing.assert_allclose(tr2.params, p - 1e-3 * g, rtol=0, atol=1e-15)


def test_adam_matches_torch_optim():
    torch = pytest.importorskip("torch")
    widths, p, x, y, mean, std, idx = _train_setup()
    tr = oracle.Trainer(widths, p, "f64")
    ref = torch.tensor(p.copy(), dtype=torch.float64, requires_grad=True)
    opt = torch.optim.Adam([ref], lr=3e-4)
    for step in range(4):
        before = tr.params.copy()
        # gradient of this step at the current parameters
        g = oracle.Trainer(widths, before, "f64").step(x, y, idx, mean, std, opt="sgd", lr=0.0,
                                                       want_grad=True)[1]
        tr.step(x, y, idx, mean, std, opt="adam", lr=3e-4)
        ref.grad = torch.from_numpy(g.copy())
        opt.step()
        np.testing.assert_allclose(tr.params, ref.detach().numpy(), rtol=1e-12, atol=1e-15)
        if step == 0:   # first Adam step moves every coordinate by ~lr*sign(g)
            big = np.abs(g) > 1e-4   # eps/|g| below 1e-4
            np.testing.assert_allclose((tr.params - before)[big], -3e-4 * np.sign(g[big]), rtol=1e-3)


def test_linear_model_converges_to_least_squares():
    # A d->1 predictor (no hidden layer) trained by full-batch SGD converges to
    # the least-squares fit of y on the normalised features plus intercept.
    rng = np.random.default_rng(10)
    n, d = 200, 5
    x = (rng.standard_normal((n, d)) * [1, 2, 3, 4, 5] + [1, -1, 0, 2, 3]).astype(np.float32)
    y = (x @ np.array([0.3, -0.2, 0.1, 0.05, 0.0]) + 0.5 + 0.1 * rng.standard_normal(n)).astype(np.float32)
    mean, std = x.mean(0).astype(np.float32), x.std(0).astype(np.float32)
    tr = oracle.Trainer([d, 1], np.zeros(d + 1), "f64")
    idx = np.arange(n, dtype=np.int32)
    for _ in range(600):
        tr.step(x, y, idx, mean, std, opt="sgd", lr=0.2)
    xz = ((x - mean) / std).astype(np.float32).astype(np.float64)
    A = np.hstack([xz, np.ones((n, 1))])
    sol = np.linalg.lstsq(A, y.astype(np.float64), rcond=None)[0]
    np.testing.assert_allclose(tr.params, sol, atol=1e-8)


# ----------------------------------------------------------------------------
# rounding analysis of the forward pass (the parity tests' radius per row)
# ----------------------------------------------------------------------------

def test_forward_bounds_output_equals_the_forward_pass():
    rng = np.random.default_rng(40)
    for mode, widths in (("f32", (16, 64, 64, 1)), ("bf16", (24, 32, 32, 32, 1))):
        params = W.xavier_params(widths, 3)
        x = rng.standard_normal((50, widths[0])).astype(np.float32)
        y, eb, fl = oracle.mlp_forward_bounds(mode, widths, params, x)
        assert np.array_equal(y, oracle.mlp_forward(mode, widths, params, x))
        assert (eb > 0).all() and (fl >= 0).all()
        if mode == "f32":
            assert (fl == 0).all()


def test_forward_bounds_radius_of_a_single_dot_product():
    # one linear layer (K = 3 inputs): radius = 4 sqrt(K + 1) 2^-24 sqrt(sum (w a)^2 + b^2)
    # + 2 2^-24 |z| for the sum, + 2 2^-24 |z| for the output's own rounding
    widths = (3, 1)
    w = np.array([0.5, -0.25, 2.0], np.float32)
    b = np.float32(0.125)
    params = np.concatenate([w, [b]]).astype(np.float32)
    x = np.array([[1.0, 2.0, 3.0]], np.float32)
    y, eb, fl = oracle.mlp_forward_bounds("f32", widths, params, x)
    z = 0.5 - 0.5 + 6.0 + 0.125
    u = 2.0 ** -24
    s2 = 0.25 + 0.25 + 36.0 + 0.125 ** 2
    assert y[0] == z
    assert np.isclose(eb[0], 4 * np.sqrt(4.0) * u * np.sqrt(s2) + 4 * u * abs(z), rtol=1e-12)


def test_forward_bounds_flip_at_a_bf16_midpoint():
    # hidden unit pre-activation exactly 1 + 2^-8 (the midpoint of bf16 1 and
    # 1 + 2^-7; round-to-nearest-even keeps 1): flagged, and its flip moves the
    # output by w2 * 2^-7 exactly; 1 + 2^-6 sits on a bf16 value: no flip
    widths = (1, 1, 1)
    for pre, want in ((1.0 + 2.0 ** -8, 3.0 * 2.0 ** -7), (1.0 + 2.0 ** -6, 0.0)):
        params = np.array([1.0, pre - 1.0, 3.0, 0.0], np.float32)   # W1 = 1, b1, W2 = 3, b2 = 0
        x = np.array([[1.0]], np.float32)
        y, eb, fl = oracle.mlp_forward_bounds("bf16", widths, params, x)
        assert fl[0] == want


def test_prefix_hits_on_presorted_sets_equal_the_plain_scan():
    wl = W.generate("tiny")
    rk, rko = oracle.hash_blocks(wl.tok, wl.tok_off)
    ik, iko = oracle.instance_keys(wl)
    want = oracle.prefix_hits(rk, rko, ik, iko)
    assert np.array_equal(oracle.prefix_hits_sorted(rk, rko, oracle.sorted_instance_keys((ik, iko))), want)
    r = oracle.route(wl, inst_sorted=oracle.sorted_instance_keys((ik, iko)))
    assert np.array_equal(r["hits"], want)
    with pytest.raises(Exception):                  # an unsorted set is refused
        oracle.prefix_hits_sorted(rk, rko, (ik, iko))


def test_vectorised_trainer_follows_the_scalar_oracle():
    # five bf16 Adam steps of the vectorised restatement against or_train_step:
    # the same losses and parameters up to fp64 summation order (an fp32 or
    # bf16 rounding point may land on the other side for a handful of values)
    from oracle.train_np import NpTrainer, bf16
    cfg = W.CONFIGS["training"]
    widths = (cfg.d, 64, 64, 1)
    rng = np.random.default_rng(50)
    x, y = W.records(rng, dataclasses.replace(cfg, hidden=(64, 64)), 600)
    mean, std = W.normaliser(np.random.default_rng(51), cfg)
    params = W.xavier_params(widths, 2)
    a = oracle.Trainer(widths, params, "bf16")
    b = NpTrainer(widths, params)
    for k in range(5):
        idx = W.minibatch_indices(9, k, 600, 256)
        la = a.step(x, y, idx, mean, std, "adam", 1e-3)
        lb = b.step(x, y, idx, mean, std, 1e-3)
        assert abs(la - lb) <= 1e-6 * la
        d = np.abs(a.params - b.params)
        assert np.mean(d <= 1e-6 * np.maximum(np.abs(a.params), 1e-3)) > 0.999
        assert d.max() <= 3e-3                     # at most a few flipped roundings, each under lr
    # the bf16 rounding itself against torch
    import torch
    v = rng.standard_normal(10000).astype(np.float32) * 3
    assert np.array_equal(bf16(v), torch.from_numpy(v).to(torch.bfloat16).to(torch.float64).numpy())
