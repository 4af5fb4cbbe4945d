"""Pins of the oracle's fallback heuristics (Algorithm 1: prefix-cache and
load aware; Algorithm 2: prefix aware with a threshold) against exhaustive
enumeration with numpy's mean / standard deviation and Python's sort, exact
threshold boundaries and the special cases the algorithms state.  No GPU.
"""
import numpy as np

import oracle

BLOCK = 16


def _m(L, h):
    # prefix match ratio of Sec. 4.1 (expected KV hit ratio), fp32
    return np.float32(BLOCK * h) / np.float32(L) if L > 0 else np.float32(0)


def _alg1_brute(L, hits, c, theta, k):
    c = c.astype(np.float64)
    least = int(np.argmin(c))                       # first index of the smallest count
    if float(c.max()) - float(c.min()) > theta:
        return [least] * len(L)
    thr = float(np.mean(c)) + float(np.float32(k)) * float(np.std(c))
    out = []
    for r in range(len(L)):
        m = [_m(L[r], h) for h in hits[r]]
        order = sorted(range(len(c)), key=lambda i: (-m[i], c[i], i))
        pick = next((i for i in order if c[i] <= thr), least)
        out.append(pick)
    return out


def _setting(seed, R=50, N=12):
    rng = np.random.default_rng(seed)
    L = rng.integers(0, 400, size=R).astype(np.int64)
    hits = np.stack([rng.integers(0, L[r] // BLOCK + 1, size=N) for r in range(R)]).astype(np.int32)
    inst = np.zeros((N, 5), np.float32)
    inst[:, 0] = rng.integers(0, 8, size=N)          # queued
    inst[:, 1] = rng.integers(0, 12, size=N)         # running
    inst[:, 2:] = rng.standard_normal((N, 3))
    return L, hits, inst


def test_alg1_matches_enumeration_with_numpy_statistics():
    for seed in range(20):
        L, hits, inst = _setting(seed)
        c = inst[:, 0].astype(np.float64) + inst[:, 1]
        for k in (0.0, 0.5, 1.0, 2.0):
            got = oracle.heuristic(L, hits, inst, mode=1, count_cols=(0, 1), theta_imbal=1e9, k=k)
            assert got.tolist() == _alg1_brute(L, hits, c, 1e9, k), (seed, k)


def test_alg1_imbalance_sends_everything_to_the_least_loaded():
    L, hits, inst = _setting(3, N=4)
    inst[:, 0] = [5, 1, 9, 1]
    got = oracle.heuristic(L, hits, inst, mode=1, count_cols=(0, -1), theta_imbal=7.0, k=1.0)
    assert (got == 1).all()                          # 9 - 1 = 8 > 7; lowest index of the two 1s
    got = oracle.heuristic(L, hits, inst, mode=1, count_cols=(0, -1), theta_imbal=8.0, k=1.0)
    assert got.tolist() == _alg1_brute(L, hits, inst[:, 0], 8.0, 1.0)   # 8 > 8 is false


def test_alg1_overload_bound_is_inclusive():
    # c = [1, 1, 3, 3]: mean 2, population std 1, so mu + 1 sigma = 3 exactly
    L = np.array([64], np.int64)
    hits = np.array([[0, 0, 4, 1]], np.int32)        # best prefix match on instance 2 (c = 3)
    inst = np.array([[1, 0], [1, 0], [3, 0], [3, 0]], np.float32)
    assert oracle.heuristic(L, hits, inst, mode=1, count_cols=(0, -1), theta_imbal=99, k=1.0)[0] == 2
    # k one fp32 ulp below 1: mu + k sigma = 3 - 2^-24 in fp64, just below 3 (fp32
    # arithmetic would round it back to 3), so instances 2 and 3 are overloaded;
    # the best of 0 and 1 (m equal, c equal) is 0
    k_less = float(np.nextafter(np.float32(1.0), np.float32(0)))
    assert oracle.heuristic(L, hits, inst, mode=1, count_cols=(0, -1), theta_imbal=99, k=k_less)[0] == 0


def test_alg1_counts_and_spread_are_fp64():
    # c_i = 2^24 + {1, 0, 3, 2}: distinct in fp64 (fp32 would round 2^24 + 1 to
    # 2^24 and 2^24 + 3 to 2^24 + 4).  No prefix match anywhere, so the order is
    # fewest requests first: instance 1.  The spread c_max - c_min is 3.
    L = np.array([64, 64], np.int64)
    hits = np.zeros((2, 4), np.int32)
    inst = np.array([[2**24, 1], [2**24, 0], [2**24, 3], [2**24, 2]], np.float32)
    assert oracle.heuristic(L, hits, inst, mode=1, count_cols=(0, 1), theta_imbal=99, k=9.0).tolist() == [1, 1]
    assert oracle.heuristic(L, hits, inst, mode=1, count_cols=(0, 1), theta_imbal=2.5, k=-9.0).tolist() == [1, 1]
    # 3 > 3.5 is false: balanced; with k = -9 no instance is eligible -> least loaded (1)
    assert oracle.heuristic(L, hits, inst, mode=1, count_cols=(0, 1), theta_imbal=3.5, k=-9.0).tolist() == [1, 1]
    # balanced, k = 0: eligible below the mean 2^24 + 1.5, i.e. instances 0 and 1
    hits[0] = [1, 0, 0, 0]                            # request 0 prefers instance 0 by prefix match
    assert oracle.heuristic(L, hits, inst, mode=1, count_cols=(0, 1), theta_imbal=3.5, k=0.0).tolist() == [0, 1]


def test_alg1_order_prefers_match_then_fewer_requests_then_index():
    L = np.array([160, 160], np.int64)
    hits = np.array([[2, 5, 5, 5], [0, 0, 0, 0]], np.int32)
    inst = np.array([[0, 0], [4, 0], [2, 0], [2, 0]], np.float32)
    got = oracle.heuristic(L, hits, inst, mode=1, count_cols=(0, -1), theta_imbal=99, k=9.0)
    assert got.tolist() == [2, 0]


def test_alg2_threshold_is_strict():
    L = np.array([32, 32], np.int64)
    hits = np.array([[0, 1, 1], [0, 0, 0]], np.int32)   # best match 0.5 on instance 1 (ties -> 1)
    inst = np.array([[3, 0], [7, 0], [2, 0]], np.float32)
    assert oracle.heuristic(L, hits, inst, mode=2, count_cols=(0, -1), tau=0.49).tolist() == [1, 2]
    assert oracle.heuristic(L, hits, inst, mode=2, count_cols=(0, -1), tau=0.5).tolist() == [2, 2]


def test_single_instance_and_empty_prompts():
    L = np.array([0, 5, 100], np.int64)
    hits = np.zeros((3, 1), np.int32)
    inst = np.array([[4, 4]], np.float32)
    for mode in (1, 2):
        assert (oracle.heuristic(L, hits, inst, mode=mode) == 0).all()
    L, hits, inst = _setting(9, R=5, N=6)
    L[:] = 0
    hits[:] = 0
    c = inst[:, 0] + inst[:, 1]
    got = oracle.heuristic(L, hits, inst, mode=1, theta_imbal=1e9, k=5.0)
    assert (got == int(np.argmin(c))).all()          # equal matches: fewest requests
