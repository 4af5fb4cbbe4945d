"""Parity bars for predictions and selections (shared by the GPU tests).

Predictions: |g - o| <= tol * max(|o|, 1e-3 s) (tol 1e-5 for fp32 paths,
2e-2 for bf16 paths).  A row whose value fp32 accumulation cannot pin to that
bar is checked at its rounding radius instead and counted: the oracle's
rounding analysis (oracle.mlp_forward_bounds) gives per row `ebound`, how far
an fp32-accumulating implementation lies from the fp64 value when every bf16
rounding point agrees, and `flip`, the output change if each bf16 rounding
point that lies within accumulation noise of a midpoint went the other way
(summed over those points, each taken alone).  Several such points in one
row interact through the later roundings, so the flip term carries a margin
of one half: allow = max(strict, ebound + 1.5 flip).

Selections: (i) exact on the GPU's own scores; (ii) equal to the oracle's
choice wherever the oracle's top-2 gap exceeds the two rows' allowances;
(iii) elsewhere the GPU's pick lies within those allowances of the oracle's
best.  Every check records its figures (rows, rows held to the strict bar,
worst error over the strict bar) for the run's report.
"""
import json
import os

import numpy as np

import oracle

STATS = []


def _allow(o, tol, ref):
    strict = tol * np.maximum(np.abs(o), 1e-3)
    if ref is None or "ebound" not in ref:
        return strict, strict, np.zeros_like(strict)
    rad = np.asarray(ref["ebound"], np.float64) + 1.5 * np.asarray(ref["flip"], np.float64)
    return np.maximum(strict, rad), strict, rad


def assert_scores_close(g, ref, tol, label=""):
    """ref: the oracle's route dict (scores, ebound, flip) or a plain array."""
    o = np.asarray(ref["scores"] if isinstance(ref, dict) else ref, np.float64)
    g = np.asarray(g, np.float64)
    allow, strict, rad = _allow(o, tol, ref if isinstance(ref, dict) else None)
    err = np.abs(g - o)
    bad = ~(err <= allow)
    held = rad <= strict
    STATS.append({"label": label, "tol": tol, "rows": int(o.size), "rows_strict": int(held.sum()),
                  "rows_over_strict": int((err > strict).sum()),
                  "worst_err_over_strict": float(np.max(err / strict)) if o.size else 0.0,
                  "worst_err_over_strict_held": float(np.max((err / strict)[held])) if held.any() else 0.0,
                  "worst_abs_err": float(err.max()) if o.size else 0.0})
    assert not bad.any(), (f"{label}: {bad.sum()} of {bad.size} predictions off; worst err/allow "
                           f"{np.max(err / allow):.3g}; worst err/strict {np.max(err / strict):.3g}")


def assert_choices(choice, scores_gpu, ref, tol):
    """ref: the oracle's route dict (scores, ebound, flip) or a plain array."""
    oracle_scores = np.asarray(ref["scores"] if isinstance(ref, dict) else ref, np.float32)
    # (i) the selector is exact on the GPU's own scores
    c_own, _ = oracle.argmin(scores_gpu)
    assert np.array_equal(choice, c_own)
    # (ii) equal to the oracle's choice wherever the oracle's top-2 gap is clear
    c_or, b_or = oracle.argmin(oracle_scores)
    o64 = oracle_scores.astype(np.float64)
    allow, _, _ = _allow(o64, tol, ref if isinstance(ref, dict) else None)
    rows = np.arange(len(choice))
    if o64.shape[1] > 1:
        order = np.argsort(o64, axis=1, kind="stable")
        second = order[:, 1]
        gap = o64[rows, second] - o64[rows, c_or]
        margin = allow[rows, c_or] + allow[rows, second]
    else:
        gap, margin = np.full(len(choice), np.inf), np.zeros(len(choice))
    clear = gap > margin
    assert np.array_equal(choice[clear], c_or[clear])
    # (iii) near ties: the GPU's pick is within the allowances of the oracle's best
    near = ~clear
    if near.any():
        picked = o64[rows, choice][near]
        assert np.all(picked - o64[rows, c_or][near] <= allow[rows, choice][near] + allow[rows, c_or][near])
    return clear.mean()


def write_stats(path):
    with open(path, "w") as f:
        for s in STATS:
            f.write(json.dumps(s) + "\n")
