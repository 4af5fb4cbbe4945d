"""Vectorised restatement of the oracle's training step (or_train_step in
lodestar_oracle.c) for runs of many steps -- test infrastructure, like the
rest of this package.

The arithmetic is the same reading, step for step (Sec. 4.3.2 online learning;
loss and optimiser are this project's readings): z-scored rows (fp32), the
forward pass with bf16 operands and fp32 layer outputs, MSE on TTFT, backprop
with bf16 operands of every product, fp32 gradients, Adam (beta1 0.9, beta2
0.999, eps 1e-8, bias corrections 1 - beta^t in fp64) on fp32 master values.
Each dot product is an fp64 matrix product (numpy) instead of a scalar loop,
so sums run in another order: results agree with or_train_step to fp64
rounding before each fp32 / bf16 rounding point (tests/test_oracle_pins.py).
"""
from __future__ import annotations

import numpy as np


def f32(a):
    """fp64 array of the fp32 values nearest to a."""
    return np.asarray(a, np.float64).astype(np.float32).astype(np.float64)


def bf16(a):
    """fp64 array of the bf16 values of a's fp32 values (round to nearest even)."""
    f = np.ascontiguousarray(np.asarray(a, np.float64).astype(np.float32))
    u = f.view(np.uint32)
    nan = ((u & np.uint32(0x7F800000)) == np.uint32(0x7F800000)) & ((u & np.uint32(0x007FFFFF)) != 0)
    r = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) & np.uint32(0xFFFF0000)
    r = np.where(nan, (u | np.uint32(0x00400000)) & np.uint32(0xFFFF0000), r).astype(np.uint32)
    return r.view(np.float32).astype(np.float64)


def zscore(x, mean, std):
    """(x - mean) / std in fp32, a std below 1e-12 taken as 1."""
    x = np.asarray(x, np.float32)
    s = np.where(np.asarray(std, np.float32) < np.float32(1e-12), np.float32(1), np.asarray(std, np.float32))
    return ((x - np.asarray(mean, np.float32)) / s).astype(np.float32)


class NpTrainer:
    """bf16-operand Adam training of the predictor (fp32 master values)."""

    def __init__(self, widths, params):
        self.w = [int(v) for v in widths]
        p = np.asarray(params, np.float64)
        self.W, self.b, off = [], [], 0
        for l in range(len(self.w) - 1):
            fi, fo = self.w[l], self.w[l + 1]
            self.W.append(p[off:off + fo * fi].reshape(fo, fi).copy())
            off += fo * fi
            self.b.append(p[off:off + fo].copy())
            off += fo
        self.mW = [np.zeros_like(a) for a in self.W]
        self.vW = [np.zeros_like(a) for a in self.W]
        self.mb = [np.zeros_like(a) for a in self.b]
        self.vb = [np.zeros_like(a) for a in self.b]
        self.t = 0

    @property
    def params(self):
        return np.concatenate([np.concatenate([W.ravel(), b]) for W, b in zip(self.W, self.b)])

    def forward(self, x):
        """x: z-scored fp32 rows -> (activations a_0.. (bf16), pre-activations z_1.. (fp32))."""
        acts, zs = [bf16(x)], []
        n = len(self.W)
        for l in range(n):
            z = f32(acts[-1] @ bf16(self.W[l]).T + f32(self.b[l]))
            zs.append(z)
            if l + 1 < n:
                acts.append(bf16(np.maximum(z, 0.0)))
        return acts, zs

    def step(self, ring_x, ring_y, idx, mean, std, lr):
        """One Adam step on rows idx; returns the minibatch loss before the update."""
        self.t += 1
        idx = np.asarray(idx)
        x = zscore(np.asarray(ring_x)[idx], mean, std)
        y = np.asarray(ring_y, np.float32)[idx].astype(np.float64)
        acts, zs = self.forward(x)
        B = len(idx)
        e = zs[-1][:, 0] - y
        loss = float(np.mean(e * e))
        dz = f32(2.0 * e / B)[:, None]
        gW, gb = [None] * len(self.W), [None] * len(self.W)
        for l in range(len(self.W) - 1, -1, -1):
            gb[l] = f32(dz.sum(axis=0))
            gW[l] = f32(bf16(dz).T @ acts[l])
            if l > 0:
                s = bf16(dz) @ bf16(self.W[l])
                dz = np.where(zs[l - 1] > 0.0, f32(s), 0.0)
        bc1, bc2 = 1.0 - 0.9 ** self.t, 1.0 - 0.999 ** self.t
        for P, G, M, V in ((self.W, gW, self.mW, self.vW), (self.b, gb, self.mb, self.vb)):
            for l in range(len(P)):
                M[l] = f32(0.9 * M[l] + 0.1 * G[l])
                V[l] = f32(0.999 * V[l] + 0.001 * G[l] * G[l])
                P[l] = f32(P[l] - lr * (M[l] / bc1) / (np.sqrt(V[l] / bc2) + 1e-8))
        return loss
