"""The pipelined scorer adds each fp32 bias inside the tensor-core product as
three bf16 terms hi = bf16(b), mid = bf16(b - hi), lo = bf16(b - hi - mid)
(both differences formed in fp32).  Their sum is b exactly, which this checks
in fp64 over fp32 values of every magnitude the biases can take, both signs,
and the values next to powers of two and to bf16 rounding ties.  No GPU."""
import numpy as np
import torch


def split(b32: torch.Tensor):
    hi = b32.to(torch.bfloat16).to(torch.float32)
    r1 = b32 - hi
    mid = r1.to(torch.bfloat16).to(torch.float32)
    lo = (r1 - mid).to(torch.bfloat16).to(torch.float32)
    return hi, mid, lo


def test_three_terms_sum_to_the_bias_exactly():
    rng = np.random.default_rng(7)
    exps = rng.integers(-100, 100, size=200000)
    mant = rng.integers(0, 1 << 23, size=200000)
    sign = rng.integers(0, 2, size=200000)
    bits = (sign.astype(np.uint32) << 31) | ((exps + 127).astype(np.uint32) << 23) | mant.astype(np.uint32)
    vals = bits.view(np.float32)
    # values at and next to powers of two and to bf16 rounding ties
    edge = []
    for e in range(-60, 61, 3):
        p = np.float32(2.0) ** e
        edge += [p, np.nextafter(p, np.float32(0)), np.nextafter(p, np.float32(np.inf)),
                 p * np.float32(1 + 2 ** -8), p * np.float32(1 + 2 ** -8 + 2 ** -23)]
    vals = np.concatenate([vals, np.array(edge, dtype=np.float32), -np.array(edge, dtype=np.float32),
                           np.array([0.0, -0.0], dtype=np.float32)])
    b = torch.from_numpy(vals)
    hi, mid, lo = split(b)
    total = hi.double() + mid.double() + lo.double()
    assert torch.equal(total, b.double())
    # and the sum of the three terms formed in fp32 is b as well
    assert torch.equal((hi + mid) + lo, b)
