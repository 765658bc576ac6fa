"""The exact three-way bf16 split that the tensor-core projection of the ridge solve feeds to the
tensor cores (no GPU needed): for an fp32 value x, hi = bf16(x), mid = bf16(x - hi) and
lo = bf16(x - hi - mid) (each rounding to nearest even, each subtraction in fp32) satisfy
hi + mid + lo = x exactly, so every bf16 x bf16 part product is exact in fp32 and the nine part
products of a tile entry and an adapter entry sum to the fp32 product up to the fp32 additions.
"""

import numpy as np
import torch


def _bf16(x32):
    return torch.from_numpy(x32).to(torch.bfloat16).to(torch.float32).numpy()


def _split(x32):
    hi = _bf16(x32)
    r1 = (x32 - hi).astype(np.float32)
    mid = _bf16(r1)
    r2 = (r1 - mid).astype(np.float32)
    lo = _bf16(r2)
    return hi, mid, lo, r1, r2


def _values(seed=0, n=200000):
    rng = np.random.default_rng(seed)
    mant = rng.uniform(1.0, 2.0, n)
    expo = rng.integers(-100, 100, n)
    sign = rng.choice([-1.0, 1.0], n)
    x = (sign * mant * np.exp2(expo)).astype(np.float32)
    # every fp32 significand pattern near 1, ties of the bf16 rounding, and powers of two
    edge = np.concatenate([
        (1.0 + np.arange(0, 1 << 16) * 2.0 ** -23).astype(np.float32),
        np.float32(1.0) + np.float32(2.0 ** -8) * np.arange(-8, 9, dtype=np.float32),
        np.exp2(np.arange(-60, 60)).astype(np.float32),
        np.array([0.0, -0.0, 3.0, -7.5, 1.0 / 3.0], dtype=np.float32),
    ])
    return np.concatenate([x, edge]).astype(np.float32)


def test_three_parts_sum_to_x_exactly():
    x = _values()
    hi, mid, lo, r1, r2 = _split(x)
    # the two fp32 subtractions are exact (each operand within a factor of two of the other)
    assert np.array_equal(r1.astype(np.float64), x.astype(np.float64) - hi.astype(np.float64))
    assert np.array_equal(r2.astype(np.float64), r1.astype(np.float64) - mid.astype(np.float64))
    # the last remainder is already a bf16 value, so the three parts add up to x with no error
    assert np.array_equal(lo, r2)
    total = hi.astype(np.float64) + mid.astype(np.float64) + lo.astype(np.float64)
    assert np.array_equal(total, x.astype(np.float64))


def test_part_products_are_exact_in_fp32():
    x = _values(1, 20000)
    y = _values(2, 20000)[: x.size]
    px = _split(x)[:3]
    py = _split(y)[:3]
    for a in px:
        for b in py:
            prod64 = a.astype(np.float64) * b.astype(np.float64)
            with np.errstate(over="ignore", under="ignore"):  # out-of-range products are skipped
                prod32 = (a * b).astype(np.float32)  # 8-bit by 8-bit significands: at most 16 bits
            # products in fp32's normal range (the test values span 2^-100 .. 2^100)
            finite = (np.abs(prod64) > 2.0 ** -126) & (np.abs(prod64) < 2.0 ** 127)
            assert np.array_equal(prod32[finite].astype(np.float64), prod64[finite])
