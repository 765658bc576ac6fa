"""The two-part fp16 split that the tensor-core projection of the ridge solve feeds to the tensor
cores (no GPU needed).  A 32-channel slice of a row (or of a column of A) is scaled by 2^e, e
chosen so that its largest magnitude m lies in [2^14, 2^15); then y = 2^e x is carried as
hi = fp16(y) and lo = fp16(y - hi), both rounded to nearest even, with y - hi computed in fp32.
The checks: y - hi is exact in fp32, |y - hi - lo| <= 2^-22 |y| (2^-25 absolute where lo is an
fp16 subnormal), nothing overflows fp16, every part product is exact in fp32, and a projection
evaluated this way slice by slice stays within the error of an fp32 evaluation.
"""

import numpy as np


def _shift(m):
    """e with m 2^e in [2^14, 2^15) (m > 0, finite, fp32-normal)."""
    return 14 - np.floor(np.log2(m)).astype(np.int64)


def _split(y32):
    hi = y32.astype(np.float16)
    r = (y32 - hi.astype(np.float32)).astype(np.float32)
    lo = r.astype(np.float16)
    return hi, lo, r


def _slices(seed=0, n=4096):
    """n slices of 32 values with magnitudes spread over 2^-60 .. 2^60 and within-slice spreads up
    to 2^40 (the small entries land in fp16's subnormal range after scaling)."""
    rng = np.random.default_rng(seed)
    base = np.exp2(rng.uniform(-60, 60, (n, 1)))
    spread = np.exp2(-rng.uniform(0, 40, (n, 32)))
    sign = rng.choice([-1.0, 1.0], (n, 32))
    x = (sign * base * spread * rng.uniform(1, 2, (n, 32))).astype(np.float32)
    x[:8, 5] = 0.0  # zeros inside a slice
    return x


def test_scaled_slice_fits_fp16_and_split_is_within_2_pow_minus_22():
    x = _slices()
    e = _shift(np.abs(x).max(axis=1).astype(np.float64))
    y = (x.astype(np.float64) * np.exp2(e)[:, None]).astype(np.float32)
    # scaling by a power of two is exact, and the largest magnitude lies in [2^14, 2^15)
    assert np.array_equal(y.astype(np.float64), x.astype(np.float64) * np.exp2(e)[:, None])
    ymax = np.abs(y).max(axis=1)
    assert np.all(ymax >= 2.0 ** 14) and np.all(ymax < 2.0 ** 15)
    hi, lo, r = _split(y)
    assert np.all(np.isfinite(hi)) and np.all(np.isfinite(lo))  # |hi| <= 2^15 < 65504
    # the fp32 remainder is exact
    assert np.array_equal(r.astype(np.float64), y.astype(np.float64) - hi.astype(np.float64))
    err = np.abs(y.astype(np.float64) - hi.astype(np.float64) - lo.astype(np.float64))
    bound = np.maximum(2.0 ** -22 * np.abs(y.astype(np.float64)), 2.0 ** -25)
    assert np.all(err <= bound)
    # relative to the slice's largest entry the error is at most 2^-22, whatever the spread
    assert np.all(err <= 2.0 ** -22 * ymax[:, None].astype(np.float64))


def test_part_products_are_exact_in_fp32():
    x = _slices(1, 512)
    a = _slices(2, 512)
    px = _split((x * np.exp2(_shift(np.abs(x).max(1)))[:, None]).astype(np.float32))[:2]
    pa = _split((a * np.exp2(_shift(np.abs(a).max(1)))[:, None]).astype(np.float32))[:2]
    for u in px:
        for v in pa:
            p64 = u.astype(np.float64) * v.astype(np.float64)  # 11-bit by 11-bit significands
            p32 = (u.astype(np.float32) * v.astype(np.float32)).astype(np.float64)
            assert np.array_equal(p32, p64)


def _project(M, A):
    """M A slice by slice (32 channels): rows of M and columns of A scaled and split, the four
    part products summed per slice (exact products, fp64 stands in for the short fp32 sum), the
    scales undone, and the slices added in fp32."""
    out = np.zeros((M.shape[0], A.shape[1]), np.float32)
    for c0 in range(0, M.shape[1], 32):
        T, S = M[:, c0:c0 + 32], A[c0:c0 + 32]
        er = _shift(np.abs(T).max(1))
        ec = _shift(np.abs(S).max(0))
        th, tl, _ = _split((T * np.exp2(er)[:, None]).astype(np.float32))
        ah, al, _ = _split((S * np.exp2(ec)[None, :]).astype(np.float32))
        D = (th.astype(np.float64) + tl) @ (ah.astype(np.float64) + al)
        D = D.astype(np.float32)
        out += (D * np.exp2(-er)[:, None].astype(np.float32)) * np.exp2(-ec)[None, :].astype(np.float32)
    return out


def test_projection_through_the_split_matches_fp64_at_fp32_accuracy():
    rng = np.random.default_rng(3)
    N, d, k = 1024, 640, 8
    X = rng.standard_normal((N, d)) * rng.uniform(0.1, 3.0, d)
    gram = (X.T @ X).astype(np.float32)
    cross = (0.01 * rng.standard_normal((N, d)).T @ X).astype(np.float32)
    A = (rng.standard_normal((d, k)) / np.sqrt(d)).astype(np.float32)
    for M in (gram, cross):
        ref = M.astype(np.float64) @ A.astype(np.float64)
        got = _project(M, A)
        fp32 = (M @ A).astype(np.float64)
        rel = np.linalg.norm(got - ref) / np.linalg.norm(ref)
        rel32 = np.linalg.norm(fp32 - ref) / np.linalg.norm(ref)
        assert rel < 1e-6 and rel < 2.0 * rel32 + 1e-7, (rel, rel32)
