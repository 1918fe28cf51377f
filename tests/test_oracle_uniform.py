"""Pins of the oracle's uniform asymmetric RTN quantizer (paper Section 2.2, Section 3.2).

None of these re-type the quantizer's formula: they check properties that the
definition fixes (nearest grid point with the stated tie rule, exact round trip
of grid-aligned groups, the zero-scale special case, power-of-two equivariance,
the error bound).
"""
import numpy as np
import pytest

import oracle

F16 = np.float16


def _all_finite_fp16():
    v = np.arange(1 << 16, dtype=np.uint16).view(F16)
    return v[np.isfinite(v)]


def _check_nearest(w, q, s, z, qmax):
    """Every code is the nearest grid point (q - z) * s; ties go to an even offset q - z.

    float64 evaluation is exact here: fp16 values and j * s (j <= 15) are multiples
    of 2^-24 below 2^17, so their differences need < 42 significant bits.
    """
    w = w.astype(np.float64)
    s = s.astype(np.float64)[..., None]
    z = z.astype(np.float64)[..., None]
    j = np.arange(qmax + 1, dtype=np.float64)
    d = np.abs(w[..., None] - (j - z[..., None]) * s[..., None])
    dmin = d.min(axis=-1, keepdims=True)
    at_min = d == dmin
    chosen = np.take_along_axis(d, q.astype(np.int64)[..., None], axis=-1)[..., 0]
    assert np.all(chosen == dmin[..., 0]), "a code is not the nearest grid point"
    tie = at_min.sum(axis=-1) > 1
    if tie.any():
        off = q.astype(np.int64) - z.astype(np.int64)
        assert np.all(off[tie] % 2 == 0), "a tie did not go to the even offset"


@pytest.mark.parametrize("bits", [3, 4])
def test_rtn_exhaustive_all_fp16(bits):
    """Every finite fp16 value against the widest grid: group [-65504, 65504, w...]."""
    qmax = (1 << bits) - 1
    vals = _all_finite_fp16()
    g = 64
    per = g - 2
    pad = (-len(vals)) % per
    body = np.concatenate([vals, np.zeros(pad, dtype=F16)]).reshape(-1, per)
    ends = np.tile(np.array([-65504, 65504], dtype=F16), (body.shape[0], 1))
    W = np.concatenate([ends, body], axis=1)
    q, s, z = oracle.quantize_uniform(W, bits, g)
    assert q.max() <= qmax and z.max() <= qmax
    _check_nearest(W.reshape(-1, 1, g)[:, 0], q, s[:, 0], z[:, 0], qmax)


@pytest.mark.parametrize("bits", [3, 4])
@pytest.mark.parametrize("lo,hi", [(-0.109375, 0.125), (-3.0, 0.5), (0.0, 0.0078125),
                                   (-1e-3, 2e-3), (-700.0, 5.0)])
def test_rtn_exhaustive_in_range(bits, lo, hi):
    """All fp16 values inside [lo, hi] against the grid the group [lo, hi, w...] selects."""
    qmax = (1 << bits) - 1
    vals = _all_finite_fp16()
    lo16, hi16 = F16(lo), F16(hi)
    vals = vals[(vals >= lo16) & (vals <= hi16)]
    g = 32
    per = g - 2
    pad = (-len(vals)) % per
    body = np.concatenate([vals, np.full(pad, lo16, dtype=F16)]).reshape(-1, per)
    ends = np.tile(np.array([lo16, hi16], dtype=F16), (body.shape[0], 1))
    W = np.concatenate([ends, body], axis=1)
    q, s, z = oracle.quantize_uniform(W, bits, g)
    # every group has the same range, hence the same scale and zero-point
    assert np.all(s == s[0, 0]) and np.all(z == z[0, 0])
    _check_nearest(W, q, s[:, 0], z[:, 0], qmax)


@pytest.mark.parametrize("g", [2, 3, 5, 8])
@pytest.mark.parametrize("bits", [3, 4])
def test_tiny_groups_bruteforce(bits, g):
    """Tiny random groups: codes are nearest grid points; range and error bound hold."""
    qmax = (1 << bits) - 1
    r = np.random.default_rng(1234 + g)
    W = (r.standard_normal((4000, g)) * r.choice([1e-3, 0.05, 3.0], size=(4000, 1))).astype(F16)
    W[:500] = np.abs(W[:500])  # all-positive groups
    W[500:1000] = -np.abs(W[500:1000])  # all-negative groups
    q, s, z = oracle.quantize_uniform(W, bits, g)
    assert q.max() <= qmax and z.max() <= qmax
    _check_nearest(W, q, s[:, 0], z[:, 0], qmax)
    wh = oracle.dequant_uniform(q, s, z, g).astype(np.float64)
    s64 = s.astype(np.float64)
    # the grid spans [lo, hi] up to one step (z and s are rounded), so the
    # reconstruction error is at most one step plus fp16 rounding of w_hat
    err = np.abs(wh - W.astype(np.float64))
    bound = s64 * (1 + 2.0 ** -6) + np.abs(wh) * 2.0 ** -11 + 2.0 ** -24
    assert np.all(err <= bound)
    # groups whose extremes are +-same magnitude have an interior error of at most s/2
    inner = (W.astype(np.float64) > -(z.astype(np.float64)) * s64) & \
            (W.astype(np.float64) < (qmax - z.astype(np.float64)) * s64)
    assert np.all(err[inner] <= 0.5 * s64.repeat(g, 1)[inner] * (1 + 2.0 ** -10)
                  + np.abs(wh[inner]) * 2.0 ** -11 + 2.0 ** -24)


@pytest.mark.parametrize("bits,g", [(4, 64), (4, 128), (3, 64), (3, 128), (4, 32)])
def test_grid_aligned_round_trip(bits, g):
    """Groups that lie exactly on a grid containing codes 0 and 2^b - 1 round-trip bit-exactly."""
    qmax = (1 << bits) - 1
    r = np.random.default_rng(7 * bits + g)
    rows = []
    truth = []
    for _ in range(200):
        s0 = float(r.integers(1, 16)) * 2.0 ** int(r.integers(-14, 4))  # <= 4 significant bits
        z0 = int(r.integers(0, qmax + 1))
        codes = r.integers(0, qmax + 1, size=g)
        codes[r.integers(0, g)] = 0
        codes[(r.integers(1, g) + 0) % g] = qmax
        codes[0], codes[1] = 0, qmax
        r.shuffle(codes)
        w = (codes - z0) * s0  # exact in fp16: <= 9 significant bits, in range
        rows.append(w)
        truth.append((codes, s0, z0))
    W = np.array(rows, dtype=np.float64).astype(F16)
    assert np.array_equal(W.astype(np.float64), np.array(rows))
    q, s, z = oracle.quantize_uniform(W, bits, g)
    for i, (codes, s0, z0) in enumerate(truth):
        assert float(s[i, 0]) == s0
        assert int(z[i, 0]) == z0
        assert np.array_equal(q[i], codes)
    assert np.array_equal(oracle.dequant_uniform(q, s, z, g), W)


def test_zero_scale_special_case():
    """An all-zero group, and one whose range rounds to a zero fp16 scale, code to 0."""
    tiny = F16(2.0 ** -24)  # smallest subnormal: (hi - lo) / 15 rounds to fp16 zero
    W = np.zeros((3, 64), dtype=F16)
    W[1, 5] = tiny
    W[2, :] = -tiny
    q, s, z = oracle.quantize_uniform(W, 4, 64)
    assert np.all(s == 0) and np.all(z == 0) and np.all(q == 0)
    assert np.all(oracle.dequant_uniform(q, s, z, 64) == 0)


@pytest.mark.parametrize("bits", [3, 4])
def test_power_of_two_equivariance(bits):
    """Scaling a group by 2^e scales the fp16 scale by 2^e and leaves codes and zeros alone."""
    W = np.random.default_rng(5).standard_normal((64, 128)).astype(F16)
    q, s, z = oracle.quantize_uniform(W, bits, 64)
    for e in (-3, 4):
        q2, s2, z2 = oracle.quantize_uniform((W.astype(np.float64) * 2.0 ** e).astype(F16), bits, 64)
        assert np.array_equal(q, q2) and np.array_equal(z, z2)
        assert np.array_equal(s.astype(np.float64) * 2.0 ** e, s2.astype(np.float64))


def test_rejects_nonfinite_and_bad_groups():
    W = np.zeros((2, 64), dtype=F16)
    W[1, 3] = np.inf
    with pytest.raises(ValueError):
        oracle.quantize_uniform(W, 4, 64)
    with pytest.raises(ValueError):
        oracle.quantize_uniform(np.zeros((2, 64), dtype=F16), 4, 48)


def _nearest_fp16_exact(v):
    """Nearest fp16 to the exact rational ``v`` (ties to even), by exhaustive search."""
    from fractions import Fraction

    allv = _all_finite_fp16()
    allv = np.unique(allv.astype(np.float64))
    i = np.searchsorted(allv, float(v))
    best = None
    for c in allv[max(i - 2, 0):i + 2]:
        d = abs(Fraction(float(c)) - v)
        m = int(np.float64(c).astype(F16).view(np.uint16)) & 1
        key = (d, m)
        if best is None or key < best[0]:
            best = (key, c)
    return best[1]


@pytest.mark.parametrize("bits", [3, 4])
def test_dequant_is_one_rounding_of_exact_product(bits):
    """w_hat is the fp16 nearest to the exact (q - z) * s, for full-precision scales."""
    from fractions import Fraction

    qmax = (1 << bits) - 1
    r = np.random.default_rng(77)
    s = (r.uniform(0.5, 1.0, size=(40, 1)) * 2.0 ** r.integers(-20, 6, size=(40, 1))).astype(F16)
    s[0, 0] = F16(0.0999755859375)  # 11 significant bits
    z = r.integers(0, qmax + 1, size=(40, 1)).astype(np.uint8)
    q = np.tile(np.arange(qmax + 1, dtype=np.uint8), (40, 4))[:, :4 * (qmax + 1)]
    g = q.shape[1]
    wh = oracle.dequant_uniform(q, s, z, g)
    for i in range(40):
        for j in range(g):
            exact = Fraction(int(q[i, j]) - int(z[i, 0])) * Fraction(float(s[i, 0]))
            assert float(wh[i, j]) == float(_nearest_fp16_exact(exact))
