"""Pins of the oracle's non-uniform Lloyd-Max LUT quantizer (paper Section 2.2, Fig. 2a).

Checks: codes in range and nearest to the LUT; groups with <= 2^b distinct values
round-trip; two hand-derived closed forms; the Lloyd fixed-point conditions
against exact rational means; monotone distortion; the exact 1-D k-means optimum
from dynamic programming as a lower bound; agreement with scikit-learn's Lloyd
k-means from the same initial levels; permutation and power-of-two invariance;
single-rounding float64 -> fp16 conversion of the levels.
"""
from fractions import Fraction

import numpy as np
import pytest

import oracle

F16 = np.float16


def _nearest_check(wg, codes, luts):
    w = wg.astype(np.float64)
    L = luts.astype(np.float64)
    d = np.abs(w[:, :, None] - L[:, None, :])
    first_min = np.argmin(d, axis=2)  # lowest index among equal distances
    assert np.array_equal(codes, first_min)


@pytest.mark.parametrize("bits,g", [(3, 128), (3, 64), (4, 128)])
def test_codes_range_sorted_nearest(bits, g):
    W = (np.random.default_rng(3).standard_t(4, size=(16, 4 * g)) * 0.02).astype(F16)
    q, lut = oracle.quantize_lut(W, bits, g)
    assert q.max() < (1 << bits)
    assert lut.shape == (16, 4, 1 << bits)
    assert np.all(np.diff(lut.astype(np.float64), axis=2) >= 0)
    _nearest_check(W.reshape(-1, g), q.reshape(-1, g), lut.reshape(-1, 1 << bits))
    wh = oracle.dequant_lut(q, lut, g)
    assert wh.dtype == F16


def test_few_distinct_values_round_trip():
    r = np.random.default_rng(11)
    rows = []
    for d in (1, 2, 5, 8):
        vals = (r.standard_normal(d) * 0.1).astype(F16)
        rows.append(r.choice(vals, size=128))
    W = np.array(rows, dtype=F16)
    q, lut = oracle.quantize_lut(W, 3, 128)
    assert np.array_equal(oracle.dequant_lut(q, lut, 128), W)
    # padding repeats the largest value
    u = np.unique(W[0])
    assert np.all(lut[0, 0] == u[0])


def test_closed_form_equally_spaced():
    """128 values i * delta, quantile initialisation, hand derivation.

    Initial levels are sorted(w)[8, 24, ..., 120] = 8, 24, ..., 120 (in units of
    delta).  Value 16 lies exactly between 8 and 24 and goes to the lower index,
    likewise 32 between 24 and 40, etc.  So the cells are {0..16}, {17..32}, ...,
    {97..112}, {113..127} with means 8, 24.5, 40.5, ..., 104.5, 120.  With those
    levels the boundaries move to 16.25, 32.5, ..., 112.25: the same cells, a fixed
    point after one update.
    """
    delta = 2.0 ** -10
    W = (np.arange(128) * delta).astype(F16)[None, :]
    q, lut = oracle.quantize_lut(W, 3, 128)
    expect = np.array([8, 24.5, 40.5, 56.5, 72.5, 88.5, 104.5, 120]) * delta
    assert np.array_equal(lut[0, 0].astype(np.float64), expect)
    cells = [range(0, 17)] + [range(16 * j + 1, 16 * j + 17) for j in range(1, 7)] + [range(113, 128)]
    for j, cell in enumerate(cells):
        assert np.all(q[0, list(cell)] == j)


def test_closed_form_separated_clusters():
    """Eight tight, well separated clusters of 16: one level per cluster at its mean."""
    r = np.random.default_rng(5)
    centres = np.array([-3.0, -2.0, -1.0, -0.25, 0.25, 1.0, 2.0, 3.0])
    vals = (centres[:, None] + r.integers(-20, 21, size=(8, 16)) * 2.0 ** -10)
    W16 = vals.astype(F16)
    W = W16.reshape(1, 128)[:, r.permutation(128)]
    q, lut = oracle.quantize_lut(W, 3, 128)
    for j in range(8):
        exact = sum(Fraction(float(v)) for v in W16[j]) / 16
        assert lut[0, 0, j] == F16(float(exact))  # one rounding of the exact mean
        assert float(lut[0, 0, j]) == float(F16(float(exact)))


def _exact_fixed_point(w, levels):
    """Nearest-level cells of ``levels`` and their exact rational means."""
    a = np.argmin(np.abs(w[:, None] - levels[None, :]), axis=1)
    means = {}
    for j in range(len(levels)):
        cell = w[a == j]
        if cell.size:
            means[j] = sum(Fraction(float(v)) for v in cell) / cell.size
    return means


def test_fixed_point_conditions_at_convergence():
    W = (np.random.default_rng(21).standard_t(4, size=(24, 128)) * 0.02).astype(F16)
    c0, trace = oracle.lloyd_max_trace(W, 3, 500)
    final = trace[-1]
    for gi in range(W.shape[0]):
        w = W[gi].astype(np.float64)
        means = _exact_fixed_point(w, final[gi])
        for j, m in means.items():
            # the float64 level is the correctly rounded exact mean of its cell
            assert final[gi, j] == float(m)


def test_distortion_monotone():
    W = (np.random.default_rng(8).standard_t(4, size=(64, 128)) * 0.04).astype(F16)
    W[:, 5] = 0.4  # a large outlier per group
    c0, trace = oracle.lloyd_max_trace(W, 3, 25)
    w = W.astype(np.float64)

    def dist(c):
        return (np.min(np.abs(w[:, :, None] - c[:, None, :]), axis=2) ** 2).sum(axis=1)

    prev = dist(c0)
    for c in trace:
        cur = dist(c)
        assert np.all(cur <= prev * (1 + 1e-12) + 1e-300)
        prev = cur


def _kmeans_1d_optimum(x, L):
    """Exact optimal L-level distortion of sorted samples x by dynamic programming."""
    x = np.sort(x)
    n = len(x)
    p1 = np.concatenate([[0.0], np.cumsum(x)])
    p2 = np.concatenate([[0.0], np.cumsum(x * x)])

    def cost(i, j):  # samples i..j-1
        m = j - i
        s = p1[j] - p1[i]
        return (p2[j] - p2[i]) - s * s / m

    INF = float("inf")
    D = [[INF] * (n + 1) for _ in range(L + 1)]
    D[0][0] = 0.0
    for l in range(1, L + 1):
        for j in range(1, n + 1):
            best = INF
            for i in range(l - 1, j):
                if D[l - 1][i] < INF:
                    best = min(best, D[l - 1][i] + cost(i, j))
            D[l][j] = best
    return min(D[l][n] for l in range(1, L + 1))


@pytest.mark.parametrize("g", [16, 24, 32])
def test_distortion_not_below_dp_optimum(g):
    W = (np.random.default_rng(g).standard_normal((12, g)) * 0.1).astype(F16)
    c0, trace = oracle.lloyd_max_trace(W, 3, 200)
    final = trace[-1] if trace else c0
    for gi in range(W.shape[0]):
        w = W[gi].astype(np.float64)
        if len(np.unique(w)) <= 8:
            continue
        d = (np.min(np.abs(w[:, None] - final[gi][None, :]), axis=1) ** 2).sum()
        opt = _kmeans_1d_optimum(w, 8)
        assert d >= opt * (1 - 1e-9) - 1e-18


def test_matches_sklearn_lloyd():
    sk = pytest.importorskip("sklearn.cluster")
    W = (np.random.default_rng(99).standard_t(4, size=(20, 128)) * 0.02).astype(F16)
    c0, trace = oracle.lloyd_max_trace(W, 3, 300)
    final = trace[-1]
    for gi in range(W.shape[0]):
        w = W[gi].astype(np.float64)[:, None]
        km = sk.KMeans(n_clusters=8, init=c0[gi][:, None], n_init=1, max_iter=300, tol=0.0,
                       algorithm="lloyd").fit(w)
        ours = np.sort(final[gi])
        theirs = np.sort(km.cluster_centers_[:, 0])
        assert np.allclose(ours, theirs, rtol=1e-12, atol=1e-15)


def test_permutation_and_scale_invariance():
    r = np.random.default_rng(4)
    W = (r.standard_t(4, size=(8, 256)) * 0.02).astype(F16)
    q, lut = oracle.quantize_lut(W, 3, 128)
    perm = np.concatenate([r.permutation(128), 128 + r.permutation(128)])
    q2, lut2 = oracle.quantize_lut(W[:, perm], 3, 128)
    assert np.array_equal(lut, lut2) and np.array_equal(q[:, perm], q2)
    q3, lut3 = oracle.quantize_lut((W.astype(np.float64) * 4).astype(F16), 3, 128)
    assert np.array_equal(q, q3)
    assert np.array_equal(lut.astype(np.float64) * 4, lut3.astype(np.float64))


def test_float64_to_fp16_single_rounding():
    """Levels are rounded once from float64: values that a float32 hop would double-round."""
    # 1 + 2^-11 is a tie between fp16 neighbours 1 and 1 + 2^-10; a hair above it
    # must round up, but float32 would first round it onto the tie and then to 1.
    x = np.array([1.0 + 2.0 ** -11 + 2.0 ** -40, 1.0 + 2.0 ** -11 - 2.0 ** -40, 1.0 + 2.0 ** -11])
    exact = []
    for v in x:
        fr = Fraction(v)
        lo = Fraction(1)
        hi = Fraction(1) + Fraction(1, 1024)
        if fr - lo < hi - fr:
            exact.append(1.0)
        elif fr - lo > hi - fr:
            exact.append(float(hi))
        else:
            exact.append(1.0)  # tie to even mantissa
    assert list(x.astype(F16).astype(np.float64)) == exact


def test_lut_levels_rounded_once_to_nearest_fp16():
    """The oracle's LUT rounding step takes float64 levels to the nearest fp16 (exact check).

    The cases sit just off fp16 ties, where a float32 intermediate would round onto
    the tie first and then to the even neighbour.
    """
    from oracle.quant import round_to_fp16

    ties = []
    for base, ulp in ((1.0, 2.0 ** -10), (0.03125, 2.0 ** -15), (-3.0, 2.0 ** -9), (2.0 ** -20, 2.0 ** -24)):
        t = base + ulp / 2
        for eps in (2.0 ** -40, -(2.0 ** -40)):
            ties.append(t + eps * max(abs(base), 2.0 ** -20))
    x = np.array(ties)
    got = round_to_fp16(x).astype(np.float64)
    for v, h in zip(x, got):
        fr = Fraction(float(v))
        cand = np.unique(np.array([np.nextafter(F16(h), F16(-np.inf)), F16(h),
                                   np.nextafter(F16(h), F16(np.inf))]).astype(np.float64))
        dists = [abs(Fraction(float(c)) - fr) for c in cand]
        assert abs(Fraction(float(h)) - fr) == min(dists)
