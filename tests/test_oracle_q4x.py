"""Pins of the Q4X oracle (Section 3.2, Fig. 3a/3b; Table 2 "Q4X W4A8G64, 4.28 BPW").

Each test checks the oracle against something other than itself: brute force,
closed forms, fixed-point conditions of the two learning steps, an exact 1-D
optimum, and a hand-written byte image.
"""
import os

import numpy as np
import pytest

import oracle
from oracle import q4x
import synth

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _w(n, k, seed, outliers=0.001):
    return synth.student_t_weights(n, k, 0.02, seed=seed, stream=64, outlier_frac=outliers).astype(np.float16)


def test_scale_is_group_absmax_and_dead_groups_decode_to_zero():
    W = _w(8, 256, 1)
    W[3, 64:128] = 0
    W[5, :64] = -0.0
    r = q4x.quantize_q4x(W)
    Wf = W.astype(np.float64).reshape(8, 4, 64)
    assert np.array_equal(r["scales"].astype(np.float64), np.abs(Wf).max(axis=2))
    assert r["books"][3, 1] == 0 and r["books"][5, 0] == 0
    assert not r["codes"][3, 64:128].any() and not r["codes"][5, :64].any()
    Wh = q4x.dequant_q4x(r["codes"], r["scales"], r["books"], r["codebooks"])
    assert not Wh[3, 64:128].astype(np.float64).any()


def test_normalised_values_reach_plus_minus_one_exactly():
    W = _w(4, 128, 2)
    s16, U, live = q4x.q4x_normalize(W)
    assert live.all()
    assert np.array_equal(np.abs(U).max(axis=2), np.full((4, 2), 1 << 20))
    # rint of the correctly rounded quotient, recomputed one element at a time
    for (r, gi, i) in [(0, 0, 5), (1, 1, 63), (3, 0, 17)]:
        want = round(float(W[r, 64 * gi + i]) / float(s16[r, gi]) * (1 << 20))
        assert U[r, gi, i] == want or abs(U[r, gi, i] - want) == 1 and \
            abs(float(W[r, 64 * gi + i]) / float(s16[r, gi]) * (1 << 20) % 1 - 0.5) < 1e-9


def test_histogram_bins_closed_form():
    U = np.array([[-(1 << 20), -(1 << 20) + 65535, -(1 << 20) + 65536, 0, (1 << 20) - 1, 1 << 20] + [0] * 58])
    H = q4x.q4x_histograms(U)
    assert H.shape == (1, 32) and H.sum() == 64
    assert H[0, 0] == 2 and H[0, 1] == 1 and H[0, 16] == 59 and H[0, 31] == 2


def test_codes_are_the_nearest_dequantized_value():
    """Brute force over the 16 candidates of every weight (ties to the lowest)."""
    W = _w(6, 192, 3)
    r = q4x.quantize_q4x(W)
    cb, s, books = r["codebooks"], r["scales"], r["books"]
    for row in range(6):
        for gi in range(3):
            cand = [float(np.float16(np.float32(s[row, gi]) * np.float32(cb[books[row, gi], j]))) for j in range(16)]
            for i in range(64):
                w = float(W[row, 64 * gi + i])
                d = [abs(w - c) for c in cand]
                assert r["codes"][row, 64 * gi + i] == d.index(min(d))


def test_dequant_is_one_rounding_of_the_exact_product():
    W = _w(5, 320, 4)
    r = q4x.quantize_q4x(W)
    Wh = q4x.dequant_q4x(r["codes"], r["scales"], r["books"], r["codebooks"])
    for row, col in [(0, 0), (2, 100), (4, 319), (3, 64)]:
        gi = col // 64
        prod = float(r["scales"][row, gi]) * float(r["codebooks"][r["books"][row, gi], r["codes"][row, col]])
        assert Wh[row, col] == np.float16(prod)  # the float64 product is exact
    assert np.all(np.abs(Wh.astype(np.float64)) <= np.repeat(r["scales"].astype(np.float64), 64, axis=1))


def test_groups_with_sixteen_levels_round_trip_exactly():
    """Every group = 2^e * (j / 8), j in -8..7 (16 values, -1 included): one
    book holds exactly these levels and every weight decodes to itself."""
    rng = np.random.default_rng(5)
    n, G = 16, 8
    W = np.empty((n, 64 * G), dtype=np.float16)
    for r in range(n):
        for gi in range(G):
            vals = np.concatenate([np.arange(-8, 8), rng.integers(-8, 8, 48)]) / 8.0
            rng.shuffle(vals)
            W[r, 64 * gi:64 * gi + 64] = (vals * 2.0 ** -int(rng.integers(3, 9))).astype(np.float16)
    r = q4x.quantize_q4x(W)
    Wh = q4x.dequant_q4x(r["codes"], r["scales"], r["books"], r["codebooks"])
    assert np.array_equal(Wh.view(np.uint16), W.view(np.uint16))


def test_kmeans_separates_two_group_shapes():
    """Half the groups spread evenly over [-1, 1], half piled near 0 with one
    +-1 outlier: no learned histogram takes members of both kinds."""
    rng = np.random.default_rng(6)
    n, G = 32, 8
    W = np.empty((n, 64 * G), dtype=np.float16)
    wide = np.zeros((n, G), dtype=bool)
    for r in range(n):
        for gi in range(G):
            if (r + gi) % 2:
                v = rng.uniform(-1, 1, 64)
                v[0] = 1.0
                wide[r, gi] = True
            else:
                v = rng.normal(0, 0.05, 64)
                v[0] = -1.0
            W[r, 64 * gi:64 * gi + 64] = (0.03 * v).astype(np.float16)
    r = q4x.quantize_q4x(W, iters=100)
    for b in range(4):
        m = r["books"] == b
        assert not (wide[m].any() and (~wide[m]).any()), b


def _assignment_is_stable(H, a):
    C = np.stack([H[a == j].mean(axis=0) if (a == j).any() else np.full(H.shape[1], np.inf) for j in range(4)])
    D = ((H[:, None, :].astype(np.float64) - C[None, :, :]) ** 2).sum(axis=2)
    return np.all(D[np.arange(len(a)), a] <= D.min(axis=1) + 1e-9)


def test_kmeans_reaches_a_fixed_point():
    W = _w(64, 512, 7)
    _, U, live = q4x.q4x_normalize(W)
    Ul = U[live]
    H = q4x.q4x_histograms(Ul)
    a, C = q4x.q4x_kmeans(H, (Ul * Ul).sum(axis=1), iters=500)
    assert _assignment_is_stable(H, a)
    for j in range(4):
        if (a == j).any():
            assert np.allclose(C[j], H[a == j].mean(axis=0), rtol=0, atol=1e-12)


def _lloyd_mse(V, levels):
    V = V.astype(np.float64)
    return (np.min(np.abs(V[:, None] - levels[None, :]), axis=1) ** 2).mean()


def test_lloyd16_fixed_point_and_monotone_distortion():
    rng = np.random.default_rng(8)
    V = np.rint(rng.standard_t(4, 5000) / 12 * (1 << 20)).astype(np.int64).clip(-(1 << 20), 1 << 20)
    trace = []
    lv = q4x.q4x_lloyd16(V, 500, trace)
    mses = [_lloyd_mse(V, t) for t in trace]
    assert all(b <= a + 1e-6 for a, b in zip(mses, mses[1:]))
    cell = np.argmin(np.abs(V[:, None].astype(np.float64) - lv[None, :]), axis=1)
    for j in range(16):
        if (cell == j).any():
            assert abs(lv[j] - V[cell == j].mean()) < 1e-6


def _kmeans_1d_optimum(x, k):
    """Exact 1-D k-means (squared error) by dynamic programming over the sorted values."""
    x = np.sort(x.astype(np.float64))
    n = x.size
    ps, ps2 = np.concatenate([[0], np.cumsum(x)]), np.concatenate([[0], np.cumsum(x * x)])

    def cost(i, j):  # points i..j-1 in one cell
        s, s2, m = ps[j] - ps[i], ps2[j] - ps2[i], j - i
        return s2 - s * s / m
    best = np.full((k + 1, n + 1), np.inf)
    best[0, 0] = 0
    for c in range(1, k + 1):
        for j in range(c, n + 1):
            best[c, j] = min(best[c - 1, i] + cost(i, j) for i in range(c - 1, j))
    return best[k, n] / n


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_lloyd16_never_beats_the_exact_optimum(seed):
    rng = np.random.default_rng(seed)
    V = rng.integers(-(1 << 20), 1 << 20, 40)
    lv = q4x.q4x_lloyd16(V, 200)
    opt = _kmeans_1d_optimum(V, 16)
    assert opt > 0 and _lloyd_mse(V, lv) >= opt * (1 - 1e-9)


def test_book_index_packing_byte_image_and_round_trip():
    books = np.array([[0, 1, 2, 3, 3, 2, 1]], dtype=np.uint8)
    # group j in bits 2(j % 4) of byte j / 4: 0 | 1<<2 | 2<<4 | 3<<6 = 0xE4; 3 | 2<<2 | 1<<4 = 0x1B
    assert list(q4x.pack_books(books)[0]) == [0xE4, 0x1B]
    rng = np.random.default_rng(9)
    b = rng.integers(0, 4, (5, 13)).astype(np.uint8)
    assert np.array_equal(q4x.unpack_books(q4x.pack_books(b), 13), b)


def test_sizes_give_the_papers_bits_per_weight():
    with open(os.path.join(GOLD, "paper_bpw.txt")) as f:
        row = next(l.split() for l in f if l.startswith("Q4X"))
    n, k = 4096, 4096
    sz = q4x.q4x_sizes(n, k)
    per_group = 8 * (sz["codes"] + sz["scales"] + sz["books"]) / (n * k)
    assert round(per_group, 2) == float(row[4])  # 4 + (16 + 2) / 64 = 4.28
    assert sz["codebooks"] == 2 * 4 * 16


def test_codebooks_are_ascending():
    r = q4x.quantize_q4x(_w(32, 512, 10))
    cb = r["codebooks"].astype(np.float64)
    assert np.all(np.diff(cb, axis=1) >= 0)


def test_dead_groups_take_no_part_in_learning():
    """Appending all-zero rows changes no codebook and no live group's codes."""
    W = _w(24, 256, 11)
    Wd = np.concatenate([W, np.zeros((8, 256), dtype=np.float16)])
    a, b = q4x.quantize_q4x(W), q4x.quantize_q4x(Wd)
    assert np.array_equal(a["codebooks"].view(np.uint16), b["codebooks"].view(np.uint16))
    assert np.array_equal(a["codes"], b["codes"][:24]) and np.array_equal(a["books"], b["books"][:24])


def test_code_packing_byte_image():
    """Codes 0..7 of k = 0..7: code j sits in nibble j/2 + 4 (j % 2), so the
    little-endian word is 0x75316420."""
    codes = np.arange(8, dtype=np.uint8)[None, :]
    assert list(q4x.pack_codes4(codes)[0]) == [0x20, 0x64, 0x31, 0x75]


def test_code_packing_matches_the_4bit_format_and_round_trips():
    rng = np.random.default_rng(12)
    c = rng.integers(0, 16, (7, 256)).astype(np.uint8)
    assert np.array_equal(q4x.pack_codes4(c), oracle.pack_codes(c, 4))
    c = rng.integers(0, 16, (5, 320)).astype(np.uint8)  # k = 5 groups: not a multiple of 128
    assert np.array_equal(q4x.unpack_codes4(q4x.pack_codes4(c), 320), c)


def test_gemv_against_exact_rational_arithmetic():
    from fractions import Fraction

    r = q4x.quantize_q4x(_w(3, 128, 13))
    x = synth.activations(2, 128, seed=13, stream=13)
    y = q4x.gemv_q4x(r, x)
    Wh = q4x.dequant_q4x(r["codes"], r["scales"], r["books"], r["codebooks"])
    for b in range(2):
        for n in range(3):
            want = sum(Fraction(float(x[b, kk])) * Fraction(float(Wh[n, kk])) for kk in range(128))
            assert abs(Fraction(y[b, n]) - want) <= abs(want) * Fraction(1, 10 ** 13) + Fraction(1, 10 ** 30)
