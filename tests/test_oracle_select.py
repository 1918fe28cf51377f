"""Pins of the oracle's per-matrix recipe selection (Sections 2.2-2.3: uniform or
non-uniform per matrix by the Frobenius error; bit-widths per layer)."""
from fractions import Fraction

import numpy as np
import pytest

from oracle import select
from oracle.pack import Recipe
import synth

U3 = Recipe(3, 64, "uniform")
U4 = Recipe(4, 64, "uniform")
L3 = Recipe(3, 64, "lut")


def test_error_is_the_exact_sum_of_squares():
    W = synth.student_t_weights(4, 128, 0.02, seed=1, stream=1).astype(np.float16)
    Wh = (W.astype(np.float32) * np.float32(0.9)).astype(np.float16)
    want = sum((Fraction(float(a)) - Fraction(float(b))) ** 2 for a, b in zip(W.ravel(), Wh.ravel()))
    assert Fraction(select.sq_error_units(W, Wh), 1 << 48) == want


def test_groups_with_eight_levels_choose_the_lut():
    """Eight unequally spaced values per group: the 3-bit LUT is lossless (its
    step 0), the uniform 3-bit grid is not."""
    rng = np.random.default_rng(2)
    levels = np.array([-0.05, -0.011, -0.002, 0.0, 0.0007, 0.003, 0.02, 0.07])
    W = levels[rng.integers(0, 8, (8, 256))].astype(np.float16)
    best, errs, _ = select.select_recipe(W, [U3, L3])
    assert errs[1] == 0 and errs[0] > 0 and best == 1


def test_ties_go_to_fewer_bits_per_weight():
    """Groups on a uniform 3-bit grid that includes both ends: uniform 3-bit and
    the LUT are both lossless; uniform 3-bit stores fewer bits."""
    rng = np.random.default_rng(3)
    s = np.float16(2.0 ** -7)
    q = rng.integers(0, 8, (8, 256))
    q[:, ::64] = 0
    q[:, 1::64] = 7
    W = ((q - 3) * float(s)).astype(np.float16)
    best, errs, bpws = select.select_recipe(W, [L3, U3, U3])
    assert errs == [0, 0, 0]
    assert bpws == [5.0, 3.3125, 3.3125] and best == 1  # then the earlier of equals


def test_budget_excludes_recipes_and_can_exclude_all():
    W = synth.student_t_weights(16, 256, 0.02, seed=4, stream=4).astype(np.float16)
    best_all, errs, _ = select.select_recipe(W, [U3, U4, L3])
    assert best_all in (1, 2)  # more bits or a fitted codebook beat 3-bit uniform here
    best, errs_b, _ = select.select_recipe(W, [U3, U4, L3], max_bpw=4.0)
    assert best == 0 and errs_b[1] is None and errs_b[2] is None
    assert select.select_recipe(W, [U4, L3], max_bpw=3.0)[0] is None


def test_q4x_candidate_bits_per_weight_and_lossless_choice():
    """Groups made of 16 shared levels (times a per-group power of two, with
    the group maximum present) are coded without error by Q4X, which must then
    win against every per-group recipe; its bits per weight are the paper's
    4 + 18/64 plus the 128-byte codebooks."""
    from fractions import Fraction

    from oracle.select import Q4X

    n, k = 16, 256
    levels = np.array([-1, -0.75, -0.5, -0.375, -0.25, -0.125, -0.0625, 0,
                       0.0625, 0.125, 0.25, 0.375, 0.5, 0.625, 0.75, 1.0])
    rng = np.random.default_rng(4)
    W = np.empty((n, k))
    for r in range(n):
        for g in range(k // 64):
            v = levels[rng.integers(0, 16, 64)]
            v[0] = 1.0  # the group maximum, so that s is the power of two below
            W[r, 64 * g:64 * g + 64] = v * 2.0 ** -int(rng.integers(3, 8))
    W = W.astype(np.float16)
    cands = [Recipe(4, 64, "uniform"), Recipe(3, 128, "lut"), Recipe(4, 64, Q4X)]
    chosen, errs, bpws = select.select_recipe(W, cands)
    assert errs[2] == 0 and all(e > 0 for e in errs[:2]) and chosen == 2
    assert Fraction(bpws[2]).limit_denominator(1 << 20) == Fraction(8 * (n * k // 2 + 2 * n * 4 + n * 1 + 128), n * k)
    with pytest.raises(ValueError):
        select.bits_per_weight(n, k, Recipe(3, 64, Q4X))
