"""Pins of the oracle's dequantize + float64 matmul and of its tolerance."""
from fractions import Fraction

import numpy as np
import pytest

import oracle
from oracle.pack import Recipe


def test_gemv_exact_on_tiny_shapes():
    """float64 products of fp16 numbers are exact; the sum agrees with exact rationals."""
    r = np.random.default_rng(2)
    W = (r.standard_normal((6, 128)) * 0.05).astype(np.float16)
    X = r.standard_normal((3, 128)).astype(np.float16)
    for rec in (Recipe(4, 64), Recipe(3, 128, "lut", 10)):
        p = oracle.quantize(W, rec)
        Wh = oracle.dequant(p, rec, 128)
        y = oracle.gemv(p, rec, X, 128)
        for b in range(3):
            for n in range(6):
                exact = sum(Fraction(float(X[b, k])) * Fraction(float(Wh[n, k])) for k in range(128))
                assert abs(y[b, n] - float(exact)) <= 1e-12 * max(1.0, abs(float(exact)))


def test_zero_weights_give_zero():
    W = np.zeros((8, 256), np.float16)
    x = np.random.default_rng(0).standard_normal((1, 256)).astype(np.float16)
    for rec in (Recipe(4, 128), Recipe(3, 64), Recipe(3, 128, "lut")):
        y = oracle.gemv(oracle.quantize(W, rec), rec, x, 256)
        assert np.all(y == 0)


def test_single_nonzero_column_selects_activation():
    """A grid-aligned one-hot row picks out one activation exactly."""
    k = 128
    W = np.zeros((4, k), np.float16)
    for n in range(4):
        W[n, 17 * n + 3] = 1.0
    x = np.random.default_rng(1).standard_normal((2, k)).astype(np.float16)
    for rec in (Recipe(4, 64), Recipe(3, 128, "lut")):
        y = oracle.gemv(oracle.quantize(W, rec), rec, x, k)
        for n in range(4):
            assert np.array_equal(y[:, n], x[:, 17 * n + 3].astype(np.float64))


def test_tolerance_closed_form():
    x = np.array([[3.0, 4.0], [0.0, 1.0]])
    Wh = np.array([[1.0, 0.0], [2.0, 2.0]])
    tol = oracle.tolerance(x, Wh)
    assert np.allclose(tol, 2e-3 * np.array([5.0, 1.0]) * np.sqrt(8.0))


def test_quantization_error_ordering():
    """Sanity on Student-t(4) weights: more bits, smaller groups and Lloyd iterations help."""
    W = (np.random.default_rng(0).standard_t(4, size=(64, 1024)) * 0.02).astype(np.float16)

    def rel(rec):
        Wh = oracle.dequant(oracle.quantize(W, rec), rec, 1024).astype(np.float64)
        return np.linalg.norm(Wh - W) / np.linalg.norm(W.astype(np.float64))

    u4g64, u4g128, u3g64 = rel(Recipe(4, 64)), rel(Recipe(4, 128)), rel(Recipe(3, 64))
    l3, l3_init = rel(Recipe(3, 128, "lut", 25)), rel(Recipe(3, 128, "lut", 0))
    assert u4g64 < u4g128 < u3g64 < 0.3
    assert l3 < 0.6 * l3_init and l3 < u3g64
