"""Dequantize-then-multiply reference and the parity tolerance (test infrastructure only).

Decode (matrix-vector, Section 2.4: "decoding is memory-bound") and prefill
(matrix-matrix, Table 2 "Prefill") both compute Y = X W_hat^T with
X [m][k] fp16 activations and W_hat [n][k] the dequantized weights.  The oracle
forms W_hat with :func:`oracle.pack.dequant` and multiplies in float64, where
every product of two fp16 numbers is exact.

Tolerance (the accuracy target of the quantized path): for every row b of X,
    max_n |y_gpu[b][n] - y_ref[b][n]| <= 2e-3 * ||x_b||_2 * max_n ||w_hat_n||_2.
"""
from __future__ import annotations

import numpy as np

from .pack import Recipe, dequant

REL_TOL = 2e-3


def gemm(p: dict, r: Recipe, X: np.ndarray, k: int) -> np.ndarray:
    """float64 [m][n] = X W_hat^T for packed weights ``p``."""
    Wh = dequant(p, r, k).astype(np.float64)
    return np.asarray(X, dtype=np.float16).astype(np.float64) @ Wh.T


def gemv(p: dict, r: Recipe, x: np.ndarray, k: int) -> np.ndarray:
    """Decode form of :func:`gemm`: ``x`` is [batch][k] (a handful of tokens)."""
    return gemm(p, r, np.atleast_2d(x), k)


def tolerance(X: np.ndarray, W_hat: np.ndarray) -> np.ndarray:
    """Per-row bound 2e-3 * ||x_b||_2 * max_n ||w_hat_n||_2 (float64)."""
    X = np.atleast_2d(np.asarray(X)).astype(np.float64)
    Wn = np.sqrt((np.asarray(W_hat).astype(np.float64) ** 2).sum(axis=1)).max(initial=0.0)
    return REL_TOL * np.sqrt((X ** 2).sum(axis=1)) * Wn


def max_abs_err(y: np.ndarray, y_ref: np.ndarray) -> np.ndarray:
    """Per-row max_n |y - y_ref| in float64."""
    d = np.abs(np.atleast_2d(y).astype(np.float64) - np.atleast_2d(y_ref).astype(np.float64))
    return d.max(axis=1, initial=0.0)
