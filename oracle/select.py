"""Per-matrix recipe selection of the oracle (test infrastructure only).

QuantX picks, per weight matrix, between uniform and non-uniform quantization
by the Frobenius norm of the quantization error (Section 2.2, closing
paragraph; Section 2.3, first paragraph), and sets bit-widths per layer to
trade memory against accuracy (Section 2.3, mixed bit-widths as in HAWQ).  The
paper's further criterion, the attention maps of Section 2.3, needs
activations and is not part of this step.  Reading:

  for every candidate recipe r (bits, group size, kind):
      bpw_r = 8 * (bytes of r's packed buffers) / (n k)
      E_r   = sum over the matrix of (w - w_hat_r)^2, exactly: fp16 values are
              integer multiples of 2^-24, so E_r * 2^48 is an integer
              (kept as a Python int; returned in units of 2^-48)
  eligible: bpw_r <= max_bpw (every candidate when max_bpw is None)
  chosen:   the eligible r with the smallest E_r, ties to the smaller bpw_r,
            then to the earlier candidate; None when none is eligible.

A candidate of kind "q4x" (bits 4, group size 64) is the shared-codebook
format of Section 3.2 (oracle/q4x.py, lloyd_iters as its step limit); its
bytes include the matrix's four codebooks.
"""
from __future__ import annotations

import numpy as np

from .pack import Recipe, dequant, packed_sizes, quantize
from .q4x import dequant_q4x, q4x_sizes, quantize_q4x

Q4X = "q4x"


def sq_error_units(W: np.ndarray, W_hat: np.ndarray) -> int:
    """sum (w - w_hat)^2 * 2^48 as an exact integer (both arrays fp16)."""
    a = (np.asarray(W, dtype=np.float16).astype(np.float64) * float(1 << 24)).astype(np.int64)
    b = (np.asarray(W_hat, dtype=np.float16).astype(np.float64) * float(1 << 24)).astype(np.int64)
    d = (a - b).ravel().astype(object)  # |d| < 2^41; squares need more than 64 bits
    return int((d * d).sum())


def _check_q4x(r: Recipe):
    if r.bits != 4 or r.group_size != 64:
        raise ValueError("a q4x candidate has 4 bits and groups of 64")


def bits_per_weight(n: int, k: int, r: Recipe) -> float:
    """8 * packed bytes / weights, as the float64 division of two integers."""
    if r.kind == Q4X:
        _check_q4x(r)
        return 8.0 * sum(q4x_sizes(n, k).values()) / (n * k)
    return 8.0 * sum(packed_sizes(n, k, r).values()) / (n * k)


def dequantized(W: np.ndarray, r: Recipe) -> np.ndarray:
    """W_hat of candidate r."""
    if r.kind == Q4X:
        _check_q4x(r)
        q = quantize_q4x(W, iters=r.lloyd_iters)
        return dequant_q4x(q["codes"], q["scales"], q["books"], q["codebooks"])
    return dequant(quantize(W, r), r, np.asarray(W).shape[1])


def select_recipe(W: np.ndarray, recipes: list, max_bpw: float | None = None):
    """(chosen index or None, [E_r in units of 2^-48], [bpw_r]) for fp16 W [n][k]."""
    W = np.asarray(W, dtype=np.float16)
    n, k = W.shape
    errs, bpws = [], []
    best = None
    for i, r in enumerate(recipes):
        bpw = bits_per_weight(n, k, r)
        bpws.append(bpw)
        if max_bpw is not None and bpw > max_bpw:
            errs.append(None)
            continue
        e = sq_error_units(W, dequantized(W, r))
        errs.append(e)
        if best is None or (e, bpw) < (errs[best], bpws[best]):
            best = i
    return best, errs, bpws
