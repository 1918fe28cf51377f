"""Per-group weight quantizers of the oracle (test infrastructure only).

Weights W are fp16 [n][k] (row n = output feature, k = input feature, as in a
linear layer).  A group is g consecutive weights of one row along k.

Uniform asymmetric RTN (``quantize_uniform``)
    The paper's uniform quantizer places 2^b equally spaced points per group
    (Section 2.2), rounds each weight to the nearest one (Section 3.2, Q4_0:
    "RTN on a group") and is asymmetric with a per-group scale and minimum
    (Section 3.2, Q4_K).  The paper prints no formula; the reading used here,
    in IEEE fp32 with round-to-nearest-even and no fused multiply-add:

      lo  = min(0, min_G w),  hi = max(0, max_G w)        range widened to hold 0
      s16 = fp16( fp32(hi - lo) / (2^b - 1) )              stored scale
      s   = (float) s16
      if s16 == 0:  z = 0 and every code is 0
      else:         z = clamp(rint(-lo / s), 0, 2^b - 1)   stored 4-bit zero-point
                    q = clamp(rint(w / s) + z, 0, 2^b - 1)
      w_hat = fp16( (float)(q - z) * s )                   exact product, one rounding

    rint rounds half to even.  Because 0 is inside [lo, hi] the zero-point fits
    in b bits, so a 4-bit nibble stores it for both b = 3 and b = 4.

Non-uniform Lloyd-Max LUT (``quantize_lut``)
    The non-uniform quantizer maps each group onto its own codebook of 2^b
    levels placed where the probability mass is (Section 2.2, Fig. 2a); the
    codebook is fit by Lloyd-Max, i.e. one-dimensional k-means.  Reading:

      0. a group with at most 2^b distinct values: the LUT is those values in
         ascending order, padded by repeating the largest;
      1. otherwise initial levels c_j = sorted(w)[floor((2j + 1) g / 2^(b+1))];
      2. up to T iterations (T = ``iters``), stopping as soon as an
         assignment equals the previous one:
           a_k = argmin_j |w_k - c_j|       (float64; ties to the lowest j)
           c_j = (sum_{a_k = j} w_k) / n_j  (sum exact, one float64 division;
                                             an empty cell keeps c_j)
      3. sort the levels ascending; LUT_j = fp16(c_j), one rounding from float64;
      4. q_k = argmin_j |w_k - LUT_j| (float64, exact; ties to the lowest j);
      5. w_hat_k = LUT_{q_k}.

    The cell sums are taken exactly: every fp16 value is an integer multiple
    of 2^-24 and |w| <= 65504 < 2^16, so sum(w * 2^24) over <= 2^7 weights is an
    integer below 2^47 and both it and its float64 image are exact.
"""
from __future__ import annotations

import numpy as np

F16, F32, F64 = np.float16, np.float32, np.float64
_TWO24 = float(1 << 24)


def round_to_fp16(x: np.ndarray) -> np.ndarray:
    """One rounding from float64 to the nearest fp16, ties to even (LUT step 3)."""
    return np.asarray(x, dtype=F64).astype(F16)


def _check_input(W: np.ndarray, g: int) -> np.ndarray:
    W = np.asarray(W)
    if W.dtype != F16 or W.ndim != 2:
        raise ValueError("W must be a 2-D float16 array")
    if g <= 0 or W.shape[1] % g != 0:
        raise ValueError("the group size must divide k")
    if not np.all(np.isfinite(W)):
        raise ValueError("W holds NaN or Inf")
    return W


def quantize_uniform(W: np.ndarray, bits: int, g: int):
    """Uniform asymmetric per-group RTN quantizer (Section 2.2; Section 3.2).

    Returns ``(codes uint8 [n][k], scales fp16 [n][k/g], zeros uint8 [n][k/g])``.
    """
    W = _check_input(W, g)
    n, k = W.shape
    qmax = F32((1 << bits) - 1)
    w = W.reshape(n, k // g, g).astype(F32)  # fp16 -> fp32 is exact
    lo = np.minimum(w.min(axis=2), F32(0))
    hi = np.maximum(w.max(axis=2), F32(0))
    s16 = ((hi - lo) / qmax).astype(F16)  # fp32 subtract, fp32 divide, round to fp16
    s = s16.astype(F32)
    dead = s == 0
    s_safe = np.where(dead, F32(1), s)
    z = np.clip(np.rint(-lo / s_safe), F32(0), qmax)
    q = np.clip(np.rint(w / s_safe[:, :, None]) + z[:, :, None], F32(0), qmax)
    z = np.where(dead, F32(0), z)
    q = np.where(dead[:, :, None], F32(0), q)
    return q.astype(np.uint8).reshape(n, k), s16, z.astype(np.uint8)


def dequant_uniform(codes: np.ndarray, scales: np.ndarray, zeros: np.ndarray, g: int) -> np.ndarray:
    """w_hat = fp16((q - z) * s) per element (Section 3.2: scale and minimum per group)."""
    n, k = codes.shape
    q = codes.reshape(n, k // g, g).astype(F32)
    z = zeros.astype(F32)[:, :, None]
    s = scales.astype(F32)[:, :, None]
    return ((q - z) * s).astype(F16).reshape(n, k)


def _argmin_abs(w: np.ndarray, c: np.ndarray) -> np.ndarray:
    """Index of the nearest level, float64 distances, ties to the lowest index."""
    return np.argmin(np.abs(w[:, :, None] - c[:, None, :]), axis=2)


def _lloyd(w: np.ndarray, wi: np.ndarray, c: np.ndarray, iters: int, trace=None):
    """Lloyd-Max iterations on a batch of groups (rows of ``w``); returns levels."""
    L = c.shape[1]
    active = np.ones(w.shape[0], dtype=bool)
    prev = None
    for _ in range(iters):
        a = _argmin_abs(w, c)
        if prev is not None:
            active &= np.any(a != prev, axis=1)
            if not active.any():
                break
        newc = c.copy()
        for j in range(L):
            m = a == j
            cnt = m.sum(axis=1)
            tot = np.where(m, wi, 0).sum(axis=1)  # exact int64
            mean = (tot.astype(F64) / _TWO24) / np.maximum(cnt, 1)
            newc[:, j] = np.where(cnt > 0, mean, c[:, j])
        c = np.where(active[:, None], newc, c)
        prev = a
        if trace is not None:
            trace.append(c.copy())
    return c


def _lut_groups(wg: np.ndarray, bits: int, iters: int, trace=None) -> np.ndarray:
    """fp16 LUTs [groups][2^b] for fp16 groups ``wg`` [groups][g]."""
    G, g = wg.shape
    L = 1 << bits
    w = wg.astype(F64)
    wi = (w * _TWO24).astype(np.int64)
    ws = np.sort(w, axis=1)
    distinct = 1 + np.count_nonzero(np.diff(ws, axis=1), axis=1)
    few = distinct <= L
    luts = np.empty((G, L), dtype=F64)
    # step 0: groups that already have at most 2^b distinct values
    for i in np.nonzero(few)[0]:
        u = np.unique(ws[i])
        luts[i] = np.concatenate([u, np.full(L - u.size, u[-1])])
    rest = np.nonzero(~few)[0]
    if rest.size:
        idx = [((2 * j + 1) * g) // (2 * L) for j in range(L)]
        c = ws[rest][:, idx]  # step 1: quantile initialisation
        c = _lloyd(w[rest], wi[rest], c, iters, trace)  # step 2
        luts[rest] = np.sort(c, axis=1, kind="stable")  # step 3 (sort)
    return round_to_fp16(luts)  # step 3


def quantize_lut(W: np.ndarray, bits: int, g: int, iters: int = 25):
    """Non-uniform per-group Lloyd-Max quantizer (Section 2.2, Fig. 2a; Table 1).

    Returns ``(codes uint8 [n][k], luts fp16 [n][k/g][2^b])``.
    """
    W = _check_input(W, g)
    if iters < 0:
        raise ValueError("iters must be >= 0")
    n, k = W.shape
    wg = W.reshape(-1, g)
    luts = _lut_groups(wg, bits, iters)
    codes = _argmin_abs(wg.astype(F64), luts.astype(F64))  # step 4
    return codes.astype(np.uint8).reshape(n, k), luts.reshape(n, k // g, 1 << bits)


def dequant_lut(codes: np.ndarray, luts: np.ndarray, g: int) -> np.ndarray:
    """w_hat_k = LUT_{q_k} of the element's group (step 5)."""
    n, k = codes.shape
    q = codes.reshape(n, k // g, g).astype(np.int64)
    return np.take_along_axis(luts, q, axis=2).reshape(n, k)


def lloyd_max_trace(wg: np.ndarray, bits: int, iters: int):
    """Levels after every Lloyd-Max update for fp16 groups ``wg`` [groups][g].

    Only for groups with more than 2^b distinct values; used by the tests that
    check the monotone decrease of the distortion.  Returns (init, [levels...]).
    """
    G, g = wg.shape
    L = 1 << bits
    w = wg.astype(F64)
    wi = (w * _TWO24).astype(np.int64)
    ws = np.sort(w, axis=1)
    idx = [((2 * j + 1) * g) // (2 * L) for j in range(L)]
    c0 = ws[:, idx]
    trace: list = []
    _lloyd(w, wi, c0.copy(), iters, trace)
    return c0, trace
