"""W.A8 decode of the oracle: 8-bit activations against uniform 3/4-bit weights
(test infrastructure only).

Paper Table 2 runs every weight format with "8-bit RTN per-token quantization
for the activation tensors" (W4A8), and Table 1 lists W3A8 next to W3A16.
Readings:

  Activations, per token b (row of x, fp16):
      m   = max_k |x[b][k]|                     exact
      s_b = fp32(m / 127)                        one fp32 division
      q   = clamp(rint(fp32(x) / s_b), -127, 127) int8, fp32 division, rint
                                                 half to even; q = 0 when m = 0
  Matmul, uniform weights (codes q_w, zero-points z, fp16 scales s_g):
      y[b][n] = s_b * sum_g s_g * sum_{k in g} (q_w[n][k] - z[n][g]) * q[b][k]
      The inner sums are exact integers; the oracle takes the rest in float64.
  Non-uniform (LUT) weights have no integer form: W.A8 decode is uniform only.
  Prefill (any weight format): the tensor cores take fp16 operands, so the
  int8 activations enter as
      x_hat[b][k] = fp16(fp32(s_b * q[b][k]))      one fp32 product, then RN
  and Y = x_hat W_hat^T is the fp16 matmul of the prefill, in float64 here.
  For uniform weights it differs from the decode form above only by the
  rounding of x_hat (at most 2^-11 of each |s_b q|).
"""
from __future__ import annotations

import numpy as np

from .pack import UNIFORM, unpack_codes, unpack_zeros

F32, F64 = np.float32, np.float64


def quantize_act(x: np.ndarray):
    """Per-token symmetric int8 RTN: (q int8 [b][k], s float32 [b])."""
    x = np.atleast_2d(np.asarray(x, dtype=np.float16)).astype(F32)  # exact
    m = np.abs(x).max(axis=1)
    s = (m / F32(127)).astype(F32)
    safe = np.where(s > 0, s, F32(1))
    q = np.clip(np.rint(x / safe[:, None]), -127, 127)
    q[s == 0] = 0
    return q.astype(np.int8), s


def int_dots(p: dict, r, q: np.ndarray, k: int) -> np.ndarray:
    """Exact integer group sums D[b][n][g] = sum_{k in g} (q_w - z) q_x (int64)."""
    if r.kind != UNIFORM:
        raise ValueError("W.A8 needs uniform weights")
    qw = unpack_codes(p["codes"], r.bits, k).astype(np.int64)  # [n][k]
    n = qw.shape[0]
    G = k // r.group_size
    z = unpack_zeros(p["zeros"], G).astype(np.int64)  # [n][G]
    off = qw.reshape(n, G, r.group_size) - z[:, :, None]
    qx = q.astype(np.int64).reshape(q.shape[0], G, r.group_size)
    return np.einsum("ngk,bgk->bng", off, qx)


def gemv_a8(p: dict, r, x: np.ndarray, k: int) -> np.ndarray:
    """float64 y [b][n] of the W.A8 decode for fp16 activations x [b][k]."""
    q, s = quantize_act(x)
    D = int_dots(p, r, q, k).astype(F64)  # exact: |D| < 2^31
    sg = p["scales"].astype(F64)  # [n][G]
    return (D * sg[None, :, :]).sum(axis=2) * s.astype(F64)[:, None]


def dequant_act(q: np.ndarray, s: np.ndarray) -> np.ndarray:
    """x_hat = s q (float64), the activations the W.A8 decode multiplies."""
    return q.astype(F64) * s.astype(F64)[:, None]


def dequant_act_f16(q: np.ndarray, s: np.ndarray) -> np.ndarray:
    """x_hat = fp16(fp32(s_b q)) [b][k], the prefill's fp16 activations."""
    prod = np.asarray(q, dtype=np.int8).astype(F32) * np.asarray(s, dtype=F32)[:, None]  # one fp32 RN product
    return prod.astype(np.float16)


def gemm_a8(W_hat: np.ndarray, x: np.ndarray) -> np.ndarray:
    """float64 Y [b][n] of the W.A8 prefill for fp16 activations x [b][k] and
    dequantized fp16 weights W_hat [n][k]."""
    q, s = quantize_act(x)
    return dequant_act_f16(q, s).astype(F64) @ np.asarray(W_hat, dtype=np.float16).astype(F64).T
