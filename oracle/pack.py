"""Packed storage of quantized weights (oracle; test infrastructure only).

The paper fixes no byte layout: Section 2.4 says only that data-mover bus widths
and the packing/unpacking kernels decide decode speed, and Section 3.2 shows
llama.cpp's Q4_0 / Q4_K / Q4X blocks for a CPU.  The layout below is this
library's contract, written out element by element so that it can be checked by
eye.  All multi-byte words are little-endian.  A row of W (fixed n) is stored
contiguously; rows follow each other with no padding (k is a multiple of 128,
so every row starts on a 16-byte boundary).

4-bit codes (k/2 bytes per row)
    Word t of a row (bytes 4t..4t+3) holds the codes of k = 8t .. 8t+7.  The
    code of k = 8t + j sits in nibble pi(j) = j // 2 + 4 * (j % 2), i.e. the
    nibbles 0..7 hold j = 0, 2, 4, 6, 1, 3, 5, 7.

3-bit codes (3k/8 bytes per row)
    A row is three planes of k/8 bytes each; plane p starts at byte p * k / 8.
    Superblock s covers k = 128 s .. 128 s + 127 and owns bytes 16 s .. 16 s + 15
    of every plane.  Inside it, word i (i = 0..3, bytes 4i..4i+3 of the
    superblock's 16 bytes) of planes 0, 1, 2 -- called A_i, B_i, C_i -- hold the
    32 codes c_0..c_31 of k = 128 s + 32 i + m (m = 0..31):
      nibble t (t = 0..7) of A_i, bits 0-2: c_t
      nibble t of B_i, bits 0-2:            c_{8+t}
      nibble t of C_i, bits 0-2:            c_{16+t}
      bit 3 of nibble t of A_i, B_i, C_i:   bits 0, 1, 2 of c_{24+t}

Zero-points (uniform only; ceil(G/2) bytes per row, G = k / g groups)
    Group j's zero-point is the low nibble of byte j // 2 when j is even and
    the high nibble when j is odd; an unused high nibble is 0.

Scales (uniform only): fp16 [n][G].  LUTs (non-uniform only): fp16 [n][G][2^b],
entries ascending.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

from .quant import quantize_uniform, dequant_uniform, quantize_lut, dequant_lut

UNIFORM, LUT = "uniform", "lut"
_PI4 = [j // 2 + 4 * (j % 2) for j in range(8)]


@dataclass(frozen=True)
class Recipe:
    """Per-matrix recipe: bit-width, group size, uniform vs non-uniform (Sections 2.1-2.3)."""

    bits: int
    group_size: int
    kind: str = UNIFORM
    lloyd_iters: int = 25


def _check_shape(k: int, bits: int):
    if bits not in (3, 4):
        raise ValueError("bits must be 3 or 4")
    if k % 128 != 0:
        raise ValueError("k must be a multiple of 128")


def pack_codes(codes: np.ndarray, bits: int) -> np.ndarray:
    """Codes uint8 [n][k] (each < 2^bits) -> packed bytes uint8 [n][k * bits / 8]."""
    codes = np.asarray(codes, dtype=np.uint8)
    n, k = codes.shape
    _check_shape(k, bits)
    if codes.size and int(codes.max()) >= (1 << bits):
        raise ValueError("code out of range")
    c = codes.astype(np.uint32)
    if bits == 4:
        c = c.reshape(n, k // 8, 8)
        words = np.zeros((n, k // 8), dtype=np.uint32)
        for j in range(8):
            words |= c[:, :, j] << np.uint32(4 * _PI4[j])
        return words.astype("<u4").view(np.uint8).reshape(n, k // 2)
    c = c.reshape(n, k // 128, 4, 32)  # [row][superblock s][word i][m]
    planes = []
    for p in range(3):  # plane p: nibbles hold c_{8p+t}, bit 3 holds bit p of c_{24+t}
        w = np.zeros((n, k // 128, 4), dtype=np.uint32)
        for t in range(8):
            w |= c[:, :, :, 8 * p + t] << np.uint32(4 * t)
            w |= ((c[:, :, :, 24 + t] >> np.uint32(p)) & np.uint32(1)) << np.uint32(4 * t + 3)
        planes.append(w.reshape(n, k // 32))
    words = np.concatenate(planes, axis=1)
    return words.astype("<u4").view(np.uint8).reshape(n, 3 * k // 8)


def unpack_codes(packed: np.ndarray, bits: int, k: int) -> np.ndarray:
    """Inverse of :func:`pack_codes`."""
    packed = np.ascontiguousarray(packed, dtype=np.uint8)
    n = packed.shape[0]
    _check_shape(k, bits)
    words = packed.view("<u4").astype(np.uint32)
    if bits == 4:
        words = words.reshape(n, k // 8)
        out = np.zeros((n, k // 8, 8), dtype=np.uint32)
        for j in range(8):
            out[:, :, j] = (words >> np.uint32(4 * _PI4[j])) & np.uint32(15)
        return out.reshape(n, k).astype(np.uint8)
    words = words.reshape(n, 3, k // 128, 4)  # [row][plane][superblock][word]
    out = np.zeros((n, k // 128, 4, 32), dtype=np.uint32)
    for p in range(3):
        w = words[:, p]
        for t in range(8):
            out[:, :, :, 8 * p + t] = (w >> np.uint32(4 * t)) & np.uint32(7)
            out[:, :, :, 24 + t] |= ((w >> np.uint32(4 * t + 3)) & np.uint32(1)) << np.uint32(p)
    return out.reshape(n, k).astype(np.uint8)


def pack_zeros(zeros: np.ndarray) -> np.ndarray:
    """Zero-points uint8 [n][G] (each < 16) -> nibble bytes uint8 [n][ceil(G/2)]."""
    zeros = np.asarray(zeros, dtype=np.uint8)
    n, G = zeros.shape
    if zeros.size and int(zeros.max()) > 15:
        raise ValueError("zero-point out of range")
    pad = np.zeros((n, G + (G % 2)), dtype=np.uint8)
    pad[:, :G] = zeros
    return (pad[:, 0::2] | (pad[:, 1::2] << 4)).astype(np.uint8)


def unpack_zeros(packed: np.ndarray, G: int) -> np.ndarray:
    packed = np.asarray(packed, dtype=np.uint8)
    out = np.empty((packed.shape[0], 2 * packed.shape[1]), dtype=np.uint8)
    out[:, 0::2] = packed & 15
    out[:, 1::2] = packed >> 4
    return out[:, :G]


def packed_sizes(n: int, k: int, r: Recipe) -> dict:
    """Bytes of each packed buffer; 0 for buffers the recipe does not use."""
    _check_shape(k, r.bits)
    G = k // r.group_size
    uni = r.kind == UNIFORM
    return {
        "codes": n * k * r.bits // 8,
        "scales": n * G * 2 if uni else 0,
        "zeros": n * ((G + 1) // 2) if uni else 0,
        "luts": 0 if uni else n * G * (1 << r.bits) * 2,
    }


def quantize(W: np.ndarray, r: Recipe) -> dict:
    """Quantize fp16 W [n][k] with recipe ``r`` and pack it."""
    n, k = W.shape
    _check_shape(k, r.bits)
    if r.kind == UNIFORM:
        q, s, z = quantize_uniform(W, r.bits, r.group_size)
        return {"codes": pack_codes(q, r.bits), "scales": s, "zeros": pack_zeros(z), "luts": None}
    if r.kind == LUT:
        q, lut = quantize_lut(W, r.bits, r.group_size, r.lloyd_iters)
        return {"codes": pack_codes(q, r.bits), "scales": None, "zeros": None, "luts": lut}
    raise ValueError("unknown kind")


def dequant(p: dict, r: Recipe, k: int) -> np.ndarray:
    """Packed weights -> fp16 W_hat [n][k]."""
    q = unpack_codes(p["codes"], r.bits, k)
    G = k // r.group_size
    if r.kind == UNIFORM:
        return dequant_uniform(q, p["scales"], unpack_zeros(p["zeros"], G), r.group_size)
    return dequant_lut(q, p["luts"], r.group_size)
