"""Q4X shared-codebook quantizer of the oracle (test infrastructure only).

Q4X (paper Section 3.2, Fig. 3a/3b, Table 2 "Q4X W4A8G64, 4.28 BPW") codes each
group of 64 weights with a 2-byte scale, a 2-bit index naming one of four
codebooks, and a 4-bit centroid index per weight.  The four codebooks, of 16
centroids each, are learned per weight matrix: a histogram is taken of every
group, four histograms that best represent all of them are learned, and each
learned histogram is reduced to 16 non-uniform samples.  The paper gives the
idea, not the arithmetic; the readings below fix every step so that another
implementation can reproduce the result exactly.

  1. Scale.  s = max_G |w| (an fp16 value, so no rounding).  A group with
     s = 0 is dead: book 0, every code 0, and it takes no part in learning.
  2. Normalised values.  U = rint(fp64(w) / fp64(s) * 2^20): the quotient is
     correctly rounded in float64, the scaling by 2^20 is exact, rint rounds
     half to even.  |U| <= 2^20; every later sum of U is an exact int64.
  3. Histograms.  32 bins over [-1, 1]: bin = min(31, (U + 2^20) >> 16); a
     group's histogram is its 32 integer counts.
  4. Learned histograms: k-means with 4 centres over the live groups'
     histograms (squared Euclidean distance).
       init: sort the live groups by M2 = sum U^2 (then by position); the
             centres start as the histograms of the groups at ranks
             floor((2j + 1) L / 8), j = 0..3, of the L live groups;
       step: assign each group to the nearest centre -- the distance summed in
             float64 over the bins in order 0..31, ties to the lowest centre;
             stop when the assignment equals the previous one; else each
             centre becomes the exact integer sum of its members' histograms
             divided by their count (one float64 division per bin), and a
             centre without members keeps its value; at most `iters` steps.
     A group's codebook index is its centre in the last assignment.
  5. Dimension reduction: each learned histogram stands for the normalised
     values of the groups assigned to it, and its 16 samples are the 16-level
     Lloyd-Max quantizer of those values (1-D k-means):
       at most 16 distinct values: those values ascending, padded by repeating
             the largest;
       else init c_j = sorted(U)[floor((2j + 1) N / 32)], then up to `iters`
             steps: nearest level (float64, ties to the lowest), stop when the
             assignment repeats, each level = exact int64 cell sum / count
             (one float64 division), an empty cell keeps its level;
       then sort ascending.  A book no group uses gets the uniform levels
       ((2j + 1) / 16 - 1) 2^20.
     Codebook entry = fp16(level / 2^20), one rounding from float64.
  6. Codes.  For a group with scale s and book b the candidates are
     w_hat_j = fp16(fp32(s) * fp32(CB[b][j])) (the fp32 product of two fp16
     values is exact, so there is one rounding); q = argmin_j |w - w_hat_j| in
     float64, ties to the lowest j.
  7. Dequantization.  w_hat = fp16(fp32(s) * fp32(CB[b][q])).
"""
from __future__ import annotations

import numpy as np

from .quant import F16, F32, F64, _check_input, round_to_fp16

GROUP = 64      # weights per group (Section 3.2: "each group of 64 weights")
BINS = 32       # histogram bins over [-1, 1]
BOOKS = 4       # learned histograms / codebooks per matrix
LEVELS = 16     # centroids per codebook (4-bit codes)
FRAC = 20       # fixed-point bits of the normalised values
_ONE = 1 << FRAC


def q4x_normalize(W: np.ndarray, g: int = GROUP):
    """Step 1-2: fp16 scales [n][k/g], int64 normalised values U [n][k/g][g], live mask."""
    W = _check_input(W, g)
    n, k = W.shape
    wg = W.reshape(n, k // g, g)
    s16 = np.abs(wg).max(axis=2)  # |fp16| and max are exact
    s = s16.astype(F64)
    live = s > 0
    u = wg.astype(F64) / np.where(live, s, 1.0)[:, :, None]  # correctly rounded
    U = np.rint(u * float(_ONE)).astype(np.int64)
    U[~live] = 0
    return s16, U, live


def q4x_histograms(U: np.ndarray) -> np.ndarray:
    """Step 3: integer histograms [groups][32] of normalised groups U [groups][g]."""
    b = np.minimum((U + _ONE) >> (FRAC + 1 - 5), BINS - 1)  # (U + 2^20) >> 16
    return np.stack([(b == j).sum(axis=1) for j in range(BINS)], axis=1).astype(np.int64)


def _sq_dist(H: np.ndarray, C: np.ndarray) -> np.ndarray:
    """float64 squared distances [groups][books], summed over the bins in order."""
    D = np.zeros((H.shape[0], C.shape[0]), dtype=F64)
    for b in range(H.shape[1]):
        diff = H[:, b:b + 1].astype(F64) - C[None, :, b]
        D = D + diff * diff
    return D


def q4x_kmeans(H: np.ndarray, M2: np.ndarray, iters: int, trace=None):
    """Step 4: (assignment [groups], centres float64 [4][32]) of the live groups."""
    L = H.shape[0]
    order = np.lexsort((np.arange(L), M2))
    C = H[order[[((2 * j + 1) * L) // (2 * BOOKS) for j in range(BOOKS)]]].astype(F64)
    a = np.zeros(L, dtype=np.int64)
    prev = None
    for _ in range(iters):
        a = np.argmin(_sq_dist(H, C), axis=1)
        if prev is not None and np.array_equal(a, prev):
            break
        for j in range(BOOKS):
            m = a == j
            cnt = int(m.sum())
            if cnt:
                C[j] = H[m].sum(axis=0).astype(F64) / cnt
        prev = a
        if trace is not None:
            trace.append((a.copy(), C.copy()))
    return a, C


def _nearest(V: np.ndarray, c: np.ndarray) -> np.ndarray:
    """Index of the nearest level for int64 values V (float64, ties to the lowest)."""
    out = np.empty(V.size, dtype=np.int64)
    cf = c.astype(F64)
    for i in range(0, V.size, 1 << 16):  # chunks keep the distance table small
        v = V[i:i + (1 << 16)].astype(F64)
        out[i:i + v.size] = np.argmin(np.abs(v[:, None] - cf[None, :]), axis=1)
    return out


def q4x_lloyd16(V: np.ndarray, iters: int, trace=None) -> np.ndarray:
    """Step 5: 16 sorted float64 levels (in units of 2^-20) for pooled values V."""
    V = np.asarray(V, dtype=np.int64).ravel()
    if V.size == 0:
        return np.array([((2 * j + 1) / LEVELS - 1.0) * _ONE for j in range(LEVELS)], dtype=F64)
    u = np.unique(V)
    if u.size <= LEVELS:
        return np.concatenate([u, np.full(LEVELS - u.size, u[-1])]).astype(F64)
    Vs = np.sort(V)
    N = V.size
    c = Vs[[((2 * j + 1) * N) // (2 * LEVELS) for j in range(LEVELS)]].astype(F64)
    prev = None
    for _ in range(iters):
        a = _nearest(V, c)
        if prev is not None and np.array_equal(a, prev):
            break
        for j in range(LEVELS):
            m = a == j
            cnt = int(m.sum())
            if cnt:
                c[j] = float(int(V[m].sum())) / cnt  # exact int64 sum, one division
        prev = a
        if trace is not None:
            trace.append(c.copy())
    return np.sort(c, kind="stable")


def q4x_candidates(s16: np.ndarray, books: np.ndarray, codebooks: np.ndarray) -> np.ndarray:
    """fp16 w_hat_j = fp16(fp32(s) * fp32(CB[book][j])) for every group: [n][G][16]."""
    cb = codebooks.astype(F32)[books]  # [n][G][16]
    return (s16.astype(F32)[:, :, None] * cb).astype(F16)


def quantize_q4x(W: np.ndarray, iters: int = 25, g: int = GROUP, trace=None) -> dict:
    """Q4X quantizer (Section 3.2, Fig. 3a): steps 1-6 of the module docstring.

    Returns ``{"codes": uint8 [n][k], "scales": fp16 [n][k/g], "books": uint8
    [n][k/g], "codebooks": fp16 [4][16]}``.
    """
    if iters < 0:
        raise ValueError("iters must be >= 0")
    s16, U, live = q4x_normalize(W, g)
    n, G, _ = U.shape
    Ul = U[live]  # [L][g] live groups in row-major group order
    books = np.zeros((n, G), dtype=np.uint8)
    levels = np.zeros((BOOKS, LEVELS), dtype=F64)
    if Ul.shape[0]:
        H = q4x_histograms(Ul)
        M2 = (Ul * Ul).sum(axis=1)
        a, _ = q4x_kmeans(H, M2, iters, trace)
        books[live] = a.astype(np.uint8)
        for j in range(BOOKS):
            levels[j] = q4x_lloyd16(Ul[a == j], iters)
    else:
        for j in range(BOOKS):
            levels[j] = q4x_lloyd16(np.zeros(0, dtype=np.int64), iters)
    codebooks = round_to_fp16(levels / float(_ONE))
    # step 6: nearest candidate, rows in chunks to bound the distance table
    codes = np.empty((n, G * g), dtype=np.uint8)
    wg = np.asarray(W).reshape(n, G, g)
    for r0 in range(0, n, 64):
        cand = q4x_candidates(s16[r0:r0 + 64], books[r0:r0 + 64], codebooks).astype(F64)
        d = np.abs(wg[r0:r0 + 64].astype(F64)[:, :, :, None] - cand[:, :, None, :])
        codes[r0:r0 + 64] = np.argmin(d, axis=3).reshape(-1, G * g)
    return {"codes": codes, "scales": s16, "books": books, "codebooks": codebooks}


def dequant_q4x(codes: np.ndarray, scales: np.ndarray, books: np.ndarray, codebooks: np.ndarray,
                g: int = GROUP) -> np.ndarray:
    """Step 7: w_hat = fp16(fp32(s) * fp32(CB[book][q])) per element."""
    n, k = codes.shape
    cb = codebooks.astype(F32)[books.astype(np.int64)]  # [n][G][16]
    q = codes.reshape(n, k // g, g).astype(np.int64)
    c = np.take_along_axis(cb, q, axis=2)
    return (scales.astype(F32)[:, :, None] * c).astype(F16).reshape(n, k)


def pack_books(books: np.ndarray) -> np.ndarray:
    """2-bit codebook indices, four groups per byte: group j of a row in bits
    2 (j % 4) .. 2 (j % 4) + 1 of byte j / 4 (Section 3.2: 'padded together for
    byte alignment'); a row is padded to whole bytes with zeros."""
    n, G = books.shape
    nb = (G + 3) // 4
    out = np.zeros((n, nb), dtype=np.uint8)
    for j in range(G):
        out[:, j // 4] |= (books[:, j].astype(np.uint8) & 3) << (2 * (j % 4))
    return out


def unpack_books(packed: np.ndarray, G: int) -> np.ndarray:
    """Inverse of :func:`pack_books` for rows of G groups."""
    n = packed.shape[0]
    out = np.zeros((n, G), dtype=np.uint8)
    for j in range(G):
        out[:, j] = (packed[:, j // 4] >> (2 * (j % 4))) & 3
    return out


_NIBBLE = [j // 2 + 4 * (j % 2) for j in range(8)]  # nibble of k = 8t + j in word t


def pack_codes4(codes: np.ndarray) -> np.ndarray:
    """4-bit codes uint8 [n][k] (k a multiple of 8) -> bytes [n][k/2] in the
    library's 4-bit layout: little-endian word t holds k = 8t..8t+7, the code of
    k = 8t + j in nibble j/2 + 4 (j % 2)."""
    c = np.asarray(codes, dtype=np.uint32)
    n, k = c.shape
    if k % 8:
        raise ValueError("k must be a multiple of 8")
    c = c.reshape(n, k // 8, 8)
    words = np.zeros((n, k // 8), dtype=np.uint32)
    for j in range(8):
        words |= (c[:, :, j] & np.uint32(15)) << np.uint32(4 * _NIBBLE[j])
    return words.astype("<u4").view(np.uint8).reshape(n, k // 2)


def unpack_codes4(packed: np.ndarray, k: int) -> np.ndarray:
    """Inverse of :func:`pack_codes4`."""
    n = packed.shape[0]
    words = np.ascontiguousarray(packed, dtype=np.uint8).reshape(n, k // 2).view("<u4").astype(np.uint32)
    out = np.zeros((n, k // 8, 8), dtype=np.uint8)
    for j in range(8):
        out[:, :, j] = (words >> np.uint32(4 * _NIBBLE[j])) & np.uint32(15)
    return out.reshape(n, k)


def pack_q4x(q: dict) -> dict:
    """The packed buffers of a :func:`quantize_q4x` result: codes [n][k/2],
    scales fp16 [n][k/64], books [n][ceil(k/256)], codebooks fp16 [4][16]."""
    return {"codes": pack_codes4(q["codes"]), "scales": q["scales"], "books": pack_books(q["books"]),
            "codebooks": q["codebooks"]}


def gemv_q4x(q: dict, x: np.ndarray) -> np.ndarray:
    """float64 y [batch][n] = x W_hat^T with W_hat from :func:`dequant_q4x`."""
    Wh = dequant_q4x(q["codes"], q["scales"], q["books"], q["codebooks"]).astype(F64)
    return np.atleast_2d(np.asarray(x, dtype=F16)).astype(F64) @ Wh.T


def q4x_sizes(n: int, k: int, g: int = GROUP) -> dict:
    """Byte sizes of a packed Q4X matrix: 4-bit codes, fp16 scales, 2-bit book
    indices (padded per row to whole bytes), and the 4 x 16 fp16 codebook."""
    G = k // g
    return {"codes": n * k // 2, "scales": 2 * n * G, "books": n * ((G + 3) // 4), "codebooks": 2 * BOOKS * LEVELS}
