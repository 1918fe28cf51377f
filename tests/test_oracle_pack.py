"""Pins of the oracle's packed layout: round trips, hand-computed byte images, sizes."""
import os

import numpy as np
import pytest

import oracle
from oracle.pack import Recipe

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _read_golden(name):
    out = {}
    with open(os.path.join(GOLD, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            key, *vals = line.split()
            out[key] = vals
    return out


@pytest.mark.parametrize("bits", [3, 4])
@pytest.mark.parametrize("k", [128, 384, 4096])
def test_codes_round_trip(bits, k):
    r = np.random.default_rng(bits * k)
    codes = r.integers(0, 1 << bits, size=(5, k)).astype(np.uint8)
    p = oracle.pack_codes(codes, bits)
    assert p.shape == (5, k * bits // 8) and p.dtype == np.uint8
    assert np.array_equal(oracle.unpack_codes(p, bits, k), codes)


def test_every_code_bit_is_used_once():
    """Setting one code to all-ones flips exactly ``bits`` distinct bits in the row."""
    for bits in (3, 4):
        k = 256
        base = oracle.pack_codes(np.zeros((1, k), np.uint8), bits)
        seen = np.zeros(base.size * 8, dtype=int)
        for kk in range(k):
            c = np.zeros((1, k), np.uint8)
            c[0, kk] = (1 << bits) - 1
            diff = np.unpackbits(oracle.pack_codes(c, bits) ^ base)
            assert diff.sum() == bits
            seen += diff
        assert np.all(seen == 1)


def test_golden_4bit_word():
    g = _read_golden("pack_4bit_word.txt")
    codes = np.zeros((1, 128), np.uint8)
    codes[0, :8] = [int(v) for v in g["codes"]]
    p = oracle.pack_codes(codes, 4)
    assert list(p[0, :4]) == [int(v, 16) for v in g["bytes"]]
    assert np.all(p[0, 4:] == 0)


def test_golden_3bit_superblock():
    g = _read_golden("pack_3bit_superblock.txt")
    codes = np.zeros((1, 128), np.uint8)
    codes[0, :32] = [int(v) for v in g["codes"]]
    p = oracle.pack_codes(codes, 3)
    assert p.shape == (1, 48)
    for plane in range(3):
        want = [int(v, 16) for v in g[f"plane{plane}"]]
        assert list(p[0, 16 * plane:16 * plane + 16]) == want


def test_zeros_nibbles():
    z = np.array([[1, 2, 3], [15, 0, 7]], dtype=np.uint8)
    p = oracle.pack_zeros(z)
    assert p.tolist() == [[0x21, 0x03], [0x0F, 0x07]]
    assert np.array_equal(oracle.unpack_zeros(p, 3), z)


def test_paper_bpw_arithmetic():
    """The bits-per-weight the paper prints follow from bits + metadata / group."""
    with open(os.path.join(GOLD, "paper_bpw.txt")) as f:
        rows = [ln.split() for ln in f if ln.strip() and not ln.startswith("#")]
    for name, bits, g, meta, printed, *_ in rows:
        bpw = int(bits) + int(meta) / int(g)
        assert round(bpw, 2) == float(printed), name


@pytest.mark.parametrize("bits,g,kind,bpw", [
    (4, 64, "uniform", 4.3125), (4, 128, "uniform", 4.15625),
    (3, 64, "uniform", 3.3125), (3, 128, "lut", 4.0), (3, 64, "lut", 5.0)])
def test_packed_sizes_bpw(bits, g, kind, bpw):
    n, k = 4, 4096
    sz = oracle.packed_sizes(n, k, Recipe(bits, g, kind))
    assert 8 * sum(sz.values()) / (n * k) == bpw
    W = (np.random.default_rng(0).standard_normal((n, k)) * 0.02).astype(np.float16)
    p = oracle.quantize(W, Recipe(bits, g, kind, 5))
    for key, nbytes in sz.items():
        arr = p[key]
        assert (0 if arr is None else arr.nbytes) == nbytes


def test_shape_checks():
    with pytest.raises(ValueError):
        oracle.pack_codes(np.zeros((1, 64), np.uint8), 4)
    with pytest.raises(ValueError):
        oracle.pack_codes(np.full((1, 128), 8, np.uint8), 3)


@pytest.mark.parametrize("bits,g,kind", [(3, 64, "uniform"), (4, 128, "uniform"), (3, 128, "lut")])
def test_rows_are_quantized_independently(bits, g, kind):
    """Every group lies within one row (Section 2.1: groups of consecutive
    weights along a row), so matrices stacked along n pack to their packed
    buffers stacked row for row: a fused projection is the same model."""
    import synth

    r = Recipe(bits, g, kind, 6)
    A = synth.student_t_weights(40, 256, 0.02, seed=1, stream=2).astype(np.float16)
    B = synth.student_t_weights(24, 256, 0.05, seed=1, stream=3).astype(np.float16)
    pa, pb, pab = oracle.quantize(A, r), oracle.quantize(B, r), oracle.quantize(np.vstack([A, B]), r)
    for key in ("codes", "scales", "zeros", "luts"):
        if pab[key] is None:
            assert pa[key] is None
            continue
        assert np.array_equal(pab[key].view(np.uint8), np.vstack([pa[key], pb[key]]).view(np.uint8)), key
