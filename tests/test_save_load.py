"""Save / load of packed matrices (host side; CPU tensors stand in for device
buffers): byte-exact round trips, and a corrupted, truncated or inconsistent
file is refused."""
import numpy as np
import pytest
import torch

import oracle
import synth
from oracle.pack import Recipe as ORecipe


@pytest.fixture(scope="module")
def qx():
    from paper_2505_07531_gb300 import build
    import os

    if not os.path.exists(build.LIB):
        build.build_library()
    import paper_2505_07531_gb300.qx as qx

    return qx


def _t(a, dtype=torch.uint8):
    return None if a is None else torch.from_numpy(np.ascontiguousarray(a).reshape(-1).view(np.uint8).copy()).view(dtype)


def _packed(qx, bits, g, kind):
    n, k = 24, 512
    W = synth.student_t_weights(n, k, 0.02, seed=bits + g, stream=77)
    rec = ORecipe(bits, g, "lut" if kind else "uniform", 25)
    p = oracle.quantize(W, rec)
    return qx.PackedMatrix(n, k, qx.Recipe(bits, g, kind), _t(p["codes"]), _t(p["scales"], torch.float16),
                           _t(p["zeros"]), _t(p["luts"], torch.float16))


def _same(a, b):
    if a is None or b is None:
        return a is None and b is None
    return torch.equal(a.view(torch.uint8), b.view(torch.uint8))


@pytest.mark.parametrize("bits,g,kind", [(4, 64, 0), (3, 128, 1), (3, 64, 0)])
def test_packed_round_trip(qx, tmp_path, bits, g, kind):
    P = _packed(qx, bits, g, kind)
    qx.save(str(tmp_path / "m.qx"), P)
    Q = qx.load(str(tmp_path / "m.qx"), device="cpu")
    assert (Q.n, Q.k, Q.recipe) == (P.n, P.k, P.recipe)
    for a, b in ((P.codes, Q.codes), (P.scales, Q.scales), (P.zeros, Q.zeros), (P.luts, Q.luts)):
        assert _same(a, b)


def test_q4x_round_trip(qx, tmp_path):
    n, k = 16, 320
    W = synth.student_t_weights(n, k, 0.02, seed=3, stream=78).astype(np.float16)
    p = oracle.pack_q4x(oracle.quantize_q4x(W))
    P = qx.Q4xMatrix(n, k, _t(p["codes"]), _t(p["scales"], torch.float16), _t(p["books"]),
                     _t(p["codebooks"], torch.float16))
    qx.save(str(tmp_path / "q.qx"), P)
    Q = qx.load(str(tmp_path / "q.qx"), device="cpu")
    assert isinstance(Q, qx.Q4xMatrix) and (Q.n, Q.k) == (n, k)
    for a, b in ((P.codes, Q.codes), (P.scales, Q.scales), (P.books, Q.books), (P.codebooks, Q.codebooks)):
        assert _same(a, b)


def test_damaged_files_are_refused(qx, tmp_path):
    P = _packed(qx, 4, 64, 0)
    path = tmp_path / "m.qx"
    qx.save(str(path), P)
    good = path.read_bytes()
    bad = bytearray(good)
    bad[100] ^= 0x40  # a code byte: checksum
    path.write_bytes(bytes(bad))
    with pytest.raises(ValueError, match="checksum"):
        qx.load(str(path), device="cpu")
    path.write_bytes(good[:-7])
    with pytest.raises(ValueError, match="length"):
        qx.load(str(path), device="cpu")
    path.write_bytes(b"XXXX" + good[4:])
    with pytest.raises(ValueError, match="magic"):
        qx.load(str(path), device="cpu")
    bad = bytearray(good)
    bad[24:28] = (3).to_bytes(4, "little")  # bits 4 -> 3: the sizes no longer match the recipe
    path.write_bytes(bytes(bad))
    with pytest.raises(ValueError, match="sizes"):
        qx.load(str(path), device="cpu")
    path.write_bytes(good[:40])
    with pytest.raises(ValueError, match="truncated"):
        qx.load(str(path), device="cpu")


@pytest.mark.gpu
def test_device_round_trip_decodes_identically(qx, cuda_dev, tmp_path):
    W = synth.student_t_weights(256, 1024, 0.02, seed=5, stream=79)
    Wd = torch.from_numpy(W).cuda()
    x = torch.from_numpy(synth.activations(4, 1024, seed=5, stream=80)).cuda()
    P = qx.quantize(Wd, qx.Recipe(3, 128, qx.LUT))
    qx.save(str(tmp_path / "l.qx"), P)
    Q = qx.load(str(tmp_path / "l.qx"))
    assert Q.codes.is_cuda and torch.equal(qx.gemv(P, x), qx.gemv(Q, x))
    P4 = qx.q4x_quantize(Wd)
    qx.save(str(tmp_path / "q.qx"), P4)
    Q4 = qx.load(str(tmp_path / "q.qx"))
    assert torch.equal(qx.q4x_gemv(P4, x), qx.q4x_gemv(Q4, x))
    assert qx.device_status() == 0
