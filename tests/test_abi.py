"""The C-ABI library loads, exports every entry point include/qx.h declares, and its
host-only logic (sizes, validation, status strings) behaves; no GPU needed."""
import ctypes
import os
import re

import pytest

import oracle
from oracle.pack import Recipe as ORecipe

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def qx():
    from paper_2505_07531_gb300 import build

    if not os.path.exists(build.LIB):
        build.build_library()
    import paper_2505_07531_gb300.qx as qx

    return qx


def _declared():
    names = []
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            src = open(os.path.join(ROOT, "include", fn)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names += re.findall(r"\b(qx_[a-z0-9_]+)\s*\(", src)
    return sorted(set(names))


def test_every_declared_symbol_is_exported(qx):
    names = _declared()
    assert "qx_gemv" in names and "qx_gemm" in names and "qx_quantize" in names
    lib = ctypes.CDLL(qx.library_path())
    for n in names:
        assert hasattr(lib, n), n


@pytest.mark.parametrize("n,k,bits,g,kind", [
    (1, 128, 4, 64, 0), (37, 384, 4, 128, 0), (5, 4096, 3, 64, 0), (3, 11008, 3, 128, 1),
    (2, 256, 4, 32, 0), (4, 512, 3, 256, 1), (7, 640, 3, 32, 0)])
def test_packed_size_matches_oracle(qx, n, k, bits, g, kind):
    got = qx.packed_size(n, k, qx.Recipe(bits, g, kind))
    want = oracle.packed_sizes(n, k, ORecipe(bits, g, "lut" if kind else "uniform"))
    assert got == want


@pytest.mark.parametrize("n,k,recipe,code", [
    (0, 128, (4, 64, 0, 0), 1),      # n < 1
    (4, 100, (4, 64, 0, 0), 2),      # k not a multiple of 128
    (4, 192, (4, 128, 0, 0), 2),     # k not a multiple of g... and of 128
    (4, 128, (5, 64, 0, 0), 2),      # bits
    (4, 128, (4, 48, 0, 0), 2),      # group size
    (4, 128, (4, 64, 1, 25), 2),     # 4-bit LUT not built
    (4, 128, (3, 64, 7, 0), 1),      # kind
    (4, 128, (3, 64, 1, -1), 1),     # lloyd iterations
])
def test_packed_size_rejects(qx, n, k, recipe, code):
    lib = qx._lib()
    s = qx._Sizes()
    r = qx._Recipe(*recipe)
    assert lib.qx_packed_size(n, k, ctypes.byref(r), ctypes.byref(s)) == code


def test_entry_points_reject_bad_arguments_before_launching(qx):
    """Validation happens on the host: these calls return without touching a GPU."""
    lib = qx._lib()
    P = qx._Packed(64, 128, qx._Recipe(4, 64, 0, 0), None, None, None, None)
    assert lib.qx_gemv(ctypes.byref(P), None, 1, None, 0, None) == 1
    assert lib.qx_gemm(None, None, 1, None, None) == 1
    assert lib.qx_dequant(ctypes.byref(P), None, None) == 1
    # misaligned codes pointer
    P2 = qx._Packed(64, 128, qx._Recipe(4, 64, 0, 0), ctypes.c_void_p(0x1008), ctypes.c_void_p(0x2000),
                    ctypes.c_void_p(0x3000), None)
    assert lib.qx_dequant(ctypes.byref(P2), ctypes.c_void_p(0x4000), None) == 3
    # batch outside 1..16
    P3 = qx._Packed(64, 128, qx._Recipe(4, 64, 0, 0), ctypes.c_void_p(0x1000), ctypes.c_void_p(0x2000),
                    ctypes.c_void_p(0x3000), None)
    assert lib.qx_gemv(ctypes.byref(P3), ctypes.c_void_p(0x4000), 17, ctypes.c_void_p(0x5000), 0, None) == 2
    assert lib.qx_gemv(ctypes.byref(P3), ctypes.c_void_p(0x4000), 0, ctypes.c_void_p(0x5000), 0, None) == 1
    assert lib.qx_gemv(ctypes.byref(P3), ctypes.c_void_p(0x4008), 1, ctypes.c_void_p(0x5000), 0, None) == 3
    assert lib.qx_gemm(ctypes.byref(P3), ctypes.c_void_p(0x4000), 0, ctypes.c_void_p(0x5000), None) == 1
    # split-k matmul: the same argument checks, and the workspace query's own
    assert lib.qx_gemm_splitk(None, None, 1, None, None, 0, 0, None) == 1
    assert lib.qx_gemm_splitk(ctypes.byref(P3), ctypes.c_void_p(0x4000), 0, ctypes.c_void_p(0x5000), None, 0, 0,
                              None) == 1
    assert lib.qx_gemm_splitk(ctypes.byref(P3), ctypes.c_void_p(0x4008), 1, ctypes.c_void_p(0x5000), None, 0, 0,
                              None) == 3
    assert lib.qx_gemm_splitk(ctypes.byref(P3), ctypes.c_void_p(0x4000), 1, ctypes.c_void_p(0x5000), None, 0, 2,
                              None) == 1  # unknown flag
    nbytes = ctypes.c_size_t(0)
    r = qx._Recipe(3, 128, 1, 0)
    assert lib.qx_gemm_splitk_workspace(4096, 4096, 1, ctypes.byref(r), None) == 1
    assert lib.qx_gemm_splitk_workspace(4096, 4096, 0, ctypes.byref(r), ctypes.byref(nbytes)) == 1
    assert lib.qx_gemm_splitk_workspace(4096, 4000, 1, ctypes.byref(r), ctypes.byref(nbytes)) == 2
    assert lib.qx_gemm_splitk_workspace(4096, 4096, 1, None, ctypes.byref(nbytes)) == 1
    # W.A8: activation and matmul argument checks
    assert lib.qx_quantize_act(None, 1, 128, None, None, None) == 1
    assert lib.qx_quantize_act(ctypes.c_void_p(0x4000), 0, 128, ctypes.c_void_p(0x5000), ctypes.c_void_p(0x6000),
                               None) == 1
    assert lib.qx_quantize_act(ctypes.c_void_p(0x4000), (1 << 24) + 1, 128, ctypes.c_void_p(0x5000),
                               ctypes.c_void_p(0x6000), None) == 2  # up to 2^24 tokens
    # W.A8 prefill activations: pointers, sizes, alignment
    A, S, X = ctypes.c_void_p(0x4000), ctypes.c_void_p(0x5000), ctypes.c_void_p(0x6000)
    assert lib.qx_dequant_act(None, S, 4, 128, X, None) == 1
    assert lib.qx_dequant_act(A, S, 0, 128, X, None) == 1
    assert lib.qx_dequant_act(A, S, 4, 120, X, None) == 2
    assert lib.qx_dequant_act(A, S, (1 << 24) + 1, 128, X, None) == 2
    assert lib.qx_dequant_act(ctypes.c_void_p(0x4008), S, 4, 128, X, None) == 3
    assert lib.qx_dequant_act(A, ctypes.c_void_p(0x5002), 4, 128, X, None) == 3
    assert lib.qx_dequant_act(A, S, 4, 128, ctypes.c_void_p(0x6008), None) == 3
    assert lib.qx_quantize_act(ctypes.c_void_p(0x4000), 1, 120, ctypes.c_void_p(0x5000), ctypes.c_void_p(0x6000),
                               None) == 2
    assert lib.qx_quantize_act(ctypes.c_void_p(0x4000), 1, 128, ctypes.c_void_p(0x5008), ctypes.c_void_p(0x6000),
                               None) == 3
    PL = qx._Packed(64, 128, qx._Recipe(3, 64, 1, 0), ctypes.c_void_p(0x1000), None, None, ctypes.c_void_p(0x2000))
    assert lib.qx_gemv_a8(ctypes.byref(PL), ctypes.c_void_p(0x4000), ctypes.c_void_p(0x5000), 1,
                          ctypes.c_void_p(0x6000), 0, None) == 2  # LUT weights: no integer form
    assert lib.qx_gemv_a8(ctypes.byref(P3), ctypes.c_void_p(0x4008), ctypes.c_void_p(0x5000), 1,
                          ctypes.c_void_p(0x6000), 0, None) == 3
    # recipe selection: candidate list and shape checks come first
    cands = (qx._Recipe * 2)(qx._Recipe(3, 64, 0, 0), qx._Recipe(4, 64, 0, 0))
    assert lib.qx_select_workspace(64, 256, cands, 0, ctypes.byref(nbytes)) == 1
    assert lib.qx_select_workspace(64, 256, cands, 17, ctypes.byref(nbytes)) == 1
    assert lib.qx_select_workspace(64, 200, cands, 2, ctypes.byref(nbytes)) == 2
    bad = (qx._Recipe * 1)(qx._Recipe(4, 64, 1, 0))  # 4-bit LUT is not built
    assert lib.qx_select_workspace(64, 256, bad, 1, ctypes.byref(nbytes)) == 2
    # Q4X: a selection candidate only, with bits 4, groups of 64, 0..1000 steps
    q4 = qx._Recipe(4, 64, qx.Q4X, 0)
    assert lib.qx_packed_size(64, 256, ctypes.byref(q4), ctypes.byref(qx._Sizes())) == 1
    for r, code in [((3, 64, qx.Q4X, 0), 2), ((4, 128, qx.Q4X, 0), 2), ((4, 64, qx.Q4X, 1001), 1),
                    ((4, 64, qx.Q4X, -1), 1), ((4, 64, 3, 0), 1)]:
        one = (qx._Recipe * 1)(qx._Recipe(*r))
        assert lib.qx_select_workspace(64, 256, one, 1, ctypes.byref(nbytes)) == code, r
    assert lib.qx_select_workspace(64, 224, (qx._Recipe * 1)(q4), 1, ctypes.byref(nbytes)) == 2  # k % 64
    ch, err, bpw = ctypes.c_int32(0), (ctypes.c_uint64 * 4)(), (ctypes.c_double * 2)()
    assert lib.qx_select_recipe(None, 64, 256, cands, 2, 0.0, None, 0, ctypes.byref(ch), err, bpw, None) == 1
    assert lib.qx_select_recipe(ctypes.c_void_p(0x4008), 64, 256, cands, 2, 0.0, None, 0, ctypes.byref(ch), err, bpw,
                                None) == 3


def test_status_strings_and_version(qx):
    lib = qx._lib()
    for code in range(7):
        assert len(lib.qx_status_string(code)) > 0
    assert lib.qx_version() >= 100


@pytest.mark.parametrize("n,k", [(1, 64), (37, 320), (64, 512), (4096, 4096), (11008, 4096), (4096, 11008)])
def test_q4x_size_matches_oracle(qx, n, k):
    assert qx.q4x_size(n, k) == oracle.q4x_sizes(n, k)


def test_q4x_shape_limits_and_workspace(qx):
    lib = qx._lib()
    s = qx._Q4xSizes()
    nbytes = ctypes.c_size_t(0)
    assert lib.qx_q4x_size(0, 64, ctypes.byref(s)) == 1
    assert lib.qx_q4x_size(4, 100, ctypes.byref(s)) == 2            # k not a multiple of 64
    assert lib.qx_q4x_size(4, 64, None) == 1
    assert lib.qx_q4x_size(1 << 19, 4096, ctypes.byref(s)) == 0     # n k = 2^31: the limit
    assert lib.qx_q4x_size((1 << 19) + 1, 4096, ctypes.byref(s)) == 2
    assert lib.qx_q4x_workspace(4, 64, None) == 1
    assert lib.qx_q4x_workspace(4, 100, ctypes.byref(nbytes)) == 2
    # per-group histograms, sums and assignments grow with the groups; the
    # value histograms of the four books are a fixed 42 MB
    a, b = qx.q4x_workspace_bytes(64, 4096), qx.q4x_workspace_bytes(4096, 4096)
    assert 4 * (2 ** 21 + 1) * 5 < a < b
    assert b - a >= (4096 - 64) * 64 * 42 - 1024


def test_q4x_entry_points_reject_bad_arguments_before_launching(qx):
    lib = qx._lib()
    A = ctypes.c_void_p
    good = qx._Q4x(64, 512, A(0x10000), A(0x20000), A(0x30000), A(0x40000))
    ws = A(0x100000)
    big = 1 << 40
    assert lib.qx_q4x_quantize(None, 25, ctypes.byref(good), ws, big, None) == 1
    assert lib.qx_q4x_quantize(A(0x1000), 25, None, ws, big, None) == 1
    nul = qx._Q4x(64, 512, A(0x10000), None, A(0x30000), A(0x40000))
    assert lib.qx_q4x_quantize(A(0x1000), 25, ctypes.byref(nul), ws, big, None) == 1
    assert lib.qx_q4x_quantize(A(0x1000), -1, ctypes.byref(good), ws, big, None) == 1
    assert lib.qx_q4x_quantize(A(0x1000), 1001, ctypes.byref(good), ws, big, None) == 1
    assert lib.qx_q4x_quantize(A(0x1000), 25, ctypes.byref(good), ws, 1024, None) == 1  # workspace too small
    assert lib.qx_q4x_quantize(A(0x1000), 25, ctypes.byref(good), None, big, None) == 1
    assert lib.qx_q4x_quantize(A(0x1008), 25, ctypes.byref(good), ws, big, None) == 3   # W alignment
    assert lib.qx_q4x_quantize(A(0x1000), 25, ctypes.byref(good), A(0x100080), big, None) == 3
    mis = qx._Q4x(64, 512, A(0x10008), A(0x20000), A(0x30000), A(0x40000))
    assert lib.qx_q4x_quantize(A(0x1000), 25, ctypes.byref(mis), ws, big, None) == 3
    odd = qx._Q4x(64, 500, A(0x10000), A(0x20000), A(0x30000), A(0x40000))
    assert lib.qx_q4x_quantize(A(0x1000), 25, ctypes.byref(odd), ws, big, None) == 2
    assert lib.qx_q4x_dequant(ctypes.byref(good), None, None) == 1
    assert lib.qx_q4x_dequant(ctypes.byref(good), A(0x5008), None) == 3
    assert lib.qx_q4x_dequant(ctypes.byref(mis), A(0x5000), None) == 3
    assert lib.qx_q4x_gemv(ctypes.byref(good), A(0x5000), 0, A(0x6000), 0, None) == 1
    assert lib.qx_q4x_gemv(ctypes.byref(good), A(0x5000), 17, A(0x6000), 0, None) == 2
    assert lib.qx_q4x_gemv(ctypes.byref(good), A(0x5000), 1, A(0x6000), 2, None) == 1   # y dtype
    assert lib.qx_q4x_gemv(ctypes.byref(good), A(0x5008), 1, A(0x6000), 0, None) == 3
    assert lib.qx_q4x_gemv(ctypes.byref(good), A(0x5000), 1, A(0x6002), 0, None) == 3
    assert lib.qx_q4x_gemv(ctypes.byref(good), None, 1, A(0x6000), 0, None) == 1


def test_q4x_gemv_multi_rejects_bad_arguments_before_launching(qx):
    lib = qx._lib()
    A = ctypes.c_void_p
    mats = (qx._Q4x * 2)(qx._Q4x(64, 512, A(0x10000), A(0x20000), A(0x30000), A(0x40000)),
                         qx._Q4x(32, 256, A(0x50000), A(0x60000), A(0x70000), A(0x80000)))
    xs = (A * 2)(A(0x1000), A(0x2000))
    ys = (A * 2)(A(0x3000), A(0x4000))
    assert lib.qx_q4x_gemv_multi(None, 1, xs, 1, ys, 0, None) == 1
    assert lib.qx_q4x_gemv_multi(mats, 0, xs, 1, ys, 0, None) == 1
    assert lib.qx_q4x_gemv_multi(mats, 9, xs, 1, ys, 0, None) == 1
    assert lib.qx_q4x_gemv_multi(mats, 2, None, 1, ys, 0, None) == 1
    assert lib.qx_q4x_gemv_multi(mats, 2, xs, 0, ys, 0, None) == 1
    assert lib.qx_q4x_gemv_multi(mats, 2, xs, 17, ys, 0, None) == 2
    assert lib.qx_q4x_gemv_multi(mats, 2, xs, 1, ys, 3, None) == 1
    bad_x = (A * 2)(A(0x1000), A(0x2008))
    assert lib.qx_q4x_gemv_multi(mats, 2, bad_x, 1, ys, 0, None) == 3
    nul_y = (A * 2)(A(0x3000), None)
    assert lib.qx_q4x_gemv_multi(mats, 2, xs, 1, nul_y, 0, None) == 1
    odd = (qx._Q4x * 2)(mats[0], qx._Q4x(32, 200, A(0x50000), A(0x60000), A(0x70000), A(0x80000)))
    assert lib.qx_q4x_gemv_multi(odd, 2, xs, 1, ys, 0, None) == 2


def test_cuda_errors_are_reported_with_their_name():
    """With no visible device, an entry point that passes validation fails in
    the CUDA runtime: QX_ERR_CUDA, and qx_last_error_string() names the error."""
    import subprocess
    import sys

    code = (
        "import ctypes, paper_2505_07531_gb300.qx as qx\n"
        "lib = qx._lib(); A = ctypes.c_void_p\n"
        "P = qx._Packed(64, 128, qx._Recipe(4, 64, 0, 0), A(0x10000), A(0x20000), A(0x30000), None)\n"
        "print(lib.qx_dequant(ctypes.byref(P), A(0x40000), None), lib.qx_last_error_string().decode())\n"
        "print(lib.qx_get_device_status(None), lib.qx_last_error_string().decode())\n"
        "print(lib.qx_selftest_wait_timeout(0, None), lib.qx_selftest_wait_timeout(2000000, None))\n")
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, cwd=ROOT, env=env, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = r.stdout.split("\n")
    for line in lines[:2]:
        status, name = line.split(" ", 1)
        assert status == "4" and name.startswith("cuda") and name != "cudaSuccess", line
    assert lines[2] == "1 1"  # limit outside 1 us .. 1 s


def test_q4x_gemm_rejects_bad_arguments_before_launching(qx):
    lib = qx._lib()
    A = ctypes.c_void_p
    good = qx._Q4x(64, 512, A(0x10000), A(0x20000), A(0x30000), A(0x40000))
    assert lib.qx_q4x_gemm(None, A(0x1000), 4, A(0x2000), None) == 1
    assert lib.qx_q4x_gemm(ctypes.byref(good), None, 4, A(0x2000), None) == 1
    assert lib.qx_q4x_gemm(ctypes.byref(good), A(0x1000), 0, A(0x2000), None) == 1
    assert lib.qx_q4x_gemm(ctypes.byref(good), A(0x1008), 4, A(0x2000), None) == 3
    assert lib.qx_q4x_gemm(ctypes.byref(good), A(0x1000), 4, A(0x2001), None) == 3
    k64 = qx._Q4x(64, 320, A(0x10000), A(0x20000), A(0x30000), A(0x40000))  # k not a multiple of 128
    assert lib.qx_q4x_gemm(ctypes.byref(k64), A(0x1000), 4, A(0x2000), None) == 2
    assert lib.qx_q4x_gemm_splitk(ctypes.byref(good), A(0x1000), 4, A(0x2000), None, 0, 2, None) == 1  # flag
    assert lib.qx_q4x_gemm_splitk(ctypes.byref(k64), A(0x1000), 4, A(0x2000), None, 0, 0, None) == 2
    nbytes = ctypes.c_size_t(0)
    assert lib.qx_q4x_gemm_splitk_workspace(64, 320, 4, ctypes.byref(nbytes)) == 2
    assert lib.qx_q4x_gemm_splitk_workspace(64, 512, 0, ctypes.byref(nbytes)) == 1
    assert lib.qx_q4x_gemm_splitk_workspace(64, 512, 4, None) == 1


def test_gemv_chain_rejects_bad_arguments_before_launching(qx):
    lib = qx._lib()
    A = ctypes.c_void_p
    P3 = qx._Packed(64, 128, qx._Recipe(4, 64, 0, 0), A(0x1000), A(0x2000), A(0x3000), None)
    mats = (qx._Packed * 1)(P3)
    xs, ys = (A * 1)(A(0x4000)), (A * 1)(A(0x5000))
    VPA = ctypes.POINTER(ctypes.c_void_p)
    g = qx._GemvGroup(ctypes.cast(mats, ctypes.POINTER(qx._Packed)), 1, ctypes.cast(xs, VPA), ctypes.cast(ys, VPA))
    assert lib.qx_gemv_chain(None, 1, 1, 0, 0, None) == 1
    assert lib.qx_gemv_chain((qx._GemvGroup * 1)(g), 0, 1, 0, 0, None) == 1
    assert lib.qx_gemv_chain((qx._GemvGroup * 1)(g), 65, 1, 0, 0, None) == 1
    assert lib.qx_gemv_chain((qx._GemvGroup * 1)(g), 1, 17, 0, 0, None) == 2   # batch
    assert lib.qx_gemv_chain((qx._GemvGroup * 1)(g), 1, 1, 0, 2, None) == 1    # unknown flag
    bad = qx._GemvGroup(ctypes.cast(mats, ctypes.POINTER(qx._Packed)), 0, ctypes.cast(xs, VPA), ctypes.cast(ys, VPA))
    assert lib.qx_gemv_chain((qx._GemvGroup * 2)(g, bad), 2, 1, 0, 0, None) == 1  # count 0 in the second group


def test_decode_step_rejects_bad_arguments_before_launching(qx):
    lib = qx._lib()
    A = ctypes.c_void_p
    P3 = qx._Packed(64, 128, qx._Recipe(4, 64, 0, 0), A(0x1000), A(0x2000), A(0x3000), None)
    mats = (qx._Packed * 1)(P3)
    xs, ys = (A * 1)(A(0x4000)), (A * 1)(A(0x5000))
    VPA = ctypes.POINTER(ctypes.c_void_p)
    g = (qx._GemvGroup * 1)(qx._GemvGroup(ctypes.cast(mats, ctypes.POINTER(qx._Packed)), 1, ctypes.cast(xs, VPA),
                                          ctypes.cast(ys, VPA)))
    c = (qx._Copy * 1)(qx._Copy(0x4000, 0x9000, 256))
    nul = (qx._Copy * 1)(qx._Copy(0x4000, None, 256))
    assert lib.qx_decode_step(c, 17, g, 1, 1, 0, 0, c, 1, 1, None) == 1
    assert lib.qx_decode_step(c, 1, g, 1, 1, 0, 0, c, -1, 1, None) == 1
    assert lib.qx_decode_step(None, 1, g, 1, 1, 0, 0, None, 0, 1, None) == 1
    assert lib.qx_decode_step(nul, 1, g, 1, 1, 0, 0, None, 0, 1, None) == 1
    assert lib.qx_decode_step(c, 1, None, 1, 1, 0, 0, None, 0, 1, None) == 1
    assert lib.qx_decode_step(c, 1, g, 1, 17, 0, 0, None, 0, 1, None) == 2
