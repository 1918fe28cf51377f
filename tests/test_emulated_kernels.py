"""Every kernel source of the library runs on host threads, compiled with
AddressSanitizer and UBSan (a stand-in for compute-sanitizer): the quantizers,
dequantizers, the exact-error reduction, the W.A8 pair, the Q4X path, the
TMA-pipelined decode GEMV and the tcgen05 matmul (its mbarriers, tensor copies,
tensor memory and MMAs are emulated with the hardware's rules checked).  Every index must stay
inside buffers of exactly the sizes the C ABI states, and the results must
equal the oracle's (bit-exact codes, LUTs, dequantized weights, exact squared
errors and int8 activations; matmuls within the tolerance).  No GPU; the
library never loads this code (tests/emulation/cuda_host.h)."""
import os
import shutil
import subprocess
import sys

import numpy as np
import pytest

import oracle
import synth
from oracle import select as oselect
from oracle.pack import Recipe as ORecipe

HERE = os.path.join(os.path.dirname(os.path.abspath(__file__)), "emulation")
ENV = dict(os.environ, ASAN_OPTIONS="detect_leaks=0", UBSAN_OPTIONS="print_stacktrace=1")


@pytest.fixture(scope="module")
def harness(emulation_dir):
    gxx = shutil.which("g++")
    if gxx is None:
        pytest.skip("g++ is not available")
    out = emulation_dir
    sys.path.insert(0, HERE)
    import translate

    exe = translate.build(gxx, str(out), "harness")
    return exe, out


def _run(harness, args, W, x=None):
    exe, out = harness
    fin, fout = str(out / "in.bin"), str(out / "out.bin")
    with open(fin, "wb") as f:
        f.write(np.ascontiguousarray(W, np.float16).tobytes())
        if x is not None:
            f.write(np.ascontiguousarray(x, np.float16).tobytes())
    r = subprocess.run([exe, *map(str, args), fin, fout], capture_output=True, text=True, env=ENV, timeout=900)
    assert r.returncode == 0 and "runtime error" not in r.stderr and "AddressSanitizer" not in r.stderr, \
        r.stderr[-3000:]
    return Reader(open(fout, "rb").read())


class Reader:
    def __init__(self, b):
        self.b, self.off = b, 0

    def take(self, count, dtype):
        a = np.frombuffer(self.b, dtype=dtype, count=count, offset=self.off)
        self.off += a.nbytes
        return a


def _weights(n, k, seed, dead_row=True):
    W = synth.student_t_weights(n, k, 0.02, seed=seed, stream=n + k, outlier_frac=0.001)
    if dead_row and n >= 3:
        W[1, :64] = 0
    return W


@pytest.mark.parametrize("n,k,bits,g,kind,sms", [  # ragged rows, every group size, 1 and 5 SMs of grid
    (1, 128, 4, 64, 0, 1), (37, 384, 4, 128, 0, 5), (130, 640, 3, 64, 0, 1), (130, 640, 3, 64, 0, 5),
    (3, 128, 3, 32, 0, 5), (9, 512, 4, 256, 0, 1), (20, 512, 3, 128, 1, 5), (11, 384, 3, 32, 1, 1),
    (3, 512, 3, 256, 1, 5), (1, 11008, 3, 128, 1, 1)])
def test_quantize_dequant_and_exact_error(harness, n, k, bits, g, kind, sms):
    W = _weights(n, k, seed=n + bits)
    rd = _run(harness, ["quant", n, k, bits, g, kind, 25, sms], W)
    rec = ORecipe(bits, g, "lut" if kind else "uniform", 25)
    ref = oracle.quantize(W, rec)
    G = k // g
    assert np.array_equal(rd.take(n * k * bits // 8, np.uint8).reshape(n, -1), ref["codes"])
    if kind == 0:
        assert np.array_equal(rd.take(n * G, np.uint16).reshape(n, G), ref["scales"].view(np.uint16))
        assert np.array_equal(rd.take(n * ((G + 1) // 2), np.uint8).reshape(n, -1), ref["zeros"])
    else:
        assert np.array_equal(rd.take(n * G * 8, np.uint16).reshape(n, G, 8), ref["luts"].view(np.uint16))
    Wh = oracle.dequant(ref, rec, k)
    assert np.array_equal(rd.take(n * k, np.uint16).reshape(n, k), Wh.view(np.uint16))
    tot = rd.take(2, np.uint64)
    assert int(tot[0]) | (int(tot[1]) << 64) == oselect.sq_error_units(W, Wh)
    assert rd.take(1, np.uint32)[0] == 0


@pytest.mark.parametrize("batch", [1, 3, 16])
@pytest.mark.parametrize("n,k,bits,g", [(37, 384, 4, 128), (33, 640, 3, 64), (1, 128, 3, 32)])
def test_int8_activations_and_w_a8_matmul(harness, n, k, bits, g, batch):
    W = _weights(n, k, seed=n + batch)
    x = synth.activations(batch, k, seed=batch, stream=n)
    rd = _run(harness, ["a8", n, k, bits, g, batch, 3], W, x)
    G = k // g
    rd.take(n * k * bits // 8 + 2 * n * G + n * ((G + 1) // 2), np.uint8)
    qr, sr = oracle.quantize_act(x)
    assert np.array_equal(rd.take(batch * k, np.int8).reshape(batch, k), qr)
    assert np.array_equal(rd.take(batch, np.float32), sr)
    y = rd.take(batch * n, np.float32).reshape(batch, n)
    rec = ORecipe(bits, g, "uniform", 25)
    ref = oracle.quantize(W, rec)
    qw = oracle.unpack_codes(ref["codes"], bits, k).astype(np.float64)
    z = np.repeat(oracle.unpack_zeros(ref["zeros"], G).astype(np.float64), g, axis=1)
    w_exact = (qw - z) * np.repeat(ref["scales"].astype(np.float64), g, axis=1)
    tol = oracle.tolerance(oracle.dequant_act(qr, sr), w_exact)
    assert np.all(oracle.max_abs_err(y, oracle.gemv_a8(ref, rec, x, k)) <= tol)


@pytest.mark.parametrize("n,k,bits,g,kind,batch,sms,split", [  # 1..16 rows of x, ragged row blocks
    (37, 384, 4, 64, 0, 1, 2, 0), (130, 640, 3, 64, 0, 4, 3, 0), (33, 256, 4, 32, 0, 8, 2, 0),
    (20, 512, 3, 128, 1, 3, 2, 0), (5, 4096, 4, 128, 0, 2, 4, 1), (70, 1152, 3, 128, 0, 1, 3, 0),
    (40, 512, 3, 128, 1, 16, 2, 0), (33, 384, 4, 64, 0, 11, 2, 0), (24, 768, 3, 32, 1, 5, 2, 0),
    # the balanced plan: blocks split between two CTAs (1), or kept whole
    # because a block would get three CTAs or no CTA would get fewer stages (0)
    (5, 4096, 4, 128, 0, 2, 3, 1), (5, 4096, 3, 128, 1, 1, 8, 0), (130, 2048, 3, 64, 0, 4, 3, 1),
    (40, 3072, 3, 128, 1, 9, 5, 0)])
def test_tma_pipelined_decode_gemv(harness, n, k, bits, g, kind, batch, sms, split):
    """qx_gemv's kernel and host plan (tensor maps, byte-balanced CTA slices):
    one matrix, the same matrix twice in one launch (with PDL set), and twice
    more the pair with the CTAs balanced stage by stage (row blocks split
    between CTAs through the workspace): within tolerance, the balanced
    launches deterministic, their flags back at zero."""
    W = _weights(n, k, seed=n + g)
    x = synth.activations(batch, k, seed=batch, stream=n)
    rd = _run(harness, ["gemv", n, k, bits, g, kind, batch, sms], W, x)
    G = k // g
    rd.take(n * k * bits // 8 + (2 * n * G + n * ((G + 1) // 2) if kind == 0 else 2 * n * G * 8), np.uint8)
    ys = [rd.take(batch * n, np.float32).reshape(batch, n) for _ in range(7)]
    assert rd.take(1, np.int32)[0] == split
    assert rd.take(1, np.uint32)[0] == 0  # every split flag back at zero
    assert rd.take(1, np.uint32)[0] == 0  # no bounded wait gave up
    rec = ORecipe(bits, g, "lut" if kind else "uniform", 25)
    ref = oracle.quantize(W, rec)
    y_ref = oracle.gemv(ref, rec, x, k)
    tol = oracle.tolerance(x, oracle.dequant(ref, rec, k))
    for y in ys:
        assert np.all(oracle.max_abs_err(y, y_ref) <= tol)
    assert np.array_equal(ys[0], ys[1]) and np.array_equal(ys[1], ys[2])
    assert np.array_equal(ys[3], ys[5]) and np.array_equal(ys[4], ys[6])


@pytest.mark.parametrize("n,k,bits,g,kind,m,sms", [  # 16-, 64- and 256-token tiles, 1..4 k splits
    (37, 384, 4, 64, 0, 5, 2), (128, 2048, 4, 128, 0, 16, 4), (200, 1024, 3, 64, 0, 40, 4),
    (64, 1152, 4, 32, 0, 1, 8), (130, 256, 4, 256, 0, 300, 2), (40, 256, 3, 128, 1, 3, 2),
    (128, 2048, 3, 128, 1, 40, 4)])  # 64-token tiles split four ways
def test_tensor_core_matmul(harness, n, k, bits, g, kind, m, sms):
    """qx_gemm (one CTA per tile), then qx_gemm_splitk twice on one workspace,
    the second with PDL: each within tolerance (fp16 output), and the split
    counters back to zero after every call."""
    W = _weights(n, k, seed=n + m)
    X = synth.activations(m, k, seed=m, stream=n)
    rd = _run(harness, ["gemm", n, k, bits, g, kind, m, sms], W, X)
    G = k // g
    rd.take(n * k * bits // 8 + (2 * n * G + n * ((G + 1) // 2) if kind == 0 else 2 * n * G * 8), np.uint8)
    rec = ORecipe(bits, g, "lut" if kind else "uniform", 25)
    ref = oracle.quantize(W, rec)
    y_ref = oracle.gemm(ref, rec, X, k)
    tol = oracle.tolerance(X, oracle.dequant(ref, rec, k)) + np.abs(y_ref).max(axis=1) * 2.0 ** -11
    for _ in range(3):
        Y = rd.take(m * n, np.float16).reshape(m, n).astype(np.float64)
        assert np.all(oracle.max_abs_err(Y, y_ref) <= tol)
        assert rd.take(1, np.uint32)[0] == 1  # counters rearmed
        rd.take(2, np.uint32)  # the plan: token tile, splits
    assert rd.take(1, np.uint32)[0] == 0


@pytest.mark.parametrize("n,k,iters,m,sms", [  # Q4X weights: a 4-way k split; a ragged 256-token prefill
    (128, 2048, 2, 16, 4), (64, 1152, 2, 300, 2)])
def test_q4x_tensor_core_matmul(harness, n, k, iters, m, sms):
    W = _weights(n, k, seed=n + m).astype(np.float16)
    X = synth.activations(m, k, seed=m, stream=n)
    rd = _run(harness, ["q4xgemm", n, k, iters, m, sms], np.concatenate([W.ravel(), X.astype(np.float16).ravel()]))
    ref = oracle.quantize_q4x(W, iters=iters)
    want = oracle.pack_q4x(ref)
    G, bb = k // 64, (k // 64 + 3) // 4
    assert np.array_equal(rd.take(n * k // 2, np.uint8).reshape(n, -1), want["codes"])
    assert np.array_equal(rd.take(n * G, np.uint16).reshape(n, G), want["scales"].view(np.uint16))
    assert np.array_equal(rd.take(n * bb, np.uint8).reshape(n, -1), want["books"])
    assert np.array_equal(rd.take(64, np.uint16).reshape(4, 16), want["codebooks"].view(np.uint16))
    y_ref = oracle.gemv_q4x(ref, X)
    Wh = oracle.dequant_q4x(ref["codes"], ref["scales"], ref["books"], ref["codebooks"])
    tol = oracle.tolerance(X, Wh) + np.abs(y_ref).max(axis=1) * 2.0 ** -11
    for _ in range(3):
        Y = rd.take(m * n, np.float16).reshape(m, n).astype(np.float64)
        assert np.all(oracle.max_abs_err(Y, y_ref) <= tol)
        assert rd.take(1, np.uint32)[0] == 1
        rd.take(2, np.uint32)
    assert rd.take(1, np.uint32)[0] == 0


def _q4x_cases():
    nan = _weights(24, 512, seed=9, dead_row=False).astype(np.float16)
    nan[4, 130] = np.float16(np.nan)
    nan[9, 0] = np.float16(np.inf)
    return {
        "ragged": (_weights(37, 320, seed=1), 3, 2, 3),
        "no_steps": (_weights(16, 128, seed=2), 0, 1, 1),
        "batch16": (_weights(130, 640, seed=3), 3, 5, 16),
        "all_zero": (np.zeros((8, 256), np.float16), 3, 2, 2),
        "few_distinct": (np.tile(np.array([-1, 0, 0.5, 1], np.float16), (8, 64)), 3, 2, 4),
        "nonfinite": (nan, 3, 2, 1),
        "three_slices": (_weights(40, 2176, seed=4), 3, 3, 2),
    }


Q4X = _q4x_cases()


@pytest.mark.parametrize("name", sorted(Q4X))
def test_q4x_learner_dequant_and_multi_matrix_decode(harness, name):
    W, iters, sms, batch = Q4X[name]
    W = np.asarray(W, np.float16)
    n, k = W.shape
    x = synth.activations(batch, k, seed=batch, stream=n)
    rd = _run(harness, ["q4x", n, k, iters, sms, batch], W, x)
    G, bb = k // 64, (k // 64 + 3) // 4
    got = {"codes": rd.take(n * k // 2, np.uint8).reshape(n, -1), "scales": rd.take(n * G, np.uint16).reshape(n, G),
           "books": rd.take(n * bb, np.uint8).reshape(n, -1), "codebooks": rd.take(64, np.uint16).reshape(4, 16)}
    bad = ~np.isfinite(W.reshape(n, G, 64).astype(np.float32)).all(axis=2)
    clean = W.copy()
    clean.reshape(n, G, 64)[bad] = 0  # a non-finite group is coded as a dead one
    ref = oracle.quantize_q4x(clean, iters=iters)
    want = oracle.pack_q4x(ref)
    assert np.array_equal(got["codes"], want["codes"])
    assert np.array_equal(got["scales"], want["scales"].view(np.uint16))
    assert np.array_equal(got["books"], want["books"])
    assert np.array_equal(got["codebooks"], want["codebooks"].view(np.uint16))
    Wh = oracle.dequant_q4x(ref["codes"], ref["scales"], ref["books"], ref["codebooks"])
    assert np.array_equal(rd.take(n * k, np.uint16).reshape(n, k), Wh.view(np.uint16))
    y0 = rd.take(batch * n, np.float32).reshape(batch, n)
    y1 = rd.take(batch * n, np.float32).reshape(batch, n)
    yh = rd.take(batch * n, np.float16).reshape(batch, n).astype(np.float64)
    # the register-dequant kernel (run when k is a multiple of 128)
    ring = rd.take(1, np.int32)[0] == 1
    assert ring == (k % 128 == 0)
    y2 = rd.take(batch * n, np.float32).reshape(batch, n)
    y3 = rd.take(batch * n, np.float32).reshape(batch, n)
    yh2 = rd.take(batch * n, np.float16).reshape(batch, n).astype(np.float64)
    assert np.array_equal(y0, y1)  # both entries of the two-matrix launch
    if ring:
        assert np.array_equal(y2, y3)
    if not bad.any():
        y_ref = oracle.gemv_q4x(ref, x)
        tol = oracle.tolerance(x, Wh)
        fp16_out = np.abs(y_ref).max(axis=1) * 2.0 ** -11
        assert np.all(oracle.max_abs_err(y0, y_ref) <= tol)
        assert np.all(oracle.max_abs_err(yh, y_ref) <= tol + fp16_out)
        if ring:
            assert np.all(oracle.max_abs_err(y2, y_ref) <= tol)
            assert np.all(oracle.max_abs_err(yh2, y_ref) <= tol + fp16_out)
    assert rd.take(1, np.uint32)[0] == (1 if bad.any() else 0)  # the non-finite status bit
