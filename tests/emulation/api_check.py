"""Every C-ABI entry point of the library, built for the host from the kernel
and API sources (tests/emulation) with AddressSanitizer and UBSan, called the
way a user calls it, on buffers of exactly the sizes the header states;
results against the oracle.  Run by tests/test_emulated_api.py in a child
process that preloads the sanitizer runtimes:  python api_check.py LIB
Exits non-zero (an assertion, or the sanitizer) on the first problem."""
from __future__ import annotations

import ctypes
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
import synth  # noqa: E402
from oracle.pack import Recipe as ORecipe  # noqa: E402
from oracle import select as oselect  # noqa: E402
import paper_2505_07531_gb300.qx as qx  # noqa: E402  (its ctypes declarations only)

qx._LIB_PATH = sys.argv[1]
L = qx._lib()
_libc = ctypes.CDLL(None)
_libc.posix_memalign.argtypes = [ctypes.POINTER(ctypes.c_void_p), ctypes.c_size_t, ctypes.c_size_t]
_keep = []


def buf(nbytes, dtype=np.uint8, fill=None):
    """A host buffer of exactly `nbytes` (256-byte aligned) as a numpy array."""
    p = ctypes.c_void_p()
    assert _libc.posix_memalign(ctypes.byref(p), 256, max(int(nbytes), 1)) == 0
    a = np.ctypeslib.as_array((ctypes.c_uint8 * int(nbytes)).from_address(p.value)).view(dtype)
    if fill is not None:
        a[...] = fill
    _keep.append(a)
    return a


def put(arr):
    """An exact-size aligned copy of a numpy array."""
    arr = np.ascontiguousarray(arr)
    b = buf(arr.nbytes, arr.dtype)
    b[...] = arr.ravel()
    return b


def P(a):
    return ctypes.c_void_p(a.ctypes.data)


def ok(code, where):
    assert code == 0, f"{where}: status {code}"


def status():
    return L.qx_get_device_status(None)


def within(y, y_ref, tol, extra_f16=False):
    y = np.asarray(y, np.float64)
    t = tol + (np.abs(y_ref).max(axis=1) * 2.0 ** -11 if extra_f16 else 0.0)
    assert np.all(oracle.max_abs_err(y, y_ref) <= t), "outside tolerance"


def packed(n, k, rec):
    """Exact-size buffers of a packed matrix and its ctypes struct."""
    sz = qx._Sizes()
    r = rec.c()
    ok(L.qx_packed_size(n, k, ctypes.byref(r), ctypes.byref(sz)), "qx_packed_size")
    bufs = [buf(sz.codes), buf(sz.scales) if sz.scales else None, buf(sz.zeros) if sz.zeros else None,
            buf(sz.luts) if sz.luts else None]
    s = qx._Packed(n, k, r, *[None if b is None else P(b) for b in bufs])
    return s, bufs


def check_per_group(n, k, bits, g, kind):
    rec = qx.Recipe(bits, g, kind)
    orec = ORecipe(bits, g, "lut" if kind else "uniform", 25)
    W = synth.student_t_weights(n, k, 0.02, seed=n + k, stream=bits, outlier_frac=0.001)
    Wd = put(W)
    S, bufs = packed(n, k, rec)
    r = rec.c()
    ok(L.qx_quantize(P(Wd), n, k, ctypes.byref(r), ctypes.byref(S), None), "qx_quantize")
    ref = oracle.quantize(W, orec)
    assert np.array_equal(bufs[0].reshape(n, -1), ref["codes"]), "codes"
    if kind == 0:
        assert np.array_equal(bufs[1].view(np.uint16), ref["scales"].view(np.uint16).ravel()), "scales"
        assert np.array_equal(bufs[2], ref["zeros"].ravel()), "zeros"
    else:
        assert np.array_equal(bufs[3].view(np.uint16), ref["luts"].view(np.uint16).ravel()), "luts"
    Wh = oracle.dequant(ref, orec, k)
    out = buf(2 * n * k, np.float16)
    ok(L.qx_dequant(ctypes.byref(S), P(out), None), "qx_dequant")
    assert np.array_equal(out.view(np.uint16), Wh.view(np.uint16).ravel()), "dequant"
    # decode: every batch chunking (8 + 4 + 1 ...), fp32 and fp16 outputs
    for batch in (1, 3, 5, 9, 16):
        x = synth.activations(batch, k, seed=batch, stream=n)
        xd, y, yh = put(x), buf(4 * batch * n, np.float32), buf(2 * batch * n, np.float16)
        ok(L.qx_gemv(ctypes.byref(S), P(xd), batch, P(y), 1, None), "qx_gemv")
        ok(L.qx_gemv(ctypes.byref(S), P(xd), batch, P(yh), 0, None), "qx_gemv f16")
        y_ref = oracle.gemv(ref, orec, x, k)
        tol = oracle.tolerance(x, Wh)
        within(y.reshape(batch, n), y_ref, tol)
        within(yh.reshape(batch, n), y_ref, tol, extra_f16=True)
    # the same matrix three times in one launch, with PDL
    x = synth.activations(2, k, seed=7, stream=n)
    xd = put(x)
    mats = (qx._Packed * 3)(S, S, S)
    ys = [buf(8 * n, np.float32) for _ in range(3)]
    ok(L.qx_gemv_multi(mats, 3, (ctypes.c_void_p * 3)(*[P(xd)] * 3), 2,
                       (ctypes.c_void_p * 3)(*[P(v) for v in ys]), 1, 1, None), "qx_gemv_multi")
    for v in ys:
        within(v.reshape(2, n), oracle.gemv(ref, orec, x, k), oracle.tolerance(x, Wh))
    # a decode step as one call: groups (S, S) and (S), each equal to its qx_gemv_multi
    VPA = ctypes.POINTER(ctypes.c_void_p)

    def group(mlist, xs, ys_):
        c = len(mlist)
        pa, xa, ya = (qx._Packed * c)(*mlist), (ctypes.c_void_p * c)(*xs), (ctypes.c_void_p * c)(*ys_)
        _keep.extend([pa, xa, ya])
        return qx._GemvGroup(ctypes.cast(pa, ctypes.POINTER(qx._Packed)), c, ctypes.cast(xa, VPA),
                             ctypes.cast(ya, VPA))

    yc = [buf(8 * n, np.float32, fill=np.nan) for _ in range(3)]
    ok(L.qx_gemv_chain((qx._GemvGroup * 2)(group([S, S], [P(xd)] * 2, [P(yc[0]), P(yc[1])]),
                                           group([S], [P(xd)], [P(yc[2])])), 2, 2, 1, 1, None), "qx_gemv_chain")
    sep = [buf(8 * n, np.float32) for _ in range(3)]
    ok(L.qx_gemv_multi((qx._Packed * 2)(S, S), 2, (ctypes.c_void_p * 2)(P(xd), P(xd)), 2,
                       (ctypes.c_void_p * 2)(P(sep[0]), P(sep[1])), 1, 1, None), "multi (S, S)")
    ok(L.qx_gemv_multi((qx._Packed * 1)(S), 1, (ctypes.c_void_p * 1)(P(xd)), 2, (ctypes.c_void_p * 1)(P(sep[2])),
                       1, 1, None), "multi (S)")
    for a_, b_ in zip(yc, sep):
        assert np.array_equal(a_, b_), "chain equals the separate calls"
    untouched = buf(8 * n, np.float32, fill=np.nan)
    bad_y = buf(8 * n + 4, np.uint8)[2:]  # misaligned output of the second group
    assert L.qx_gemv_chain((qx._GemvGroup * 2)(group([S], [P(xd)], [P(untouched)]),
                                               group([S], [P(xd)], [ctypes.c_void_p(bad_y.ctypes.data)])),
                           2, 2, 1, 1, None) == 3, "misaligned y"
    assert np.isnan(untouched).all(), "nothing launched when a later group is invalid"
    # the whole step in one call: host x in, the groups, host y out, synchronize
    hx = put(x)
    dx = buf(x.nbytes, np.float16)
    dys = [buf(8 * n, np.float32) for _ in range(3)]
    hys = [buf(8 * n, np.float32, fill=np.nan) for _ in range(3)]
    cin = (qx._Copy * 1)(qx._Copy(dx.ctypes.data, hx.ctypes.data, x.nbytes))
    cout = (qx._Copy * 3)(*[qx._Copy(h.ctypes.data, d.ctypes.data, h.nbytes) for h, d in zip(hys, dys)])
    steps = (qx._GemvGroup * 2)(group([S, S], [P(dx)] * 2, [P(dys[0]), P(dys[1])]), group([S], [P(dx)], [P(dys[2])]))
    ok(L.qx_decode_step(cin, 1, steps, 2, 2, 1, 1, cout, 3, 1, None), "qx_decode_step")
    for a_, b_ in zip(hys, sep):
        assert np.array_equal(a_, b_), "decode step equals the separate calls"
    assert L.qx_decode_step(cin, 17, steps, 2, 2, 1, 1, cout, 3, 1, None) == 1, "too many copies"
    assert L.qx_decode_step(None, 1, steps, 2, 2, 1, 1, cout, 3, 1, None) == 1, "missing copy list"
    # prefill: one CTA per tile, split-k (twice on one workspace, the second with PDL), no-alloc
    for m in (3, 17, 200):
        X = synth.activations(m, k, seed=m, stream=n)
        Xd = put(X)
        y_ref = oracle.gemm(ref, orec, X, k)
        tol = oracle.tolerance(X, Wh)
        Y = buf(2 * m * n, np.float16)
        ok(L.qx_gemm(ctypes.byref(S), P(Xd), m, P(Y), None), "qx_gemm")
        within(Y.reshape(m, n), y_ref, tol, extra_f16=True)
        nb = ctypes.c_size_t(0)
        ok(L.qx_gemm_splitk_workspace(n, k, m, ctypes.byref(r), ctypes.byref(nb)), "workspace")
        ws = buf(max(nb.value, 256), fill=0)
        Ys = [buf(2 * m * n, np.float16) for _ in range(2)]
        for i, flags in enumerate((0, 1)):
            ok(L.qx_gemm_splitk(ctypes.byref(S), P(Xd), m, P(Ys[i]), P(ws), ws.nbytes, flags, None), "splitk")
            within(Ys[i].reshape(m, n), y_ref, tol, extra_f16=True)
            assert not ws[:65536].any(), "split counters not rearmed"
        assert np.array_equal(Ys[0], Ys[1]), "split-k repeat"
        Yn = buf(2 * m * n, np.float16)
        code = L.qx_gemm_splitk_noalloc(ctypes.byref(S), P(Xd), m, P(Yn), None)
        if nb.value <= 4 << 20:
            ok(code, "noalloc")
            assert np.array_equal(Yn, Ys[0]), "no-alloc equals the workspace call"
    if kind == 0:  # W.A8
        batch = 3
        x = synth.activations(batch, k, seed=11, stream=n)
        xd, q, s, y = put(x), buf(batch * k, np.int8), buf(4 * batch, np.float32), buf(4 * batch * n, np.float32)
        ok(L.qx_quantize_act(P(xd), batch, k, P(q), P(s), None), "qx_quantize_act")
        qr, sr = oracle.quantize_act(x)
        assert np.array_equal(q.reshape(batch, k), qr) and np.array_equal(s, sr), "int8 activations"
        ok(L.qx_gemv_a8(ctypes.byref(S), P(q), P(s), batch, P(y), 1, None), "qx_gemv_a8")
        qw = oracle.unpack_codes(ref["codes"], bits, k).astype(np.float64)
        z = np.repeat(oracle.unpack_zeros(ref["zeros"], k // g).astype(np.float64), g, axis=1)
        w_exact = (qw - z) * np.repeat(ref["scales"].astype(np.float64), g, axis=1)
        within(y.reshape(batch, n), oracle.gemv_a8(ref, orec, x, k), oracle.tolerance(oracle.dequant_act(qr, sr),
                                                                                      w_exact))
    # W.A8 prefill activations for more tokens than a decode batch, any weight format
    m = 19
    x = synth.activations(m, k, seed=12, stream=n)
    q, s, xh = buf(m * k, np.int8), buf(4 * m, np.float32), buf(2 * m * k, np.float16)
    ok(L.qx_quantize_act(P(put(x)), m, k, P(q), P(s), None), "qx_quantize_act (prefill)")
    ok(L.qx_dequant_act(P(q), P(s), m, k, P(xh), None), "qx_dequant_act")
    qr, sr = oracle.quantize_act(x)
    assert np.array_equal(q.reshape(m, k), qr) and np.array_equal(s, sr), "prefill int8 activations"
    assert np.array_equal(xh.view(np.uint16), oracle.dequant_act_f16(qr, sr).view(np.uint16).ravel()), "x_hat"
    assert status() == 0


def check_select(n, k):
    W = synth.student_t_weights(n, k, 0.02, seed=5, stream=6, outlier_frac=0.001)
    cands = [qx.Recipe(3, 64, qx.UNIFORM), qx.Recipe(3, 128, qx.LUT), qx.Recipe(4, 64, qx.UNIFORM),
             qx.Recipe(4, 128, qx.UNIFORM), qx.Recipe(4, 64, qx.Q4X, 4)]
    c = len(cands)
    arr = (qx._Recipe * c)(*[r.c() for r in cands])
    names = {qx.UNIFORM: "uniform", qx.LUT: "lut", qx.Q4X: oselect.Q4X}
    orecs = [ORecipe(r.bits, r.group_size, names[r.kind], r.lloyd_iters) for r in cands]
    Wd = put(W)
    for budget in (0.0, 4.3):
        nb = ctypes.c_size_t(0)
        ok(L.qx_select_workspace(n, k, arr, c, ctypes.byref(nb)), "qx_select_workspace")
        ws = buf(nb.value)
        chosen, err, bpw = ctypes.c_int32(-1), (ctypes.c_uint64 * (2 * c))(), (ctypes.c_double * c)()
        ok(L.qx_select_recipe(P(Wd), n, k, arr, c, budget, P(ws), ws.nbytes, ctypes.byref(chosen), err, bpw, None),
           "qx_select_recipe")
        want = oselect.select_recipe(W, orecs, max_bpw=budget or None)
        got_e = [None if err[2 * i] == err[2 * i + 1] == 2 ** 64 - 1 else err[2 * i] | (err[2 * i + 1] << 64)
                 for i in range(c)]
        assert chosen.value == (-1 if want[0] is None else want[0]), f"chosen {chosen.value} vs {want[0]}"
        assert got_e == [None if e is None else int(e) for e in want[1]], "exact errors"
        assert list(bpw) == list(want[2]), "bits per weight"
    # a Q4X candidate outside bits 4 / group 64 is not built
    bad = (qx._Recipe * 1)(qx._Recipe(4, 128, qx.Q4X, 4))
    assert L.qx_select_workspace(n, k, bad, 1, ctypes.byref(nb)) == 2
    assert status() == 0


def check_q4x(n, k, iters):
    W = synth.student_t_weights(n, k, 0.02, seed=n, stream=k, outlier_frac=0.001).astype(np.float16)
    sz = qx._Q4xSizes()
    ok(L.qx_q4x_size(n, k, ctypes.byref(sz)), "qx_q4x_size")
    codes, scales, books, cbs = buf(sz.codes), buf(sz.scales), buf(sz.books), buf(sz.codebooks)
    M = qx._Q4x(n, k, P(codes), P(scales), P(books), P(cbs))
    nb = ctypes.c_size_t(0)
    ok(L.qx_q4x_workspace(n, k, ctypes.byref(nb)), "qx_q4x_workspace")
    ws = buf(nb.value)
    ok(L.qx_q4x_quantize(P(put(W)), iters, ctypes.byref(M), P(ws), ws.nbytes, None), "qx_q4x_quantize")
    ref = oracle.quantize_q4x(W, iters=iters)
    want = oracle.pack_q4x(ref)
    assert np.array_equal(codes, want["codes"].ravel()), "q4x codes"
    assert np.array_equal(scales.view(np.uint16), want["scales"].view(np.uint16).ravel()), "q4x scales"
    assert np.array_equal(books, want["books"].ravel()), "q4x books"
    assert np.array_equal(cbs.view(np.uint16), want["codebooks"].view(np.uint16).ravel()), "q4x codebooks"
    Wh = oracle.dequant_q4x(ref["codes"], ref["scales"], ref["books"], ref["codebooks"])
    out = buf(2 * n * k, np.float16)
    ok(L.qx_q4x_dequant(ctypes.byref(M), P(out), None), "qx_q4x_dequant")
    assert np.array_equal(out.view(np.uint16), Wh.view(np.uint16).ravel()), "q4x dequant"
    for batch in (1, 5, 16):
        x = synth.activations(batch, k, seed=batch, stream=n)
        xd = put(x)
        y = buf(4 * batch * n, np.float32)
        ok(L.qx_q4x_gemv(ctypes.byref(M), P(xd), batch, P(y), 1, None), "qx_q4x_gemv")
        within(y.reshape(batch, n), oracle.gemv_q4x(ref, x), oracle.tolerance(x, Wh))
        ys = [buf(4 * batch * n, np.float32) for _ in range(2)]
        ok(L.qx_q4x_gemv_multi((qx._Q4x * 2)(M, M), 2, (ctypes.c_void_p * 2)(P(xd), P(xd)), batch,
                               (ctypes.c_void_p * 2)(*[P(v) for v in ys]), 1, None), "qx_q4x_gemv_multi")
        assert np.array_equal(ys[0], y) and np.array_equal(ys[1], y), "multi-matrix equals one matrix"
    if k % 128 == 0:
        for m in (5, 40):
            X = synth.activations(m, k, seed=m, stream=n)
            Xd = put(X)
            y_ref = oracle.gemv_q4x(ref, X)
            tol = oracle.tolerance(X, Wh)
            Y = buf(2 * m * n, np.float16)
            ok(L.qx_q4x_gemm(ctypes.byref(M), P(Xd), m, P(Y), None), "qx_q4x_gemm")
            within(Y.reshape(m, n), y_ref, tol, extra_f16=True)
            wb = ctypes.c_size_t(0)
            ok(L.qx_q4x_gemm_splitk_workspace(n, k, m, ctypes.byref(wb)), "q4x workspace")
            gws = buf(max(wb.value, 256), fill=0)
            Ys = buf(2 * m * n, np.float16)
            ok(L.qx_q4x_gemm_splitk(ctypes.byref(M), P(Xd), m, P(Ys), P(gws), gws.nbytes, 1, None), "q4x splitk")
            within(Ys.reshape(m, n), y_ref, tol, extra_f16=True)
            assert not gws[:65536].any(), "split counters not rearmed"
    else:
        X = put(synth.activations(2, k, seed=1, stream=n))
        assert L.qx_q4x_gemm(ctypes.byref(M), P(X), 2, P(buf(4 * n, np.float16)), None) == 2, "k % 128"
    assert status() == 0
    # a group holding NaN raises the non-finite status and is coded as dead
    bad = W.copy()
    bad[0, 3] = np.float16(np.nan)
    ok(L.qx_q4x_quantize(P(put(bad)), iters, ctypes.byref(M), P(ws), ws.nbytes, None), "qx_q4x_quantize NaN")
    assert status() == 6, "non-finite status"
    assert status() == 0, "status cleared"


def main():
    check_per_group(37, 384, 4, 64, 0)
    check_per_group(40, 256, 3, 128, 1)
    check_select(64, 512)
    check_q4x(37, 384, 2)
    print("api ok")


if __name__ == "__main__":
    main()
