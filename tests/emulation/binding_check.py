"""The Python binding (paper_2505_07531_gb300/qx.py) driven against the host
build of the library (tests/emulation) under AddressSanitizer and UBSan: the
wrappers the GPU tests call, with host tensors standing in for device tensors
(256-byte aligned, as the device allocator's blocks are); results against the
oracle, or against the separate calls a combined call replaces.  Run by
tests/test_emulated_api.py in a child process that preloads the sanitizer
runtimes:  python binding_check.py LIB
Exits non-zero (an assertion, or the sanitizer) on the first problem."""
from __future__ import annotations

import ctypes
import math
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import torch  # noqa: E402

import oracle  # noqa: E402
import synth  # noqa: E402
from oracle import select as oselect  # noqa: E402
from oracle.pack import Recipe as ORecipe  # noqa: E402
import paper_2505_07531_gb300.qx as qx  # noqa: E402

qx._LIB_PATH = sys.argv[1]
_HOST = set()  # data pointers of the tensors that stand for host memory


def _aligned(shape, dtype, zero=False):
    shape = tuple(int(s) for s in shape)
    nbytes = math.prod(shape) * torch.empty((), dtype=dtype).element_size()
    base = torch.zeros(nbytes + 256, dtype=torch.uint8) if zero else torch.empty(nbytes + 256, dtype=torch.uint8)
    off = (-base.data_ptr()) % 256
    return base[off:off + nbytes].view(dtype).view(shape)


def _shape(size):
    return tuple(size[0]) if len(size) == 1 and isinstance(size[0], (tuple, list, torch.Size)) else size


class _HostTorch:
    """The torch module, whose empty/zeros give aligned host tensors whatever
    device they are asked for."""

    def __getattr__(self, name):
        return getattr(torch, name)

    @staticmethod
    def empty(*size, dtype=torch.float32, device=None, **kw):
        return _aligned(_shape(size), dtype)

    @staticmethod
    def zeros(*size, dtype=torch.float32, device=None, **kw):
        return _aligned(_shape(size), dtype, zero=True)


qx.torch = _HostTorch()
qx._stream = lambda dev: ctypes.c_void_p(None)
qx._on_device = lambda t: t.data_ptr() not in _HOST


def dev(a):
    """An aligned "device" tensor holding numpy array a."""
    t = _aligned(a.shape, {np.float16: torch.float16, np.float32: torch.float32}[a.dtype.type])
    t.copy_(torch.from_numpy(np.ascontiguousarray(a)))
    return t


def host(shape, dtype):
    t = _aligned(shape, dtype)
    _HOST.add(t.data_ptr())
    return t


def bits(t):
    return t.numpy().view(np.uint16)


def check_q4x(n, k, iters):
    W = synth.student_t_weights(n, k, 0.02, seed=3, stream=n + k, outlier_frac=0.001).astype(np.float16)
    P = qx.q4x_quantize(dev(W), iters)
    assert qx.device_status() == 0
    ref = oracle.quantize_q4x(W, iters=iters)
    want = oracle.pack_q4x(ref)
    got = P.to_numpy()
    for key in ("codes", "scales", "books", "codebooks"):
        assert np.array_equal(np.ascontiguousarray(got[key]).view(np.uint8).ravel(),
                              np.ascontiguousarray(want[key]).view(np.uint8).ravel()), key
    Wh = oracle.dequant_q4x(ref["codes"], ref["scales"], ref["books"], ref["codebooks"])
    assert np.array_equal(bits(qx.q4x_dequant(P)), Wh.view(np.uint16))
    # decode: one matrix, then two in one launch (each row's sum is the same)
    x = synth.activations(3, k, seed=1, stream=k)
    y = qx.q4x_gemv(P, dev(x), out_dtype=torch.float32).numpy()
    assert np.all(oracle.max_abs_err(y, oracle.gemv_q4x(ref, x)) <= oracle.tolerance(x, Wh))
    x2 = synth.activations(3, k, seed=2, stream=k)
    ya, yb = qx.q4x_gemv_multi([P, P], [dev(x), dev(x2)])
    assert np.array_equal(bits(ya), bits(qx.q4x_gemv(P, dev(x))))
    assert np.array_equal(bits(yb), bits(qx.q4x_gemv(P, dev(x2))))
    # prefill on the (emulated) tensor cores, one CTA per tile and k split
    X = synth.activations(5, k, seed=5, stream=k)
    y_ref = oracle.gemv_q4x(ref, X)
    tol = oracle.tolerance(X, Wh) + np.abs(y_ref).max(axis=1) * 2.0 ** -11
    Y = qx.q4x_gemm(P, dev(X)).numpy().astype(np.float64)
    assert np.all(oracle.max_abs_err(Y, y_ref) <= tol)
    need = ctypes.c_size_t(0)
    assert qx._lib().qx_q4x_gemm_splitk_workspace(n, k, 5, ctypes.byref(need)) == 0
    ws = _aligned((max(int(need.value), 256),), torch.uint8, zero=True)
    Ys = qx.q4x_gemm_splitk(P, dev(X), workspace=ws).numpy().astype(np.float64)
    assert np.all(oracle.max_abs_err(Ys, y_ref) <= tol)
    assert qx.device_status() == 0


def check_select():
    W = synth.student_t_weights(32, 256, 0.02, seed=8, stream=9, outlier_frac=0.001).astype(np.float16)
    cands = [qx.Recipe(4, 64, qx.UNIFORM), qx.Recipe(4, 64, qx.Q4X, 2), qx.Recipe(3, 128, qx.LUT, 3)]
    orecs = [ORecipe(4, 64, "uniform"), ORecipe(4, 64, oselect.Q4X, 2), ORecipe(3, 128, "lut", 3)]
    for budget in (None,):  # budgets: tests/emulation/api_check.py
        got = qx.select_recipe(dev(W), cands, budget)
        want = oselect.select_recipe(W, orecs, budget)
        assert got[0] == want[0] and got[1] == [None if e is None else int(e) for e in want[1]], budget
        assert got[2] == want[2]


def check_chain_and_step():
    rec = qx.Recipe(3, 128, qx.LUT, 3)
    shapes = {"q": (64, 256), "k": (32, 256), "down": (48, 512)}
    mats = {nm: qx.quantize(dev(synth.student_t_weights(n, k, 0.02, seed=i, stream=n).astype(np.float16)), rec)
            for i, (nm, (n, k)) in enumerate(shapes.items())}
    batch = 2
    xa = dev(synth.activations(batch, 256, seed=1, stream=1))
    xd = dev(synth.activations(batch, 512, seed=2, stream=2))
    groups = [(["q", "k"], xa), (["down"], xd)]
    sep = {}
    for names, x in groups:
        for nm, y in zip(names, qx.gemv_multi([mats[nm] for nm in names], [x] * len(names))):
            sep[nm] = y
    ys = {nm: qx.torch.zeros((batch, P.n), dtype=torch.float16) for nm, P in mats.items()}
    qx.GemvChain([([mats[nm] for nm in names], [x] * len(names), [ys[nm] for nm in names])
                  for names, x in groups])()
    for nm in mats:
        assert np.array_equal(bits(ys[nm]), bits(sep[nm])), nm
    # the step with its copies: host x in, the q projection, host y out
    hx = host(xa.shape, torch.float16)
    hx.copy_(xa)
    xs = qx.torch.zeros(xa.shape, dtype=torch.float16)
    yd = qx.torch.zeros((batch, 64), dtype=torch.float16)
    hy = host(yd.shape, torch.float16)
    step = qx.DecodeStep([([mats["q"]], [xs], [yd])], h2d=[(xs, hx)], d2h=[(hy, yd)])
    step()
    assert torch.equal(xs, xa) and np.array_equal(bits(hy), bits(sep["q"]))
    try:  # a pair in the wrong direction is refused before any call
        qx.DecodeStep([([mats["q"]], [xs], [ys["q"]])], h2d=[(hx, xs)])
        raise AssertionError("wrong-direction copy accepted")
    except ValueError:
        pass
    assert qx.device_status() == 0


def check_stacked():
    """q, k, v stacked along n: the same packed rows and, per 128-row tile, the
    same prefill outputs bit for bit."""
    r = qx.Recipe(4, 128, qx.UNIFORM)
    k, m = 256, 20
    Ws = [synth.student_t_weights(n, k, 0.02, seed=7, stream=i).astype(np.float16)
          for i, n in enumerate((256, 128, 128))]
    parts = [qx.quantize(dev(W), r) for W in Ws]
    S = qx.quantize(dev(np.vstack(Ws)), r)
    for key in ("codes", "scales", "zeros"):
        assert torch.equal(getattr(S, key).view(torch.uint8),
                           torch.cat([getattr(P, key).view(torch.uint8) for P in parts])), key
    X = dev(synth.activations(m, k, seed=3, stream=m))
    Y = qx.gemm(S, X)
    Yp = torch.cat([qx.gemm(P, X) for P in parts], dim=1)
    assert torch.equal(Y.view(torch.int16), Yp.view(torch.int16))
    assert qx.device_status() == 0


def check_a8_prefill():
    """W.A8 prefill: int8 codes and scales for more tokens than a decode batch,
    x_hat bit-exact, and the matmul on x_hat within tolerance, for per-group
    and Q4X weights."""
    k, m = 256, 37
    x = synth.activations(m, k, seed=11, stream=12)
    x[4] = 0  # a dead token
    q, s = qx.quantize_act(dev(x))
    qr, sr = oracle.quantize_act(x)
    assert np.array_equal(q.numpy(), qr) and np.array_equal(s.numpy().view(np.uint32), sr.view(np.uint32))
    xh = qx.dequant_act(q, s)
    xr = oracle.dequant_act_f16(qr, sr)
    assert np.array_equal(bits(xh), xr.view(np.uint16))
    W = synth.student_t_weights(72, k, 0.02, seed=13, stream=14).astype(np.float16)
    for rec, orec in [((4, 128, qx.UNIFORM), ORecipe(4, 128, "uniform")), ((3, 128, qx.LUT, 3), ORecipe(3, 128, "lut", 3))]:
        P = qx.quantize(dev(W), qx.Recipe(*rec))
        Wh = oracle.dequant(oracle.quantize(W, orec), orec, k)
        y_ref = oracle.gemm_a8(Wh, x)
        tol = oracle.tolerance(xr, Wh) + np.abs(y_ref).max(axis=1) * 2.0 ** -11
        Y = qx.gemm_a8(P, dev(x)).numpy().astype(np.float64)
        assert np.all(oracle.max_abs_err(Y, y_ref) <= tol), rec
    P4 = qx.q4x_quantize(dev(W), 2)
    ref = oracle.quantize_q4x(W, iters=2)
    Wh = oracle.dequant_q4x(ref["codes"], ref["scales"], ref["books"], ref["codebooks"])
    y_ref = oracle.gemm_a8(Wh, x)
    Y = qx.gemm_a8(P4, dev(x)).numpy().astype(np.float64)
    assert np.all(oracle.max_abs_err(Y, y_ref) <= oracle.tolerance(xr, Wh) + np.abs(y_ref).max(axis=1) * 2.0 ** -11)
    assert qx.device_status() == 0


def main():
    check_a8_prefill()
    check_q4x(37, 384, 2)
    check_select()
    check_chain_and_step()
    check_stacked()
    print("binding ok")


if __name__ == "__main__":
    main()
