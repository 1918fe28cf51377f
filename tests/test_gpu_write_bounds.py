"""Out-of-bounds writes, caught without a sanitizer: every output buffer of
every entry point sits between two 4 KiB guard bands of a known byte pattern,
on ragged shapes; after the call the bands must be untouched and the results
equal to those of the same call on plain buffers."""
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu

GUARD = 4096
CANARY = 0xA5


@pytest.fixture(scope="module")
def qx(cuda_dev):
    import paper_2505_07531_gb300.qx as qx

    qx._lib()
    return qx


class Guarded:
    """A device buffer of `nbytes` between two guard bands."""

    def __init__(self, nbytes, dtype=torch.uint8):
        self.nbytes = nbytes
        self.buf = torch.full((nbytes + 2 * GUARD,), CANARY, dtype=torch.uint8, device="cuda")
        self.t = self.buf[GUARD:GUARD + nbytes].view(dtype)

    def intact(self):
        bands = torch.cat([self.buf[:GUARD], self.buf[GUARD + self.nbytes:]])
        return bool((bands == CANARY).all())


def _g(nbytes, dtype=torch.uint8):
    return None if not nbytes else Guarded(nbytes, dtype)


def _packed_guarded(qx, n, k, rec):
    sz = qx.packed_size(n, k, rec)
    g = {"codes": _g(sz["codes"]), "scales": _g(sz["scales"], torch.float16),
         "zeros": _g(sz["zeros"]), "luts": _g(sz["luts"], torch.float16)}
    P = qx.PackedMatrix(n, k, rec, *[None if g[key] is None else g[key].t for key in ("codes", "scales", "zeros", "luts")])
    return P, [v for v in g.values() if v is not None]


@pytest.mark.parametrize("n,k,bits,gs,kind", [(37, 384, 4, 64, 0), (130, 640, 3, 128, 1), (33, 640, 3, 64, 0)])
def test_per_group_entry_points_stay_in_bounds(qx, n, k, bits, gs, kind):
    rec = qx.Recipe(bits, gs, kind)
    W = torch.from_numpy(synth.student_t_weights(n, k, 0.02, seed=n, stream=k)).cuda()
    P, bands = _packed_guarded(qx, n, k, rec)
    qx.quantize(W, rec, out=P)
    ref = qx.quantize(W, rec)
    for a, b in ((P.codes, ref.codes), (P.scales, ref.scales), (P.zeros, ref.zeros), (P.luts, ref.luts)):
        assert (a is None and b is None) or torch.equal(a.view(torch.uint8), b.view(torch.uint8))
    Wo = Guarded(2 * n * k, torch.float16)
    qx.dequant(P, out=Wo.t.view(n, k))
    assert torch.equal(Wo.t.view(n, k), qx.dequant(ref))
    bands.append(Wo)
    for batch in (1, 3, 9):
        x = torch.from_numpy(synth.activations(batch, k, seed=batch, stream=n)).cuda()
        y = Guarded(4 * batch * n, torch.float32)
        qx.gemv(P, x, out=y.t.view(batch, n))
        assert torch.equal(y.t.view(batch, n), qx.gemv(ref, x, out_dtype=torch.float32))
        bands.append(y)
    for m in (5, 17):
        X = torch.from_numpy(synth.activations(m, k, seed=m, stream=n)).cuda()
        Y = Guarded(2 * m * n, torch.float16)
        qx.gemm(P, X, out=Y.t.view(m, n))
        Ys = Guarded(2 * m * n, torch.float16)
        qx.gemm_splitk(P, X, out=Ys.t.view(m, n))
        assert torch.equal(Y.t.view(m, n), qx.gemm(ref, X))
        assert torch.equal(Ys.t.view(m, n), qx.gemm_splitk(ref, X))
        bands += [Y, Ys]
    if kind == 0:  # W.A8: int8 activations and their scales, then the integer-dot matmul
        batch = 3
        x = torch.from_numpy(synth.activations(batch, k, seed=7, stream=n)).cuda()
        q, s = Guarded(batch * k, torch.int8), Guarded(4 * batch, torch.float32)
        qx._check(qx._lib().qx_quantize_act(qx._ptr(x), batch, k, qx._ptr(q.t), qx._ptr(s.t),
                                            qx._stream(x.device)), "qx_quantize_act")
        q2, s2 = qx.quantize_act(x)
        assert torch.equal(q.t.view(batch, k), q2) and torch.equal(s.t, s2)
        y = Guarded(4 * batch * n, torch.float32)
        qx.gemv_a8(P, q.t.view(batch, k), s.t, out=y.t.view(batch, n))
        assert torch.equal(y.t.view(batch, n), qx.gemv_a8(ref, q2, s2, out_dtype=torch.float32))
        bands += [q, s, y]
        # W.A8 prefill: more tokens than a decode batch, then x_hat
        m = 20
        X = torch.from_numpy(synth.activations(m, k, seed=8, stream=n)).cuda()
        q, s, xh = Guarded(m * k, torch.int8), Guarded(4 * m, torch.float32), Guarded(2 * m * k, torch.float16)
        qx._check(qx._lib().qx_quantize_act(qx._ptr(X), m, k, qx._ptr(q.t), qx._ptr(s.t),
                                            qx._stream(X.device)), "qx_quantize_act")
        qx.dequant_act(q.t.view(m, k), s.t, out=xh.t.view(m, k))
        q2, s2 = qx.quantize_act(X)
        assert torch.equal(xh.t.view(m, k), qx.dequant_act(q2, s2))
        bands += [q, s, xh]
    assert qx.device_status() == 0
    assert all(b.intact() for b in bands)


def test_q4x_entry_points_stay_in_bounds(qx):
    n, k = 37, 320
    W = torch.from_numpy(synth.student_t_weights(n, k, 0.02, seed=1, stream=2)).cuda()
    sz = qx.q4x_size(n, k)
    g = [Guarded(sz["codes"]), Guarded(sz["scales"], torch.float16), Guarded(sz["books"]),
         Guarded(sz["codebooks"], torch.float16)]
    P = qx.Q4xMatrix(n, k, *[b.t for b in g])
    qx.q4x_quantize(W, out=P)
    ref = qx.q4x_quantize(W)
    for a, b in ((P.codes, ref.codes), (P.scales, ref.scales), (P.books, ref.books), (P.codebooks, ref.codebooks)):
        assert torch.equal(a.view(torch.uint8), b.view(torch.uint8))
    Wo = Guarded(2 * n * k, torch.float16)
    qx.q4x_dequant(P, out=Wo.t.view(n, k))
    assert torch.equal(Wo.t.view(n, k), qx.q4x_dequant(ref))
    g.append(Wo)
    mats = [P, ref, P]
    for batch in (1, 5, 16):
        xs = [torch.from_numpy(synth.activations(batch, k, seed=batch, stream=i)).cuda() for i in range(3)]
        ys = [Guarded(4 * batch * n, torch.float32) for _ in mats]
        qx.q4x_gemv_multi(mats, xs, outs=[y.t.view(batch, n) for y in ys])
        for x, y in zip(xs, ys):
            assert torch.equal(y.t.view(batch, n), qx.q4x_gemv(ref, x, out_dtype=torch.float32))
        g += ys
    assert qx.device_status() == 0
    assert all(b.intact() for b in g)
