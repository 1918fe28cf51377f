"""A decode step as one library call (qx_gemv_chain, bound once by GemvChain):
bit-identical to the separate qx_gemv_multi calls it replaces."""
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def qx(cuda_dev):
    import paper_2505_07531_gb300.qx as qx

    qx._lib()
    return qx


@pytest.mark.parametrize("batch", [1, 4, 9])
def test_chain_equals_the_separate_calls(qx, batch):
    rec = qx.Recipe(3, 128, qx.LUT)
    shapes = {"q": (256, 512), "k": (128, 512), "o": (512, 512), "down": (512, 1024)}
    mats = {nm: qx.quantize(torch.from_numpy(synth.student_t_weights(n, k, 0.02, seed=i, stream=n)).cuda(), rec)
            for i, (nm, (n, k)) in enumerate(shapes.items())}
    xa = torch.from_numpy(synth.activations(batch, 512, seed=1, stream=1)).cuda()
    xd = torch.from_numpy(synth.activations(batch, 1024, seed=2, stream=2)).cuda()
    groups = [(["q", "k"], xa), (["o"], xa), (["down"], xd)]
    ys = {nm: torch.full((batch, P.n), float("nan"), device="cuda") for nm, P in mats.items()}
    chain = qx.GemvChain([([mats[nm] for nm in names], [x] * len(names), [ys[nm] for nm in names])
                          for names, x in groups])
    chain()
    for names, x in groups:
        sep = qx.gemv_multi([mats[nm] for nm in names], [x] * len(names), out_dtype=torch.float32, pdl=True)
        for nm, y in zip(names, sep):
            assert torch.equal(ys[nm], y), nm
    assert qx.device_status() == 0


@pytest.mark.parametrize("fused", [False, True])
def test_decode_step_copies_in_and_out(qx, fused):
    """qx_decode_step (qx_decode_step_fused): pinned host x in, the groups, host
    y out, synchronized: the host outputs equal the device results of the
    separate calls."""
    rec = qx.Recipe(4, 128, qx.UNIFORM)
    mats = [qx.quantize(torch.from_numpy(synth.student_t_weights(n, 512, 0.02, seed=n, stream=1)).cuda(), rec)
            for n in (256, 384)]
    hx = torch.from_numpy(synth.activations(2, 512, seed=3, stream=3)).pin_memory()
    dx = torch.empty(hx.shape, dtype=hx.dtype, device="cuda")
    dys = [torch.empty((2, P.n), dtype=torch.float16, device="cuda") for P in mats]
    hys = [torch.full((2, P.n), float("nan"), dtype=torch.float16).pin_memory() for P in mats]
    step = qx.DecodeStep([(mats, [dx, dx], dys)], h2d=[(dx, hx)], d2h=list(zip(hys, dys)), fused=fused)
    # the step is captured as a graph on its first call and replayed after: every
    # call copies the host buffers' current contents in and the results out
    for seed in (3, 4, 5):
        hx.copy_(torch.from_numpy(synth.activations(2, 512, seed=seed, stream=3)))
        for h in hys:
            h.fill_(float("nan"))
        step()
        ref = qx.gemv_multi(mats, [hx.cuda(), hx.cuda()])
        for h, r in zip(hys, ref):
            assert torch.equal(h, r.cpu()), seed
    assert qx.device_status() == 0


def test_decode_step_copies_of_any_alignment(qx):
    """Pinned host buffers are copied by the library's copy kernel: two copies
    each way, a host x starting 2 bytes past a 16-byte boundary, a y of 400
    bytes and a host y at an odd element offset; the host outputs equal the
    separate calls, call after call."""
    rec = qx.Recipe(4, 128, qx.UNIFORM)
    mats = [qx.quantize(torch.from_numpy(synth.student_t_weights(n, 512, 0.02, seed=n, stream=4)).cuda(), rec)
            for n in (200, 384)]
    hbuf = torch.empty(1 + 512, dtype=torch.float16).pin_memory()
    hx = hbuf[1:].view(1, 512)  # 2 bytes past the pinned buffer's start
    hx2 = torch.empty((1, 512), dtype=torch.float16).pin_memory()
    dx = torch.empty((1, 512), dtype=torch.float16, device="cuda")
    dx2 = torch.empty((1, 512), dtype=torch.float16, device="cuda")
    dys = [torch.empty((1, P.n), dtype=torch.float16, device="cuda") for P in mats]
    ybuf = torch.empty(1 + 200, dtype=torch.float16).pin_memory()
    hys = [ybuf[1:].view(1, 200), torch.empty((1, 384), dtype=torch.float16).pin_memory()]
    step = qx.DecodeStep([(mats, [dx, dx2], dys)], h2d=[(dx, hx), (dx2, hx2)], d2h=list(zip(hys, dys)))
    for seed in (7, 8, 9):
        hx.copy_(torch.from_numpy(synth.activations(1, 512, seed=seed, stream=1)))
        hx2.copy_(torch.from_numpy(synth.activations(1, 512, seed=seed, stream=2)))
        for h in hys:
            h.fill_(float("nan"))
        step()
        ref = qx.gemv_multi(mats, [hx.cuda(), hx2.cuda()])
        for h, r in zip(hys, ref):
            assert torch.equal(h, r.cpu()), seed
    assert qx.device_status() == 0


def test_decode_step_with_pageable_host_memory(qx):
    """Host buffers that are not pinned: the step is issued call by call (a
    graph's copy nodes take pinned memory), with the same results."""
    rec = qx.Recipe(3, 128, qx.LUT)
    P = qx.quantize(torch.from_numpy(synth.student_t_weights(256, 512, 0.02, seed=1, stream=2)).cuda(), rec)
    hx = torch.from_numpy(synth.activations(1, 512, seed=6, stream=3))
    dx = torch.empty(hx.shape, dtype=hx.dtype, device="cuda")
    dy = torch.empty((1, 256), dtype=torch.float16, device="cuda")
    hy = torch.full((1, 256), float("nan"), dtype=torch.float16)
    step = qx.DecodeStep([([P], [dx], [dy])], h2d=[(dx, hx)], d2h=[(hy, dy)])
    for _ in range(2):
        step()
        assert torch.equal(hy, qx.gemv(P, hx.cuda()).cpu())
    assert qx.device_status() == 0


@pytest.mark.parametrize("bits,g,kind", [(3, 128, 1), (4, 64, 0)])
@pytest.mark.parametrize("batch", [1, 2, 5, 16])
def test_fused_launch_equals_the_chain(qx, bits, g, kind, batch):
    """qx_gemv_fused: the groups of a chain in one persistent launch, its CTAs
    balanced slice by slice (blocks split between CTAs summed through the
    workspace): bit for bit the same as the balanced launches one group at a
    time (QX_GEMV_SEPARATE), and within fp32 summation order (fp16 outputs:
    one rounding) of the chain, whose CTAs take whole blocks.  With fp16
    outputs the third group reads the first group's output as its x, which the
    launch may read only once every CTA has finished the first group (the
    outputs start as NaN, so an early read shows).  Three calls in a row share
    one workspace: each launch leaves its counters zero for the next."""
    rec = qx.Recipe(bits, g, kind)
    shapes = {"q": (256, 512), "k": (96, 512), "up": (1000, 512), "o": (512, 256), "down": (384, 1024)}
    mats = {nm: qx.quantize(torch.from_numpy(synth.student_t_weights(n, k, 0.02, seed=i, stream=n)).cuda(), rec)
            for i, (nm, (n, k)) in enumerate(shapes.items())}
    xa = torch.from_numpy(synth.activations(batch, 512, seed=1, stream=1)).cuda()
    xd = torch.from_numpy(synth.activations(batch, 1024, seed=2, stream=2)).cuda()
    for dt in (torch.float16, torch.float32):
        ys = {nm: torch.empty((batch, P.n), dtype=dt, device="cuda") for nm, P in mats.items()}
        yss = {nm: torch.empty((batch, P.n), dtype=dt, device="cuda") for nm, P in mats.items()}
        handoff = dt == torch.float16
        xo_ref = torch.from_numpy(synth.activations(batch, 256, seed=3, stream=3)).cuda()

        def groups_for(out):
            xo = out["q"] if handoff else xo_ref
            return [(["q", "k"], [xa, xa]), (["up"], [xa]), (["o"], [xo]), (["down"], [xd])]

        def chain(out, **kw):
            return qx.GemvChain([([mats[nm] for nm in names], xs, [out[nm] for nm in names])
                                 for names, xs in groups_for(out)], **kw)

        fused, separate = chain(ys, fused=True), chain(yss, separate=True)
        for rep in range(3):
            for y in list(ys.values()) + list(yss.values()):
                y.fill_(float("nan"))
            fused()
            separate()
            ref = {}
            for names, xs in groups_for(ys):
                xs_ref = [ref["q"] if handoff and x is ys["q"] else x for x in xs]
                ref.update(zip(names, qx.gemv_multi([mats[nm] for nm in names], xs_ref, out_dtype=dt, pdl=True)))
            for nm in mats:
                assert torch.equal(ys[nm], yss[nm]), (nm, rep)
                r = ref[nm].float()
                tol = 4e-5 * r.abs().amax(dim=1, keepdim=True) + (r.abs() * 2.0 ** -10 if handoff else 0.0)
                assert torch.all((ys[nm].float() - r).abs() <= tol), (nm, rep)
        assert qx.device_status() == 0
