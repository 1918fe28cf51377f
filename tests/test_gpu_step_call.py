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


def test_decode_step_copies_in_and_out(qx):
    """qx_decode_step: pinned host x in, the groups, host y out, synchronized:
    the host outputs equal the device results of the separate calls."""
    rec = qx.Recipe(4, 128, qx.UNIFORM)
    mats = [qx.quantize(torch.from_numpy(synth.student_t_weights(n, 512, 0.02, seed=n, stream=1)).cuda(), rec)
            for n in (256, 384)]
    hx = torch.from_numpy(synth.activations(2, 512, seed=3, stream=3)).pin_memory()
    dx = torch.empty(hx.shape, dtype=hx.dtype, device="cuda")
    dys = [torch.empty((2, P.n), dtype=torch.float16, device="cuda") for P in mats]
    hys = [torch.full((2, P.n), float("nan"), dtype=torch.float16).pin_memory() for P in mats]
    step = qx.DecodeStep([(mats, [dx, dx], dys)], h2d=[(dx, hx)], d2h=list(zip(hys, dys)))
    step()
    ref = qx.gemv_multi(mats, [hx.cuda(), hx.cuda()])
    for h, r in zip(hys, ref):
        assert torch.equal(h, r.cpu())
    assert qx.device_status() == 0
