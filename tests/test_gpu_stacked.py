"""A fused projection: matrices that read the same activations and share a
per-group recipe, stacked along n, quantize to their packed buffers stacked
row for row (every group lies within one row, Section 2.1), and the tensor-core
prefill of the stacked matrix equals the separate prefills column for column,
bit for bit (a 128-row W tile never straddles two of them)."""
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def qx(cuda_dev):
    import paper_2505_07531_gb300.qx as qx

    qx._lib()
    return qx


@pytest.mark.parametrize("rec,m", [((4, 128, 0), 576), ((3, 64, 0), 40), ((3, 128, 1), 300)])
def test_stacked_qkv_is_the_same_model(qx, rec, m):
    r = qx.Recipe(*rec, 6)
    k = 1024
    Ws = [torch.from_numpy(synth.student_t_weights(n, k, 0.02, seed=7, stream=i)).cuda()
          for i, n in enumerate((384, 128, 256))]
    parts = [qx.quantize(W, r) for W in Ws]
    S = qx.quantize(torch.cat(Ws), r)
    assert qx.device_status() == 0
    for key in ("codes", "scales", "zeros", "luts"):
        t = getattr(S, key)
        if t is None:
            continue
        assert torch.equal(t.view(torch.uint8), torch.cat([getattr(P, key).view(torch.uint8) for P in parts])), key
    X = torch.from_numpy(synth.activations(m, k, seed=3, stream=m)).cuda()
    Y = qx.gemm(S, X)
    Yp = torch.cat([qx.gemm(P, X) for P in parts], dim=1)
    assert qx.device_status() == 0
    assert torch.equal(Y.view(torch.int16), Yp.view(torch.int16))
