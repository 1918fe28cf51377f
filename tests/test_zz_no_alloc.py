"""qx_gemm_splitk_noalloc: the split-k tensor-core matmul with the library's
static scratch in place of a caller workspace.  Same results as the oracle
(and bit-identical to qx_gemm_splitk, which runs the same plan), no device
memory allocated by the calls, and a refusal when the plan needs more scratch
than the library holds.  Collected last (its name), so that the rest of the
suite runs first."""

import numpy as np
import pytest
import torch

import oracle
import synth
from oracle.pack import Recipe as ORecipe


def test_noalloc_rejects_bad_arguments_before_launching():
    """Host validation refuses a null struct, m = 0 and a misaligned X before
    any launch.  The calls run in a child process that sees no CUDA device, so
    that the placeholder addresses below can never reach a kernel: were the
    validation ever to let one through, the call would fail in the CUDA
    runtime (QX_ERR_CUDA = 4), not launch."""
    import os
    import subprocess
    import sys

    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    code = (
        "import ctypes, paper_2505_07531_gb300.qx as qx\n"
        "lib = qx._lib(); A = ctypes.c_void_p\n"
        "P = qx._Packed(64, 128, qx._Recipe(4, 64, 0, 0), A(0x1000), A(0x2000), A(0x3000), None)\n"
        "print(lib.qx_gemm_splitk_noalloc(None, None, 1, None, None),\n"
        "      lib.qx_gemm_splitk_noalloc(ctypes.byref(P), A(0x4000), 0, A(0x5000), None),\n"
        "      lib.qx_gemm_splitk_noalloc(ctypes.byref(P), A(0x4008), 1, A(0x5000), None))\n")
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, cwd=root, env=env, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    assert r.stdout.split() == ["1", "1", "3"]  # QX_ERR_INVALID_ARG twice, then QX_ERR_ALIGNMENT


@pytest.fixture(scope="module")
def qx(cuda_dev):
    import paper_2505_07531_gb300.qx as qx

    qx._lib()
    return qx


def _orecipe(bits, g, kind):
    return ORecipe(bits, g, "lut" if kind else "uniform", 25)


@pytest.mark.gpu
@pytest.mark.parametrize("bits,g,kind", [(3, 128, 1), (4, 64, 0)])
def test_noalloc_matches_oracle_and_workspace_path(qx, bits, g, kind):
    n, k = 1000, 4096  # 8 ragged W tiles, k split across CTAs
    rec = _orecipe(bits, g, kind)
    W = synth.student_t_weights(n, k, 0.02, seed=900 + bits, stream=g)
    ref = oracle.quantize(W, rec)
    Wh = oracle.dequant(ref, rec, k)
    P = qx.quantize(torch.from_numpy(W).cuda(), qx.Recipe(bits, g, kind))
    for m in (1, 5, 16, 40):
        assert m > 16 or qx.gemm_splitk_workspace_bytes(n, k, m, P.recipe) > 0
        X = synth.activations(m, k, seed=m, stream=91)
        Xd = torch.from_numpy(X).cuda()
        Y = qx.gemm_splitk_noalloc(P, Xd)
        Y2 = qx.gemm_splitk_noalloc(P, Xd)
        Yw = qx.gemm_splitk(P, Xd)
        assert qx.device_status() == 0
        assert torch.equal(Y, Y2) and torch.equal(Y, Yw)
        err = oracle.max_abs_err(Y.cpu().numpy(), oracle.gemm(ref, rec, X, k))
        assert np.all(err <= oracle.tolerance(X, Wh)), err


@pytest.mark.gpu
def test_noalloc_allocates_nothing(qx):
    n, k, m = 4096, 4096, 16
    P = qx.quantize(synth.student_t_weights_torch(n, k, 0.02, seed=3, stream=3, device="cuda"),
                    qx.Recipe(3, 128, 1))
    X = synth.activations_torch(m, k, seed=3, stream=4, device="cuda")
    Y = torch.empty((m, n), dtype=torch.float16, device="cuda")
    qx.gemm_splitk_noalloc(P, X, out=Y)  # first call: module and symbol lookup
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for _ in range(20):
        qx.gemm_splitk_noalloc(P, X, out=Y)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert qx.device_status() == 0
    assert free1 == free0


@pytest.mark.gpu
def test_noalloc_refuses_plans_larger_than_its_scratch(qx):
    # 21632 x 1920 at m = 1 splits into 507 units: 4.2 MB of workspace > 4 MiB
    n, k = 21632, 1920
    rec = qx.Recipe(4, 128, 0)
    assert qx.gemm_splitk_workspace_bytes(n, k, 1, rec) > 4 << 20
    P = qx.PackedMatrix.empty(n, k, rec, torch.device("cuda"))
    X = torch.zeros((1, k), dtype=torch.float16, device="cuda")
    with pytest.raises(qx.QxError) as e:
        qx.gemm_splitk_noalloc(P, X)
    assert e.value.code == 2
