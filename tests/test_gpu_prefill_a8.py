"""GPU parity of the W.A8 prefill (Tables 1-2: 8-bit per-token RTN
activations): int8 codes and scales for prefill-sized token counts and their
fp16 form x_hat = fp16(fp32(s_b q)) bit-exact with the CPU oracle; the
tensor-core matmul on x_hat within
max_n |y - y_ref| <= 2e-3 * ||x_hat_b||_2 * max_n ||w_hat_n||_2 (+ the fp16
rounding of the output) for every token b."""
import numpy as np
import pytest
import torch

import oracle
import synth
from oracle.pack import Recipe as ORecipe

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def qx(cuda_dev):
    import paper_2505_07531_gb300.qx as qx

    qx._lib()
    return qx


def _check(Y, W_hat, x):
    y_ref = oracle.gemm_a8(W_hat, x)
    q, s = oracle.quantize_act(x)
    tol = oracle.tolerance(oracle.dequant_act_f16(q, s), W_hat) + np.abs(y_ref).max(axis=1) * 2.0 ** -11
    assert np.all(oracle.max_abs_err(Y.cpu().numpy().astype(np.float64), y_ref) <= tol)


@pytest.mark.parametrize("m,k", [(17, 128), (576, 1024), (2048, 4096)])
def test_activation_codes_and_x_hat_bit_exact(qx, m, k):
    x = synth.activations(m, k, seed=m, stream=k)
    x[1] = 0  # a dead token
    q, s = qx.quantize_act(torch.from_numpy(x).cuda())
    qr, sr = oracle.quantize_act(x)
    assert np.array_equal(q.cpu().numpy(), qr)
    assert np.array_equal(s.cpu().numpy().view(np.uint32), sr.view(np.uint32))
    xh = qx.dequant_act(q, s)
    assert np.array_equal(xh.cpu().numpy().view(np.uint16), oracle.dequant_act_f16(qr, sr).view(np.uint16))
    assert qx.device_status() == 0


@pytest.mark.parametrize("bits,g,kind,m", [(4, 128, 0, 576), (3, 64, 0, 300), (3, 128, 1, 40)])
@pytest.mark.parametrize("splitk", [False, True])
def test_prefill_per_group_weights(qx, bits, g, kind, m, splitk):
    n, k = 384, 1024
    W = synth.student_t_weights(n, k, 0.02, seed=bits, stream=g).astype(np.float16)
    rec = ORecipe(bits, g, "lut" if kind else "uniform", 25)
    P = qx.quantize(torch.from_numpy(W).cuda(), qx.Recipe(bits, g, kind))
    x = synth.activations(m, k, seed=3, stream=m)
    Y = qx.gemm_a8(P, torch.from_numpy(x).cuda(), splitk=splitk)
    assert qx.device_status() == 0
    _check(Y, oracle.dequant(oracle.quantize(W, rec), rec, k), x)


def test_prefill_q4x_weights(qx):
    n, k, m = 256, 512, 200
    W = synth.student_t_weights(n, k, 0.02, seed=5, stream=6).astype(np.float16)
    P = qx.q4x_quantize(torch.from_numpy(W).cuda(), 6)
    ref = oracle.quantize_q4x(W, iters=6)
    W_hat = oracle.dequant_q4x(ref["codes"], ref["scales"], ref["books"], ref["codebooks"])
    x = synth.activations(m, k, seed=7, stream=8)
    for splitk in (False, True):
        Y = qx.gemm_a8(P, torch.from_numpy(x).cuda(), splitk=splitk)
        assert qx.device_status() == 0
        _check(Y, W_hat, x)
