"""Failure detection without a GPU fault: a bounded wait that runs out records
QX_ERR_TIMEOUT in the device status word and returns; the context stays
usable (no trap, no hang, no fault)."""
import time

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


def test_bounded_wait_gives_up_and_reports_timeout(qx):
    qx.device_status()  # read and clear whatever an earlier call left
    t0 = time.perf_counter()
    qx.selftest_wait_timeout(20000)  # 20 ms
    assert qx.device_status() == 5  # QX_ERR_TIMEOUT, read and cleared
    assert time.perf_counter() - t0 < 10.0
    assert qx.device_status() == 0


def test_context_is_usable_after_a_timeout(qx):
    qx.selftest_wait_timeout(1000)
    assert qx.device_status() == 5
    n, k = 96, 512
    W = synth.student_t_weights(n, k, 0.02, seed=4, stream=900)
    x = synth.activations(2, k, seed=4, stream=901)
    P = qx.quantize(torch.from_numpy(W).cuda(), qx.Recipe(3, 128, qx.LUT))
    y = qx.gemv(P, torch.from_numpy(x).cuda(), out_dtype=torch.float32).cpu().numpy()
    assert qx.device_status() == 0
    rec = ORecipe(3, 128, "lut", 25)
    ref = oracle.quantize(W, rec)
    assert np.array_equal(P.to_numpy()["codes"], ref["codes"])
    tol = oracle.tolerance(x, oracle.dequant(ref, rec, k))
    assert np.all(oracle.max_abs_err(y, oracle.gemv(ref, rec, x, k)) <= tol)
