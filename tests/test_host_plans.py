"""Host logic of the split-k planner (qx_gemm_splitk_plan): no GPU needed."""
import numpy as np
import pytest


@pytest.fixture(scope="module")
def qx():
    import paper_2505_07531_gb300.qx as qx

    qx._lib()
    return qx


@pytest.mark.parametrize("n,k,m,want", [
    (4096, 4096, 16, (16, 4)),     # decode: 32 W tiles split four ways for 152 SMs
    (4096, 4096, 1, (16, 4)),
    (11008, 4096, 16, (16, 3)),
    (4096, 11008, 16, (16, 4)),
    (1024, 1024, 576, (64, 1)),    # vision prefill: 64-token tiles fill 72 SMs; a split costs more
    (4096, 1024, 576, (256, 1)),   # enough 256-token tiles already
    (1024, 4096, 576, (64, 2)),    # 64-token tiles, two splits
    (11008, 4096, 2048, (256, 1)),  # full prefill: no split
])
def test_plans_of_the_benchmark_shapes(qx, n, k, m, want):
    bn, sp, nbytes = qx.gemm_splitk_plan(n, k, m, 152)
    assert (bn, sp) == want
    tiles = -(-m // bn) * -(-n // 128)
    assert nbytes == (65536 + tiles * sp * bn * 128 * 4 if sp > 1 else 0)


def test_plan_invariants_over_random_shapes(qx):
    rng = np.random.default_rng(0)
    for _ in range(400):
        n = int(rng.integers(1, 40000))
        k = 128 * int(rng.integers(1, 200))
        m = int(rng.choice([1, 3, 16, 17, 64, 100, 576, 2048, 5000]))
        sms = int(rng.choice([1, 8, 132, 152]))
        bn, sp, nbytes = qx.gemm_splitk_plan(n, k, m, sms)
        assert bn in (16, 64, 256) and (bn == 16) == (m <= 16)
        assert 1 <= sp <= min(16, k // 128)
        assert bn != 256 or sp == 1
        tiles = -(-m // bn) * -(-n // 128)
        assert nbytes == (65536 + tiles * sp * bn * 128 * 4 if sp > 1 else 0)
        if sp > 1:
            assert tiles <= 65536 // 16  # the counter region holds every tile's four counters


def test_plan_rejects_bad_arguments(qx):
    import ctypes
    lib = qx._lib()
    a, b, c = ctypes.c_int32(), ctypes.c_int32(), ctypes.c_size_t()
    assert lib.qx_gemm_splitk_plan(64, 128, 1, 152, None, ctypes.byref(b), ctypes.byref(c)) == 1
    assert lib.qx_gemm_splitk_plan(64, 128, 0, 152, ctypes.byref(a), ctypes.byref(b), ctypes.byref(c)) == 1
    assert lib.qx_gemm_splitk_plan(64, 128, 1, 0, ctypes.byref(a), ctypes.byref(b), ctypes.byref(c)) == 1
    assert lib.qx_gemm_splitk_plan(64, 100, 1, 152, ctypes.byref(a), ctypes.byref(b), ctypes.byref(c)) == 2
