"""GPU parity of the Q4X shared-codebook path (Section 3.2, Fig. 3a/3b) through
the C ABI: scales, book indices, codebooks, codes and dequantized weights
bit-exact with the CPU oracle; the decode matmul within
max_n |y - y_ref| <= 2e-3 * ||x_b||_2 * max_n ||w_hat_n||_2 for every row b."""
import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def qx(cuda_dev):
    import paper_2505_07531_gb300.qx as qx

    qx._lib()
    return qx


def _weights(n, k, seed, outliers=0.001):
    return synth.student_t_weights(n, k, 0.02, seed=seed, stream=3 * n + k, outlier_frac=outliers).astype(np.float16)


CASES = [  # n, k, iters -- ragged book bytes (k/64 not a multiple of 4), early and late stops
    (64, 512, 25),
    (37, 320, 25),
    (130, 640, 3),
    (1, 64, 25),
    (16, 128, 0),
    (256, 1024, 25),
    (300, 704, 25),
    (96, 4096, 1),
]


def _ids(c):
    return "n%d_k%d_it%d" % c


def _assert_same(P, ref):
    got, want = P.to_numpy(), oracle.pack_q4x(ref)
    assert np.array_equal(got["scales"].view(np.uint16), want["scales"].view(np.uint16)), "scales"
    assert np.array_equal(got["books"], want["books"]), "book indices"
    assert np.array_equal(got["codebooks"].view(np.uint16), want["codebooks"].view(np.uint16)), "codebooks"
    assert np.array_equal(got["codes"], want["codes"]), "codes"


@pytest.fixture(scope="module")
def learned(qx):
    out = {}
    for c in CASES:
        n, k, iters = c
        W = _weights(n, k, seed=sum(c))
        P = qx.q4x_quantize(torch.from_numpy(W).cuda(), iters)
        assert qx.device_status() == 0
        out[c] = (W, P, oracle.quantize_q4x(W, iters=iters))
    return out


@pytest.mark.parametrize("c", CASES, ids=_ids)
def test_learned_buffers_bit_exact(learned, c):
    _, P, ref = learned[c]
    _assert_same(P, ref)


@pytest.mark.parametrize("c", CASES, ids=_ids)
def test_dequant_bit_exact(qx, learned, c):
    _, P, ref = learned[c]
    want = oracle.dequant_q4x(ref["codes"], ref["scales"], ref["books"], ref["codebooks"])
    assert np.array_equal(qx.q4x_dequant(P).cpu().numpy().view(np.uint16), want.view(np.uint16))


@pytest.mark.parametrize("batch", [1, 3, 4, 8, 16])
@pytest.mark.parametrize("c", CASES, ids=_ids)
def test_gemv_within_tolerance(qx, learned, c, batch):
    _, P, ref = learned[c]
    x = synth.activations(batch, c[1], seed=batch, stream=c[0])
    y = qx.q4x_gemv(P, torch.from_numpy(x).cuda(), out_dtype=torch.float32).cpu().numpy()
    assert qx.device_status() == 0
    Wh = oracle.dequant_q4x(ref["codes"], ref["scales"], ref["books"], ref["codebooks"])
    assert np.all(oracle.max_abs_err(y, oracle.gemv_q4x(ref, x)) <= oracle.tolerance(x, Wh))


@pytest.mark.parametrize("m", [1, 5, 17, 200])
@pytest.mark.parametrize("c", CASES, ids=_ids)
def test_tensor_core_matmul_within_tolerance(qx, learned, c, m):
    """Prefill on the tensor cores (qx_q4x_gemm and the split-k form) against
    the oracle; k must be a multiple of 128, else the call is refused."""
    _, P, ref = learned[c]
    X = torch.from_numpy(synth.activations(m, c[1], seed=m, stream=c[0] + 2)).cuda()
    if c[1] % 128:
        with pytest.raises(qx.QxError):
            qx.q4x_gemm(P, X)
        return
    Xn = X.cpu().numpy()
    y_ref = oracle.gemv_q4x(ref, Xn)
    Wh = oracle.dequant_q4x(ref["codes"], ref["scales"], ref["books"], ref["codebooks"])
    tol = oracle.tolerance(Xn, Wh) + np.abs(y_ref).max(axis=1) * 2.0 ** -11  # fp16 output
    Y = qx.q4x_gemm(P, X).cpu().numpy().astype(np.float64)
    Ys = qx.q4x_gemm_splitk(P, X).cpu().numpy().astype(np.float64)
    assert qx.device_status() == 0
    assert np.all(oracle.max_abs_err(Y, y_ref) <= tol)
    assert np.all(oracle.max_abs_err(Ys, y_ref) <= tol)


def test_split_k_repeats_and_pdl_are_bit_identical(qx, learned):
    _, P, _ = learned[(96, 4096, 1)]
    X = torch.from_numpy(synth.activations(16, 4096, seed=3, stream=3)).cuda()
    a = qx.q4x_gemm_splitk(P, X)
    b = qx.q4x_gemm_splitk(P, X)
    c = qx.q4x_gemm_splitk(P, X, pdl=True)
    assert qx.device_status() == 0
    assert torch.equal(a, b) and torch.equal(b, c)


def test_gemv_fp16_output(qx, learned):
    c = CASES[5]
    _, P, ref = learned[c]
    x = synth.activations(4, c[1], seed=7, stream=7)
    y = qx.q4x_gemv(P, torch.from_numpy(x).cuda()).cpu().numpy()
    y_ref = oracle.gemv_q4x(ref, x)
    Wh = oracle.dequant_q4x(ref["codes"], ref["scales"], ref["books"], ref["codebooks"])
    # fp16 output adds at most half an ulp of the result
    tol = oracle.tolerance(x, Wh) + np.abs(y_ref).max(axis=1) * 2.0 ** -11
    assert np.all(oracle.max_abs_err(y, y_ref) <= tol)


@pytest.mark.parametrize("batch", [1, 4, 16])
def test_gemv_multi_over_mixed_shapes(qx, learned, batch):
    """One launch over all eight parity matrices (different n, k and
    codebooks): every output within tolerance, and equal to the one-matrix
    call bit for bit (the same per-row arithmetic)."""
    cs = CASES
    mats = [learned[c][1] for c in cs]
    xs = [torch.from_numpy(synth.activations(batch, c[1], seed=batch, stream=c[0] + 1)).cuda() for c in cs]
    ys = qx.q4x_gemv_multi(mats, xs, out_dtype=torch.float32)
    assert qx.device_status() == 0
    for c, P, x, y in zip(cs, mats, xs, ys):
        ref = learned[c][2]
        Wh = oracle.dequant_q4x(ref["codes"], ref["scales"], ref["books"], ref["codebooks"])
        xn = x.cpu().numpy()
        assert np.all(oracle.max_abs_err(y.cpu().numpy(), oracle.gemv_q4x(ref, xn)) <= oracle.tolerance(xn, Wh))
        one = qx.q4x_gemv(P, x, out_dtype=torch.float32)
        assert torch.equal(one, y)


def test_repeat_is_bit_identical(qx):
    """Every reduction of the learner is an integer reduction: the result does
    not depend on how the threads were scheduled."""
    W = torch.from_numpy(_weights(200, 1024, seed=21)).cuda()
    a, b = qx.q4x_quantize(W).to_numpy(), qx.q4x_quantize(W).to_numpy()
    for key in a:
        assert np.array_equal(a[key], b[key]), key


def _degenerate():
    rng = np.random.default_rng(5)
    cases = {}
    cases["all_zero"] = np.zeros((8, 256), np.float16)
    w = np.zeros((8, 256), np.float16)
    w[5, 70] = 0.25
    cases["one_live_group"] = w
    cases["identical_groups"] = np.tile(np.linspace(-1, 1, 64).astype(np.float16), (12, 4))
    cases["few_distinct"] = np.tile(np.array([-1, 0, 0.5, 1], np.float16), (8, 64))
    cases["integers"] = rng.integers(-20, 21, size=(32, 512)).astype(np.float16)
    cases["subnormals"] = (rng.standard_normal((16, 256)) * 2.0 ** -20).astype(np.float16)
    w = _weights(16, 256, seed=6)
    w[3, :64] = np.float16(65504)
    w[3, 64:128] = np.float16(-65504)
    w[4, 128:192] = np.float16(6e-8)  # the smallest subnormal
    cases["extremes"] = w
    w = _weights(16, 512, seed=8)
    w[2, 0] = np.float16(3.0)  # one outlier sets its group's scale
    cases["outlier"] = w
    return cases


DEGENERATE = _degenerate()


@pytest.mark.parametrize("name", sorted(DEGENERATE))
def test_degenerate_matrices_bit_exact(qx, name):
    W = DEGENERATE[name]
    P = qx.q4x_quantize(torch.from_numpy(W).cuda())
    assert qx.device_status() == 0
    ref = oracle.quantize_q4x(W)
    _assert_same(P, ref)
    want = oracle.dequant_q4x(ref["codes"], ref["scales"], ref["books"], ref["codebooks"])
    assert np.array_equal(qx.q4x_dequant(P).cpu().numpy().view(np.uint16), want.view(np.uint16))


def test_nonfinite_group_is_flagged_and_coded_as_dead(qx):
    """A group holding NaN or Inf raises QX_ERR_NONFINITE and is coded as a
    dead group; the rest equals the oracle on the matrix with that group zero."""
    W = _weights(24, 512, seed=9)
    bad = W.copy()
    bad[4, 130] = np.float16(np.nan)
    bad[9, 0] = np.float16(np.inf)
    P = qx.q4x_quantize(torch.from_numpy(bad).cuda())
    assert qx.device_status() == 6  # QX_ERR_NONFINITE
    clean = W.copy()
    clean[4, 128:192] = 0
    clean[9, 0:64] = 0
    _assert_same(P, oracle.quantize_q4x(clean))


@pytest.mark.parametrize("shape", [(96, 512), (37, 384)])
def test_select_recipe_with_q4x_candidate(qx, shape):
    """Recipe selection with a Q4X candidate beside per-group ones: the same
    choice, exact errors and bits per weight as the oracle, with budgets that
    keep or exclude Q4X (its 128 codebook bytes count)."""
    from oracle import select as oselect
    from oracle.pack import Recipe as ORecipe
    n, k = shape
    W = _weights(n, k, seed=700 + n)
    spec = [(3, 64, qx.UNIFORM, "uniform", 25), (4, 64, qx.Q4X, oselect.Q4X, 6), (3, 128, qx.LUT, "lut", 25),
            (4, 128, qx.UNIFORM, "uniform", 25)]
    cands = [qx.Recipe(b, g, kd, it) for b, g, kd, _, it in spec]
    orecs = [ORecipe(b, g, name, it) for b, g, _, name, it in spec]
    Wd = torch.from_numpy(W).cuda()
    for max_bpw in (None, 4.35, 4.2):
        got = qx.select_recipe(Wd, cands, max_bpw)
        want = oselect.select_recipe(W, orecs, max_bpw)
        assert got[0] == want[0] and got[1] == want[1] and got[2] == want[2], max_bpw
    assert qx.device_status() == 0


def test_select_recipe_q4x_lossless(qx):
    """Groups drawn from 16 shared levels with their maximum present: Q4X codes
    them without error and is chosen over the per-group recipes."""
    rng = np.random.default_rng(9)
    levels = np.array([-1, -0.75, -0.5, -0.375, -0.25, -0.125, -0.0625, 0,
                       0.0625, 0.125, 0.25, 0.375, 0.5, 0.625, 0.75, 1.0])
    W = levels[rng.integers(0, 16, (32, 512))]
    W[:, ::64] = 1.0
    W = (W * 2.0 ** -rng.integers(3, 8, (32, 8)).repeat(64, axis=1)).astype(np.float16)
    best, errs, _ = qx.select_recipe(torch.from_numpy(W).cuda(),
                                     [qx.Recipe(4, 64, qx.UNIFORM), qx.Recipe(4, 64, qx.Q4X)])
    assert best == 1 and errs[1] == 0 and errs[0] > 0


@pytest.mark.slow
def test_full_size_llama_projection(qx):
    """4096 x 4096 (a Llama-7B attention projection), the default 25 steps:
    every buffer bit-exact, and the decode matmul at batch 1 and 4."""
    n = k = 4096
    W = _weights(n, k, seed=11)
    P = qx.q4x_quantize(torch.from_numpy(W).cuda())
    assert qx.device_status() == 0
    ref = oracle.quantize_q4x(W)
    _assert_same(P, ref)
    Wh = oracle.dequant_q4x(ref["codes"], ref["scales"], ref["books"], ref["codebooks"])
    assert np.array_equal(qx.q4x_dequant(P).cpu().numpy().view(np.uint16), Wh.view(np.uint16))
    for batch in (1, 4):
        x = synth.activations(batch, k, seed=batch, stream=11)
        y = qx.q4x_gemv(P, torch.from_numpy(x).cuda(), out_dtype=torch.float32).cpu().numpy()
        assert np.all(oracle.max_abs_err(y, oracle.gemv_q4x(ref, x)) <= oracle.tolerance(x, Wh))
    # a 512-token prefill on the tensor cores
    X = synth.activations(512, k, seed=5, stream=11)
    Y = qx.q4x_gemm(P, torch.from_numpy(X).cuda()).cpu().numpy().astype(np.float64)
    y_ref = oracle.gemv_q4x(ref, X)
    assert np.all(oracle.max_abs_err(Y, y_ref) <= oracle.tolerance(X, Wh) + np.abs(y_ref).max(axis=1) * 2.0 ** -11)
