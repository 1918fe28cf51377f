"""GPU parity through the C ABI: packed codes, scales, zeros, LUTs and dequantized
weights bit-exact with the CPU oracle; GEMV and GEMM outputs within
max_n |y - y_ref| <= 2e-3 * ||x_b||_2 * max_n ||w_hat_n||_2 for every row b."""
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


def _orecipe(bits, g, kind, iters=25):
    return ORecipe(bits, g, "lut" if kind else "uniform", iters)


def _weights(n, k, seed, sigma=0.02, outliers=0.001):
    return synth.student_t_weights(n, k, sigma, seed=seed, stream=n * 7 + k, outlier_frac=outliers)


CASES = [  # n, k, bits, g, kind -- ragged n, several groups/superblocks per row
    (64, 512, 4, 64, 0),
    (37, 384, 4, 128, 0),
    (130, 640, 3, 64, 0),
    (96, 1024, 3, 128, 1),
    (33, 256, 4, 32, 0),
    (17, 512, 3, 256, 1),
    (50, 768, 3, 32, 1),
    (257, 256, 4, 256, 0),
    (1, 128, 3, 128, 0),
    (3, 128, 4, 128, 0),
]


def _ids(c):
    return "n%d_k%d_b%d_g%d_%s" % (c[0], c[1], c[2], c[3], "lut" if c[4] else "u")


@pytest.fixture(scope="module")
def packed(qx):
    """Quantize every case once on the GPU and once in the oracle."""
    out = {}
    for c in CASES:
        n, k, bits, g, kind = c
        W = _weights(n, k, seed=sum(c))
        P = qx.quantize(torch.from_numpy(W).cuda(), qx.Recipe(bits, g, kind))
        assert qx.device_status() == 0
        out[c] = (W, P, oracle.quantize(W, _orecipe(bits, g, kind)))
    return out


@pytest.mark.parametrize("case", CASES, ids=_ids)
def test_quantize_bit_exact(packed, case):
    W, P, ref = packed[case]
    got = P.to_numpy()
    assert np.array_equal(got["codes"], ref["codes"])
    for key in ("scales", "zeros", "luts"):
        if ref[key] is None:
            assert got[key] is None
        else:
            assert np.array_equal(got[key].view(np.uint16) if got[key].dtype == np.float16 else got[key],
                                  ref[key].view(np.uint16) if ref[key].dtype == np.float16 else ref[key]), key


@pytest.mark.parametrize("case", CASES, ids=_ids)
def test_dequant_bit_exact(qx, packed, case):
    W, P, ref = packed[case]
    n, k, bits, g, kind = case
    Wh = qx.dequant(P).cpu().numpy()
    want = oracle.dequant(ref, _orecipe(bits, g, kind), k)
    assert np.array_equal(Wh.view(np.uint16), want.view(np.uint16))


def _check_matmul(y_gpu, y_ref, X, Wh):
    tol = oracle.tolerance(X, Wh)
    err = oracle.max_abs_err(y_gpu, y_ref)
    assert np.all(err <= tol), (err, tol)
    return err / np.maximum(tol, 1e-300)


@pytest.mark.parametrize("batch", [1, 2, 3, 4, 5, 8, 16])
@pytest.mark.parametrize("case", CASES, ids=_ids)
def test_gemv_tolerance(qx, packed, case, batch):
    W, P, ref = packed[case]
    n, k, bits, g, kind = case
    x = synth.activations(batch, k, seed=batch, stream=k)
    y_ref = oracle.gemv(ref, _orecipe(bits, g, kind), x, k)
    Wh = oracle.dequant(ref, _orecipe(bits, g, kind), k)
    xd = torch.from_numpy(x).cuda()
    for dt in (torch.float16, torch.float32):
        y = qx.gemv(P, xd, out_dtype=dt).cpu().numpy()
        assert y.shape == (batch, n)
        _check_matmul(y, y_ref, x, Wh)


@pytest.mark.parametrize("m", [1, 7, 128, 200])
@pytest.mark.parametrize("case", CASES, ids=_ids)
def test_gemm_tolerance(qx, packed, case, m):
    W, P, ref = packed[case]
    n, k, bits, g, kind = case
    X = synth.activations(m, k, seed=m, stream=3 * k)
    Y = qx.gemm(P, torch.from_numpy(X).cuda())
    assert qx.device_status() == 0
    Y = Y.cpu().numpy()
    y_ref = oracle.gemm(ref, _orecipe(bits, g, kind), X, k)
    _check_matmul(Y, y_ref, X, oracle.dequant(ref, _orecipe(bits, g, kind), k))


def test_gemm_many_tiles(qx):
    """Several W-row tiles and token tiles, ragged in both, k spanning > 4 stages."""
    n, k, m = 300, 1280, 333
    for bits, g, kind in ((4, 64, 0), (3, 128, 1), (3, 64, 0)):
        W = _weights(n, k, seed=bits + g + kind)
        ref = oracle.quantize(W, _orecipe(bits, g, kind))
        P = qx.quantize(torch.from_numpy(W).cuda(), qx.Recipe(bits, g, kind))
        X = synth.activations(m, k, seed=5, stream=k)
        Y = qx.gemm(P, torch.from_numpy(X).cuda()).cpu().numpy()
        assert qx.device_status() == 0
        _check_matmul(Y, oracle.gemm(ref, _orecipe(bits, g, kind), X, k), X,
                      oracle.dequant(ref, _orecipe(bits, g, kind), k))


def test_config_single_layer_512(qx):
    """512 x 512 Student-t(4), sigma 0.02, 0.1% outliers at 10 sigma, seed 0; U4 g64; x 1 x 512."""
    W = synth.student_t_weights(512, 512, 0.02, seed=0, stream=0, outlier_frac=0.001)
    x = synth.activations(1, 512, seed=0, stream=1)
    rec = _orecipe(4, 64, 0)
    ref = oracle.quantize(W, rec)
    P = qx.quantize(torch.from_numpy(W).cuda(), qx.Recipe(4, 64, 0))
    got = P.to_numpy()
    assert np.array_equal(got["codes"], ref["codes"])
    assert np.array_equal(got["scales"].view(np.uint16), ref["scales"].view(np.uint16))
    assert np.array_equal(got["zeros"], ref["zeros"])
    y = qx.gemv(P, torch.from_numpy(x).cuda(), out_dtype=torch.float32).cpu().numpy()
    _check_matmul(y, oracle.gemv(ref, rec, x, 512), x, oracle.dequant(ref, rec, 512))


def test_nonfinite_weight_sets_status(qx):
    W = torch.zeros((4, 128), dtype=torch.float16, device="cuda")
    W[2, 5] = float("nan")
    qx.quantize(W, qx.Recipe(4, 64, 0))
    assert qx.device_status() == 6
    assert qx.device_status() == 0  # read clears it
    W[2, 5] = float("inf")
    qx.quantize(W, qx.Recipe(3, 128, 1))
    assert qx.device_status() == 6
    assert qx.device_status() == 0


MULTI_GROUPS = [  # matrices of one launch share bits and kind
    [(2048, 4096, 3, 128, 1), (512, 4096, 3, 128, 1), (256, 11008, 3, 64, 1)],
    [(300, 512, 4, 64, 0), (77, 1024, 4, 128, 0), (5, 256, 4, 32, 0), (640, 384, 4, 64, 0)],
    [(129, 640, 3, 64, 0), (3, 128, 3, 32, 0)],
    [(1, 128, 4, 128, 0)] * 8,
]


@pytest.fixture(scope="module")
def multi_packed(qx):
    """Each group quantized once on the GPU and once in the oracle."""
    out = []
    for gi, group in enumerate(MULTI_GROUPS):
        Ps, refs = [], []
        for i, (n, k, bits, g, kind) in enumerate(group):
            W = _weights(n, k, seed=97 + i + 10 * gi)
            Ps.append(qx.quantize(torch.from_numpy(W).cuda(), qx.Recipe(bits, g, kind)))
            refs.append(oracle.quantize(W, _orecipe(bits, g, kind)))
        out.append((Ps, refs))
    return out


@pytest.mark.parametrize("pdl", [False, True])
@pytest.mark.parametrize("batch", [1, 3, 6])
@pytest.mark.parametrize("gi", range(len(MULTI_GROUPS)))
def test_gemv_multi(qx, multi_packed, gi, batch, pdl):
    """One launch over several matrices (slices spanning matrix boundaries)."""
    group = MULTI_GROUPS[gi]
    Ps, refs = multi_packed[gi]
    xs = [synth.activations(batch, k, seed=i, stream=gi) for i, (n, k, bits, g, kind) in enumerate(group)]
    xds = [torch.from_numpy(x).cuda() for x in xs]
    if pdl:  # the flag's contract: the previous kernel must not write these weights
        torch.cuda.synchronize()
    ys = qx.gemv_multi(Ps, xds, out_dtype=torch.float32, pdl=pdl)
    for (n, k, bits, g, kind), ref, x, y in zip(group, refs, xs, ys):
        rec = _orecipe(bits, g, kind)
        _check_matmul(y.cpu().numpy(), oracle.gemv(ref, rec, x, k), x, oracle.dequant(ref, rec, k))


def test_gemv_multi_rejects_mixed_kinds(qx):
    a = qx.quantize(torch.zeros((4, 128), dtype=torch.float16, device="cuda"), qx.Recipe(4, 64, 0))
    b = qx.quantize(torch.zeros((4, 128), dtype=torch.float16, device="cuda"), qx.Recipe(3, 128, 1))
    x = torch.zeros((1, 128), dtype=torch.float16, device="cuda")
    with pytest.raises(qx.QxError):
        qx.gemv_multi([a, b], [x, x])


def test_gemv_pdl_chain_orders_activations(qx):
    """A decode that reads the previous decode's output under PDL sees the finished
    output: the chained result equals the same chain run without PDL, bit for bit."""
    W1 = _weights(4096, 4096, seed=1)
    W2 = _weights(2048, 4096, seed=2)
    P1 = qx.quantize(torch.from_numpy(W1).cuda(), qx.Recipe(3, 128, 1))
    P2 = qx.quantize(torch.from_numpy(W2).cuda(), qx.Recipe(3, 128, 1))
    x = torch.from_numpy(synth.activations(1, 4096, seed=3, stream=3)).cuda()
    y1 = torch.empty((1, 4096), dtype=torch.float16, device="cuda")
    outs = []
    for pdl in (False, True):
        torch.cuda.synchronize()
        for _ in range(20):
            qx.gemv_multi([P1], [x], outs=[y1], pdl=pdl)
            (y2,) = qx.gemv_multi([P2], [y1], pdl=pdl)
        outs.append(y2.clone())
    torch.cuda.synchronize()
    assert torch.equal(outs[0], outs[1])


@pytest.mark.parametrize("bits,g,kind", [(4, 32, 0), (3, 32, 1)])
def test_gemv_longest_rows(qx, bits, g, kind):
    """k = 32768 (the largest k the decode kernel takes), batch 3: the host splits the batch."""
    n, k = 40, 32768
    W = _weights(n, k, seed=k + bits)
    ref = oracle.quantize(W, _orecipe(bits, g, kind))
    P = qx.quantize(torch.from_numpy(W).cuda(), qx.Recipe(bits, g, kind))
    x = synth.activations(3, k, seed=1, stream=2)
    y = qx.gemv(P, torch.from_numpy(x).cuda(), out_dtype=torch.float32).cpu().numpy()
    rec = _orecipe(bits, g, kind)
    _check_matmul(y, oracle.gemv(ref, rec, x, k), x, oracle.dequant(ref, rec, k))


WRAP_CASES = [  # enough rows that every CTA cycles its shared-memory ring several times
    (20000, 128, 3, 128, 1),
    (20000, 256, 3, 64, 0),
    (20000, 512, 4, 64, 0),
    (6000, 4096, 3, 128, 0),
]


@pytest.mark.parametrize("batch", [1, 3, 4])
@pytest.mark.parametrize("case", WRAP_CASES, ids=_ids)
def test_gemv_ring_wraps(qx, case, batch):
    n, k, bits, g, kind = case
    W = _weights(n, k, seed=n + k)
    rec = _orecipe(bits, g, kind)
    ref = oracle.quantize(W, rec)
    P = qx.quantize(torch.from_numpy(W).cuda(), qx.Recipe(bits, g, kind))
    x = synth.activations(batch, k, seed=batch, stream=n)
    y = torch.full((batch, n), float("nan"), dtype=torch.float32, device="cuda")
    qx.gemv(P, torch.from_numpy(x).cuda(), out=y)
    assert qx.device_status() == 0
    _check_matmul(y.cpu().numpy(), oracle.gemv(ref, rec, x, k), x, oracle.dequant(ref, rec, k))


# Mixed per-layer recipe (paper Sections 2.1 and 2.3): each matrix carries its
# own recipe.  A two-layer stack shaped like the LLaVA language layers (Q/K
# 3-bit LUT g128, V/O and MLP 4-bit uniform g64) is decoded through the
# launch sequence q,k | v | o | gate,up | down captured in one CUDA graph
# with programmatic dependent launch, and a vision-shaped set of matrices
# (4-bit uniform g128) is prefilled with qx_gemm.
STACK = [("q", 256, 256, (3, 128, 1)), ("k", 256, 256, (3, 128, 1)), ("v", 256, 256, (4, 64, 0)),
         ("o", 256, 256, (4, 64, 0)), ("gate", 640, 256, (4, 64, 0)), ("up", 640, 256, (4, 64, 0)),
         ("down", 256, 640, (4, 64, 0))]


@pytest.mark.gpu
def test_mixed_recipe_stack_decode_graph(qx):
    layers = []
    for li in range(2):
        L = {}
        for i, (nm, n, k, (bits, g, kind)) in enumerate(STACK):
            W = _weights(n, k, seed=300 + 10 * li + i)
            L[nm] = (qx.quantize(torch.from_numpy(W).cuda(), qx.Recipe(bits, g, kind)),
                     oracle.quantize(W, _orecipe(bits, g, kind)), (bits, g, kind))
        layers.append(L)
    xa = synth.activations(1, 256, seed=1, stream=41)
    xo = synth.activations(1, 256, seed=1, stream=42)
    xm = synth.activations(1, 256, seed=1, stream=43)
    xd = synth.activations(1, 640, seed=1, stream=44)
    dx = {nm: torch.from_numpy(x).cuda() for nm, x in (("a", xa), ("o", xo), ("m", xm), ("d", xd))}
    ys = [{nm: torch.empty((1, n), dtype=torch.float32, device="cuda") for nm, n, _, _ in STACK} for _ in layers]
    chain = [(["q", "k"], "a"), (["v"], "a"), (["o"], "o"), (["gate", "up"], "m"), (["down"], "d")]
    s = torch.cuda.Stream()

    def body():
        for L, Y in zip(layers, ys):
            for names, xn in chain:
                qx.gemv_multi([L[nm][0] for nm in names], [dx[xn]] * len(names), outs=[Y[nm] for nm in names],
                              pdl=True)

    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        body()
    for Y in ys:
        for y in Y.values():
            y.fill_(float("nan"))
    g.replay()
    torch.cuda.synchronize()
    assert qx.device_status() == 0
    xs = {"a": xa, "o": xo, "m": xm, "d": xd}
    for L, Y in zip(layers, ys):
        for names, xn in chain:
            for nm in names:
                P, ref, (bits, g_, kind) = L[nm]
                k = P.k
                rec = _orecipe(bits, g_, kind)
                _check_matmul(Y[nm].cpu().numpy(), oracle.gemv(ref, rec, xs[xn], k), xs[xn], oracle.dequant(ref, rec, k))


@pytest.mark.gpu
def test_mixed_recipe_vision_prefill(qx):
    M = 300  # two token tiles, ragged
    for i, (n, k) in enumerate(((256, 256), (1024, 256), (256, 1024))):
        W = _weights(n, k, seed=400 + i)
        P = qx.quantize(torch.from_numpy(W).cuda(), qx.Recipe(4, 128, 0))
        ref = oracle.quantize(W, _orecipe(4, 128, 0))
        X = synth.activations(M, k, seed=4, stream=50 + i)
        rec = _orecipe(4, 128, 0)
        y_ref, Wh = oracle.gemm(ref, rec, X, k), oracle.dequant(ref, rec, k)
        for gemm in (qx.gemm, qx.gemm_splitk):  # 256-token tiles; 64-token tiles split along k
            Y = gemm(P, torch.from_numpy(X).cuda())
            assert qx.device_status() == 0
            _check_matmul(Y.cpu().numpy(), y_ref, X, Wh)


# ---------------------------------------------------------------- split-k tensor-core matmul
@pytest.mark.parametrize("m", [1, 3, 16, 17, 200])
@pytest.mark.parametrize("case", CASES, ids=_ids)
def test_gemm_splitk_tolerance(qx, packed, case, m):
    W, P, ref = packed[case]
    n, k, bits, g, kind = case
    X = synth.activations(m, k, seed=m + 1, stream=5 * k)
    Y = qx.gemm_splitk(P, torch.from_numpy(X).cuda())
    assert qx.device_status() == 0
    rec = _orecipe(bits, g, kind)
    _check_matmul(Y.cpu().numpy(), oracle.gemm(ref, rec, X, k), X, oracle.dequant(ref, rec, k))


@pytest.mark.parametrize("bits,g,kind", [(3, 128, 1), (4, 64, 0), (3, 64, 0)])
def test_gemm_splitk_deterministic_and_rearmed(qx, bits, g, kind):
    """A ragged 1000-row matrix (8 W tiles) with k = 4096 split across CTAs: the
    result does not depend on which split finishes last, every call leaves the
    workspace counters at zero, and a short workspace is refused."""
    n, k = 1000, 4096
    rec = _orecipe(bits, g, kind)
    W = _weights(n, k, seed=500 + bits + g)
    ref = oracle.quantize(W, rec)
    Wh = oracle.dequant(ref, rec, k)
    P = qx.quantize(torch.from_numpy(W).cuda(), qx.Recipe(bits, g, kind))
    for m in (1, 5, 16):
        nbytes = qx.gemm_splitk_workspace_bytes(n, k, m, P.recipe)
        assert nbytes > 0
        ws = torch.zeros(nbytes, dtype=torch.uint8, device="cuda")
        X = synth.activations(m, k, seed=m, stream=77)
        Xd = torch.from_numpy(X).cuda()
        Y1 = qx.gemm_splitk(P, Xd, workspace=ws)
        Y2 = qx.gemm_splitk(P, Xd, workspace=ws)
        assert qx.device_status() == 0
        assert torch.equal(Y1, Y2)
        assert int(ws[:65536].count_nonzero()) == 0  # the counter region
        _check_matmul(Y1.cpu().numpy(), oracle.gemm(ref, rec, X, k), X, Wh)
    with pytest.raises(qx.QxError) as e:
        qx.gemm_splitk(P, Xd, workspace=torch.zeros(256, dtype=torch.uint8, device="cuda"))
    assert e.value.code == 1


def test_gemm_splitk_pdl_chain_orders_inputs(qx):
    """Under PDL a split-k call that reads the previous call's output (and shares
    its workspace) sees the finished output: the chain equals the same chain run
    without PDL, bit for bit."""
    P1 = qx.quantize(torch.from_numpy(_weights(4096, 4096, seed=11)).cuda(), qx.Recipe(3, 128, 1))
    P2 = qx.quantize(torch.from_numpy(_weights(1024, 4096, seed=12)).cuda(), qx.Recipe(4, 64, 0))
    for m in (16, 300):
        X = torch.from_numpy(synth.activations(m, 4096, seed=m, stream=13)).cuda()
        outs = []
        for pdl in (False, True):
            torch.cuda.synchronize()
            for _ in range(10):
                Y1 = qx.gemm_splitk(P1, X, pdl=pdl)
                Y2 = qx.gemm_splitk(P2, Y1, pdl=pdl)
            outs.append(Y2.clone())
        torch.cuda.synchronize()
        assert qx.device_status() == 0
        assert torch.equal(outs[0], outs[1])


# ---------------------------------------------------------------- full sizes, sampled rows
# The Llama-7B-shaped layer of the decode benchmark in 3-bit LUT g128.  The
# weights are drawn on the GPU and quantized there; for each matrix a seeded
# sample of rows is also quantized by the oracle (quantization is row-local,
# so those rows' codes and outputs are unique) and every output of those rows
# is checked.
LLAMA_LAYER = [("q_proj", 4096, 4096, 0.01), ("k_proj", 4096, 4096, 0.01), ("v_proj", 4096, 4096, 0.02),
               ("o_proj", 4096, 4096, 0.02), ("gate_proj", 11008, 4096, 0.04), ("up_proj", 11008, 4096, 0.04),
               ("down_proj", 4096, 11008, 0.04)]
SAMPLE_ROWS = 48


@pytest.fixture(scope="module")
def llama_layer(qx):
    rec = _orecipe(3, 128, 1)
    out = {}
    for i, (nm, n, k, sigma) in enumerate(LLAMA_LAYER):
        W = synth.student_t_weights_torch(n, k, sigma, seed=7, stream=i, device="cuda")
        P = qx.quantize(W, qx.Recipe(3, 128, 1))
        rows = np.sort(np.random.default_rng(i).choice(n, size=SAMPLE_ROWS, replace=False))
        ref = oracle.quantize(W[torch.from_numpy(rows).cuda()].cpu().numpy(), rec)
        out[nm] = (P, rows, ref, oracle.dequant(ref, rec, k))
        del W
    assert qx.device_status() == 0
    return out


def test_full_size_decode_layer_sampled(qx, llama_layer):
    """The decode benchmark's launch configuration: q,k,v | o | gate,up | down as
    four qx_gemv_multi launches with programmatic dependent launch, captured in
    one CUDA graph, batch 1."""
    chain = [(["q_proj", "k_proj", "v_proj"], 4096), (["o_proj"], 4096), (["gate_proj", "up_proj"], 4096),
             (["down_proj"], 11008)]
    xs = [synth.activations(1, k, seed=0, stream=60 + j) for j, (_, k) in enumerate(chain)]
    dx = [torch.from_numpy(x).cuda() for x in xs]
    ys = {nm: torch.empty((1, n), dtype=torch.float16, device="cuda") for nm, n, _, _ in LLAMA_LAYER}
    s = torch.cuda.Stream()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        for (names, _), x in zip(chain, dx):
            qx.gemv_multi([llama_layer[nm][0] for nm in names], [x] * len(names), outs=[ys[nm] for nm in names],
                          pdl=True)
    for y in ys.values():
        y.fill_(float("nan"))
    g.replay()
    torch.cuda.synchronize()
    assert qx.device_status() == 0
    rec = _orecipe(3, 128, 1)
    for (names, k), x in zip(chain, xs):
        for nm in names:
            P, rows, ref, Wh = llama_layer[nm]
            _check_matmul(ys[nm].float().cpu().numpy()[:, rows], oracle.gemv(ref, rec, x, k), x, Wh)


@pytest.mark.parametrize("m", [1, 4, 16])
def test_full_size_tensor_core_decode_sampled(qx, llama_layer, m):
    """qx_gemm_splitk as a decode matmul (16-token tiles, k split) on the layer's shapes."""
    rec = _orecipe(3, 128, 1)
    for nm in ("q_proj", "gate_proj", "down_proj"):
        P, rows, ref, Wh = llama_layer[nm]
        X = synth.activations(m, P.k, seed=m, stream=70)
        Y = qx.gemm_splitk(P, torch.from_numpy(X).cuda())
        assert qx.device_status() == 0
        _check_matmul(Y.cpu().numpy()[:, rows], oracle.gemm(ref, rec, X, P.k), X, Wh)


def test_full_size_prefill_sampled(qx, llama_layer):
    """Prefill of 2048 tokens against 11008x4096 and 4096x11008 (the GEMM benchmark's shapes)."""
    rec = _orecipe(3, 128, 1)
    for nm in ("gate_proj", "down_proj"):
        P, rows, ref, Wh = llama_layer[nm]
        X = synth.activations(2048, P.k, seed=2, stream=80)
        Y = qx.gemm(P, torch.from_numpy(X).cuda())
        assert qx.device_status() == 0
        _check_matmul(Y.cpu().numpy()[:, rows], oracle.gemm(ref, rec, X, P.k), X, Wh)


# ---------------------------------------------------------------- recipe selection
SELECT_CANDIDATES = [(3, 64, 0), (3, 128, 1), (4, 64, 0), (4, 128, 0), (3, 64, 1)]


@pytest.mark.parametrize("shape", [(96, 512), (130, 256)])
def test_select_recipe_matches_oracle(qx, shape):
    """Same choice and the same exact errors (integers in units of 2^-48) as the
    oracle, with no budget and with budgets that exclude candidates or all."""
    from oracle import select as oselect
    n, k = shape
    W = _weights(n, k, seed=600 + n)
    cands = [qx.Recipe(b, g, kd) for b, g, kd in SELECT_CANDIDATES]
    orecs = [_orecipe(b, g, kd) for b, g, kd in SELECT_CANDIDATES]
    Wd = torch.from_numpy(W).cuda()
    for max_bpw in (None, 4.2, 3.3):
        got = qx.select_recipe(Wd, cands, max_bpw)
        want = oselect.select_recipe(W, orecs, max_bpw)
        assert got[0] == want[0] and got[1] == want[1] and got[2] == want[2], max_bpw


def test_select_recipe_lossless_lut_closed_form(qx):
    """Eight unequally spaced values per group: the 3-bit LUT is exact (error 0) and chosen."""
    rng = np.random.default_rng(12)
    levels = np.array([-0.05, -0.011, -0.002, 0.0, 0.0007, 0.003, 0.02, 0.07])
    W = levels[rng.integers(0, 8, (64, 512))].astype(np.float16)
    best, errs, _ = qx.select_recipe(torch.from_numpy(W).cuda(), [qx.Recipe(3, 64, 0), qx.Recipe(3, 64, 1)])
    assert best == 1 and errs[1] == 0 and errs[0] > 0


# ---------------------------------------------------------------- W.A8 decode
@pytest.mark.parametrize("batch", [1, 3, 16])
def test_quantize_act_bit_exact(qx, batch):
    from oracle import act8
    x = synth.activations(batch, 1280, seed=batch, stream=90)
    x[0, 7] = 0  # a zero element
    q, s = qx.quantize_act(torch.from_numpy(x).cuda())
    qr, sr = act8.quantize_act(x)
    assert np.array_equal(q.cpu().numpy(), qr) and np.array_equal(s.cpu().numpy().view(np.uint32), sr.view(np.uint32))


A8_CASES = [c for c in CASES if c[4] == 0]  # uniform recipes only


@pytest.mark.parametrize("batch", [1, 2, 5, 16])
@pytest.mark.parametrize("case", A8_CASES, ids=_ids)
def test_gemv_a8_tolerance(qx, packed, case, batch):
    """Within 2e-3 ||x_hat_b|| max_n ||w_n|| of the oracle's W.A8 product, w the
    unrounded (q - z) s the integer path multiplies."""
    from oracle import act8
    W, P, ref = packed[case]
    n, k, bits, g, kind = case
    rec = _orecipe(bits, g, kind)
    x = synth.activations(batch, k, seed=batch, stream=91)
    q, s = qx.quantize_act(torch.from_numpy(x).cuda())
    for dt in (torch.float16, torch.float32):
        y = qx.gemv_a8(P, q, s, out_dtype=dt)
        assert qx.device_status() == 0
        y_ref = act8.gemv_a8(ref, rec, x, k)
        qw = oracle.unpack_codes(ref["codes"], bits, k).astype(np.float64)
        z = np.repeat(oracle.unpack_zeros(ref["zeros"], k // g).astype(np.float64), g, axis=1)
        w_exact = (qw - z) * np.repeat(ref["scales"].astype(np.float64), g, axis=1)
        qr, sr = act8.quantize_act(x)
        _check_matmul(y.float().cpu().numpy(), y_ref, act8.dequant_act(qr, sr), w_exact)


def test_gemv_a8_full_size_sampled(qx, llama_layer):
    """4-bit uniform g128 on the q_proj / down_proj shapes: sampled rows, batch 4."""
    from oracle import act8
    rec = _orecipe(4, 128, 0)
    for nm, n, k in (("q", 4096, 4096), ("down", 4096, 11008)):
        W = synth.student_t_weights_torch(n, k, 0.02, seed=9, stream=n + k, device="cuda")
        P = qx.quantize(W, qx.Recipe(4, 128, 0))
        rows = np.sort(np.random.default_rng(n + k).choice(n, size=SAMPLE_ROWS, replace=False))
        ref = oracle.quantize(W[torch.from_numpy(rows).cuda()].cpu().numpy(), rec)
        x = synth.activations(4, k, seed=4, stream=92)
        q, s = qx.quantize_act(torch.from_numpy(x).cuda())
        y = qx.gemv_a8(P, q, s, out_dtype=torch.float32).cpu().numpy()[:, rows]
        assert qx.device_status() == 0
        qw = oracle.unpack_codes(ref["codes"], 4, k).astype(np.float64)
        z = np.repeat(oracle.unpack_zeros(ref["zeros"], k // 128).astype(np.float64), 128, axis=1)
        w_exact = (qw - z) * np.repeat(ref["scales"].astype(np.float64), 128, axis=1)
        qr, sr = act8.quantize_act(x)
        _check_matmul(y, act8.gemv_a8(ref, rec, x, k), act8.dequant_act(qr, sr), w_exact)


# ---------------------------------------------------------------- degenerate groups
def _degenerate_weights(g):
    """Rows of groups that take the quantizers' special paths: all zero, one
    constant (positive and negative), a few distinct values, subnormals whose
    scale underflows, fp16 extremes, and a single outlier among zeros."""
    k = 4 * g
    rows = []
    rows.append(np.zeros(k))
    rows.append(np.full(k, 0.0371))
    rows.append(np.full(k, -2.5))
    rows.append(np.tile(np.array([-0.25, 0.0, 0.125, 0.5]), k // 4))
    rows.append(np.tile(np.array([6e-8, -1.2e-7, 0.0, 3e-8]), k // 4))  # fp16 subnormals
    ext = np.zeros(k)
    ext[::3] = 65504.0
    ext[1::3] = -65504.0
    rows.append(ext)
    one = np.zeros(k)
    one[g // 2] = 7.0
    one[g + 3] = -0.001
    rows.append(one)
    rng = np.random.default_rng(g)
    rows.append(rng.choice([-1.0, -0.5, 0.0, 0.5, 1.0, 2.0, -3.0, 0.25, 9.0], k))  # nine distinct values
    return np.stack(rows).astype(np.float16)


@pytest.mark.parametrize("bits,g,kind", [(4, 64, 0), (3, 64, 0), (4, 128, 0), (3, 128, 1), (3, 32, 1)])
def test_degenerate_groups_bit_exact(qx, bits, g, kind):
    W = _degenerate_weights(g)
    n, k = W.shape
    k_pad = max(k, 128)  # k must be a multiple of 128
    if k_pad != k:
        W = np.concatenate([W, np.zeros((n, k_pad - k), dtype=np.float16)], axis=1)
        k = k_pad
    rec = _orecipe(bits, g, kind)
    ref = oracle.quantize(W, rec)
    P = qx.quantize(torch.from_numpy(W).cuda(), qx.Recipe(bits, g, kind))
    assert qx.device_status() == 0
    got = P.to_numpy()
    assert np.array_equal(got["codes"], ref["codes"])
    for key in ("scales", "luts"):
        if ref[key] is not None:
            assert np.array_equal(got[key].view(np.uint16), ref[key].view(np.uint16)), key
    if ref["zeros"] is not None:
        assert np.array_equal(got["zeros"], ref["zeros"])
    Wh = oracle.dequant(ref, rec, k)
    assert np.array_equal(qx.dequant(P).cpu().numpy().view(np.uint16), Wh.view(np.uint16))
    # the decode forms its products and 16-pair sums in fp16: the row of fp16
    # extremes (row 5) is outside that range by design and is left out here
    x = synth.activations(2, k, seed=g, stream=93)
    y = qx.gemv(P, torch.from_numpy(x).cuda(), out_dtype=torch.float32).cpu().numpy()
    keep = [r for r in range(n) if r != 5]
    _check_matmul(y[:, keep], oracle.gemv(ref, rec, x, k)[:, keep], x, Wh[keep])


# ---------------------------------------------------------------- heavy-tailed activations
def _massive_activations(batch, k, seed):
    """N(0, 1) activations with eight 'massive' channels of |x| 100..1000 (the
    outlier channels of LLM residual streams), the same channels in every row."""
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((batch, k))
    ch = rng.choice(k, size=8, replace=False)
    x[:, ch] = rng.choice([-1.0, 1.0], size=(batch, 8)) * rng.uniform(100.0, 1000.0, size=(batch, 8))
    return x.astype(np.float16)


@pytest.mark.parametrize("batch", [1, 2, 4, 16])
@pytest.mark.parametrize("n,k,bits,g,kind", [(512, 4096, 3, 128, 1), (384, 11008, 4, 64, 0)])
def test_gemv_heavy_tailed_activations(qx, n, k, bits, g, kind, batch):
    """Batches of 1 and 2 form fp16 products and their sums over 8 weight pairs
    on the CUDA cores before the fp32 sum; larger batches accumulate in fp32 on
    the tensor cores.  With massive activation channels (and the weights' 10
    sigma outliers) both stay within the tolerance."""
    W = synth.student_t_weights(n, k, 0.04, seed=n, stream=k, outlier_frac=0.001)
    rec = _orecipe(bits, g, kind)
    ref = oracle.quantize(W, rec)
    Wh = oracle.dequant(ref, rec, k)
    P = qx.quantize(torch.from_numpy(W).cuda(), qx.Recipe(bits, g, kind))
    x = _massive_activations(batch, k, seed=batch)
    y = qx.gemv(P, torch.from_numpy(x).cuda(), out_dtype=torch.float32).cpu().numpy()
    assert qx.device_status() == 0
    _check_matmul(y, oracle.gemv(ref, rec, x, k), x, Wh)
