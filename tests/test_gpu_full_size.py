"""Full-size parity on the benchmark's shapes and launch configurations.

Quantization is row-local (every group lies within one row), so the oracle
quantizes only a seeded sample of 48 rows of each matrix, whose codes are then
unique, and every output of those rows is compared with the oracle's float64
matmul within max_n |y - y_ref| <= 2e-3 ||x_b||_2 max_n ||w_hat_n||_2.

* The Llama-7B-shaped layer with 4-bit uniform g128 and 3-bit uniform g64
  weights through the decode chain q,k,v | o | gate,up | down (four
  qx_gemv_multi launches with PDL in one CUDA graph) at batch 1, 4 and 16, and
  through the same chain with its CTAs balanced slice by slice (qx_gemv_fused:
  one launch, and one launch per group).
* One LLaVA-v1.6-7B-shaped language layer with the mixed per-matrix recipe of
  the recipe table (q, k: 3-bit LUT g128; v, o, gate, up, down: 4-bit uniform
  g64) through its five-launch chain.
* One CLIP-L/14-shaped vision layer prefilled at 576 tokens, q, k, v stacked as
  one 3072 x 1024 matrix, through qx_gemm_splitk with PDL in one CUDA graph.
Paper: Section 2.1 and 2.3 (recipes per layer and per sub-model), Section 2.4
and Table 2 (decode and prefill)."""
import os

import numpy as np
import pytest
import torch

import oracle
import synth
from oracle.pack import Recipe as ORecipe

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SAMPLE_ROWS = 48
LLAMA = [("q_proj", 4096, 4096, 0.01), ("k_proj", 4096, 4096, 0.01), ("v_proj", 4096, 4096, 0.02),
         ("o_proj", 4096, 4096, 0.02), ("gate_proj", 11008, 4096, 0.04), ("up_proj", 11008, 4096, 0.04),
         ("down_proj", 4096, 11008, 0.04)]
LLAMA_CHAIN = [["q_proj", "k_proj", "v_proj"], ["o_proj"], ["gate_proj", "up_proj"], ["down_proj"]]


@pytest.fixture(scope="module")
def qx(cuda_dev):
    import paper_2505_07531_gb300.qx as qx

    qx._lib()
    return qx


def _orecipe(rec):
    return ORecipe(rec.bits, rec.group_size, "lut" if rec.kind == 1 else "uniform", 25)


def _sampled(qx, name_shapes, recipes, seed):
    """Quantize each full matrix on the GPU; the oracle quantizes its sampled rows."""
    out = {}
    for i, (nm, n, k, sigma) in enumerate(name_shapes):
        rec = recipes[nm]
        W = synth.student_t_weights_torch(n, k, sigma, seed=seed, stream=i, device="cuda")
        P = qx.quantize(W, rec)
        rows = np.sort(np.random.default_rng(seed * 100 + i).choice(n, size=SAMPLE_ROWS, replace=False))
        orec = _orecipe(rec)
        ref = oracle.quantize(W[torch.from_numpy(rows).cuda()].cpu().numpy(), orec)
        out[nm] = (P, rows, ref, orec, oracle.dequant(ref, orec, k))
        del W
    assert qx.device_status() == 0
    return out


def _check(y_rows, ref, orec, X, k, Wh):
    y_ref = oracle.gemm(ref, orec, X, k) if X.shape[0] > 1 else oracle.gemv(ref, orec, X, k)
    tol = oracle.tolerance(X, Wh)
    err = oracle.max_abs_err(y_rows.astype(np.float64), y_ref)
    assert np.all(err <= tol), (err, tol)


def _chain_graph(qx, chain, mats, xs, ys):
    s = torch.cuda.Stream()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        for names in chain:
            qx.gemv_multi([mats[nm][0] for nm in names], [xs[nm] for nm in names], outs=[ys[nm] for nm in names],
                          pdl=True)
    return g


@pytest.mark.parametrize("bits,g", [(4, 128), (3, 64)])
def test_llama_layer_uniform_decode_chain(qx, bits, g):
    rec = qx.Recipe(bits, g, qx.UNIFORM)
    mats = _sampled(qx, LLAMA, {nm: rec for nm, *_ in LLAMA}, seed=30 + bits)
    for batch in (1, 4, 16):
        xk = {k: synth.activations(batch, k, seed=batch, stream=600 + k) for k in (4096, 11008)}
        xs = {nm: torch.from_numpy(xk[k]).cuda() for nm, n, k, _ in LLAMA}
        ys = {nm: torch.full((batch, n), float("nan"), dtype=torch.float16, device="cuda") for nm, n, _, _ in LLAMA}
        g_ = _chain_graph(qx, LLAMA_CHAIN, mats, xs, ys)
        g_.replay()
        torch.cuda.synchronize()
        assert qx.device_status() == 0
        # the same chain with its CTAs balanced slice by slice: one launch, and
        # one balanced launch per group (bit for bit the same)
        yb = {}
        for mode in ("fused", "separate"):
            yb[mode] = {nm: torch.full((batch, n), float("nan"), dtype=torch.float16, device="cuda")
                        for nm, n, _, _ in LLAMA}
            qx.GemvChain([([mats[nm][0] for nm in names], [xs[nm] for nm in names], [yb[mode][nm] for nm in names])
                          for names in LLAMA_CHAIN], **{mode: True})()
        torch.cuda.synchronize()
        assert qx.device_status() == 0
        for nm, n, k, _ in LLAMA:
            P, rows, ref, orec, Wh = mats[nm]
            assert torch.equal(yb["fused"][nm], yb["separate"][nm]), nm
            for y in (ys[nm], yb["fused"][nm]):
                _check(y.float().cpu().numpy()[:, rows], ref, orec, xk[k], k, Wh)


def test_llava_language_layer_mixed_recipe_decode(qx):
    table = qx.recipe_table(os.path.join(ROOT, "paper_2505_07531_gb300", "recipes", "llava_v1_6_7b.json"))
    lang = table["language"]["matrices"]
    sig = {"q_proj": 0.01, "k_proj": 0.01, "v_proj": 0.02, "o_proj": 0.02}
    shapes = [(nm, n, k, sig.get(nm, 0.04)) for nm, n, k, _ in lang]
    mats = _sampled(qx, shapes, {nm: r for nm, _, _, r in lang}, seed=41)
    # launches group matrices that share the activations and the recipe
    chain = [["q_proj", "k_proj"], ["v_proj"], ["o_proj"], ["gate_proj", "up_proj"], ["down_proj"]]
    src = {"q_proj": 0, "k_proj": 0, "v_proj": 0, "o_proj": 1, "gate_proj": 2, "up_proj": 2, "down_proj": 3}
    xn = [synth.activations(1, k, seed=5, stream=700 + j) for j, k in enumerate((4096, 4096, 4096, 11008))]
    xs = {nm: torch.from_numpy(xn[src[nm]]).cuda() for nm, *_ in shapes}
    ys = {nm: torch.full((1, n), float("nan"), dtype=torch.float16, device="cuda") for nm, n, _, _ in shapes}
    g_ = _chain_graph(qx, chain, mats, xs, ys)
    g_.replay()
    torch.cuda.synchronize()
    assert qx.device_status() == 0
    for nm, n, k, _ in shapes:
        P, rows, ref, orec, Wh = mats[nm]
        _check(ys[nm].float().cpu().numpy()[:, rows], ref, orec, xn[src[nm]], k, Wh)


def test_clip_vision_layer_prefill_stacked_qkv(qx):
    table = qx.recipe_table(os.path.join(ROOT, "paper_2505_07531_gb300", "recipes", "llava_v1_6_7b.json"))
    vis = table["vision"]["matrices"]
    rec = vis[0][3]
    M = 576
    qkv = [m for m in vis if m[0] in ("q_proj", "k_proj", "v_proj")]
    rest = [m for m in vis if m[0] not in ("q_proj", "k_proj", "v_proj")]
    n3, k1 = sum(m[1] for m in qkv), qkv[0][2]
    shapes = [("qkv_proj", n3, k1, 0.02)] + [(nm, n, k, 0.02 if k == n else 0.04) for nm, n, k, _ in rest]
    mats = _sampled(qx, shapes, {nm: rec for nm, *_ in shapes}, seed=52)
    X = {k: synth.activations(M, k, seed=5, stream=800 + k) for k in (1024, 4096)}
    Xd = {k: torch.from_numpy(v).cuda() for k, v in X.items()}
    Ys = {nm: torch.full((M, n), float("nan"), dtype=torch.float16, device="cuda") for nm, n, _, _ in shapes}
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):  # sizes the stream's split-k workspace before capture
        for nm, n, k, _ in shapes:
            qx.gemm_splitk(mats[nm][0], Xd[k], out=Ys[nm], pdl=True)
    torch.cuda.synchronize()
    g_ = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_, stream=s):
        for nm, n, k, _ in shapes:
            qx.gemm_splitk(mats[nm][0], Xd[k], out=Ys[nm], pdl=True)
    for y in Ys.values():
        y.fill_(float("nan"))
    g_.replay()
    torch.cuda.synchronize()
    assert qx.device_status() == 0
    for nm, n, k, _ in shapes:
        P, rows, ref, orec, Wh = mats[nm]
        y_ref = oracle.gemm(ref, orec, X[k], k)
        # fp16 output: one more rounding of each result (2^-11 of |y|)
        tol = oracle.tolerance(X[k], Wh) + np.abs(y_ref).max(axis=1) * 2.0 ** -11
        err = oracle.max_abs_err(Ys[nm].float().cpu().numpy()[:, rows].astype(np.float64), y_ref)
        assert np.all(err <= tol), (nm, err.max(), tol.min())
