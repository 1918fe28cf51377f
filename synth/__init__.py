"""Seeded synthetic inputs for the quantized-matmul path.

This module draws weight matrices and activations and nothing else: it holds none
of the quantization, packing or matmul arithmetic.  Both the CPU oracle's tests
and the GPU tests and benchmark take their inputs from here, so the two sides
always see the same fp16 values.

Distributions (stand-ins for the LLaVA / Llama / CLIP weights of the paper's
Section 3, which are not available here):

* weights: Student-t with nu = 4, scaled to standard deviation ``sigma``
  (Var t_4 = 2, so the draw is multiplied by sigma / sqrt(2)); the heavy tail
  mimics the peaked, long-tailed per-layer weight histograms of Section 2.1
  (Fig. 1).  t_4 is drawn exactly as Z / sqrt(V / 4) with V ~ chi^2_4 = 2 Gamma(2).
* optional outliers: floor(frac * N * K) distinct positions replaced by
  +-mult * sigma with a random sign (the "critical outliers" of Section 2.2).
* activations: N(0, 1).

Every array is rounded once to fp16 (round to nearest even) from float64.

Random streams: numpy's Philox counter-based generator keyed by (seed, stream);
``stream`` identifies the matrix (or activation) inside a configuration so that
each matrix has its own independent draw.  ``*_torch`` variants draw the same
distributions with torch's generator on any device; they are used where the
matrices are too large to draw on one host core in reasonable time (the full
language/vision stacks) and are not value-identical to the numpy variants.
"""
from __future__ import annotations

import math

import numpy as np

__all__ = [
    "rng",
    "student_t_weights",
    "activations",
    "student_t_weights_torch",
    "activations_torch",
]


def rng(seed: int, stream: int) -> np.random.Generator:
    """Counter-based generator for one (seed, stream) pair."""
    return np.random.Generator(np.random.Philox(key=[int(seed), int(stream)]))


def student_t_weights(
    n: int,
    k: int,
    sigma: float,
    seed: int = 0,
    stream: int = 0,
    outlier_frac: float = 0.0,
    outlier_mult: float = 10.0,
) -> np.ndarray:
    """[n][k] fp16 weights, Student-t(4) with standard deviation ``sigma``."""
    g = rng(seed, stream)
    z = g.standard_normal((n, k))
    v = 2.0 * g.standard_gamma(2.0, (n, k))  # chi^2 with 4 degrees of freedom
    w = z / np.sqrt(v / 4.0) * (sigma / math.sqrt(2.0))
    cnt = int(math.floor(outlier_frac * n * k))
    if cnt > 0:
        pos = g.choice(n * k, size=cnt, replace=False)
        sign = np.where(g.integers(0, 2, size=cnt) == 0, -1.0, 1.0)
        w.reshape(-1)[pos] = sign * outlier_mult * sigma
    return w.astype(np.float16)


def activations(b: int, k: int, seed: int = 0, stream: int = 1) -> np.ndarray:
    """[b][k] fp16 activations drawn from N(0, 1)."""
    return rng(seed, stream).standard_normal((b, k)).astype(np.float16)


def student_t_weights_torch(n, k, sigma, seed=0, stream=0, device="cpu",
                            outlier_frac=0.0, outlier_mult=10.0):
    """Same distribution as :func:`student_t_weights`, drawn with torch on ``device``."""
    import torch

    gen = torch.Generator(device=device)
    gen.manual_seed((int(seed) << 20) ^ int(stream))
    z = torch.randn((n, k), generator=gen, device=device, dtype=torch.float32)
    # chi^2_4 = -2 ln(U1 U2): sum of two independent Exp(1/2) variables.
    u = torch.rand((2, n, k), generator=gen, device=device, dtype=torch.float32)
    u = u.clamp_min_(1e-30)
    v = -2.0 * (torch.log(u[0]) + torch.log(u[1]))
    w = z / torch.sqrt(v / 4.0) * (sigma / math.sqrt(2.0))
    cnt = int(math.floor(outlier_frac * n * k))
    if cnt > 0:
        pos = torch.randperm(n * k, generator=gen, device=device)[:cnt]
        sign = torch.randint(0, 2, (cnt,), generator=gen, device=device).float() * 2 - 1
        w.view(-1)[pos] = sign * outlier_mult * sigma
    return w.to(torch.float16)


def activations_torch(b, k, seed=0, stream=1, device="cpu"):
    """[b][k] fp16 N(0, 1) activations drawn with torch on ``device``."""
    import torch

    gen = torch.Generator(device=device)
    gen.manual_seed((int(seed) << 20) ^ int(stream))
    return torch.randn((b, k), generator=gen, device=device, dtype=torch.float32).to(torch.float16)
