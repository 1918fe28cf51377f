"""CPU oracle for per-group 3/4-bit weight quantization fused into matmul.

TEST INFRASTRUCTURE ONLY.  This package is a plain, slow, obviously-correct
restatement of what the quantized-matmul path computes, written in numpy with
float64 wherever the definition does not fix another precision.  Only the test
suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may
import it; the product path (the CUDA library and its Python binding) never does
and shares no code with it.

Modules
-------
``quant``   uniform asymmetric RTN quantizer and the non-uniform Lloyd-Max LUT
            quantizer, per group of g consecutive weights along K
            (paper Section 2.2, Section 3.2 "Q4_0"/"Q4_K", Table 1 "G128").
``pack``    the packed byte layout of codes and zero-points (the paper fixes none;
            Section 2.4 says only that packing/unpacking kernels set decode time).
``matmul``  dequantize + float64 matvec / matmul and the parity tolerance.
``act8``    W.A8 decode: per-token 8-bit RTN activations against uniform
            weights with integer group sums (Tables 1-2: W3A8, W4A8).
``select``  per-matrix recipe selection by the exact Frobenius error under a
            bits-per-weight budget (Sections 2.2-2.3).
``q4x``     the Q4X shared-codebook quantizer (Section 3.2, Fig. 3a: groups of
            64, per-group fp16 scale and 2-bit book index, 4 learned books of 16
            centroids per matrix).

Every function names the passage (section, table or figure of the paper) it
follows; where the paper is silent the docstring states the reading taken.
"""
from .quant import (  # noqa: F401
    quantize_uniform,
    dequant_uniform,
    quantize_lut,
    dequant_lut,
    lloyd_max_trace,
)
from .pack import (  # noqa: F401
    Recipe,
    pack_codes,
    unpack_codes,
    pack_zeros,
    unpack_zeros,
    packed_sizes,
    quantize,
    dequant,
)
from .matmul import gemv, gemm, tolerance, max_abs_err  # noqa: F401
from .q4x import (  # noqa: F401
    quantize_q4x,
    dequant_q4x,
    pack_books,
    unpack_books,
    q4x_sizes,
    pack_codes4,
    unpack_codes4,
    pack_q4x,
    gemv_q4x,
)
from .select import select_recipe, sq_error_units, bits_per_weight  # noqa: F401
from .act8 import quantize_act, gemv_a8, dequant_act, dequant_act_f16, gemm_a8  # noqa: F401
