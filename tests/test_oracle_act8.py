"""Pins of the oracle's W.A8 decode (Table 2: 8-bit per-token RTN activations;
Table 1: W3A8)."""
from fractions import Fraction

import numpy as np
import pytest

import oracle
from oracle import act8
from oracle.pack import Recipe
import synth


def test_activation_grid_closed_form():
    """x = j 2^-7 for j = -127..127: the scale is 2^-7 exactly and q = j."""
    j = np.arange(-127, 128)
    x = (j * 2.0 ** -7).astype(np.float16)[None, :]
    q, s = act8.quantize_act(x)
    assert s[0] == np.float32(2.0 ** -7) and np.array_equal(q[0].astype(int), j)


def test_activation_ties_round_half_to_even_and_dead_tokens():
    x = np.zeros((2, 8), dtype=np.float16)
    x[0, :4] = np.array([127, 2.5, 3.5, -2.5]) * 2.0 ** -7
    q, s = act8.quantize_act(x)
    assert list(q[0, :4]) == [127, 2, 4, -2]
    assert s[1] == 0 and not q[1].any()


def test_activation_codes_stay_in_range_and_reach_the_end():
    x = synth.activations(4, 512, seed=1, stream=1)
    q, s = act8.quantize_act(x)
    assert np.abs(q.astype(int)).max() == 127
    assert np.all(np.abs(q.astype(int)).max(axis=1) == 127)


def _tiny(bits, g):
    W = synth.student_t_weights(3, 128, 0.02, seed=bits + g, stream=2).astype(np.float16)
    r = Recipe(bits, g, "uniform")
    return W, r, oracle.quantize(W, r)


@pytest.mark.parametrize("bits,g", [(4, 64), (3, 32), (4, 128)])
def test_matmul_against_exact_rational_arithmetic(bits, g):
    W, r, p = _tiny(bits, g)
    x = synth.activations(2, 128, seed=3, stream=3)
    q, s = act8.quantize_act(x)
    qw = oracle.unpack_codes(p["codes"], bits, 128).astype(int)
    z = oracle.unpack_zeros(p["zeros"], 128 // g).astype(int)
    y = act8.gemv_a8(p, r, x, 128)
    for b in range(2):
        for n in range(3):
            tot = Fraction(0)
            for gi in range(128 // g):
                d = sum((qw[n, k] - z[n, gi]) * int(q[b, k]) for k in range(gi * g, gi * g + g))
                tot += Fraction(float(p["scales"][n, gi])) * d
            want = tot * Fraction(float(s[b]))
            assert abs(Fraction(y[b, n]) - want) <= abs(want) * Fraction(1, 10 ** 14) + Fraction(1, 10 ** 30)


def test_matmul_equals_dequantized_operands():
    """y = x_hat (q_w - z) s^T with both sides dequantized without rounding."""
    W, r, p = _tiny(4, 64)
    x = synth.activations(3, 128, seed=4, stream=4)
    q, s = act8.quantize_act(x)
    qw = oracle.unpack_codes(p["codes"], 4, 128).astype(np.float64)
    z = np.repeat(oracle.unpack_zeros(p["zeros"], 2).astype(np.float64), 64, axis=1)
    sw = np.repeat(p["scales"].astype(np.float64), 64, axis=1)
    want = act8.dequant_act(q, s) @ ((qw - z) * sw).T
    assert np.allclose(act8.gemv_a8(p, r, x, 128), want, rtol=1e-12, atol=0)


def test_lut_weights_have_no_integer_path():
    W = synth.student_t_weights(2, 128, 0.02, seed=5, stream=5).astype(np.float16)
    r = Recipe(3, 64, "lut")
    with pytest.raises(ValueError):
        act8.gemv_a8(oracle.quantize(W, r), r, synth.activations(1, 128, seed=1, stream=1), 128)


# ---------------------------------------------------------------- W.A8 prefill
def test_prefill_activations_closed_form():
    """x = j 2^-7: s = 2^-7, q = j and x_hat = x exactly, so the prefill is the
    plain product with x."""
    j = np.arange(-127, 129)[:256].reshape(2, 128)
    j[j > 127] = 0
    x = (j * 2.0 ** -7).astype(np.float16)
    q, s = act8.quantize_act(x)
    xh = act8.dequant_act_f16(q, s)
    assert np.array_equal(xh.view(np.uint16), x.view(np.uint16))
    W = synth.student_t_weights(24, 128, 0.02, seed=2, stream=3).astype(np.float16)
    assert np.array_equal(act8.gemm_a8(W, x), x.astype(np.float64) @ W.astype(np.float64).T)


def test_prefill_largest_activation_round_trips():
    """s_b = fp32(m / 127) is within 2^-24 of m / 127, so fp16(fp32(127 s_b))
    lands back on the fp16 value m: the largest |x| of every token is kept
    exactly (including fp16 subnormals)."""
    x = synth.activations(64, 256, seed=4, stream=5)
    x[3] *= np.float16(2.0 ** -20)  # a token in the subnormal range
    q, s = act8.quantize_act(x)
    xh = act8.dequant_act_f16(q, s)
    for b in range(x.shape[0]):
        i = int(np.argmax(np.abs(x[b].astype(np.float64))))
        assert abs(int(q[b, i])) == 127 and xh[b, i] == x[b, i], b


def test_prefill_matches_the_integer_decode_form_within_one_rounding():
    """For uniform weights the prefill and the decode (exact integer group
    sums) differ only by x_hat's rounding: |diff| <= 2^-11 sum_k |s_b q_k w_hat_k|."""
    k = 256
    r = Recipe(4, 64, "uniform")
    W = synth.student_t_weights(40, k, 0.02, seed=6, stream=7).astype(np.float16)
    x = synth.activations(5, k, seed=8, stream=9)
    x[2] = 0  # a dead token: zero output
    p = oracle.quantize(W, r)
    Wh = oracle.dequant(p, r, k)
    y_pre, y_dec = act8.gemm_a8(Wh, x), act8.gemv_a8(p, r, x, k)
    q, s = act8.quantize_act(x)
    bound = 2.0 ** -11 * (np.abs(act8.dequant_act(q, s)) @ np.abs(Wh.astype(np.float64)).T)
    assert np.all(np.abs(y_pre - y_dec) <= bound * (1 + 1e-9) + 1e-300)
    assert not y_pre[2].any()
    # a dropped scale or a transposed operand is far outside that bound
    assert np.abs(y_pre - y_dec).max() < 1e-2 * np.abs(y_dec).max()
