"""Pins for the oracle's GEMM (CPU only).

The float64 GEMM (plain definition) is checked against the exact factored GEMM
of App. B.1 Eq. (factor), and the exact GEMM against a direct element-by-element
sum in rational arithmetic -- three formulations that share no accumulation.
"""
from fractions import Fraction

import numpy as np

from paper_2605_31035_gb300 import synth


def _quant(oracle, t, mode=0):
    return oracle.quantize(synth.bf16_bits(t), mode=mode)


def test_exact_gemm_against_rationals(oracle):
    a = _quant(oracle, synth.activations(3, 64, 31, 32))
    b = _quant(oracle, synth.weights(4, 64, 33, 0.02, 0.5))
    C = oracle.gemm_exact(a, b)
    books = [[Fraction(oracle.fp4_value(f, p)) for p in range(8)] for f in (0, 1)]

    def deq(q, r, k):
        codes, scales, s32 = q
        s = int(scales[r, k // 16])
        nib = (int(codes[r, k // 2]) >> (4 * (k & 1))) & 0xF
        v = books[s >> 7][nib & 7] * (-1 if nib & 8 else 1)
        return v * Fraction(oracle.e4m3_value(s & 0x7F)) * Fraction(s32)

    for m in range(3):
        for n in range(4):
            ref = sum(deq(a, m, k) * deq(b, n, k) for k in range(64))
            assert C[m, n] == float(ref), (m, n)


def test_f64_gemm_against_exact(oracle):
    a = _quant(oracle, synth.activations(16, 512, 41, 42))
    b = _quant(oracle, synth.weights(24, 512, 43, 0.02, 0.5))
    Cd = oracle.gemm_f64(a, b)
    Ce = oracle.gemm_exact(a, b)
    A = oracle.dequant_rows_f64(a[0], a[1], a[2], range(16))
    B = oracle.dequant_rows_f64(b[0], b[1], b[2], range(24))
    D = np.abs(A) @ np.abs(B).T
    assert np.all(np.abs(Cd - Ce) <= 1e-12 * D + 1e-300)


def test_gemm_modes_and_zero(oracle):
    """E1M2-only operands are integers times scales; the f64 GEMM of an
    all-zero operand is exactly zero."""
    x = synth.activations(8, 128, 51, None)
    for mode in (1, 2):
        a = _quant(oracle, x, mode)
        b = _quant(oracle, synth.weights(8, 128, 52, 0.02), mode)
        assert np.allclose(oracle.gemm_f64(a, b), oracle.gemm_exact(a, b), rtol=1e-13, atol=0)
    z = oracle.quantize(np.zeros((8, 128), np.uint16))
    b = _quant(oracle, synth.weights(8, 128, 53, 0.02))
    assert not oracle.gemm_f64(z, b).any() and not oracle.gemm_exact(z, b).any()


def test_dequantize_definition(oracle):
    """Dequantize = sign * v * s8 * s32 rounded once to fp32 (App. B.2/B.3)."""
    codes, scales, s32 = _quant(oracle, synth.activations(4, 64, 61, 62))
    out = oracle.dequantize(codes, scales, s32)
    ref = oracle.dequant_rows_f64(codes, scales, s32, range(4)).astype(np.float32)
    assert np.array_equal(out, ref)
