"""Pins of the oracle's 128-point rotation (reading R11) and of Algorithm 1
on fp32 inputs (CPU only).

The rotation is checked against an independent formulation, the dense
Sylvester matrix built by the Kronecker recursion H_2n = [[H, H], [H, -H]],
on inputs whose butterfly sums are exact in fp32 (so both sides round only
the final product by c), and against float64 on general inputs."""
import math
import struct
from fractions import Fraction

import numpy as np
import pytest

from paper_2605_31035_gb300 import synth

HERE = __import__("os").path.dirname(__import__("os").path.abspath(__file__))


def golden():
    d = {}
    for line in open(f"{HERE}/golden/rht_constants.txt"):
        line = line.split("#")[0].strip()
        if line:
            k, v = (t.strip() for t in line.split("="))
            d[k] = int(v, 0)
    return d


def sylvester(n=128):
    H = np.array([[1.0]])
    while H.shape[0] < n:
        H = np.block([[H, H], [H, -H]])
    return H


def c32():
    return np.float32(struct.unpack("<f", struct.pack("<I", golden()["c_bits"]))[0])


def bits_of(x):
    """bf16 bit patterns of values that are exact in bf16."""
    torch = __import__("torch")
    t = torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16)
    assert np.array_equal(t.float().numpy(), np.asarray(x, np.float32))
    return synth.bf16_bits(t)


def test_scale_constant_and_sylvester_matrix():
    from decimal import Decimal, getcontext
    getcontext().prec = 50
    exact = Decimal(1) / Decimal(128).sqrt()
    c = c32()
    u = struct.unpack("<I", struct.pack("<f", c))[0]
    dist = [abs(Decimal(float(struct.unpack("<f", struct.pack("<I", u + d))[0])) - exact) for d in (-1, 0, 1)]
    assert dist[1] < dist[0] and dist[1] < dist[2]
    H = sylvester()
    assert np.array_equal(H @ H.T, 128 * np.eye(128))


def test_unit_vectors_give_scaled_hadamard_columns(oracle):
    H, c = sylvester(), c32()
    x = np.zeros((5, 256), np.float32)
    js = [0, 1, 77, 127, 128 + 5]
    for r, j in enumerate(js):
        x[r, j] = 1.0
    y = oracle.rht(bits_of(x))
    for r, j in enumerate(js):
        k0 = (j // 128) * 128
        expect = (H[:, j - k0] * np.float64(c)).astype(np.float32)
        assert np.array_equal(y[r, k0:k0 + 128], expect)
        other = np.delete(np.arange(256), np.arange(k0, k0 + 128))
        assert np.all(y[r, other] == 0)


@pytest.mark.parametrize("with_signs", [False, True])
def test_butterfly_equals_dense_product_on_exact_inputs(oracle, with_signs):
    """Integer inputs in [-8, 8]: every butterfly sum is an exact fp32 integer,
    so the oracle must equal fl32((H v) * c) computed from the dense matrix."""
    rng = np.random.default_rng(7)
    x = rng.integers(-8, 9, (6, 384)).astype(np.float32)
    signs = rng.integers(0, 256, 16).astype(np.uint8) if with_signs else None
    y = oracle.rht(bits_of(x), signs)
    H, c = sylvester(), np.float64(c32())
    sgn = np.ones(128)
    if with_signs:
        sgn = np.where((signs[np.arange(128) // 8] >> (np.arange(128) % 8)) & 1, -1.0, 1.0)
    for r in range(x.shape[0]):
        for k0 in range(0, 384, 128):
            v = x[r, k0:k0 + 128].astype(np.float64) * sgn
            expect = ((H @ v) * c).astype(np.float32)   # H v exact, one rounding of the product
            assert np.array_equal(y[r, k0:k0 + 128], expect), (r, k0)


def test_rotation_close_to_float64_and_orthogonal(oracle):
    x = synth.activations(8, 1024, 31, 32)
    b = synth.bf16_bits(x)
    xf = (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    y = oracle.rht(b).astype(np.float64)
    H = sylvester() / math.sqrt(128.0)
    ref = np.concatenate([xf[:, k:k + 128] @ H.T for k in range(0, 1024, 128)], axis=1)
    l1 = np.concatenate([np.repeat(np.abs(xf[:, k:k + 128]).sum(1, keepdims=True), 128, 1)
                         for k in range(0, 1024, 128)], axis=1)
    assert np.all(np.abs(y - ref) <= 8 * 2.0 ** -24 * l1 / math.sqrt(128.0))
    assert np.allclose((y ** 2).sum(1), (xf ** 2).sum(1), rtol=1e-5)


def test_quantize_f32_equals_bf16_path_on_bf16_values(oracle):
    b = synth.bf16_bits(synth.activations(16, 512, 41, 42))
    xf = (b.astype(np.uint32) << 16).view(np.float32)
    for mode in (0, 1, 2):
        q1, q2 = oracle.quantize(b, mode), oracle.quantize_f32(xf, mode)
        assert np.array_equal(q1[0], q2[0]) and np.array_equal(q1[1], q2[1]) and q1[2] == q2[2]


def test_quantize_f32_brute_force(oracle):
    """fp32 inputs with full 24-bit significands (s32 = 1): every code is the
    codebook value nearest the fp32 quotient fl32(|a|/s8), ties to the even
    payload; the type bit follows the exact error comparison when it is not
    within fp32 noise."""
    rng = np.random.default_rng(9)
    rows, nb = 12, 8
    x = (rng.standard_normal((rows, nb * 16)) * rng.choice([0.3, 3.0, 30.0], (rows, 1))).astype(np.float32)
    x[0, 0] = 2688.0  # s32 = 1
    codes, scales, s32 = oracle.quantize_f32(x)
    assert s32 == 1.0
    books = [[oracle.fp4_value(f, p) for p in range(8)] for f in (0, 1)]
    for r in range(rows):
        for b in range(nb):
            a = x[r, b * 16:(b + 1) * 16]
            T = scales[r, b] >> 7
            s8 = np.float32(oracle.e4m3_value(scales[r, b] & 0x7F))
            for i in range(16):
                nib = (codes[r, b * 8 + i // 2] >> (4 * (i & 1))) & 0xF
                assert (nib >> 3) == (1 if math.copysign(1, a[i]) < 0 else 0)
                y = Fraction(float(np.float32(np.abs(a[i]) / s8))) if s8 > 0 else Fraction(0)
                d = [abs(Fraction(books[T][p]) - y) for p in range(8)]
                best = min(range(8), key=lambda p: (d[p], p % 2))
                if T == 0 or y <= 7:  # E1M2 saturates at 7
                    assert (nib & 7) == best, (r, b, i)
