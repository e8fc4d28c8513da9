"""Pins of the training-side quantizer orientations in the oracle.

* quantize_2d (Algorithm 1 with 16 x 16 weight blocks, Sec. 3.2; reading R12)
  is pinned against the 1D oracle on tiles that reduce to one row (identical
  rows, a single nonzero row), against exact rational arithmetic on small
  dyadic tiles, and by the sign and power-of-two invariances.
* transpose_2d is pinned through the dequantizer: the transposed codes decode
  to the transpose of the decoded tensor, bit for bit.
* quantize_colwise is by definition the row-wise oracle on the transpose;
  its test checks the orientation of the output against single columns.
"""
import math
from fractions import Fraction

import numpy as np
import pytest
import torch

from paper_2605_31035_gb300 import synth


def bf16_bits_of(values):
    t = torch.tensor(np.asarray(values, np.float32)).to(torch.bfloat16)
    assert np.array_equal(t.float().numpy(), np.asarray(values, np.float32)), "value not exact in bf16"
    return t.view(torch.int16).numpy().view(np.uint16)


def test_2d_tiles_of_identical_rows_match_1d(oracle):
    """A tile whose 16 rows are equal has the row's block max, and its tree
    sum is 16 x the row's error exactly, so codes and scale bytes equal the 1D
    quantization of the row (with the same s32)."""
    base = synth.bf16_bits(synth.activations(2, 256, 41, 42))
    x = np.repeat(base, 16, axis=0)                 # tile 0: row 0 x 16, tile 1: row 1 x 16
    for mode in (0, 1, 2):
        c2, s2, t2 = oracle.quantize_2d(x, mode)
        c1, s1, t1 = oracle.quantize(base, mode, s32=t2)
        assert t2 == oracle.quantize(x, mode)[2]
        assert np.array_equal(c2, np.repeat(c1, 16, axis=0))
        assert np.array_equal(s2, np.repeat(s1, 16, axis=0))


def test_2d_single_nonzero_row_matches_1d(oracle):
    """Zero rows add exact zeros to the tile's max and error, so a tile with one
    nonzero row quantizes that row as the 1D oracle does; a 1-row tensor (a
    ragged tile of one row) likewise."""
    row = synth.bf16_bits(synth.activations(1, 512, 43, 44))
    x = np.zeros((16, 512), np.uint16)
    x[5] = row[0]
    for mode in (0, 1, 2):
        c2, s2, t2 = oracle.quantize_2d(x, mode)
        c1, s1, t1 = oracle.quantize(row, mode)
        assert t2 == t1
        assert np.array_equal(c2[5], c1[0]) and np.array_equal(s2[5], s1[0])
        assert np.all(c2[np.arange(16) != 5] == 0)
        assert np.all(s2 == s2[5])
        c3, s3, t3 = oracle.quantize_2d(row, mode)
        assert t3 == t1 and np.array_equal(c3, c1) and np.array_equal(s3, s1)


def _exact_tile_error(tile, s8, fmt, book):
    out = Fraction(0)
    for a in tile.ravel():
        y = Fraction(abs(float(a)))
        best = min(range(8), key=lambda p: (abs(Fraction(book[p]) * Fraction(s8) - y), p % 2))
        out += (Fraction(book[best]) * Fraction(s8) - y) ** 2
    return out


def test_2d_brute_force_dyadic_tiles(oracle):
    """With s32 = 1: each tile's scale byte is the torch E4M3 cast of
    tile_max / c, every code is the nearest codebook value (ties to the even
    payload) of |a| / s8, and the chosen format has the smaller exact tile
    error whenever the two differ by more than fp32 noise (ties -> E1M2)."""
    rng = np.random.default_rng(9)
    grid = np.array([0, 0.25, 0.5, 0.75, 1, 1.25, 1.5, 2, 2.5, 3, 3.5, 4, 5, 6, 7, 8, 10, 12], np.float32)
    rows, K = 48, 64
    x = (rng.choice(grid, (rows, K)) * rng.choice([-1, 1], (rows, K))).astype(np.float32)
    scale_t = 2.0 ** rng.integers(-3, 3, (rows // 16, K // 16))   # per-tile power of two
    x = (x.reshape(rows // 16, 16, K // 16, 16) * scale_t[:, None, :, None]).reshape(rows, K).astype(np.float32)
    x[0, 0] = 2688.0                                              # s32 = 1 exactly
    bits = bf16_bits_of(x)
    codes, scales, s32 = oracle.quantize_2d(bits)
    assert s32 == 1.0
    books = [[oracle.fp4_value(f, p) for p in range(8)] for f in (0, 1)]
    checked = 0
    for t in range(rows // 16):
        for b in range(K // 16):
            tile = x[16 * t:16 * t + 16, 16 * b:16 * b + 16].astype(np.float64)
            sb = scales[16 * t:16 * t + 16, b]
            assert np.all(sb == sb[0])
            T, s8 = sb[0] >> 7, oracle.e4m3_value(sb[0] & 0x7F)
            B = np.float32(np.abs(tile).max())
            ref = torch.tensor([float(B / np.float32(7.0 if T else 6.0))], dtype=torch.float32)
            assert int(ref.to(torch.float8_e4m3fn).view(torch.uint8)) == sb[0] & 0x7F
            for i in range(16):
                for k in range(16):
                    nib = (codes[16 * t + i, 8 * b + k // 2] >> (4 * (k & 1))) & 0xF
                    a = tile[i, k]
                    assert (nib >> 3) == (1 if math.copysign(1, a) < 0 else 0)
                    y = Fraction(abs(float(a))) / Fraction(s8) if s8 > 0 else Fraction(0)
                    best = min(range(8), key=lambda p: (abs(Fraction(books[T][p]) - y), p % 2))
                    assert (nib & 7) == best
            errs = []
            for fmt in (0, 1):
                s8f = oracle.e4m3_value(oracle.e4m3_rne(float(np.float32(B / np.float32(6.0 if fmt == 0 else 7.0)))))
                errs.append(_exact_tile_error(tile, s8f, fmt, books[fmt]))
            if errs[0] != errs[1] and abs(errs[0] - errs[1]) > Fraction(1, 10 ** 5) * max(errs):
                assert T == (0 if errs[0] < errs[1] else 1)
                checked += 1
            if errs[0] == errs[1]:
                assert T == 1
    assert checked > 0


def test_2d_random_tiles_codes_and_choice(oracle):
    """Full-precision tiles (Student-t values with outlier columns, computed
    s32): every code is reading R4 applied to the fp32 quotient fl32(a / s8)
    with a = fl32(|x| / s32), the scale byte is the E4M3 cast of
    fl32(tile_max / c), and the chosen format has the smaller exact tile
    error (rational sum over the 256 elements of the R4 codes) whenever the
    two exact errors differ by more than 64 u of the larger: the tree of
    fp32 row sums cannot reverse such a comparison."""
    rng = np.random.default_rng(21)
    rows, K = 64, 96
    z = rng.standard_normal((4, rows, K)).astype(np.float32)
    x = z[0] / np.sqrt((z[1] ** 2 + z[2] ** 2 + z[3] ** 2) / 3.0) * 0.5
    x[:, rng.integers(0, K, 3)] *= 30.0
    bits = torch.tensor(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    xf = (bits.astype(np.uint32) << 16).view(np.float32)
    codes, scales, s32 = oracle.quantize_2d(bits)
    books = [[oracle.fp4_value(f, p) for p in range(8)] for f in (0, 1)]
    u = Fraction(1, 2 ** 24)

    def r4(yq, book):
        yy = Fraction(float(yq))
        return min(range(8), key=lambda p: (abs(Fraction(book[p]) - yy), p % 2))

    decided = 0
    for t in range(rows // 16):
        for b in range(K // 16):
            a = np.abs(xf[16 * t:16 * t + 16, 16 * b:16 * b + 16]) / np.float32(s32)   # fl32(|x| / s32)
            B = np.float32(a.max())
            sb = scales[16 * t:16 * t + 16, b]
            assert np.all(sb == sb[0])
            T = sb[0] >> 7
            errs, s8s = [], []
            for fmt in (0, 1):
                code = oracle.e4m3_rne(float(np.float32(B / np.float32(6.0 if fmt == 0 else 7.0))))
                s8 = oracle.e4m3_value(code)
                s8s.append((code, s8))
                e = Fraction(0)
                for v in a.ravel():
                    q = r4(np.float32(v) / np.float32(s8), books[fmt]) if s8 > 0 else 0
                    e += (Fraction(books[fmt][q]) * Fraction(s8) - Fraction(float(v))) ** 2
                errs.append(e)
            assert sb[0] & 0x7F == s8s[T][0]
            s8 = s8s[T][1]
            for i in range(16):
                for k in range(16):
                    nib = (codes[16 * t + i, 8 * b + k // 2] >> (4 * (k & 1))) & 0xF
                    q = r4(np.float32(a[i, k]) / np.float32(s8), books[T]) if s8 > 0 else 0
                    assert (nib & 7) == q, (t, b, i, k)
            if abs(errs[0] - errs[1]) > 64 * u * max(errs):
                assert T == (0 if errs[0] < errs[1] else 1), (t, b)
                decided += 1
    assert decided >= (rows // 16) * (K // 16) // 2


def test_2d_negation_and_power_of_two(oracle):
    """Negating X flips only the nibble sign bits; X x 2^k leaves codes and
    scale bytes unchanged and scales s32 by 2^k."""
    x = synth.activations(40, 128, 45, 46)
    c, s, t = oracle.quantize_2d(synth.bf16_bits(x))
    cn, sn, tn = oracle.quantize_2d(synth.bf16_bits(-x))
    assert tn == t and np.array_equal(sn, s) and np.array_equal(cn, c ^ 0x88)
    c4, s4, t4 = oracle.quantize_2d(synth.bf16_bits(x * 4))
    assert t4 == 4 * t and np.array_equal(c4, c) and np.array_equal(s4, s)


def test_transpose_2d_through_the_decoder(oracle):
    """The transposed codes and scales decode to the transpose of the decoded
    tensor bit for bit; transposing twice is the identity; a 1D-quantized
    tensor whose tile rows differ in scale is rejected."""
    x = synth.bf16_bits(synth.weights(48, 80, 47, 0.02, 0.5))
    c, s, t = oracle.quantize_2d(x)
    ct, st = oracle.transpose_2d(c, s)
    assert ct.shape == (80, 24) and st.shape == (80, 3)
    assert np.array_equal(oracle.dequantize(ct, st, t), oracle.dequantize(c, s, t).T)
    c2, s2 = oracle.transpose_2d(ct, st)
    assert np.array_equal(c2, c) and np.array_equal(s2, s)
    c1, s1, _ = oracle.quantize(x)
    if not np.all(s1.reshape(3, 16, 5) == s1.reshape(3, 16, 5)[:, :1, :]):
        with pytest.raises(ValueError):
            oracle.transpose_2d(c1, s1)


def test_colwise_orientation(oracle):
    """Column c of an [R, C] tensor quantized down its rows (with the tensor's
    s32) gives row c of the column-wise codes and scales."""
    x = synth.bf16_bits(synth.activations(64, 24, 48, 49))
    ct, st, t = oracle.quantize_colwise(x)
    assert ct.shape == (24, 32) and st.shape == (24, 4)
    amax = np.float32(np.abs((x.astype(np.uint32) << 16).view(np.float32)).max())
    assert np.float32(t) == np.float32(amax / np.float32(2688.0))
    for c in (0, 7, 23):
        cc, sc, _ = oracle.quantize(np.ascontiguousarray(x[:, c][None, :]), s32=t)
        assert np.array_equal(ct[c], cc[0]) and np.array_equal(st[c], sc[0])
