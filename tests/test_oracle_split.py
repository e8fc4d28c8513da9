"""Pins of the oracle's native-operand split (CPU only).

A MixFP4 operand is rewritten as main + residual E2M1 operands sharing its
block scales.  What fixes the split is arithmetic on the Table 1 codebooks:
for every nibble and type bit the two parts' decoded values must add up to
the MixFP4 value exactly, both parts must be E2M1 codes, and the residual's
magnitude is 0 or 1.  These are checked through the oracle's dequantizer,
which is pinned separately against the codebooks.
"""
import numpy as np
import pytest
import torch

from paper_2605_31035_gb300 import synth

pytestmark = pytest.mark.filterwarnings("ignore")


def _one_block(nibbles, scale_byte):
    codes = np.zeros((1, 8), np.uint8)
    for i, n in enumerate(nibbles):
        codes[0, i // 2] |= (n & 0xF) << (4 * (i % 2))
    return codes, np.array([[scale_byte]], np.uint8)


@pytest.mark.parametrize("T", [0, 1])
def test_parts_sum_to_mixfp4_value_for_every_nibble(oracle, T):
    nibbles = list(range(16))
    s8 = 0x38  # E4M3 1.0
    codes, scales = _one_block(nibbles, (T << 7) | s8)
    codes = np.tile(codes, (1, 8))          # K = 128: two 64-K scale tiles
    scales = np.tile(scales, (1, 8))
    main, res, _ = oracle.split_native(codes, scales)
    full = oracle.dequantize(codes, scales, 1.0)
    e2m1_scales = scales & 0x7F              # T = 0: both parts decode as E2M1
    m = oracle.dequantize(main, e2m1_scales, 1.0)
    r = oracle.dequantize(res, e2m1_scales, 1.0)
    assert np.array_equal(m.astype(np.float64) + r, full.astype(np.float64))
    assert set(np.abs(r).ravel().tolist()) <= {0.0, 1.0}
    if T == 0:
        assert np.array_equal(main, codes) and not res.any()
    else:
        # magnitudes 5 and 7 are the only ones outside the E2M1 codebook
        mags = np.abs(full[0, :16])
        assert np.array_equal(np.abs(r[0, :16]) == 1.0, np.isin(mags, [5.0, 7.0]))


def test_quantized_tensor_round_trip(oracle):
    x = synth.activations(37, 256, 4242, 4243)
    codes, scales, s32 = oracle.quantize(synth.bf16_bits(x))
    main, res, sf = oracle.split_native(codes, scales)
    rows = range(codes.shape[0])
    full = oracle.dequant_rows_f64(codes, scales, s32, rows)   # exact values
    plain = scales & 0x7F
    parts = oracle.dequant_rows_f64(main, plain, s32, rows) + oracle.dequant_rows_f64(res, plain, s32, rows)
    assert np.array_equal(parts, full)
    assert (scales >> 7).any() and res.any()  # both types occur in this tensor
    assert sf.size == oracle.sf_tiled_bytes(37, 256) == 256 * 16


def test_e2m1_only_tensor_has_no_residual(oracle):
    x = synth.activations(20, 512, 4244, None)
    codes, scales, _ = oracle.quantize(synth.bf16_bits(x), mode=1)
    main, res, _ = oracle.split_native(codes, scales)
    assert np.array_equal(main, codes) and not res.any()


def test_tiled_scales_hold_each_scale_once(oracle):
    """Every scale magnitude lands in exactly one byte of the tiled array and
    the padding rows are zero; which byte is the tensor core's layout."""
    rng = np.random.default_rng(7)
    rows, K = 300, 192
    codes = rng.integers(0, 256, (rows, K // 2), dtype=np.uint8)
    scales = rng.integers(1, 127, (rows, K // 16), dtype=np.uint8) | (rng.integers(0, 2, (rows, K // 16)) << 7).astype(np.uint8)
    _, _, sf = oracle.split_native(codes, scales)
    assert sf.size == 512 * 256 * K // 16 // 256 * 2 // 2
    assert np.array_equal(np.sort(sf[sf != 0]), np.sort((scales & 0x7F).ravel()))
