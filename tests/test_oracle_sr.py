"""Pins of stochastic rounding in the oracle (reading R13; the paper's SR
ablation appendix and Sec. 4.2 pre-training recipe).

* The generator: Philox4x32-10 against its published known-answer vectors
  (tests/golden/philox_kat.txt).
* The rounding: every code is one of the two codebook neighbours of
  m = |a| / s8; values on the grid round to themselves for every draw;
  scales and format choices equal Algorithm 1's; the frequency of rounding
  up matches (m - l) / (u - l) and the mean decoded value is unbiased, both
  within binomial bounds over many independent draws.
"""
import os

import numpy as np
import pytest

from paper_2605_31035_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def test_philox_known_answers(oracle):
    n = 0
    for line in open(os.path.join(GOLDEN, "philox_kat.txt")):
        if line.startswith("#") or not line.strip():
            continue
        w = [int(t, 16) for t in line.split()]
        assert list(oracle.philox4x32_10(w[0:4], w[4:6])) == w[6:10]
        n += 1
    assert n == 3


def test_uniform_definition(oracle):
    """eps of element e is word e % 4 of the block e // 4, top 24 bits."""
    seed, offset = 0x0123456789ABCDEF, 77
    for e in (0, 1, 5, 4095, (1 << 33) + 3):
        w = oracle.philox4x32_10([(e // 4) & 0xFFFFFFFF, (e // 4) >> 32, offset, 0],
                                 [seed & 0xFFFFFFFF, seed >> 32])
        assert oracle.sr_uniform(seed, offset, e) == float(w[e % 4] >> 8) * 2.0 ** -24


def _neighbours(oracle, fmt, m):
    vals = sorted(oracle.fp4_value(fmt, p) for p in range(8))
    lo = max(v for v in vals if v <= m)
    up = [v for v in vals if v > m]
    return lo, (up[0] if up else None)


def test_codes_are_neighbours_and_scales_follow_algorithm_1(oracle):
    x = synth.bf16_bits(synth.activations(24, 256, 61, 62))
    c0, s0, t0 = oracle.quantize(x)
    for seed in (1, 2, 3):
        c, s, t = oracle.quantize_sr(x, seed)
        assert t == t0 and np.array_equal(s, s0)
        xs = (x.astype(np.uint32) << 16).view(np.float32)
        for r in range(0, 24, 5):
            for k in range(0, 256, 7):
                sc = s[r, k // 16]
                fmt, s8 = sc >> 7, oracle.e4m3_value(sc & 0x7F)
                a = np.float32(xs[r, k] / np.float32(t))
                m = float(np.float32(abs(a) / np.float32(s8))) if s8 > 0 else 0.0
                nib = (c[r, k // 2] >> (4 * (k % 2))) & 0xF
                v = oracle.fp4_value(fmt, nib & 7)
                lo, up = _neighbours(oracle, fmt, m)
                assert v in (lo, up) and (nib >> 3) == (1 if np.signbit(xs[r, k]) else 0)


def test_grid_values_round_to_themselves(oracle):
    """A tensor whose values sit on the MixFP4 grid (s32 a power of two, block
    maxima 6 s8 or 7 s8) has m on the grid, so every draw gives Algorithm 1's
    codes."""
    rng = np.random.default_rng(4)
    e2m1 = np.array([0, .5, 1, 1.5, 2, 3, 4, 6], np.float32)
    rows = []
    for r in range(16):
        blk = rng.choice(e2m1, 16) * rng.choice([-1, 1], 16)
        blk[0] = 6.0
        rows.append(blk * np.float32(2.0 ** (r % 5 - 2)))
        ints = rng.integers(0, 8, 16).astype(np.float32) * rng.choice([-1, 1], 16)
        ints[0] = 7.0
        rows.append(ints * np.float32(2.0 ** (r % 3)))
    x = np.zeros((16, 48), np.float32)
    x[:, :32] = np.concatenate(rows).reshape(16, 32)
    x[0, 32] = 2688.0 / 64         # an anchor block of its own: s32 = 1/64
    import torch
    bits = torch.tensor(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    c0, s0, t0 = oracle.quantize(bits)
    assert np.log2(t0) == int(np.log2(t0))
    for seed in range(5):
        c, s, t = oracle.quantize_sr(bits, seed, offset=seed * 3)
        assert np.array_equal(c, c0) and np.array_equal(s, s0)


@pytest.mark.parametrize("fmt,m", [(0, 0.3), (0, 1.2), (0, 2.7), (0, 4.5), (1, 0.25), (1, 3.6), (1, 6.9)])
def test_frequency_of_rounding_up(oracle, fmt, m):
    """Over 4000 independent uniforms, the share of draws rounding up is within
    5 binomial standard deviations of (m - l) / (u - l)."""
    m = float(np.float32(m))
    lo, up = _neighbours(oracle, fmt, m)
    p = (m - lo) / (up - lo)
    n = 4000
    hits = sum(oracle.fp4_value(fmt, oracle.sr_payload(fmt, m, oracle.sr_uniform(9, 0, e))) == up
               for e in range(n))
    assert abs(hits / n - p) <= 5 * np.sqrt(p * (1 - p) / n) + 1e-9


def test_mean_decoded_value_is_unbiased(oracle):
    """Averaged over 400 seeds, each element's decoded SR value is within 5
    standard errors of the input it rounds, except where m = |a| / s8 lies at
    or above the codebook maximum, which saturates (the clamp of the paper's
    formula)."""
    x = synth.bf16_bits(synth.activations(2, 64, 63, None))
    _, s, t = oracle.quantize(x)
    acc = np.zeros((2, 64))
    n = 400
    for seed in range(n):
        c, sc, _ = oracle.quantize_sr(x, seed)
        acc += oracle.dequantize(c, sc, t)
    xs = (x.astype(np.uint32) << 16).view(np.float32)
    s8 = np.array([[oracle.e4m3_value(b & 0x7F) for b in row] for row in s]).repeat(16, axis=1)
    vmax = np.array([[7.0 if b >> 7 else 6.0 for b in row] for row in s]).repeat(16, axis=1)
    a = (xs / np.float32(t)).astype(np.float32)
    m = (np.abs(a) / s8.astype(np.float32)).astype(np.float32)
    inside = m < vmax
    assert inside.sum() > 100
    step = 2.0 * s8 * t                              # the widest gap of either codebook
    err = np.abs(acc / n - xs.astype(np.float64))
    assert np.all(err[inside] <= 5 * step[inside] / (2 * np.sqrt(n)) + 1e-6 * np.abs(xs[inside]))
