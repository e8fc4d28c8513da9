"""Pins for the oracle's number formats (CPU only).

The codebooks are checked against the values printed in Table 1 and Sec. 2.1 /
3.1 / App. B.2 (tests/golden), the E4M3 cast against PyTorch's float8_e4m3fn
conversion (a library routine), and FP4 rounding against an independent
midpoint-threshold formulation.
"""
import os
from fractions import Fraction

import numpy as np
import pytest
import torch

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _lines(name):
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                yield line.split()


def _payload(fmt, field):
    bits = field.replace(".", "")
    assert len(bits) == 3
    return int(bits, 2)


def test_table1_named_codes(oracle):
    """Table 1: every named E2M1 / E1M2 code decodes to the printed value."""
    seen = 0
    for parts in _lines("table1_fp4_formats.txt"):
        if parts[0] != "code":
            continue
        _, fmt, _, field, value = parts
        p = _payload(fmt, field)
        got = oracle.fp4_value(0, p) if fmt == "E2M1" else oracle.e1m2_stored_value(p)
        assert got == float(value), (fmt, field, got, value)
        seen += 1
    assert seen == 10


def test_codebooks_match_paper(oracle):
    """Sec. 2.1 / 3.1 / App. B.2 codebooks, by payload 0..7."""
    books = {parts[1]: [float(v) for v in parts[2:]]
             for parts in _lines("table1_fp4_formats.txt") if parts[0] == "codebook"}
    assert [oracle.fp4_value(0, p) for p in range(8)] == books["E2M1"]
    assert [oracle.e1m2_stored_value(p) for p in range(8)] == books["E1M2_stored"]
    assert [oracle.fp4_value(1, p) for p in range(8)] == books["E1M2_x2"]
    # Sec. 3.1: the x2 remapped E1M2 lattice is the NVINT4 lattice, and the
    # x2 value of a payload is the payload read as an unsigned integer.
    assert books["E1M2_x2"] == books["NVINT4"]
    assert [oracle.fp4_value(1, p) for p in range(8)] == [float(p) for p in range(8)]


def test_alg1_constants(oracle):
    c = {parts[0]: parts[1:] for parts in _lines("alg1_constants.txt")}
    d = int(c["tensor_divisor"][0])
    assert d == 6 * 448 == 7 * 384
    e4 = [parts for parts in _lines("alg1_constants.txt") if parts[0] == "e4m3"]
    for _, value, code in e4:
        assert oracle.e4m3_rne(float(value)) == int(code, 16)
        assert oracle.e4m3_value(int(code, 16)) == float(value)
    assert oracle.e4m3_rne(d / 6) == 0x7E and oracle.e4m3_rne(d / 7) == 0x7C


def test_e4m3_grid_definition(oracle):
    """Eq. 1 with W_E=4, W_M=3, bias 7: subnormal step 2^-9, max 448, 127 finite codes."""
    vals = [oracle.e4m3_value(c) for c in range(0x7F)]
    assert vals[0] == 0.0 and vals[1] == 2.0 ** -9 and vals[7] == 7 * 2.0 ** -9
    assert vals[8] == 2.0 ** -6 and vals[0x7E] == 448.0
    assert all(a < b for a, b in zip(vals, vals[1:]))


def _e4m3_probe_set():
    """All floats in [0, 464] whose low 16 mantissa bits are in a set that
    exercises the round and sticky bits, plus a seeded random sample."""
    hi = np.arange(0, 0x43E8 + 1, dtype=np.uint32) << 16
    lows = np.array([0x0000, 0x0001, 0x7FFF, 0x8000, 0x8001, 0xFFFF, 0x4000, 0xC000], np.uint32)
    bits = (hi[:, None] | lows[None, :]).ravel()
    rng = np.random.default_rng(7)
    bits = np.concatenate([bits, rng.integers(0, 0x43E80000, 200000, dtype=np.uint32)])
    f = bits.view(np.float32)
    return f[(f >= 0) & (f <= 464.0)]


def test_e4m3_rne_matches_torch(oracle):
    """The oracle's E4M3 cast agrees with torch float8_e4m3fn on [0, 464]."""
    f = _e4m3_probe_set()
    ref = torch.from_numpy(f).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    got = np.array([oracle.e4m3_rne(float(v)) for v in f], np.uint8)
    bad = np.nonzero(ref != got)[0]
    assert bad.size == 0, [(float(f[i]), int(ref[i]), int(got[i])) for i in bad[:5]]


def test_e4m3_saturates_at_448(oracle):
    for v in [448.0, 463.99, 464.0, 500.0, 1e6, 3.0e38]:
        assert oracle.e4m3_rne(v) == 0x7E


def _rne_by_midpoints(book, y):
    """Independent formulation: walk the sorted codebook, round at midpoints,
    break exact midpoint ties toward the even payload, clamp at the top."""
    for p in range(7):
        lo, hi = Fraction(book[p]), Fraction(book[p + 1])
        mid = (lo + hi) / 2
        if y < mid:
            return p
        if y == mid:
            return p if p % 2 == 0 else p + 1
    return 7


@pytest.mark.parametrize("fmt", [0, 1])
def test_fp4_rne_against_midpoints(oracle, fmt):
    book = [oracle.fp4_value(fmt, p) for p in range(8)]
    ys = set()
    for p in range(8):
        for v in (book[p], (book[p] + book[min(p + 1, 7)]) / 2):
            f = np.float32(v)
            ys.update([float(f), float(np.nextafter(f, np.float32(0))), float(np.nextafter(f, np.float32(100)))])
    rng = np.random.default_rng(fmt)
    ys.update(float(v) for v in rng.uniform(0, 9, 5000).astype(np.float32))
    ys.update([0.0, 6.5, 7.49, 7.5, 8.0, 1e9])
    for y in sorted(ys):
        if y < 0:
            continue
        assert oracle.fp4_rne(fmt, y) == _rne_by_midpoints(book, Fraction(y)), (fmt, y)


def test_e2m1_rounding_ties_to_even(oracle):
    # E2M1 midpoints and their even-payload results (Sec. 2.1 codebook).
    expect = {0.25: 0, 0.75: 2, 1.25: 2, 1.75: 4, 2.5: 4, 3.5: 6, 5.0: 6}
    for y, p in expect.items():
        assert oracle.fp4_rne(0, y) == p
    # E1M2 (x2): half-integers round to the even integer.
    for k in range(7):
        assert oracle.fp4_rne(1, k + 0.5) == (k if k % 2 == 0 else k + 1)
    assert oracle.fp4_rne(1, 7.5) == 7 and oracle.fp4_rne(0, 7.0) == 7
