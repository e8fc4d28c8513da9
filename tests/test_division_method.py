"""Host checks of the division methods inside the CUDA quantizer (CPU only).

The quantizer evaluates every IEEE division of Algorithm 1 (x/s32, B/6, B/7,
|a|/s8) without a divide instruction: with the two-instruction division by a
known divisor where it is exact, and with Markstein's fma correction for the
few tensor scales s32 where the former is not.  tests/native/markstein_check.c
enumerates every significand pair the quantizer can present (bf16 numerators x
all fp32 s32 significands, all fp32 numerators x all E4M3 significands, B/6
and B/7) plus exponent edges down to 2^-102 and requires bit equality with C's
IEEE '/'; tests/native/known_divisor_check.c does the same for the other
method and its acceptance rule.
"""
import os
import shutil
import subprocess

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)


@pytest.mark.skipif(shutil.which("gcc") is None, reason="needs gcc")
def test_markstein_division_matches_ieee(tmp_path):
    exe = tmp_path / "markstein_check"
    subprocess.check_call(["gcc", "-O2", "-ffp-contract=off", "-fopenmp", "-std=c11",
                           os.path.join(HERE, "native", "markstein_check.c"), "-o", str(exe), "-lm"])
    res = subprocess.run([str(exe)], capture_output=True, text=True, timeout=600)
    assert res.returncode == 0, res.stdout + res.stderr
    lines = [l for l in res.stdout.splitlines() if "mismatches=" in l]
    assert len(lines) == 7 and all(l.endswith("mismatches=0") for l in lines), res.stdout


@pytest.mark.skipif(shutil.which("gcc") is None, reason="needs gcc")
def test_known_divisor_division_matches_ieee(tmp_path):
    """The two-instruction division RN(a*zh + RN(a*zl)) (Brisebarre, Muller,
    Raina 2004) that the quantizer uses for |a|/s8, B/6, B/7 and, when its
    run-time check accepts s32, for x/s32.  tests/native/known_divisor_check.c
    enumerates every significand pair for the fixed divisors, replays the
    kernel's acceptance rule for every fp32 significand of s32, and requires
    the IEEE quotient at other exponents for every accepted one."""
    exe = tmp_path / "known_divisor_check"
    subprocess.check_call(["gcc", "-O2", "-ffp-contract=off", "-fopenmp", "-std=c11",
                           os.path.join(HERE, "native", "known_divisor_check.c"), "-o", str(exe), "-lm"])
    res = subprocess.run([str(exe)], capture_output=True, text=True, timeout=600)
    assert res.returncode == 0, res.stdout + res.stderr
    lines = [l for l in res.stdout.splitlines() if "mismatches=" in l]
    assert len(lines) == 3 and all(l.endswith("mismatches=0") for l in lines), res.stdout
    rejected = int(res.stdout.split("rejected=")[1].split()[0])
    assert 0 < rejected < 1000, res.stdout  # a handful of s32 significands fall back to Markstein


def _rn32_bits(x):
    """Binary32 nearest to the rational x (ties to even), as bits."""
    from fractions import Fraction
    import struct
    f = np.float32(float(x))
    cands = [np.nextafter(f, np.float32(-np.inf)), f, np.nextafter(f, np.float32(np.inf))]
    bits = [struct.unpack("<I", struct.pack("<f", c))[0] for c in cands]
    best = min(range(3), key=lambda i: (abs(Fraction(float(cands[i])) - x), bits[i] & 1))
    return bits[best]


def test_block_scale_divisor_constants():
    """The fixed (zh, zl) pairs of the divisors 6 and 7 in quant_core.cuh are
    RN(1/b) and RN(RN(1 - b zh) / b), recomputed here in exact rational
    arithmetic."""
    import re
    import struct
    from fractions import Fraction
    src = open(os.path.join(ROOT, "paper_2605_31035_gb300", "csrc", "quant_core.cuh")).read()
    for b in (6, 7):
        zh_bits = int(re.search(rf"kZh{b}Bits = (0x[0-9a-f]+)u", src).group(1), 16)
        zl_bits = int(re.search(rf"kZl{b}Bits = (0x[0-9a-f]+)u", src).group(1), 16)
        assert zh_bits == _rn32_bits(Fraction(1, b))
        zh = Fraction(struct.unpack("<f", struct.pack("<I", zh_bits))[0])
        r_bits = _rn32_bits(1 - b * zh)
        r = Fraction(struct.unpack("<f", struct.pack("<I", r_bits))[0])
        assert zl_bits == _rn32_bits(r / b)
