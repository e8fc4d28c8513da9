"""Host check of the division method inside the CUDA quantizer (CPU only).

The quantizer evaluates every IEEE division of Algorithm 1 (x/s32, B/6, B/7,
|a|/s8) with Markstein's fma correction instead of a divide instruction.
tests/native/markstein_check.c enumerates every significand pair the
quantizer can present (bf16 numerators x all fp32 s32 significands, all fp32
numerators x all E4M3 significands, B/6 and B/7) plus exponent edges down to
2^-102 and requires bit equality with C's IEEE '/'.
"""
import os
import shutil
import subprocess

import pytest

HERE = os.path.dirname(os.path.abspath(__file__))


@pytest.mark.skipif(shutil.which("gcc") is None, reason="needs gcc")
def test_markstein_division_matches_ieee(tmp_path):
    exe = tmp_path / "markstein_check"
    subprocess.check_call(["gcc", "-O2", "-ffp-contract=off", "-fopenmp", "-std=c11",
                           os.path.join(HERE, "native", "markstein_check.c"), "-o", str(exe), "-lm"])
    res = subprocess.run([str(exe)], capture_output=True, text=True, timeout=600)
    assert res.returncode == 0, res.stdout + res.stderr
    lines = [l for l in res.stdout.splitlines() if "mismatches=" in l]
    assert len(lines) == 7 and all(l.endswith("mismatches=0") for l in lines), res.stdout
