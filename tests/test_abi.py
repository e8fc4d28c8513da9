"""C ABI of libmixfp4.so (CPU only): the library builds and loads, exports
every entry point include/mixfp4.h declares, and rejects invalid arguments
with the documented status codes before touching the GPU."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2605_31035_gb300 import build, ops
    build.build()
    return ops.lib()


def declared_functions():
    text = open(os.path.join(ROOT, "include", "mixfp4.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(mixfp4_\w+)\s*\(", text)))


def test_exports_every_declared_symbol(lib):
    names = declared_functions()
    assert {"mixfp4_quantize", "mixfp4_dequantize", "mixfp4_gemm"} <= set(names)
    for n in names:
        assert hasattr(lib, n), n


def test_version_and_status_strings(lib):
    assert lib.mixfp4_version() >= 100
    for code in range(0, -8, -1):
        assert lib.mixfp4_status_string(code)
    assert lib.mixfp4_status_string(0) == b"ok"


def test_quantize_validation(lib):
    fake = ctypes.c_void_p(1 << 20)  # never dereferenced: validation fails first
    ws = ctypes.c_void_p(1 << 21)
    q = lib.mixfp4_quantize
    assert q(fake, 7, 4, 32, 32, fake, fake, fake, ws, 0, 0, None) == -4        # dtype
    assert q(fake, 0, 4, 24, 24, fake, fake, fake, ws, 0, 0, None) == -2        # K % 16
    assert q(fake, 0, 4, 32, 16, fake, fake, fake, ws, 0, 0, None) == -2        # ldx < K
    assert q(fake, 0, -1, 32, 32, fake, fake, fake, ws, 0, 0, None) == -2       # rows < 0
    assert q(fake, 0, 4, 32, 32, fake, fake, fake, ws, 4, 0, None) == -7        # mode
    assert q(fake, 0, 4, 32, 32, fake, fake, fake, ws, 0, 2, None) == -7        # scale flag
    assert q(None, 0, 4, 32, 32, fake, fake, fake, ws, 0, 0, None) == -1        # x null
    assert q(fake, 0, 4, 32, 32, fake, fake, fake, None, 0, 0, None) == -1      # workspace
    assert q(ctypes.c_void_p((1 << 20) + 2), 0, 4, 32, 32, fake, fake, fake, ws, 0, 0, None) == -3
    assert q(fake, 0, 4, 32, 40, fake, fake, fake, ws, 0, 1, None) == -3        # ldx % 16


def test_quantize_rht_validation(lib):
    fake = ctypes.c_void_p(1 << 20)
    ws = ctypes.c_void_p(1 << 21)
    q = lib.mixfp4_quantize_rht
    assert q(fake, 0, 4, 64, 64, None, fake, fake, fake, ws, 0, 0, None) == -2       # K % 128
    assert q(fake, 7, 4, 128, 128, None, fake, fake, fake, ws, 0, 0, None) == -4     # dtype
    assert q(fake, 0, 4, 128, 128, None, fake, fake, fake, None, 0, 0, None) == -1   # workspace
    assert q(fake, 0, 4, 128, 128, None, fake, fake, fake, ws, 5, 0, None) == -7     # mode
    assert q(ctypes.c_void_p((1 << 20) + 2), 0, 4, 128, 128, None, fake, fake, fake, ws, 0, 0, None) == -3


def test_dequantize_and_gemm_validation(lib):
    fake = ctypes.c_void_p(1 << 20)
    assert lib.mixfp4_dequantize(fake, fake, fake, 4, 24, fake, None) == -2
    assert lib.mixfp4_dequantize(None, fake, fake, 4, 32, fake, None) == -1
    assert lib.mixfp4_dequantize(fake, fake, fake, 4, 32, ctypes.c_void_p((1 << 20) + 16), None) == -3
    g = lib.mixfp4_gemm
    assert g(fake, fake, fake, fake, fake, fake, 4, 4, 128, fake, 4, None, None) == -2   # K % 256
    assert g(fake, fake, fake, fake, fake, fake, 4, 8, 256, fake, 4, None, None) == -2   # ldc < N
    assert g(fake, fake, fake, fake, fake, fake, -1, 4, 256, fake, 4, None, None) == -2
    assert g(fake, fake, fake, fake, fake, fake, 4, 4, 256, None, 4, None, None) == -1
    assert g(fake, fake, fake, fake, fake, fake, 4, 4, 256, ctypes.c_void_p((1 << 20) + 2), 4, None, None) == -3
    assert g(None, fake, fake, fake, fake, fake, 4, 4, 256, fake, 4, None, None) == -1


def test_header_documents_each_entry_point():
    text = open(os.path.join(ROOT, "include", "mixfp4.h")).read()
    for name in ("mixfp4_quantize", "mixfp4_dequantize", "mixfp4_gemm"):
        block = text[:text.index(f"int {name}(")]
        doc = block[block.rindex("/*"):]
        assert any(s in doc for s in ("Algorithm 1", "App. B")), name
        assert "device" in doc.lower()


def test_product_path_has_no_oracle_or_cpu_fallback():
    pkg = os.path.join(ROOT, "paper_2605_31035_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                src = open(os.path.join(dirpath, f)).read()
                assert "import oracle" not in src and "from oracle" not in src, f
                assert "liboracle" not in src, f


def test_native_variant_validation(lib):
    fake = ctypes.c_void_p(1 << 20)
    odd = ctypes.c_void_p((1 << 20) + 8)
    s = lib.mixfp4_split_native
    assert s(fake, fake, 4, 96, fake, fake, fake, None) == -2          # K % 64
    assert s(fake, fake, -1, 64, fake, fake, fake, None) == -2
    assert s(fake, fake, 4, 64, fake, None, fake, None) == -1          # residual output
    assert s(fake, fake, 4, 64, fake, fake, odd, None) == -3           # tiled scales alignment
    assert s(fake, fake, 0, 64, None, None, None, None) == 0           # empty: nothing to do
    g = lib.mixfp4_gemm_native
    args = lambda **kw: [kw.get(k, fake) for k in ("am", "ar", "asf", "ats", "bm", "br", "bsf", "bts")]
    assert g(*args(), 4, 4, 128, fake, 4, None, None) == -2                      # K % 256
    assert g(*args(), 4, 8, 256, fake, 4, None, None) == -2                      # ldc < N
    assert g(*args(), 4, 4, 256, None, 4, None, None) == -1                      # C
    assert g(*args(am=None), 4, 4, 256, fake, 4, None, None) == -1               # A main codes
    assert g(*args(bsf=None), 4, 4, 256, fake, 4, None, None) == -1              # B scales
    assert g(*args(ar=odd), 4, 4, 256, fake, 4, None, None) == -3                # residual alignment
    assert g(*args(), 0, 4, 256, fake, 4, None, None) == 0                       # empty M


def test_training_orientation_validation(lib):
    fake = ctypes.c_void_p(1 << 20)
    ws = ctypes.c_void_p(1 << 21)
    c = lib.mixfp4_quantize_colwise
    assert c(fake, 0, 24, 32, 32, fake, fake, fake, ws, 0, 0, None) == -2       # R % 16
    assert c(fake, 0, 32, 24, 32, fake, fake, fake, ws, 0, 0, None) == -2       # C % 16
    assert c(fake, 0, 32, 32, 16, fake, fake, fake, ws, 0, 0, None) == -2       # ldx < C
    assert c(fake, 7, 32, 32, 32, fake, fake, fake, ws, 0, 0, None) == -4       # dtype
    assert c(fake, 0, 32, 32, 32, fake, fake, fake, None, 0, 0, None) == -1     # workspace
    assert c(fake, 0, 32, 32, 32, fake, fake, fake, ws, 4, 0, None) == -7       # mode
    assert c(ctypes.c_void_p((1 << 20) + 16), 0, 32, 32, 32, fake, fake, fake, ws, 0, 0, None) == -3
    q = lib.mixfp4_quantize_2d
    assert q(fake, 0, 5, 24, 24, fake, fake, fake, ws, 0, 0, None) == -2        # K % 16
    assert q(fake, 0, 5, 32, 32, None, fake, fake, ws, 0, 0, None) == -1        # codes
    assert q(fake, 0, 5, 32, 40, fake, fake, fake, ws, 0, 1, None) == -3        # ldx % 16
    assert q(fake, 0, 5, 32, 32, fake, fake, fake, ws, 0, 3, None) == -7        # scale flag
    t = lib.mixfp4_transpose_2d
    assert t(fake, fake, 24, 32, fake, fake, None) == -2                        # rows % 16
    assert t(fake, fake, 32, 24, fake, fake, None) == -2                        # K % 16
    assert t(fake, None, 32, 32, fake, fake, None) == -1
    assert t(fake, fake, 32, 32, ctypes.c_void_p((1 << 20) + 4), fake, None) == -3
    assert t(fake, fake, 0, 32, None, None, None) == 0                          # empty


def test_stochastic_rounding_validation(lib):
    fake = ctypes.c_void_p(1 << 20)
    ws = ctypes.c_void_p(1 << 21)
    q = lib.mixfp4_quantize_sr
    assert q(fake, 0, 4, 24, 24, fake, fake, fake, ws, 0, 0, 1, 0, None) == -2       # K % 16
    assert q(fake, 0, 4, 32, 32, fake, fake, fake, None, 0, 0, 1, 0, None) == -1     # workspace
    assert q(fake, 0, 4, 32, 32, fake, fake, fake, ws, 9, 0, 1, 0, None) == -7       # mode
    assert q(fake, 0, 0, 32, 32, None, None, fake, ws, 0, 1, 1, 0, None) == 0       # empty, scale given
    c = lib.mixfp4_quantize_colwise_sr
    assert c(fake, 0, 24, 32, 32, fake, fake, fake, ws, 0, 0, 1, 0, None) == -2      # R % 16
    assert c(fake, 3, 32, 32, 32, fake, fake, fake, ws, 0, 0, 1, 0, None) == -4      # dtype


def test_fewrows_native_validation(lib):
    fake = ctypes.c_void_p(1 << 20)
    g = lib.mixfp4_gemm_native_fewrows
    assert g(fake, fake, fake, fake, fake, fake, 65, 128, 256, fake, 128, None, None) == -2   # M > 64
    assert g(fake, fake, fake, fake, fake, fake, 16, 128, 128, fake, 128, None, None) == -2   # K % 256
    assert g(fake, fake, fake, None, fake, fake, 16, 128, 256, fake, 128, None, None) == -1   # B codes
    assert g(fake, fake, fake, fake, fake, fake, 16, 128, 256, ctypes.c_void_p((1 << 20) + 2), 128, None, None) == -3
    assert g(fake, fake, fake, fake, fake, fake, 0, 128, 256, fake, 128, None, None) == 0     # empty


def test_colwise_rht_validation(lib):
    fake = ctypes.c_void_p(1 << 20)
    ws = ctypes.c_void_p(1 << 21)
    c = lib.mixfp4_quantize_colwise_rht
    assert c(fake, 0, 64, 32, 32, None, fake, fake, fake, ws, 0, 0, None) == -2      # R % 128
    assert c(fake, 0, 128, 24, 24, None, fake, fake, fake, ws, 0, 0, None) == -2     # C % 16
    assert c(fake, 0, 128, 32, 32, None, fake, fake, fake, None, 0, 0, None) == -1   # workspace
    assert c(fake, 0, 0, 32, 32, None, None, None, fake, ws, 0, 1, None) == 0        # empty


def test_fake_quantize_validation(lib):
    fake = ctypes.c_void_p(1 << 20)
    ws = ctypes.c_void_p(1 << 21)
    f = lib.mixfp4_fake_quantize
    #        x     dt rows K   ldx cand g   ts    ws  flag out  odt ldo ch    stream
    assert f(fake, 7, 4, 64, 64, 15, 16, fake, ws, 0, fake, 1, 64, fake, None) == -4    # input dtype
    assert f(fake, 0, 4, 64, 64, 15, 16, fake, ws, 0, fake, 5, 64, fake, None) == -4    # output dtype
    assert f(fake, 0, 4, 64, 64, 0, 16, fake, ws, 0, fake, 1, 64, fake, None) == -7     # empty set
    assert f(fake, 0, 4, 64, 64, 16, 16, fake, ws, 0, fake, 1, 64, fake, None) == -7    # unknown candidate
    assert f(fake, 0, 4, 64, 64, 15, 12, fake, ws, 0, fake, 1, 64, fake, None) == -7    # block size
    assert f(fake, 0, 4, 64, 64, 15, 16, fake, ws, 2, fake, 1, 64, fake, None) == -7    # scale flag
    assert f(fake, 0, 4, 48, 48, 15, 32, fake, ws, 0, fake, 1, 48, fake, None) == -2    # K % g
    assert f(fake, 0, 4, 24, 24, 15, 8, fake, ws, 0, fake, 1, 24, fake, None) == -2     # K % 16
    assert f(fake, 0, 4, 64, 64, 15, 16, fake, ws, 0, fake, 1, 48, fake, None) == -2    # ldo < K
    assert f(fake, 0, 4, 64, 64, 15, 16, None, ws, 0, fake, 1, 64, fake, None) == -1    # tensor scale
    assert f(fake, 0, 4, 64, 64, 15, 16, fake, None, 0, fake, 1, 64, fake, None) == -1  # workspace
    assert f(fake, 0, 4, 64, 64, 15, 16, fake, ws, 0, None, 1, 64, fake, None) == -1    # out
    assert f(fake, 0, 4, 64, 64, 15, 16, fake, ws, 0, ctypes.c_void_p((1 << 20) + 16), 1, 64, fake,
             None) == -3                                                                  # out alignment
    assert f(fake, 0, 4, 64, 64, 15, 16, fake, ws, 0, fake, 1, 72, fake, None) == -3    # ldo % 16
    assert f(fake, 0, 4, 64, 64, 15, 16, fake, ws, 0, fake, 1, 64, ctypes.c_void_p((1 << 20) + 1),
             None) == -3                                                                  # choice alignment


def test_four_six_mode_only_where_declared(lib):
    fake = ctypes.c_void_p(1 << 20)
    ws = ctypes.c_void_p(1 << 21)
    assert lib.mixfp4_quantize(fake, 0, 4, 32, 32, fake, fake, fake, ws, 4, 0, None) == -7   # past FOUR_SIX
    assert lib.mixfp4_quantize_colwise(fake, 0, 32, 32, 32, fake, fake, fake, ws, 3, 0, None) == -7
    assert lib.mixfp4_quantize_2d(fake, 0, 32, 32, 32, fake, fake, fake, ws, 3, 0, None) == -7
    assert lib.mixfp4_quantize_noalloc(fake, 0, 4, 32, 32, fake, fake, fake, 4, None) == -7
