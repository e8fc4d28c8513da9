"""MixFP4 CPU oracle -- TEST INFRASTRUCTURE ONLY.

A plain C restatement of the MixFP4 method (arXiv 2605.31035), wrapped with
ctypes over numpy arrays.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package.  The CUDA product path (``paper_2605_31035_gb300``) never imports it,
and the two share no code.

Function map (paper passages are cited in ``mixfp4_oracle.c``):
  e4m3_value / e4m3_rne     E4M3 block scale grid and its RNE cast (Alg. 1)
  fp4_value / fp4_rne       Table 1 / App. B.2 codebooks with the x2 E1M2 remap
  quantize                  Algorithm 1 with type-in-scale packing (App. B.3)
  dequantize                App. B.2/B.3 decode times the tensor scale
  gemm_f64                  C = A_deq B_deq^T in float64
  gemm_exact                App. B.1 Eq. (factor), exact integer accumulation
  split_native              MixFP4 operand as the sum of two E2M1 operands with
                            shared scales, plus the tensor core's tiled scale
                            layout (the native FP4 GEMM variant)
  quantize_colwise          Algorithm 1 along the other dimension (blocks of 16
                            rows in one column): quantize of the transpose, the
                            WGRAD / DGRAD operand orientation (Sec. 3.2)
  quantize_2d               Algorithm 1 with 16 x 16 tiles (2D weight blocks of
                            the training flow, Sec. 3.2), reading R12
  transpose_2d              the transposed operand of a 2D-quantized tensor
  philox4x32_10             Salmon et al.'s counter-based generator (SC'11)
  quantize_sr               Algorithm 1 with stochastic rounding of the chosen
                            format's codes (reading R13); quantize_colwise_sr
                            the same down the columns
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "mixfp4_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")

MODE_MIX, MODE_E2M1_ONLY, MODE_E1M2_ONLY, MODE_FOUR_SIX = 0, 1, 2, 3
# Candidates of the ablation quantizer (reading R14), bit c of a candidate mask.
CAND_E2M1_6, CAND_E1M2, CAND_E2M1_4, CAND_E3M0 = 1, 2, 4, 8


def build(force: bool = False) -> str:
    """Compile the oracle with IEEE-strict flags (no FMA contraction)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["gcc", "-O2", "-ffp-contract=off", "-fno-fast-math", "-std=c11", "-fPIC", "-shared",
             _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


_lib = None


def _L():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        I64 = ctypes.c_int64
        lib.oracle_e4m3_value.restype = ctypes.c_double
        lib.oracle_e4m3_value.argtypes = [ctypes.c_int]
        lib.oracle_e4m3_rne.restype = ctypes.c_int
        lib.oracle_e4m3_rne.argtypes = [ctypes.c_float]
        lib.oracle_fp4_value.restype = ctypes.c_double
        lib.oracle_fp4_value.argtypes = [ctypes.c_int, ctypes.c_int]
        lib.oracle_e1m2_stored_value.restype = ctypes.c_double
        lib.oracle_e1m2_stored_value.argtypes = [ctypes.c_int]
        lib.oracle_fp4_rne.restype = ctypes.c_int
        lib.oracle_fp4_rne.argtypes = [ctypes.c_int, ctypes.c_float]
        lib.oracle_quantize.restype = ctypes.c_int
        lib.oracle_quantize.argtypes = [P, I64, I64, I64, ctypes.c_int, ctypes.c_int, P, P, P, P, P]
        lib.oracle_quantize_f32.restype = ctypes.c_int
        lib.oracle_quantize_f32.argtypes = [P, I64, I64, I64, ctypes.c_int, ctypes.c_int, P, P, P, P, P]
        lib.oracle_rht.restype = ctypes.c_int
        lib.oracle_rht.argtypes = [P, I64, I64, I64, P, P]
        lib.oracle_dequantize.restype = None
        lib.oracle_dequantize.argtypes = [P, P, ctypes.c_float, I64, I64, P]
        lib.oracle_gemm_f64.restype = None
        lib.oracle_gemm_f64.argtypes = [P, P, ctypes.c_float, P, P, ctypes.c_float, I64, I64, I64, P]
        lib.oracle_gemm_exact.restype = None
        lib.oracle_gemm_exact.argtypes = [P, P, ctypes.c_float, P, P, ctypes.c_float, I64, I64, I64, P]
        lib.oracle_dequant_row_f64.restype = None
        lib.oracle_dequant_row_f64.argtypes = [P, P, ctypes.c_float, I64, I64, P]
        lib.oracle_split_native.argtypes = [P, P, I64, I64, P, P, P]
        lib.oracle_split_native.restype = ctypes.c_int
        lib.oracle_quantize_2d.restype = ctypes.c_int
        lib.oracle_quantize_2d.argtypes = [P, I64, I64, I64, ctypes.c_int, ctypes.c_int, P, P, P]
        lib.oracle_quantize_2d_f32.restype = ctypes.c_int
        lib.oracle_quantize_2d_f32.argtypes = [P, I64, I64, I64, ctypes.c_int, ctypes.c_int, P, P, P]
        lib.oracle_philox4x32_10.restype = None
        lib.oracle_philox4x32_10.argtypes = [P, P, P]
        lib.oracle_sr_uniform.restype = ctypes.c_float
        lib.oracle_sr_uniform.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint64]
        lib.oracle_sr_payload.restype = ctypes.c_int
        lib.oracle_sr_payload.argtypes = [ctypes.c_int, ctypes.c_float, ctypes.c_float]
        lib.oracle_quantize_sr.restype = ctypes.c_int
        lib.oracle_quantize_sr.argtypes = [P, I64, I64, I64, ctypes.c_int, ctypes.c_int, P, ctypes.c_uint64,
                                           ctypes.c_uint64, P, P]
        lib.oracle_cand_value.restype = ctypes.c_double
        lib.oracle_cand_value.argtypes = [ctypes.c_int, ctypes.c_int]
        lib.oracle_cand_divisor.restype = ctypes.c_float
        lib.oracle_cand_divisor.argtypes = [ctypes.c_int]
        lib.oracle_cand_rne.restype = ctypes.c_int
        lib.oracle_cand_rne.argtypes = [ctypes.c_int, ctypes.c_float]
        lib.oracle_fake_quantize.restype = ctypes.c_int
        lib.oracle_fake_quantize.argtypes = [P, I64, I64, I64, ctypes.c_int, ctypes.c_int, ctypes.c_int, P, P, P]
        lib.oracle_f32_to_bf16.restype = ctypes.c_uint16
        lib.oracle_f32_to_bf16.argtypes = [ctypes.c_float]
        lib.oracle_f32_to_bf16_array.restype = None
        lib.oracle_f32_to_bf16_array.argtypes = [P, I64, P]
        lib.oracle_transpose_2d.restype = ctypes.c_int
        lib.oracle_transpose_2d.argtypes = [P, P, I64, I64, P, P]
        _lib = lib
    return _lib


def _p(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.c_void_p)


def e4m3_value(code: int) -> float:
    return _L().oracle_e4m3_value(int(code))


def e4m3_rne(v: float) -> int:
    return _L().oracle_e4m3_rne(float(v))


def fp4_value(fmt: int, payload: int) -> float:
    """fmt 0 = E2M1, 1 = E1M2 (x2 remapped)."""
    return _L().oracle_fp4_value(int(fmt), int(payload))


def e1m2_stored_value(payload: int) -> float:
    return _L().oracle_e1m2_stored_value(int(payload))


def fp4_rne(fmt: int, y: float) -> int:
    return _L().oracle_fp4_rne(int(fmt), float(y))


def quantize(x_bf16_bits: np.ndarray, mode: int = MODE_MIX, s32: float | None = None,
             want_errors: bool = False):
    """Algorithm 1 on a [rows, K] tensor given as uint16 bf16 bit patterns.

    Returns (codes uint8 [rows, K/2], scales uint8 [rows, K/16], s32 float)
    and, with want_errors, the per-block S of each candidate.
    """
    x = np.ascontiguousarray(x_bf16_bits, dtype=np.uint16)
    rows, K = x.shape
    codes = np.zeros((rows, K // 2), np.uint8)
    scales = np.zeros((rows, K // 16), np.uint8)
    s = np.array([0.0 if s32 is None else s32], np.float32)
    e2 = np.zeros((rows, K // 16), np.float32)
    e1 = np.zeros((rows, K // 16), np.float32)
    rc = _L().oracle_quantize(_p(x), rows, K, K, int(mode), 0 if s32 is None else 1, _p(s),
                              _p(codes), _p(scales), _p(e2), _p(e1))
    if rc != 0:
        raise ValueError("oracle_quantize rejected the input (non-finite value or K % 16 != 0)")
    if want_errors:
        return codes, scales, float(s[0]), e2, e1
    return codes, scales, float(s[0])


def quantize_f32(x: np.ndarray, mode: int = MODE_MIX, s32: float | None = None, want_errors: bool = False):
    """Algorithm 1 on a [rows, K] float32 tensor (same steps as quantize)."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    rows, K = x.shape
    codes = np.zeros((rows, K // 2), np.uint8)
    scales = np.zeros((rows, K // 16), np.uint8)
    s = np.array([0.0 if s32 is None else s32], np.float32)
    e2 = np.zeros((rows, K // 16), np.float32)
    e1 = np.zeros((rows, K // 16), np.float32)
    rc = _L().oracle_quantize_f32(_p(x), rows, K, K, int(mode), 0 if s32 is None else 1, _p(s),
                                  _p(codes), _p(scales), _p(e2), _p(e1))
    if rc != 0:
        raise ValueError("oracle_quantize_f32 rejected the input (non-finite value or K % 16 != 0)")
    if want_errors:
        return codes, scales, float(s[0]), e2, e1
    return codes, scales, float(s[0])


def rht(x_bf16_bits: np.ndarray, signs: np.ndarray | None = None) -> np.ndarray:
    """The 128-point rotation (reading R11) of a [rows, K] bf16 tensor, K % 128 == 0.
    signs: 16 uint8 (bit i negates element i of every chunk) or None.  Returns fp32."""
    x = np.ascontiguousarray(x_bf16_bits, dtype=np.uint16)
    rows, K = x.shape
    y = np.zeros((rows, K), np.float32)
    sg = None if signs is None else np.ascontiguousarray(signs, np.uint8)
    if sg is not None and sg.size != 16:
        raise ValueError("signs must hold 16 bytes")
    if _L().oracle_rht(_p(x), rows, K, K, None if sg is None else _p(sg), _p(y)) != 0:
        raise ValueError("oracle_rht needs K % 128 == 0")
    return y


def dequantize(codes: np.ndarray, scales: np.ndarray, s32: float) -> np.ndarray:
    codes = np.ascontiguousarray(codes, np.uint8)
    scales = np.ascontiguousarray(scales, np.uint8)
    rows, K = codes.shape[0], codes.shape[1] * 2
    out = np.zeros((rows, K), np.float32)
    _L().oracle_dequantize(_p(codes), _p(scales), float(s32), rows, K, _p(out))
    return out


def dequant_rows_f64(codes: np.ndarray, scales: np.ndarray, s32: float, rows) -> np.ndarray:
    codes = np.ascontiguousarray(codes, np.uint8)
    scales = np.ascontiguousarray(scales, np.uint8)
    K = codes.shape[1] * 2
    rows = list(rows)
    out = np.zeros((len(rows), K), np.float64)
    buf = np.zeros(K, np.float64)
    for i, r in enumerate(rows):
        _L().oracle_dequant_row_f64(_p(codes), _p(scales), float(s32), K, int(r), _p(buf))
        out[i] = buf
    return out


def gemm_f64(a, b) -> np.ndarray:
    """a, b: (codes, scales, s32) triples; returns C = A_deq B_deq^T (float64)."""
    ac, as_, as32 = a
    bc, bs, bs32 = b
    ac, as_, bc, bs = (np.ascontiguousarray(t, np.uint8) for t in (ac, as_, bc, bs))
    M, N, K = ac.shape[0], bc.shape[0], ac.shape[1] * 2
    C = np.zeros((M, N), np.float64)
    _L().oracle_gemm_f64(_p(ac), _p(as_), float(as32), _p(bc), _p(bs), float(bs32), M, N, K, _p(C))
    return C


def gemm_exact(a, b) -> np.ndarray:
    """Exact App. B.1 factored GEMM, returned as float64 (rounded once)."""
    ac, as_, as32 = a
    bc, bs, bs32 = b
    ac, as_, bc, bs = (np.ascontiguousarray(t, np.uint8) for t in (ac, as_, bc, bs))
    M, N, K = ac.shape[0], bc.shape[0], ac.shape[1] * 2
    C = np.zeros((M, N), np.longdouble)
    _L().oracle_gemm_exact(_p(ac), _p(as_), float(as32), _p(bc), _p(bs), float(bs32), M, N, K, _p(C))
    return C.astype(np.float64)


def sf_tiled_bytes(rows: int, K: int) -> int:
    """Size of the tiled block-scale array: rows rounded up to 256, K/16 bytes each."""
    return ((rows + 255) // 256) * 256 * (K // 16)


def split_native(codes: np.ndarray, scales: np.ndarray):
    """Native E2M1 operands of a MixFP4 tensor: (main codes, residual codes,
    tiled ue4m3 scales); see oracle_split_native in mixfp4_oracle.c."""
    codes = np.ascontiguousarray(codes, np.uint8)
    scales = np.ascontiguousarray(scales, np.uint8)
    rows, K = codes.shape[0], codes.shape[1] * 2
    main = np.zeros_like(codes)
    res = np.zeros_like(codes)
    sf = np.zeros(sf_tiled_bytes(rows, K), np.uint8)
    rc = _L().oracle_split_native(_p(codes), _p(scales), rows, K, _p(main), _p(res), _p(sf))
    if rc != 0:
        raise ValueError(f"oracle_split_native failed ({rc})")
    return main, res, sf


def quantize_colwise(x_bf16_bits: np.ndarray, mode: int = MODE_MIX, s32: float | None = None):
    """Algorithm 1 with each block running down a column (16 consecutive rows):
    by definition the row-wise quantization of the transpose.  Returns codes
    [C, R/2], scales [C, R/16] and s32 for an [R, C] input."""
    return quantize(np.ascontiguousarray(np.asarray(x_bf16_bits, np.uint16).T), mode, s32)


def quantize_2d(x_bf16_bits: np.ndarray, mode: int = MODE_MIX, s32: float | None = None):
    """Algorithm 1 with 16 x 16 blocks (reading R12) on a [rows, K] bf16 tensor;
    codes [rows, K/2] and scales [rows, K/16] (each tile's scale byte repeated
    on its rows), s32."""
    x = np.ascontiguousarray(x_bf16_bits, dtype=np.uint16)
    rows, K = x.shape
    codes = np.zeros((rows, K // 2), np.uint8)
    scales = np.zeros((rows, K // 16), np.uint8)
    s = np.array([0.0 if s32 is None else s32], np.float32)
    rc = _L().oracle_quantize_2d(_p(x), rows, K, K, int(mode), 0 if s32 is None else 1, _p(s),
                                 _p(codes), _p(scales))
    if rc != 0:
        raise ValueError("oracle_quantize_2d rejected the input (non-finite value or K % 16 != 0)")
    return codes, scales, float(s[0])


def quantize_2d_f32(x: np.ndarray, mode: int = MODE_MIX, s32: float | None = None):
    """quantize_2d on a [rows, K] float32 tensor."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    rows, K = x.shape
    codes = np.zeros((rows, K // 2), np.uint8)
    scales = np.zeros((rows, K // 16), np.uint8)
    s = np.array([0.0 if s32 is None else s32], np.float32)
    rc = _L().oracle_quantize_2d_f32(_p(x), rows, K, K, int(mode), 0 if s32 is None else 1, _p(s),
                                     _p(codes), _p(scales))
    if rc != 0:
        raise ValueError("oracle_quantize_2d_f32 rejected the input")
    return codes, scales, float(s[0])


def transpose_2d(codes: np.ndarray, scales: np.ndarray):
    """Codes and scales of the transpose of a 2D-quantized tensor (rows % 16 == 0,
    K % 16 == 0): codes_t [K, rows/2], scales_t [K, rows/16]."""
    codes = np.ascontiguousarray(codes, np.uint8)
    scales = np.ascontiguousarray(scales, np.uint8)
    rows, K = codes.shape[0], codes.shape[1] * 2
    ct = np.zeros((K, rows // 2), np.uint8)
    st = np.zeros((K, rows // 16), np.uint8)
    rc = _L().oracle_transpose_2d(_p(codes), _p(scales), rows, K, _p(ct), _p(st))
    if rc != 0:
        raise ValueError(f"oracle_transpose_2d failed ({rc})")
    return ct, st


def philox4x32_10(ctr, key):
    """The four output words of Philox4x32-10 for a 4-word counter and 2-word key."""
    c = np.ascontiguousarray(np.asarray(ctr, np.uint32))
    k = np.ascontiguousarray(np.asarray(key, np.uint32))
    out = np.zeros(4, np.uint32)
    _L().oracle_philox4x32_10(_p(c), _p(k), _p(out))
    return out


def sr_uniform(seed: int, offset: int, e: int) -> float:
    return _L().oracle_sr_uniform(int(seed), int(offset), int(e))


def sr_payload(fmt: int, m: float, eps: float) -> int:
    return _L().oracle_sr_payload(int(fmt), float(m), float(eps))


def quantize_sr(x_bf16_bits: np.ndarray, seed: int, offset: int = 0, mode: int = MODE_MIX,
                s32: float | None = None):
    """Algorithm 1 with stochastic rounding (reading R13) on a [rows, K] bf16 tensor."""
    x = np.ascontiguousarray(x_bf16_bits, dtype=np.uint16)
    rows, K = x.shape
    codes = np.zeros((rows, K // 2), np.uint8)
    scales = np.zeros((rows, K // 16), np.uint8)
    s = np.array([0.0 if s32 is None else s32], np.float32)
    rc = _L().oracle_quantize_sr(_p(x), rows, K, K, int(mode), 0 if s32 is None else 1, _p(s), int(seed),
                                 int(offset), _p(codes), _p(scales))
    if rc != 0:
        raise ValueError("oracle_quantize_sr rejected the input")
    return codes, scales, float(s[0])


def quantize_colwise_sr(x_bf16_bits: np.ndarray, seed: int, offset: int = 0, mode: int = MODE_MIX,
                        s32: float | None = None):
    """quantize_sr of the transpose (element index c * R + r of an [R, C] input)."""
    return quantize_sr(np.ascontiguousarray(np.asarray(x_bf16_bits, np.uint16).T), seed, offset, mode, s32)


def quantize_colwise_rht(x_bf16_bits: np.ndarray, signs: np.ndarray | None = None, mode: int = MODE_MIX,
                         s32: float | None = None):
    """The 128-point rotation (R11) of every 128-row chunk of each column of an
    [R, C] tensor, then Algorithm 1 down the columns: by definition
    quantize_f32(rht(X^T))."""
    xt = np.ascontiguousarray(np.asarray(x_bf16_bits, np.uint16).T)
    return quantize_f32(rht(xt, signs), mode, s32)


def cand_value(c: int, p: int) -> float:
    """Magnitude of payload p under candidate c (reading R14)."""
    return _L().oracle_cand_value(int(c), int(p))


def cand_divisor(c: int) -> float:
    return _L().oracle_cand_divisor(int(c))


def cand_rne(c: int, y: float) -> int:
    return _L().oracle_cand_rne(int(c), float(y))


def fake_quantize(x_bf16_bits: np.ndarray, candidates: int, block: int = 16, s32: float | None = None,
                  out_bf16: bool = False):
    """Quantize-dequantize of a [rows, K] bf16 tensor under a candidate set
    (mask of CAND_*) and block size g (reading R14): (out, choice, s32), out
    fp32 [rows, K] (bf16 bits when out_bf16), choice uint8 [rows, K/g]."""
    x = np.ascontiguousarray(x_bf16_bits, dtype=np.uint16)
    rows, K = x.shape
    out = np.zeros((rows, K), np.float32)
    choice = np.zeros((rows, K // block if block else 0), np.uint8)
    s = np.array([0.0 if s32 is None else s32], np.float32)
    rc = _L().oracle_fake_quantize(_p(x), rows, K, K, int(candidates), int(block), 0 if s32 is None else 1,
                                   _p(s), _p(out), _p(choice))
    if rc != 0:
        raise ValueError("oracle_fake_quantize rejected the arguments or the input")
    if out_bf16:
        out = f32_to_bf16_array(out)
    return out, choice, float(s[0])


def f32_to_bf16_array(f: np.ndarray) -> np.ndarray:
    """bf16 bits (round to nearest even) of a float32 array."""
    f = np.ascontiguousarray(f, dtype=np.float32)
    out = np.zeros(f.shape, np.uint16)
    _L().oracle_f32_to_bf16_array(_p(f), f.size, _p(out))
    return out


def f32_to_bf16(v: float) -> int:
    return _L().oracle_f32_to_bf16(float(v))
