"""Host checks of the bit-level formulas inside the CUDA kernels (CPU only):
each formula is restated here with the semantics of its PTX instructions
(`prmt`, `lop3`, fp32 operations through numpy float32) and compared with the
oracle or with the plain definition, exhaustively or on dense grids that
include every tie.  The GPU parity tests check the kernels themselves; these
pin the derivations the kernels rely on.

* the E1M2 main / residual split (native FP4 variant): eight `lop3` per word
* the few-row native kernel's residual of a stored code (four `lop3` per word)
  and its residual scale bytes (`prmt` sign replication)
* branch-free E3M0 rounding (candidate-set ablation, reading R14)
* the stochastic-rounding payload shared by both formats (reading R13)
* the 16 x 16 nibble transpose in registers (2D transpose)
* the decode of a code word to f16 operands in the GEMM (reading R8)
"""
import numpy as np
import pytest

M32 = 0xFFFFFFFF


def prmt(a: int, b: int, sel: int) -> int:
    """PTX prmt.b32 default mode: result byte i = byte (sel >> 4i) & 7 of
    {a.b0..a.b3, b.b0..b.b3}."""
    bs = [(a >> (8 * i)) & 0xFF for i in range(4)] + [(b >> (8 * i)) & 0xFF for i in range(4)]
    return sum(bs[(sel >> (4 * i)) & 7] << (8 * i) for i in range(4))


def lop3(a: int, b: int, c: int, lut: int) -> int:
    """PTX lop3.b32: bit k of the result is bit (a_k b_k c_k) of the table,
    a the most significant index bit (the table is f(0xF0, 0xCC, 0xAA))."""
    r = 0
    for k in range(32):
        idx = (((a >> k) & 1) << 2) | (((b >> k) & 1) << 1) | ((c >> k) & 1)
        r |= ((lut >> idx) & 1) << k
    return r


def split_e1m2_word(w: int, tmask: int):
    """The native kernels' split, instruction by instruction."""
    r1, r2, l1 = w >> 1, w >> 2, (w << 1) & M32
    m0 = lop3(r1, w, r2, 0xE0)
    m1 = lop3(r1, l1, w, 0xF4)
    t = lop3(m0, m1, 0x22222222, 0xD8)
    t = lop3(t, w | l1, 0x44444444, 0xD8)
    t = lop3(t, w, 0x88888888, 0xD8)
    r = lop3(l1, r1, 0x22222222, 0x80)
    r = lop3(r, w, 0x88888888, 0xF8)
    main = lop3(t, w, tmask, 0xE4)
    return main, r & tmask


@pytest.mark.parametrize("t", [0, 1])
def test_lop3_split_matches_oracle_for_every_nibble_and_position(oracle, t):
    """Every nibble value in every one of the 8 positions of a word, for an
    E2M1 (t = 0) and an E1M2 (t = 1) block, against oracle.split_native."""
    rows = []
    for pos in range(8):
        for nib in range(16):
            rows.append((nib << (4 * pos)) | (((nib + 5) & 15) << (4 * ((pos + 3) % 8))))
    codes = np.zeros((len(rows), 32), np.uint8)     # one 64-element row per word (K = 64)
    for i, w in enumerate(rows):
        codes[i, :4] = np.frombuffer(np.uint32(w).tobytes(), np.uint8)
    scales = np.full((len(rows), 4), 0x38 | (t << 7), np.uint8)
    main, res, _ = oracle.split_native(codes, scales)
    for i, w in enumerate(rows):
        m, r = split_e1m2_word(w, M32 if t else 0)
        assert m == int(np.frombuffer(main[i, :4].tobytes(), np.uint32)[0]), (hex(w), t)
        assert r == int(np.frombuffer(res[i, :4].tobytes(), np.uint32)[0]), (hex(w), t)


def residual_word(w: int) -> int:
    """The few-row native kernel's residual codes of eight nibbles,
    instruction by instruction: payload {0,1,2,3,4,4,4,2}[p], sign kept."""
    r1, r2, l1, l2 = w >> 1, w >> 2, (w << 1) & M32, (w << 2) & M32
    a = lop3(0x22222222, r1, l1, 0xBF)
    b = lop3(0x44444444, l1, l2, 0x7F)
    c = lop3(w, a, b, 0x80)
    return lop3(c, r2, 0x11111111, 0x70)


def prmt_sign_replicate(a: int) -> int:
    """prmt.b32 d, a, 0, 0xBA98: selector nibbles 8..B pick bytes 0..3 of a
    with the sign-replicate bit set, so each byte becomes 0xFF or 0x00 by its
    bit 7."""
    return sum((0xFF if (a >> (8 * i)) & 0x80 else 0) << (8 * i) for i in range(4))


def residual_scales(sw: int) -> int:
    return sw & prmt_sign_replicate(sw) & 0x7F7F7F7F


@pytest.mark.parametrize("t", [0, 1])
def test_fewrows_residual_reconstructs_every_value(oracle, t):
    """The stored code read as E2M1 (scale with the type bit cleared) plus the
    residual code (scale from residual_scales) equals the MixFP4 value of the
    stored code, for every nibble in every position and both block types;
    values from the oracle's dequantizer.  Scale 0x38 (1.0) and 0x01 (the
    smallest subnormal) both checked."""
    for scale in (0x38, 0x01):
        sbyte = scale | (t << 7)
        rows = []
        for pos in range(8):
            for nib in range(16):
                rows.append((nib << (4 * pos)) | (((nib + 5) & 15) << (4 * ((pos + 3) % 8))))
        codes = np.zeros((len(rows), 8), np.uint8)       # K = 16: one block per row
        res = np.zeros_like(codes)
        for i, w in enumerate(rows):
            codes[i, :4] = np.frombuffer(np.uint32(w).tobytes(), np.uint8)
            res[i, :4] = np.frombuffer(np.uint32(residual_word(w)).tobytes(), np.uint8)
        sw = sbyte * 0x01010101
        main_scale = np.full((len(rows), 1), (sw & 0x7F7F7F7F) & 0xFF, np.uint8)
        res_scale = np.full((len(rows), 1), residual_scales(sw) & 0xFF, np.uint8)
        want = oracle.dequantize(codes, np.full((len(rows), 1), sbyte, np.uint8), 1.0).astype(np.float64)
        got = (oracle.dequantize(codes, main_scale, 1.0).astype(np.float64)
               + oracle.dequantize(res, res_scale, 1.0).astype(np.float64))
        assert np.array_equal(got, want), (t, scale)


def f32(v):
    return np.float32(v)


def e3m0_round_kernel(y: float) -> float:
    """candidates.cu: round up iff mantissa + exponent bit 0 > 2^22, cap 16,
    below 1/4 the neighbours 0 and 1/4 (tie 1/8 to 0)."""
    u = int(np.float32(y).view(np.uint32))
    up = (u & 0x007FFFFF) + ((u >> 23) & 1) > 0x00400000
    p2 = min(float(np.uint32((u & 0x7F800000) + (0x00800000 if up else 0)).view(np.float32)), 16.0)
    return max(p2, 0.25) if y > 0.125 else 0.0


def test_e3m0_branch_free_rounding_matches_oracle(oracle):
    vals = [oracle.cand_value(3, p) for p in range(8)]
    ys = set()
    for v in vals + [(vals[i] + vals[i + 1]) / 2 for i in range(7)] + [32.0, 1e6, 1e-40, 0.0]:
        f = f32(v)
        ys.update([float(f), float(np.nextafter(f, f32(0))), float(np.nextafter(f, f32(1e9)))])
    rng = np.random.default_rng(11)
    ys.update(rng.uniform(0, 40, 20000).astype(np.float32).tolist())
    ys.update((2.0 ** rng.uniform(-30, 20, 20000)).astype(np.float32).tolist())
    for y in ys:
        assert e3m0_round_kernel(y) == vals[oracle.cand_rne(3, y)], y


def sr_payload_kernel(e1m2: bool, m: float, eps: float) -> int:
    """quant_core.cuh sr_payload: power-of-two gaps make the neighbour fraction
    an exact scaling and floor (fp32 throughout)."""
    m, eps = f32(m), f32(eps)
    sc = f32(1.0) if e1m2 else f32(2.0 if m < 2 else (1.0 if m < 4 else 0.5))
    add = 0 if e1m2 else (2 if m >= 2 else 0) + (2 if m >= 4 else 0)
    v = f32(m * sc)
    fl = np.floor(v)
    p = int(fl) + add + (1 if eps < f32(v - fl) else 0)
    return p if m < (7.0 if e1m2 else 6.0) else 7


def test_sr_payload_matches_oracle(oracle):
    rng = np.random.default_rng(12)
    ms = np.concatenate([rng.uniform(0, 8, 1500), np.arange(0, 8, 0.125), np.arange(0, 8, 0.5) + 1e-6,
                         [6.0, 7.0, 7.5, 100.0]]).astype(np.float32)
    es = np.concatenate([rng.uniform(0, 1, 8), [0.0, 0.25, 0.5, 0.75, 1 - 2 ** -24]]).astype(np.float32)
    for m in ms:
        for e in es:
            assert sr_payload_kernel(False, m, e) == oracle.sr_payload(0, float(m), float(e)), (m, e)
            assert sr_payload_kernel(True, m, e) == oracle.sr_payload(1, float(m), float(e)), (m, e)


def transpose_nibbles16(lo, hi):
    """train.cu transpose_nibbles16: swap the off-diagonal 8 x 8 blocks, then
    16-bit fields, bytes and nibbles inside every 8 x 8 block."""
    lo, hi = list(lo), list(hi)
    for r in range(8):
        lo[r + 8], hi[r] = hi[r], lo[r + 8]
    for w in (lo, hi):
        for r in range(16):
            if r & 7 < 4:
                x, y = w[r], w[r + 4]
                w[r], w[r + 4] = prmt(x, y, 0x5410), prmt(x, y, 0x7632)
        for r in range(16):
            if r & 3 < 2:
                x, y = w[r], w[r + 2]
                w[r], w[r + 2] = prmt(x, y, 0x6240), prmt(x, y, 0x7351)
        for r in range(0, 16, 2):
            x, y = w[r], w[r + 1]
            w[r] = (x & 0x0F0F0F0F) | ((y << 4) & 0xF0F0F0F0)
            w[r + 1] = ((x >> 4) & 0x0F0F0F0F) | (y & 0xF0F0F0F0)
    return lo, hi


def test_register_nibble_transpose_is_the_transpose():
    rng = np.random.default_rng(13)
    for trial in range(50):
        M = rng.integers(0, 16, (16, 16))
        lo = [sum(int(M[r, c]) << (4 * c) for c in range(8)) for r in range(16)]
        hi = [sum(int(M[r, c + 8]) << (4 * c) for c in range(8)) for r in range(16)]
        L, H = transpose_nibbles16(lo, hi)
        for c in range(16):
            for r in range(16):
                w = L[c] if r < 8 else H[c]
                assert (w >> (4 * (r % 8))) & 0xF == M[r, c]


# gemm.cu decode8: f16 high bytes of u = 2 v by payload, E2M1 and E1M2.
LUT = {0: (0x42403C00, 0x4A484644), 1: (0x46444000, 0x4B4A4948)}


def decode8_kernel(w: int, t: int):
    """gemm.cu decode8 before the scale multiply: the eight f16 bit patterns
    of a code word, element 2j from the low nibble of byte j."""
    lo, hi = LUT[t]
    wp = w & 0x77777777
    ws = (w * 16) & M32
    u0 = prmt(lo, hi, wp & 0xFFFF)
    u1 = prmt(lo, hi, (wp >> 16) & 0xFFFF)          # __umulhi(wp, 0x10000)
    g0 = prmt(w, ws, 0x1504)
    g1 = prmt(w, ws, 0x3726)
    v0 = u0 | (g0 & 0x80808080)
    v1 = u1 | (g1 & 0x80808080)
    words = [prmt(v0, 0, 0x1404), prmt(v0, 0, 0x3424), prmt(v1, 0, 0x1404), prmt(v1, 0, 0x3424)]
    return [(x >> (16 * h)) & 0xFFFF for x in words for h in (0, 1)]


@pytest.mark.parametrize("t", [0, 1])
def test_gemm_decode_gives_the_exact_f16_of_twice_each_value(oracle, t):
    """Every nibble in every position decodes to the f16 of 2 v with the
    nibble's sign (negative zero for 0x8), v the oracle's magnitude of the
    payload (the E2M1 value, or the E1M2 payload in x2 units, R3); the GEMM
    epilogue removes the factor 4 that the two doubled operands carry."""
    for pos in range(8):
        for nib in range(16):
            w = (nib << (4 * pos)) | (((nib * 7 + 3) & 15) << (4 * ((pos + 5) % 8)))
            got = decode8_kernel(w, t)
            for e in range(8):
                n = (w >> (4 * e)) & 0xF
                v = 2.0 * oracle.fp4_value(t, n & 7)
                want = np.float16(-v if n & 8 else v)
                assert got[e] == int(want.view(np.uint16)), (hex(w), t, e)
