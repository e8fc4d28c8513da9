// Algorithm 1 (Sec. 3.2) for one 16-element block, shared by the quantizer
// kernels: the per-tensor constants, the divisions by a known divisor, the
// E2M1 / E1M2 candidates with their error sums in the pinned order, the
// selection and the nibble packing.  The design notes (division methods and
// their checks, tiny values, the E1M2 clamp) are at the top of quantize.cu.
#pragma once
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "kernels.cuh"
#include "ptx.cuh"

namespace mixfp4 {
namespace {

constexpr int kQuantThreads = 256;

// Correctly rounded a / b (per lane) given nb = -b and r = RN(1/b) (Markstein).
__device__ __forceinline__ u64 div_rn2(u64 a, u64 nb, u64 r) {
  u64 q0 = mul2(a, r);
  u64 e = fma2(q0, nb, a);
  return fma2(e, r, q0);
}

// RN(a*zh + RN(a*zl)) (per lane): a / b for a divisor b whose (zh, zl) pass
// the checks described above.
__device__ __forceinline__ u64 div_kd2(u64 a, u64 zh, u64 zl) { return fma2(a, zh, mul2(a, zl)); }

// (zh, zl) of a divisor b: RN(1/b) and RN(RN(1 - b*zh)/b); (0, 0) for b = 0.
__device__ __forceinline__ float2 kd_consts(float b) {
  if (!(b > 0.0f)) return make_float2(0.0f, 0.0f);
  const float zh = __frcp_rn(b);
  return make_float2(zh, __fdiv_rn(__fmaf_rn(-b, zh, 1.0f), b));
}

// The same pair for a divisor whose (zh, zl) is checked before use (the
// tensor scale, see markstein_needed): zl by Markstein's correction with the
// reciprocal zh instead of a correctly rounded division (cheaper on the
// critical path of every CTA; a zl that were off would only send the tensor
// to the Markstein path).
__device__ __forceinline__ float2 kd_consts_checked(float b) {
  if (!(b > 0.0f)) return make_float2(0.0f, 0.0f);
  const float zh = __frcp_rn(b);
  const float r = __fmaf_rn(-b, zh, 1.0f);
  const float q0 = __fmul_rn(r, zh);
  return make_float2(zh, __fmaf_rn(__fmaf_rn(-q0, b, r), zh, q0));
}

// (zh, zl) of the block-scale divisors 6 and 7 (kd_consts(6), kd_consts(7),
// fixed bit patterns: 6 * RN(1/6) = 1 + 2^-25, so zl = RN(-2^-25 / 6); the
// pairs are recomputed from their definition by a CPU test).
constexpr uint32_t kZh6Bits = 0x3e2aaaabu, kZl6Bits = 0xb1aaaaabu;
constexpr uint32_t kZh7Bits = 0x3e124925u, kZl7Bits = 0xb1db6db7u;

__device__ __forceinline__ uint32_t lo32(u64 v) { return (uint32_t)v; }
__device__ __forceinline__ uint32_t hi32(u64 v) { return (uint32_t)(v >> 32); }

struct TensorConsts {
  float s32;       // per-tensor scale, possibly rescaled to [1, 2)
  float r32;       // RN(1/s32), or 0 when s32 == 0
  float2 kd32;     // (zh, zl) of s32
  float2 kd6, kd7; // (zh, zl) of 6 and 7
  int k;           // |x| is multiplied by 2^k when `scaled`
  int scaled;
};

// Per-tensor constants, derived by every thread (a persistent thread handles
// many blocks, so this costs a few instructions per block at most).
__device__ __forceinline__ TensorConsts tensor_consts(float* tensor_scale, const uint32_t* amax_word,
                                                      int scale_given) {
  float s32;
  if (scale_given) {
    s32 = *tensor_scale;
  } else {
    s32 = __fdiv_rn(__uint_as_float(*amax_word), 2688.0f);  // 6*448 = 7*384
    if (blockIdx.x == 0 && threadIdx.x == 0) *tensor_scale = s32;
  }
  TensorConsts c;
  c.scaled = !(s32 == 0.0f || (s32 >= 0x1p-20f && s32 <= 0x1p100f));
  c.k = 0;
  if (c.scaled) {
    c.k = -ilogbf(s32);
    s32 = scalbnf(s32, c.k);  // exact, now in [1, 2)
  }
  c.s32 = s32;
  c.r32 = (s32 > 0.0f) ? __frcp_rn(s32) : 0.0f;
  c.kd32 = kd_consts_checked(s32);
  c.kd6 = make_float2(__uint_as_float(kZh6Bits), __uint_as_float(kZl6Bits));
  c.kd7 = make_float2(__uint_as_float(kZh7Bits), __uint_as_float(kZl7Bits));
  return c;
}

// E2M1 codes of four pairs packed into one word (pair j in byte j, first
// element low), and each pair decoded back to f16x2.
__device__ __forceinline__ uint32_t e2m1_quad(const float (&lo)[4], const float (&hi)[4], uint32_t (&h2)[4]) {
  uint32_t word;
  asm("{ .reg .b8 t0, t1, t2, t3;\n"
      " cvt.rn.satfinite.e2m1x2.f32 t0, %6, %5;\n"
      " cvt.rn.satfinite.e2m1x2.f32 t1, %8, %7;\n"
      " cvt.rn.satfinite.e2m1x2.f32 t2, %10, %9;\n"
      " cvt.rn.satfinite.e2m1x2.f32 t3, %12, %11;\n"
      " cvt.rn.f16x2.e2m1x2 %1, t0;\n cvt.rn.f16x2.e2m1x2 %2, t1;\n"
      " cvt.rn.f16x2.e2m1x2 %3, t2;\n cvt.rn.f16x2.e2m1x2 %4, t3;\n"
      " mov.b32 %0, {t0, t1, t2, t3}; }"
      : "=r"(word), "=r"(h2[0]), "=r"(h2[1]), "=r"(h2[2]), "=r"(h2[3])
      : "f"(lo[0]), "f"(hi[0]), "f"(lo[1]), "f"(hi[1]), "f"(lo[2]), "f"(hi[2]), "f"(lo[3]), "f"(hi[3]));
  return word;
}

// Four byte values (each in the low byte of a word) packed into one word.
__device__ __forceinline__ uint32_t pack_low_bytes(uint32_t b0, uint32_t b1, uint32_t b2, uint32_t b3) {
  return prmt(prmt(b0, b1, 0x0040u), prmt(b2, b3, 0x0040u), 0x5410u);
}

// Sign nibble bits of 8 elements held in 4 bf16 pairs: element 2j -> bit 3 of
// byte j, element 2j+1 -> bit 7 (the sign bits of the code word).
__device__ __forceinline__ uint32_t sign_bits(uint32_t w0, uint32_t w1, uint32_t w2, uint32_t w3) {
  const uint32_t x = prmt(w0, w1, 0x7351u);   // [w0.b1, w1.b1, w0.b3, w1.b3]
  const uint32_t y = prmt(w2, w3, 0x7351u);
  const uint32_t even = prmt(x, y, 0x5410u);  // byte j bit 7 = sign of element 2j
  const uint32_t odd = prmt(x, y, 0x7632u);   // byte j bit 7 = sign of element 2j+1
  return (odd & 0x80808080u) | ((even >> 4) & 0x08080808u);
}

// |X_FP8| = |x| / s32 of 16 bf16 elements held as 8 pairs, as packed fp32
// pairs (element 2j in the low lane); kScaled / kMarkstein as described at
// the top of quantize.cu.
template <bool kScaled, bool kMarkstein>
__device__ __forceinline__ void x_fp8_magnitudes(const uint32_t w[8], const TensorConsts& tc, u64 a[8]) {
  const u64 ns32 = pack2(-tc.s32, -tc.s32), r32 = pack2(tc.r32, tc.r32);
  const u64 zh32 = pack2(tc.kd32.x, tc.kd32.x), zl32 = pack2(tc.kd32.y, tc.kd32.y);
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const uint32_t u = w[j] & 0x7FFF7FFFu;
    uint32_t lo = u << 16, hi = u & 0xFFFF0000u;
    if (kScaled) {
      lo = __float_as_uint(scalbnf(__uint_as_float(lo), tc.k));
      hi = __float_as_uint(scalbnf(__uint_as_float(hi), tc.k));
    }
    a[j] = kMarkstein ? div_rn2(bits2(lo, hi), ns32, r32) : div_kd2(bits2(lo, hi), zh32, zl32);
  }
}

// Algorithm 1 for one 16-element block held as 8 bf16 pairs.
//
// Tiny-value note: with s32 in [2^-20, 2^100], an element with |x| < 2^-102
// has |a| < 2^-82.  Its code magnitude is 0 under either candidate (every
// nonzero block scale is >= 2^-9, and a zero block scale forces 0), and its
// squared error is below 2^-160, which cannot change a binary32 sum.  So
// whether its quotient is correctly rounded does not affect any output.  The
// same holds for |a| < 2^-102 in the |a|/s8 step and for B < 2^-102, where
// both block scales round to E4M3 zero anyway.
//
// E1M2 clamp: when s8 = E4M3(b7) is normal (>= 2^-6) and b7 = fl32(B/7) did
// not saturate, s8 >= b7 / (1 + 2^-4), so |a|/s8 <= 7 * 1.0625 * (1 + 2^-23)
// < 7.5 and RNE never exceeds 7; only other blocks need the clamp.
// kMarkstein selects the x / s32 method (see the header); the other divisions
// always take the two-instruction form.
// Algorithm 1 from X_FP8 on, for one 16-element block: a holds |X_FP8| =
// |x| / s32 as packed pairs (element 2j in the low lane).  Returns the code
// words without their sign bits and the scale byte.
//
// kTile: the block is one row of a 16 x 16 tile whose 16 rows sit on the
// 16 lanes of a half-warp (2D blocks, reading R12): the block max becomes the
// tile max and each candidate's error sum becomes the pairwise tree of the 16
// rows' sums, lane i combining with lane i ^ 1, then i ^ 2, i ^ 4, i ^ 8
// (fp32 addition is commutative, so every lane ends with the same tree
// sum), so all 16 lanes choose the same format and scale.  Every lane of the
// warp must call it together.
template <int kMode, bool kTile = false>
__device__ __forceinline__ void block_core(const u64 a[8], const TensorConsts& tc, const float4* __restrict__ tab,
                                           uint32_t& mag_lo, uint32_t& mag_hi, uint32_t& scale_byte);

__device__ __forceinline__ float tile_max16(float v) {
#pragma unroll
  for (int m = 1; m < 16; m <<= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, m));
  return v;
}
__device__ __forceinline__ float tile_tree16(float v) {
#pragma unroll
  for (int m = 1; m < 16; m <<= 1) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, m));
  return v;
}

template <int kMode, bool kScaled, bool kMarkstein, bool kTile = false>
__device__ __forceinline__ void quantize_block(const uint32_t w[8], const TensorConsts& tc,
                                               const float4* __restrict__ tab, uint32_t& code_lo,
                                               uint32_t& code_hi, uint32_t& scale_byte) {
  u64 a[8];
  x_fp8_magnitudes<kScaled, kMarkstein>(w, tc, a);
  uint32_t mlo, mhi;
  block_core<kMode, kTile>(a, tc, tab, mlo, mhi, scale_byte);
  code_lo = mlo | sign_bits(w[0], w[1], w[2], w[3]);
  code_hi = mhi | sign_bits(w[4], w[5], w[6], w[7]);
}

// One E2M1 candidate of a block with scale table entry t = {s8, zh, zl}:
// the payload bytes (element 2j low) packed into two words and, with kErr,
// the R5 error sum (even / odd chains in the two lanes of a packed pair).
template <bool kErr, bool kTile>
__device__ __forceinline__ void e2m1_candidate(const u64 a[8], const float4 t, uint32_t& p_lo, uint32_t& p_hi,
                                               float& S) {
  const u64 zh8 = pack2(t.y, t.y), zl8 = pack2(t.z, t.z);
  const uint16_t ns8h = __half_as_ushort(__float2half_rn(-t.x));  // exact: E4M3 values are f16 values
  u64 acc = 0;  // (+0, +0): even / odd chains
  uint32_t pw[2];
#pragma unroll
  for (int g = 0; g < 2; ++g) {
    float ylo[4], yhi[4];
    uint32_t hq[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) unpack2(div_kd2(a[4 * g + i], zh8, zl8), ylo[i], yhi[i]);
    pw[g] = e2m1_quad(ylo, yhi, hq);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      if (!kErr) continue;
      const int j = 4 * g + i;
      float alo, ahi, dlo, dhi;
      unpack2(a[j], alo, ahi);
      // d = |a| - q s8 (exact), with q taken straight from its f16 decode
      asm("{ .reg .f16 ql, qh; mov.b32 {ql, qh}, %2;\n"
          " fma.rn.f32.f16 %0, ql, %3, %4;\n fma.rn.f32.f16 %1, qh, %3, %5; }"
          : "=f"(dlo), "=f"(dhi) : "r"(hq[i]), "h"(ns8h), "f"(alo), "f"(ahi));
      const u64 d = pack2(dlo, dhi);
      acc = fma2(d, d, acc);
    }
  }
  p_lo = pw[0];
  p_hi = pw[1];
  S = 0.0f;
  if (kErr) {
    float se, so;
    unpack2(acc, se, so);
    S = se + so;
    if (kTile) S = tile_tree16(S);
  }
}

template <int kMode, bool kTile>
__device__ __forceinline__ void block_core(const u64 a[8], const TensorConsts& tc, const float4* __restrict__ tab,
                                           uint32_t& mag_lo, uint32_t& mag_hi, uint32_t& scale_byte) {
  // Block max of |X_FP8|.
  float v[16];
#pragma unroll
  for (int j = 0; j < 8; ++j) unpack2(a[j], v[2 * j], v[2 * j + 1]);
  float B = max3f(max3f(v[0], v[1], v[2]), max3f(v[3], v[4], v[5]), max3f(v[6], v[7], v[8]));
  B = max3f(B, max3f(v[9], v[10], v[11]), max3f(v[12], v[13], max3f(v[14], v[15], 0.0f)));
  if (kTile) B = tile_max16(B);

  // Candidate block scales s8 = E4M3(fl32(B/6)), E4M3(fl32(B/7)) and RN(1/s8).
  const u64 bq = div_kd2(pack2(B, B), pack2(tc.kd6.x, tc.kd7.x), pack2(tc.kd6.y, tc.kd7.y));
  float b6, b7;
  unpack2(bq, b6, b7);

  if (kMode == MIXFP4_MODE_FOUR_SIX) {
    // {E2M1(6), E2M1(4)} (Sec. 2.4, reading R14): the second scale from
    // fl32(B/4) = B/4 exactly; both candidates are E2M1 (T = 0) and the later
    // one, E2M1(4), wins a tie.
    const uint32_t sc = cvt_e4m3x2(__fmul_rn(B, 0.25f), b6);  // low byte: B/6 code, high: B/4
    const uint32_t c6 = sc & 0x7Fu, c4 = (sc >> 8) & 0x7Fu;
    uint32_t p6lo, p6hi, p4lo, p4hi;
    float S6, S4;
    e2m1_candidate<true, kTile>(a, tab[c6], p6lo, p6hi, S6);
    e2m1_candidate<true, kTile>(a, tab[c4], p4lo, p4hi, S4);
    const bool four = S4 <= S6;
    mag_lo = four ? p4lo : p6lo;
    mag_hi = four ? p4hi : p6hi;
    scale_byte = four ? c4 : c6;
    return;
  }

  const uint32_t sc = cvt_e4m3x2(b7, b6);  // low byte: E2M1 scale code, high: E1M2
  const uint32_t c2 = sc & 0x7Fu, c1 = (sc >> 8) & 0x7Fu;

  float S2 = 0.0f, S1 = 0.0f;
  uint32_t p2lo = 0, p2hi = 0, p1lo = 0, p1hi = 0;
  if (kMode != MIXFP4_MODE_E1M2_ONLY)
    e2m1_candidate<kMode == MIXFP4_MODE_MIX, kTile>(a, tab[c2], p2lo, p2hi, S2);
  if (kMode != MIXFP4_MODE_E2M1_ONLY) {
    // E1M2 candidate (x2 units: integers 0..7).
    const float4 t = tab[c1];
    const u64 ns8 = pack2(-t.x, -t.x), zh8 = pack2(t.y, t.y), zl8 = pack2(t.z, t.z);
    const u64 magic = pack2(12582912.0f, 12582912.0f);    // 1.5 * 2^23
    const u64 nmagic = pack2(-12582912.0f, -12582912.0f);
    const bool clamp = !(t.x >= 0x1p-6f && b7 <= 448.0f);
    u64 acc = 0;
    uint32_t pb[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const u64 y = div_kd2(a[j], zh8, zl8);
      const u64 tq = add2(y, magic);  // RNE to an integer in the low mantissa bits
      uint32_t tlo = lo32(tq), thi = hi32(tq);
      if (clamp) {
        tlo = min(tlo, 0x4B400007u);
        thi = min(thi, 0x4B400007u);
      }
      pb[j] = tlo + (thi << 4);  // low byte: payload pair (first element low)
      if (kMode == MIXFP4_MODE_MIX) {
        const u64 q = add2(bits2(tlo, thi), nmagic);
        const u64 d = fma2(q, ns8, a[j]);
        acc = fma2(d, d, acc);
      }
    }
    p1lo = pack_low_bytes(pb[0], pb[1], pb[2], pb[3]);
    p1hi = pack_low_bytes(pb[4], pb[5], pb[6], pb[7]);
    if (kMode == MIXFP4_MODE_MIX) {
      float se, so;
      unpack2(acc, se, so);
      S1 = se + so;
      if (kTile) S1 = tile_tree16(S1);
    }
  }
  int T;
  if (kMode == MIXFP4_MODE_E2M1_ONLY) T = 0;
  else if (kMode == MIXFP4_MODE_E1M2_ONLY) T = 1;
  else T = (S2 < S1) ? 0 : 1;  // strict "<" of Algorithm 1

  mag_lo = T ? p1lo : p2lo;
  mag_hi = T ? p1hi : p2hi;
  scale_byte = T ? (0x80u | c1) : c2;
}

// ---- stochastic rounding (reading R13) --------------------------------------
// Philox4x32-10 (J. K. Salmon, M. A. Moraes, R. O. Dror, D. E. Shaw, "Parallel
// random numbers: as easy as 1, 2, 3", SC'11): ten rounds of two 32 x 32-bit
// products (multipliers 0xD2511F53, 0xCD9E8D57), key bumped by
// (0x9E3779B9, 0xBB67AE85) between rounds.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int round = 0; round < 10; ++round) {
    if (round > 0) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    const uint32_t lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
    const uint32_t lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
  }
  return c;
}

// Stochastic payloads of a magnitude m = |a| / s8 (exact fp32 arithmetic
// throughout): with l <= m < u the codebook neighbours, u iff eps < (m - l) /
// (u - l); m at or above the largest value saturates.  Branch-free (lanes of
// a warp hold blocks of either type and any magnitude): every gap u - l is a
// power of two (E2M1: 1/2 below 2, 1 below 4, 2 below 6; E1M2: 1), so
// v = m / (u - l) is an exact scaling, l's position is floor(v), and
// (m - l) / (u - l) = v - floor(v) exactly.
// One routine for both formats, its constants chosen per lane: E1M2 has gap
// 1 everywhere and saturates at 7; E2M1 as described, saturating at 6.
__device__ __forceinline__ uint32_t sr_payload(bool e1m2, float m, float eps) {
  const float sc = e1m2 ? 1.0f : (m < 2.0f ? 2.0f : (m < 4.0f ? 1.0f : 0.5f));
  // payload of l: E1M2 floor(m); E2M1 2 m below 2 (0..3), m + 2 below 4 (4, 5), 6 below 6
  const uint32_t add = e1m2 ? 0u : (m >= 2.0f ? 2u : 0u) + (m >= 4.0f ? 2u : 0u);
  const float v = m * sc, fl = floorf(v);
  const uint32_t p = (uint32_t)fl + add + (eps < v - fl ? 1u : 0u);
  return m < (e1m2 ? 7.0f : 6.0f) ? p : 7u;
}

// Algorithm 1 for one block (format and scale exactly as quantize_block
// chooses them), then the chosen format's codes rounded stochastically.  e0 is
// the logical index of the block's first element (a multiple of 16): element
// e0 + i draws word i % 4 of Philox4x32-10 with counter (e0 / 4 + i / 4,
// offset) and key seed, eps = (word >> 8) * 2^-24.
template <int kMode, bool kScaled, bool kMarkstein>
__device__ __forceinline__ void quantize_block_sr(const uint32_t w[8], const TensorConsts& tc,
                                                  const float4* __restrict__ tab, uint64_t seed, uint64_t offset,
                                                  uint64_t e0, uint32_t& code_lo, uint32_t& code_hi,
                                                  uint32_t& scale_byte) {
  u64 a[8];
  const u64 ns32 = pack2(-tc.s32, -tc.s32), r32 = pack2(tc.r32, tc.r32);
  const u64 zh32 = pack2(tc.kd32.x, tc.kd32.x), zl32 = pack2(tc.kd32.y, tc.kd32.y);
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const uint32_t u = w[j] & 0x7FFF7FFFu;
    uint32_t lo = u << 16, hi = u & 0xFFFF0000u;
    if (kScaled) {
      lo = __float_as_uint(scalbnf(__uint_as_float(lo), tc.k));
      hi = __float_as_uint(scalbnf(__uint_as_float(hi), tc.k));
    }
    a[j] = kMarkstein ? div_rn2(bits2(lo, hi), ns32, r32) : div_kd2(bits2(lo, hi), zh32, zl32);
  }
  uint32_t unused_lo, unused_hi;
  block_core<kMode>(a, tc, tab, unused_lo, unused_hi, scale_byte);
  const float4 t = tab[scale_byte & 0x7Fu];
  const bool e1m2 = (scale_byte >> 7) != 0;
  const u64 zh8 = pack2(t.y, t.y), zl8 = pack2(t.z, t.z);
  uint32_t bytes[8];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const uint64_t c = e0 / 4 + (uint64_t)q;
    const uint4 r = philox4x32_10(make_uint4((uint32_t)c, (uint32_t)(c >> 32), (uint32_t)offset,
                                             (uint32_t)(offset >> 32)),
                                  (uint32_t)seed, (uint32_t)(seed >> 32));
    const uint32_t rw[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
    for (int h = 0; h < 2; ++h) {  // pair j = 2q + h holds elements 4q + 2h, 4q + 2h + 1
      const int j = 2 * q + h;
      float mlo, mhi;
      unpack2(div_kd2(a[j], zh8, zl8), mlo, mhi);  // fl32(|a| / s8), as Algorithm 1's quotient
      const float elo = __uint2float_rn(rw[2 * h] >> 8) * 0x1p-24f;
      const float ehi = __uint2float_rn(rw[2 * h + 1] >> 8) * 0x1p-24f;
      const uint32_t plo = sr_payload(e1m2, mlo, elo), phi = sr_payload(e1m2, mhi, ehi);
      bytes[j] = plo | (phi << 4);
    }
  }
  code_lo = pack_low_bytes(bytes[0], bytes[1], bytes[2], bytes[3]) | sign_bits(w[0], w[1], w[2], w[3]);
  code_hi = pack_low_bytes(bytes[4], bytes[5], bytes[6], bytes[7]) | sign_bits(w[4], w[5], w[6], w[7]);
}

// E4M3 code -> {s8, zh, zl, 0} table of the block scales (zh, zl: see div_kd2),
// filled by the CTA's first 128 threads.
__device__ __forceinline__ void fill_scale_table(float4* tab) {
  for (int i = threadIdx.x; i < 128; i += blockDim.x) {
    float s8 = 0.0f, unused;
    if (i < 0x7F) f16x2_to_f32(cvt_f16x2_from_e4m3x2((uint16_t)i), s8, unused);
    const float2 kd = kd_consts(s8);
    tab[i] = make_float4(s8, kd.x, kd.y, 0.0f);
  }
}

// x / s32 may take the two-instruction division when it returns the IEEE
// quotient for all 128 bf16 significands (the quotient scales exactly with
// x's exponent) and its correction term a*zl stays normal for every quotient
// that can matter (|a| >= 2^-82; see the tiny-value note): the remainder
// 1 - s32*zh is 0 or at least 2^-44 in magnitude.  The reference quotient is
// Markstein's form, which equals the IEEE quotient for every bf16 numerator
// significand and every fp32 divisor significand (checked exhaustively on the
// host).  Threads 0..127 check one significand each; every thread of the CTA
// must call this (it ends with a CTA barrier) and all get the same answer:
// true = use Markstein's form.
__device__ __forceinline__ bool markstein_needed(const TensorConsts& tc) {
  bool kd_ok = true;
  if (threadIdx.x < 128 && !tc.scaled) {
    const float xs = __uint_as_float(0x3F800000u | (threadIdx.x << 16));
    const u64 x2 = pack2(xs, xs);
    const u64 q = div_kd2(x2, pack2(tc.kd32.x, tc.kd32.x), pack2(tc.kd32.y, tc.kd32.y));
    const u64 ref = div_rn2(x2, pack2(-tc.s32, -tc.s32), pack2(tc.r32, tc.r32));
    const float rem = __fmaf_rn(-tc.s32, tc.kd32.x, 1.0f);
    kd_ok = tc.s32 > 0.0f && lo32(q) == lo32(ref) && (rem == 0.0f || fabsf(rem) >= 0x1p-44f);
  }
  return !__syncthreads_and(kd_ok);
}

template <bool kContig>
__device__ __forceinline__ const uint16_t* block_src(const uint16_t* x, int64_t b, int64_t kblocks, int64_t ldx) {
  if (kContig) return x + b * 16;
  const int64_t row = b / kblocks;
  return x + row * ldx + (b - row * kblocks) * 16;
}

// ---- 128-point Walsh-Hadamard rotation before quantization ----------------
// Reading R11 of the random Hadamard transform (Sec. 4.1 "+RHT", Sec. 3.2): each
// 128-element chunk of a row along K is rotated on its own: elements whose bit
// in the caller's 128-bit sign vector is set are negated, the Sylvester
// product H_128 v is formed by the radix-2 butterfly in fp32 with strides
// 1, 2, 4, ..., 64 in that order ((a, b) -> (a + b, a - b)), and every value
// is multiplied by c = RN(1/sqrt(128)).  Algorithm 1 then runs on the fp32
// values.  Threads hold one 16-element block each, so the 8 lanes 8g..8g+7 of
// a warp hold one chunk (block t of the chunk on lane 8g + t): strides 1-8 run
// inside a thread, strides 16, 32, 64 between lanes by shuffles.
constexpr uint32_t kRhtScaleBits = 0x3DB504F3u;  // RN(1/sqrt(128))

// Sign masks of this thread's 16 chunk positions 16 * (lane & 7) + e, as bf16
// word masks (bit 15: element 2j, bit 31: element 2j + 1).
__device__ __forceinline__ void rht_sign_words(const uint8_t* __restrict__ signs, int lane, uint32_t sw[8]) {
  uint32_t bits = 0;
  if (signs) {
    const int pos = lane & 7;
    bits = (uint32_t)__ldg(signs + 2 * pos) | ((uint32_t)__ldg(signs + 2 * pos + 1) << 8);
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) sw[j] = (((bits >> (2 * j)) & 1u) << 15) | (((bits >> (2 * j + 1)) & 1u) << 31);
}

// The rotated block of this thread as packed fp32 pairs (element 2j low).
// Every lane of the 8-lane group must call this together.
__device__ __forceinline__ void rht_rotate(const uint32_t w[8], const uint32_t sw[8], int lane, u64 y[8]) {
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const uint32_t u = w[j] ^ sw[j];
    const float lo = __uint_as_float(u << 16), hi = __uint_as_float(u & 0xFFFF0000u);
    y[j] = pack2(__fadd_rn(lo, hi), __fsub_rn(lo, hi));  // stride 1
  }
#pragma unroll
  for (int h = 1; h < 8; h <<= 1)  // strides 2, 4, 8 (h pairs apart)
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if ((j & h) == 0) {
        const u64 a = y[j], b = y[j + h];
        y[j] = add2(a, b);
        y[j + h] = sub2(a, b);
      }
  const unsigned gmask = 0xFFu << (lane & 24);
#pragma unroll
  for (int m = 1; m < 8; m <<= 1) {  // strides 16, 32, 64: partner lane ^ m
    // lower lane: own + other; upper lane: other - own (fma with -1 rounds the same)
    const float k = (lane & m) ? -1.0f : 1.0f;
    const u64 kk = pack2(k, k);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const uint32_t olo = __shfl_xor_sync(gmask, lo32(y[j]), m);
      const uint32_t ohi = __shfl_xor_sync(gmask, hi32(y[j]), m);
      y[j] = fma2(y[j], kk, bits2(olo, ohi));
    }
  }
  const float c = __uint_as_float(kRhtScaleBits);
  const u64 cc = pack2(c, c);
#pragma unroll
  for (int j = 0; j < 8; ++j) y[j] = mul2(y[j], cc);
}

// Sign nibble bits of 8 fp32 values held in 4 pairs: element 2j -> bit 3 of
// byte j, element 2j + 1 -> bit 7.
__device__ __forceinline__ uint32_t f32_sign_bits(const u64 y[4]) {
  const uint32_t e = prmt(prmt(lo32(y[0]), lo32(y[1]), 0x0073u), prmt(lo32(y[2]), lo32(y[3]), 0x0073u), 0x5410u);
  const uint32_t o = prmt(prmt(hi32(y[0]), hi32(y[1]), 0x0073u), prmt(hi32(y[2]), hi32(y[3]), 0x0073u), 0x5410u);
  return (o & 0x80808080u) | ((e >> 4) & 0x08080808u);
}

// Algorithm 1 on one rotated block: x / s32 for fp32 numerators by
// Markstein's correction (correctly rounded for every fp32 numerator down to
// the tiny-value bound, see the header), then the common core.
template <int kMode, bool kScaled>
__device__ __forceinline__ void rht_block(const u64 y[8], const TensorConsts& tc, const float4* __restrict__ tab,
                                          uint32_t& code_lo, uint32_t& code_hi, uint32_t& scale_byte) {
  u64 a[8];
  const u64 ns32 = pack2(-tc.s32, -tc.s32), r32 = pack2(tc.r32, tc.r32);
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    uint32_t lo = lo32(y[j]) & 0x7FFFFFFFu, hi = hi32(y[j]) & 0x7FFFFFFFu;
    if (kScaled) {
      lo = __float_as_uint(scalbnf(__uint_as_float(lo), tc.k));
      hi = __float_as_uint(scalbnf(__uint_as_float(hi), tc.k));
    }
    a[j] = div_rn2(bits2(lo, hi), ns32, r32);
  }
  uint32_t mlo, mhi;
  block_core<kMode>(a, tc, tab, mlo, mhi, scale_byte);
  code_lo = mlo | f32_sign_bits(y);
  code_hi = mhi | f32_sign_bits(y + 4);
}

// Rotation + Algorithm 1 (rht_quantize_kernel): the grid stride is a multiple
// of 8 blocks, so the 8 lanes of a chunk stay together at every step.
}  // namespace
}  // namespace mixfp4
