// MixFP4 online quantizer (Algorithm 1, Sec. 3.2), tensor amax, and decoder
// (App. B.2/B.3) for sm_103a.
//
// Design (HBM-bound, 2.5625 algorithmic bytes per element):
//   * one thread owns one 16-element block: a single 256-bit coalesced load
//     (a warp reads 1 KiB of contiguous bf16), one 64-bit code store and one
//     scale-byte store (a warp writes 256 B and 32 B contiguous);
//   * all per-element fp32 work runs on packed f32x2 instructions;
//   * every division of Algorithm 1 (x/s32, B/6, B/7, |a|/s8) is evaluated as
//     IEEE round-to-nearest by Markstein's correction (P. Markstein, "Computation
//     of elementary functions on the IBM RISC System/6000 processor", 1990;
//     Muller et al., Handbook of Floating-Point Arithmetic, Sec. 4.9):
//         q0 = RN(a*r),  e = RN(a - q0*b) (exact via fma),  q = RN(q0 + e*r)
//     with r = RN(1/b).  It returns RN(a/b) whenever a >= 2^-102 and the
//     quotient is normal; smaller numerators only occur where their exact
//     value cannot change a code or an error sum (see the tiny-value note in
//     quantize_block), and tensors whose s32 lies outside [2^-20, 2^100] are
//     first rescaled by an exact power of two;
//   * E2M1 rounding uses cvt.rn.satfinite.e2m1x2 (RNE, saturating) and E4M3
//     scale rounding cvt.rn.satfinite.e4m3x2; E1M2 rounding adds 1.5*2^23
//     (RNE to an integer) and clamps the integer to 7.
#include <cuda_runtime.h>
#include <cstdint>

#include "ptx.cuh"
#include "kernels.cuh"

namespace mixfp4 {

namespace {

constexpr int kQuantThreads = 256;

// Correctly rounded a / b (per lane) given nb = -b and r = RN(1/b).
__device__ __forceinline__ u64 div_rn2(u64 a, u64 nb, u64 r) {
  u64 q0 = mul2(a, r);
  u64 e = fma2(q0, nb, a);
  return fma2(e, r, q0);
}

__device__ __forceinline__ uint32_t lo32(u64 v) { return (uint32_t)v; }
__device__ __forceinline__ uint32_t hi32(u64 v) { return (uint32_t)(v >> 32); }

struct TensorConsts {
  float s32;   // per-tensor scale, possibly rescaled to [1, 2)
  float r32;   // RN(1/s32), or 0 when s32 == 0
  float r6, r7;  // RN(1/6), RN(1/7)
  int k;       // |x| is multiplied by 2^k when `scaled`
  int scaled;
};

// Derive the per-tensor constants once per CTA (thread 0), broadcast via smem.
__device__ __forceinline__ TensorConsts tensor_consts(float* tensor_scale,
                                                      const uint32_t* amax_word, int scale_given,
                                                      TensorConsts* sh) {
  if (threadIdx.x == 0) {
    float s32;
    if (scale_given) {
      s32 = *tensor_scale;
    } else {
      s32 = __fdiv_rn(__uint_as_float(*amax_word), 2688.0f);  // 6*448 = 7*384
      if (blockIdx.x == 0) *tensor_scale = s32;
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
    c.r6 = __frcp_rn(6.0f);
    c.r7 = __frcp_rn(7.0f);
    *sh = c;
  }
  __syncthreads();
  return *sh;
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
template <int kMode, bool kScaled>
__device__ __forceinline__ void quantize_block(const uint32_t w[8], const TensorConsts& tc,
                                               uint32_t& code_lo, uint32_t& code_hi,
                                               uint32_t& scale_byte) {
  // |x| as packed fp32 pairs (element 2j in the low lane).
  u64 a[8];
  const u64 ns32 = pack2(-tc.s32, -tc.s32), r32 = pack2(tc.r32, tc.r32);
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    uint32_t lo = (w[j] << 16) & 0x7FFF0000u, hi = w[j] & 0x7FFF0000u;
    if (kScaled) {
      lo = __float_as_uint(scalbnf(__uint_as_float(lo), tc.k));
      hi = __float_as_uint(scalbnf(__uint_as_float(hi), tc.k));
    }
    a[j] = div_rn2(bits2(lo, hi), ns32, r32);  // X_FP8 = X / s32 (magnitudes)
  }
  // Block max of |X_FP8|.
  float v[16];
#pragma unroll
  for (int j = 0; j < 8; ++j) unpack2(a[j], v[2 * j], v[2 * j + 1]);
  float B = max3f(max3f(v[0], v[1], v[2]), max3f(v[3], v[4], v[5]), max3f(v[6], v[7], v[8]));
  B = max3f(B, max3f(v[9], v[10], v[11]), max3f(v[12], v[13], max3f(v[14], v[15], 0.0f)));

  // Candidate block scales s8 = E4M3(fl32(B/6)), E4M3(fl32(B/7)).
  u64 bq = div_rn2(pack2(B, B), pack2(-6.0f, -7.0f), pack2(tc.r6, tc.r7));
  float b6, b7;
  unpack2(bq, b6, b7);
  const uint32_t sc = cvt_e4m3x2(b7, b6);  // low byte: E2M1 scale code, high: E1M2
  float s8_2, s8_1;
  f16x2_to_f32(cvt_f16x2_from_e4m3x2((uint16_t)sc), s8_2, s8_1);

  // Sign nibble bits: element 2j -> bit 3 of code byte j, 2j+1 -> bit 7.
  uint32_t sgn[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) sgn[j] = ((w[j] >> 12) & 0x08u) | ((w[j] >> 24) & 0x80u);

  float S2 = 0.0f, S1 = 0.0f;
  uint32_t pay2[8], pay1[8];
  if (kMode != MIXFP4_MODE_E1M2_ONLY) {
    // E2M1 candidate.
    const float rr = (s8_2 > 0.0f) ? __frcp_rn(s8_2) : 0.0f;
    const u64 ns8 = pack2(-s8_2, -s8_2), r8 = pack2(rr, rr);
    u64 acc = 0;  // (+0, +0): even / odd chains
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      u64 y = div_rn2(a[j], ns8, r8);
      float ylo, yhi;
      unpack2(y, ylo, yhi);
      const uint32_t c = cvt_e2m1x2(yhi, ylo);
      pay2[j] = c;
      float qlo, qhi;
      f16x2_to_f32(cvt_f16x2_from_e2m1x2(c), qlo, qhi);
      u64 d = fma2(pack2(qlo, qhi), ns8, a[j]);  // |a| - q s8 (exact)
      acc = fma2(d, d, acc);
    }
    float se, so;
    unpack2(acc, se, so);
    S2 = se + so;
  }
  if (kMode != MIXFP4_MODE_E2M1_ONLY) {
    // E1M2 candidate (x2 units: integers 0..7).
    const float rr = (s8_1 > 0.0f) ? __frcp_rn(s8_1) : 0.0f;
    const u64 ns8 = pack2(-s8_1, -s8_1), r8 = pack2(rr, rr);
    const u64 magic = pack2(12582912.0f, 12582912.0f);    // 1.5 * 2^23
    const u64 nmagic = pack2(-12582912.0f, -12582912.0f);
    u64 acc = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      u64 y = div_rn2(a[j], ns8, r8);
      u64 t = add2(y, magic);  // RNE to an integer in the low mantissa bits
      const uint32_t tlo = min(lo32(t), 0x4B400007u), thi = min(hi32(t), 0x4B400007u);
      pay1[j] = (tlo & 7u) | ((thi & 7u) << 4);
      u64 q = add2(bits2(tlo, thi), nmagic);
      u64 d = fma2(q, ns8, a[j]);
      acc = fma2(d, d, acc);
    }
    float se, so;
    unpack2(acc, se, so);
    S1 = se + so;
  }
  int T;
  if (kMode == MIXFP4_MODE_E2M1_ONLY) T = 0;
  else if (kMode == MIXFP4_MODE_E1M2_ONLY) T = 1;
  else T = (S2 < S1) ? 0 : 1;  // strict "<" of Algorithm 1

  code_lo = 0;
  code_hi = 0;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    uint32_t p;
    if (kMode == MIXFP4_MODE_E2M1_ONLY) p = pay2[j];
    else if (kMode == MIXFP4_MODE_E1M2_ONLY) p = pay1[j];
    else p = T ? pay1[j] : pay2[j];
    const uint32_t byte = (p | sgn[j]) & 0xFFu;
    if (j < 4) code_lo |= byte << (8 * j);
    else code_hi |= byte << (8 * (j - 4));
  }
  scale_byte = T ? (0x80u | ((sc >> 8) & 0x7Fu)) : (sc & 0x7Fu);
}

template <int kMode, bool kContig>
__global__ void __launch_bounds__(kQuantThreads)
quantize_kernel(const uint16_t* __restrict__ x, int64_t nblocks, int64_t kblocks, int64_t ldx,
                uint8_t* __restrict__ codes, uint8_t* __restrict__ scales, float* tensor_scale,
                const uint32_t* amax_word, int scale_given) {
  __shared__ TensorConsts sh;
  const TensorConsts tc = tensor_consts(tensor_scale, amax_word, scale_given, &sh);
  const int64_t b = (int64_t)blockIdx.x * kQuantThreads + threadIdx.x;
  if (b >= nblocks) return;
  const uint16_t* src;
  if (kContig) {
    src = x + b * 16;
  } else {
    const int64_t row = b / kblocks;
    src = x + row * ldx + (b - row * kblocks) * 16;
  }
  uint32_t w[8];
  ldg256_stream(src, w);
  uint32_t lo, hi, sb;
  if (tc.scaled) quantize_block<kMode, true>(w, tc, lo, hi, sb);
  else quantize_block<kMode, false>(w, tc, lo, hi, sb);
  stg64(codes + b * 8, lo, hi);
  scales[b] = (uint8_t)sb;
}

// max |x| over the tensor as the bit pattern of a non-negative fp32 (bf16
// magnitudes order like unsigned 16-bit integers).
template <bool kContig>
__global__ void __launch_bounds__(256)
amax_kernel(const uint16_t* __restrict__ x, int64_t nblocks, int64_t kblocks, int64_t ldx,
            uint32_t* amax_word) {
  uint32_t m = 0;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t b = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; b < nblocks; b += stride) {
    const uint16_t* src;
    if (kContig) {
      src = x + b * 16;
    } else {
      const int64_t row = b / kblocks;
      src = x + row * ldx + (b - row * kblocks) * 16;
    }
    uint32_t w[8];
    ldg256_stream(src, w);
#pragma unroll
    for (int j = 0; j < 8; ++j) m = __vmaxu2(m, w[j] & 0x7FFF7FFFu);
  }
  m = max(m & 0xFFFFu, m >> 16);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = max(m, __shfl_xor_sync(0xffffffffu, m, o));
  __shared__ uint32_t red[8];
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = m;
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int i = 1; i < (int)(blockDim.x >> 5); ++i) m = max(m, red[i]);
    if (m) atomicMax(amax_word, m << 16);
  }
}

// out = fl32(sign * v * s8 * s32): v * s8 is exact in fp32, one rounding.
__global__ void __launch_bounds__(256)
dequantize_kernel(const uint8_t* __restrict__ codes, const uint8_t* __restrict__ scales,
                  const float* tensor_scale, int64_t nblocks, float* __restrict__ out) {
  const int64_t b = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= nblocks) return;
  const float s32 = *tensor_scale;
  const uint2 c = *reinterpret_cast<const uint2*>(codes + b * 8);
  const uint32_t s = scales[b];
  float s8, unused;
  f16x2_to_f32(cvt_f16x2_from_e4m3x2((uint16_t)(s & 0x7Fu)), s8, unused);
  const bool e1m2 = (s >> 7) != 0;
  uint32_t o[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    const uint32_t word = i < 8 ? c.x : c.y;
    const uint32_t nib = (word >> (4 * (i & 7))) & 0xFu;
    const uint32_t p = nib & 7u;
    float vv;
    if (e1m2) {
      vv = (float)p;  // x2 remapped E1M2: the payload as an integer
    } else {
      // E2M1 {0, .5, 1, 1.5, 2, 3, 4, 6}: (1 + m/2) * 2^(e-1), subnormal m/2.
      const uint32_t e = p >> 1, m = p & 1u;
      vv = e ? ldexpf(1.0f + 0.5f * (float)m, (int)e - 1) : 0.5f * (float)m;
    }
    float val = __fmul_rn(__fmul_rn(vv, s8), s32);
    o[i] = __float_as_uint(val) ^ ((nib & 8u) << 28);
  }
  stg256(out + b * 16, o);
  stg256(out + b * 16 + 8, o + 8);
}

}  // namespace

int launch_amax(const uint16_t* x, int64_t rows, int64_t K, int64_t ldx, uint32_t* amax_word,
                cudaStream_t stream) {
  const int64_t kblocks = K / 16, nblocks = rows * kblocks;
  if (nblocks == 0) return 0;
  int64_t grid = (nblocks + 255) / 256;
  if (grid > 152 * 16) grid = 152 * 16;
  if (ldx == K) amax_kernel<true><<<(unsigned)grid, 256, 0, stream>>>(x, nblocks, kblocks, ldx, amax_word);
  else amax_kernel<false><<<(unsigned)grid, 256, 0, stream>>>(x, nblocks, kblocks, ldx, amax_word);
  return 0;
}

int launch_quantize(const uint16_t* x, int64_t rows, int64_t K, int64_t ldx, uint8_t* codes,
                    uint8_t* scales, float* tensor_scale, const uint32_t* amax_word, int mode,
                    int scale_given, cudaStream_t stream) {
  const int64_t kblocks = K / 16, nblocks = rows * kblocks;
  const int64_t grid = (nblocks + kQuantThreads - 1) / kQuantThreads;
  if (grid == 0) return 0;
#define MIXFP4_LAUNCH_Q(MODE)                                                              \
  do {                                                                                     \
    if (ldx == K)                                                                          \
      quantize_kernel<MODE, true><<<(unsigned)grid, kQuantThreads, 0, stream>>>(            \
          x, nblocks, kblocks, ldx, codes, scales, tensor_scale, amax_word, scale_given);   \
    else                                                                                   \
      quantize_kernel<MODE, false><<<(unsigned)grid, kQuantThreads, 0, stream>>>(           \
          x, nblocks, kblocks, ldx, codes, scales, tensor_scale, amax_word, scale_given);   \
  } while (0)
  switch (mode) {
    case MIXFP4_MODE_MIX: MIXFP4_LAUNCH_Q(MIXFP4_MODE_MIX); break;
    case MIXFP4_MODE_E2M1_ONLY: MIXFP4_LAUNCH_Q(MIXFP4_MODE_E2M1_ONLY); break;
    default: MIXFP4_LAUNCH_Q(MIXFP4_MODE_E1M2_ONLY); break;
  }
#undef MIXFP4_LAUNCH_Q
  return 0;
}

int launch_dequantize(const uint8_t* codes, const uint8_t* scales, const float* tensor_scale,
                      int64_t rows, int64_t K, float* out, cudaStream_t stream) {
  const int64_t nblocks = rows * (K / 16);
  const int64_t grid = (nblocks + 255) / 256;
  if (grid == 0) return 0;
  dequantize_kernel<<<(unsigned)grid, 256, 0, stream>>>(codes, scales, tensor_scale, nblocks, out);
  return 0;
}

}  // namespace mixfp4
