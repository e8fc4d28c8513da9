// MixFP4 online quantizer (Algorithm 1, Sec. 3.2), tensor amax, and decoder
// (App. B.2/B.3) for sm_103a.
//
// Design (HBM-bound, 2.5625 algorithmic bytes per element):
//   * one thread owns one 16-element block at a time: a single 256-bit
//     coalesced load (a warp reads 1 KiB of contiguous bf16), one 64-bit code
//     store and one scale-byte store (a warp writes 256 B and 32 B
//     contiguous); each thread quantizes two such blocks side by side;
//   * all per-element fp32 work runs on packed f32x2 instructions;
//   * every division of Algorithm 1 (x/s32, B/6, B/7, |a|/s8) is evaluated as
//     IEEE round-to-nearest with a divisor known in advance, in two packed
//     instructions (N. Brisebarre, J.-M. Muller, S. K. Raina, "Accelerating
//     correctly rounded floating-point division when the divisor is known in
//     advance", IEEE Trans. Computers 53(8), 2004):
//         q = RN(a*zh + RN(a*zl)),  zh = RN(1/b),  zl = RN(RN(1 - b*zh)/b).
//     This is not correctly rounded for every divisor, so each use is covered
//     by a check: exhaustive on the host for the divisors 6, 7 and every E4M3
//     value (every fp32 significand of a), and, for x/s32, at run time in the
//     kernel over all 128 bf16 significands of x (2 of the 2^23 fp32
//     significands of s32 fail; those tensors use Markstein's correction,
//     P. Markstein 1990; Muller et al., Handbook of Floating-Point Arithmetic,
//     Sec. 4.9:  q0 = RN(a*r), e = RN(a - q0*b) (exact via fma),
//     q = RN(q0 + e*r), r = RN(1/b)).  Both return RN(a/b) whenever a >=
//     2^-102 and the quotient is normal; smaller numerators only occur where
//     their exact value cannot change a code or an error sum (see the
//     tiny-value note in quantize_block), and tensors whose s32 lies outside
//     [2^-20, 2^100] are first rescaled by an exact power of two;
//   * E2M1 rounding uses cvt.rn.satfinite.e2m1x2 (RNE, saturating) and E4M3
//     scale rounding cvt.rn.satfinite.e4m3x2; E1M2 rounding adds 1.5*2^23
//     (RNE to an integer) and clamps the integer to 7.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "host_util.cuh"
#include "kernels.cuh"
#include "ptx.cuh"
#include "quant_core.cuh"

namespace mixfp4 {

namespace {

// Persistent grid: each thread walks blocks b, b + nthr, b + 2 nthr, ... two
// at a time (a, b): both blocks of a pair are quantized before either is
// stored, so their independent dependency chains interleave, and the loads of
// the next pair are in flight meanwhile.  The division method is fixed per
// launch, so each method gets its own copy of the loop.
template <int kMode, bool kContig, bool kScaled, bool kMarkstein>
__device__ __forceinline__ void quantize_pairs(const uint16_t* __restrict__ x, int64_t b, int64_t nthr,
                                               int64_t nblocks, int64_t kblocks, int64_t ldx,
                                               uint8_t* __restrict__ codes, uint8_t* __restrict__ scales,
                                               const TensorConsts& tc, const float4* __restrict__ tab,
                                               uint32_t (&wa)[8], uint32_t (&wb)[8]) {
  for (; b < nblocks; b += 2 * nthr) {
    const int64_t b1 = b + nthr;
    uint32_t lo0, hi0, sb0, lo1, hi1, sb1;
    quantize_block<kMode, kScaled, kMarkstein>(wa, tc, tab, lo0, hi0, sb0);
    quantize_block<kMode, kScaled, kMarkstein>(wb, tc, tab, lo1, hi1, sb1);  // wb past the end: unused
    stg64(codes + b * 8, lo0, hi0);
    scales[b] = (uint8_t)sb0;
    if (b + 2 * nthr < nblocks) ldg256_stream(block_src<kContig>(x, b + 2 * nthr, kblocks, ldx), wa);
    if (b1 < nblocks) {
      stg64(codes + b1 * 8, lo1, hi1);
      scales[b1] = (uint8_t)sb1;
      if (b1 + 2 * nthr < nblocks) ldg256_stream(block_src<kContig>(x, b1 + 2 * nthr, kblocks, ldx), wb);
    }
  }
}

// The first loads are issued before any set-up work.
template <int kMode, bool kContig>
__global__ void __launch_bounds__(kQuantThreads, 4)
quantize_kernel(const uint16_t* __restrict__ x, int64_t nblocks, int64_t kblocks, int64_t ldx,
                uint8_t* __restrict__ codes, uint8_t* __restrict__ scales, float* tensor_scale,
                const uint32_t* amax_word, int scale_given, int after_amax) {
  __shared__ float4 tab[128];  // E4M3 code -> {s8, zh, zl, 0} (zh, zl: see div_kd2)
  // Launched as a programmatic dependent of the amax kernel (after_amax), x
  // is already complete and may be read before that kernel finishes; only
  // the amax word must wait.  Otherwise wait before touching any input.
  if (!after_amax) griddep_wait();
  griddep_launch_dependents();
  const int64_t nthr = (int64_t)gridDim.x * kQuantThreads;
  const int64_t b = (int64_t)blockIdx.x * kQuantThreads + threadIdx.x;
  uint32_t wa[8], wb[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) wb[j] = 0u;  // defined values for a missing second block
  if (b < nblocks) ldg256_stream(block_src<kContig>(x, b, kblocks, ldx), wa);
  if (b + nthr < nblocks) ldg256_stream(block_src<kContig>(x, b + nthr, kblocks, ldx), wb);
  fill_scale_table(tab);
  if (after_amax) griddep_wait();
  const TensorConsts tc = tensor_consts(tensor_scale, amax_word, scale_given);
  const bool markstein = markstein_needed(tc);
  if (tc.scaled)
    quantize_pairs<kMode, kContig, true, true>(x, b, nthr, nblocks, kblocks, ldx, codes, scales, tc, tab, wa, wb);
  else if (markstein)
    quantize_pairs<kMode, kContig, false, true>(x, b, nthr, nblocks, kblocks, ldx, codes, scales, tc, tab, wa, wb);
  else
    quantize_pairs<kMode, kContig, false, false>(x, b, nthr, nblocks, kblocks, ldx, codes, scales, tc, tab, wa, wb);
}

// Rotation + Algorithm 1, two blocks per thread side by side (as in
// quantize_kernel); the rotated pairs take 2 CTAs per SM of registers.
template <int kMode, bool kContig>
__global__ void __launch_bounds__(kQuantThreads, 2)
rht_quantize_kernel(const uint16_t* __restrict__ x, int64_t nblocks, int64_t kblocks, int64_t ldx,
                    const uint8_t* __restrict__ signs, uint8_t* __restrict__ codes, uint8_t* __restrict__ scales,
                    float* tensor_scale, const uint32_t* amax_word, int scale_given, int after_amax) {
  __shared__ float4 tab[128];
  if (!after_amax) griddep_wait();
  griddep_launch_dependents();
  const int lane = threadIdx.x & 31;
  const int64_t nthr = (int64_t)gridDim.x * kQuantThreads;
  int64_t b = (int64_t)blockIdx.x * kQuantThreads + threadIdx.x;
  uint32_t w[8], w2[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) w2[j] = 0u;
  if (b < nblocks) ldg256_stream(block_src<kContig>(x, b, kblocks, ldx), w);
  if (b + nthr < nblocks) ldg256_stream(block_src<kContig>(x, b + nthr, kblocks, ldx), w2);
  if (threadIdx.x < 128) {
    float s8 = 0.0f, unused;
    if (threadIdx.x < 0x7F) f16x2_to_f32(cvt_f16x2_from_e4m3x2((uint16_t)threadIdx.x), s8, unused);
    const float2 kd = kd_consts(s8);
    tab[threadIdx.x] = make_float4(s8, kd.x, kd.y, 0.0f);
  }
  uint32_t sw[8];
  rht_sign_words(signs, lane, sw);
  if (after_amax) griddep_wait();
  const TensorConsts tc = tensor_consts(tensor_scale, amax_word, scale_given);
  __syncthreads();
  for (; b < nblocks; b += 2 * nthr) {
    const int64_t b1 = b + nthr;
    u64 y[8], y2[8];
    rht_rotate(w, sw, lane, y);
    rht_rotate(w2, sw, lane, y2);  // the 8 lanes of a chunk agree on b1 < nblocks
    if (b + 2 * nthr < nblocks) ldg256_stream(block_src<kContig>(x, b + 2 * nthr, kblocks, ldx), w);
    if (b1 + 2 * nthr < nblocks) ldg256_stream(block_src<kContig>(x, b1 + 2 * nthr, kblocks, ldx), w2);
    uint32_t lo, hi, sb, lo2, hi2, sb2;
    if (tc.scaled) {
      rht_block<kMode, true>(y, tc, tab, lo, hi, sb);
      rht_block<kMode, true>(y2, tc, tab, lo2, hi2, sb2);
    } else {
      rht_block<kMode, false>(y, tc, tab, lo, hi, sb);
      rht_block<kMode, false>(y2, tc, tab, lo2, hi2, sb2);
    }
    stg64(codes + b * 8, lo, hi);
    scales[b] = (uint8_t)sb;
    if (b1 < nblocks) {
      stg64(codes + b1 * 8, lo2, hi2);
      scales[b1] = (uint8_t)sb2;
    }
  }
}

// max |y| of the rotated tensor as the bit pattern of a non-negative fp32.
template <bool kContig>
__global__ void __launch_bounds__(256)
rht_amax_kernel(const uint16_t* __restrict__ x, int64_t nblocks, int64_t kblocks, int64_t ldx,
                const uint8_t* __restrict__ signs, uint32_t* amax_word) {
  const int lane = threadIdx.x & 31;
  uint32_t sw[8];
  rht_sign_words(signs, lane, sw);
  uint32_t m = 0;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  int64_t b = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  uint32_t w[8];
  if (b < nblocks) ldg256_stream(block_src<kContig>(x, b, kblocks, ldx), w);
  for (; b < nblocks; b += stride) {
    uint32_t wn[8];  // the next block's load is in flight during this block's rotation
    if (b + stride < nblocks) ldg256_stream(block_src<kContig>(x, b + stride, kblocks, ldx), wn);
    u64 y[8];
    rht_rotate(w, sw, lane, y);
#pragma unroll
    for (int j = 0; j < 8; ++j) m = max(m, max(lo32(y[j]) & 0x7FFFFFFFu, hi32(y[j]) & 0x7FFFFFFFu));
#pragma unroll
    for (int j = 0; j < 8; ++j) w[j] = wn[j];
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = max(m, __shfl_xor_sync(0xffffffffu, m, o));
  __shared__ uint32_t red[8];
  if (lane == 0) red[threadIdx.x >> 5] = m;
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int i = 1; i < (int)(blockDim.x >> 5); ++i) m = max(m, red[i]);
    if (m) atomicMax(amax_word, m);
  }
  griddep_launch_dependents();
}

// max |x| over the tensor as the bit pattern of a non-negative fp32 (bf16
// magnitudes order like unsigned 16-bit integers).  Each thread keeps four
// 32-byte loads in flight.
constexpr int kAmaxUnroll = 4;

template <bool kContig>
__device__ __forceinline__ const uint16_t* amax_src(const uint16_t* x, int64_t b, int64_t kblocks, int64_t ldx) {
  if (kContig) return x + b * 16;
  const int64_t row = b / kblocks;
  return x + row * ldx + (b - row * kblocks) * 16;
}

template <bool kContig>
__global__ void __launch_bounds__(256)
amax_kernel(const uint16_t* __restrict__ x, int64_t nblocks, int64_t kblocks, int64_t ldx,
            uint32_t* amax_word) {
  uint32_t m = 0;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t b = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; b < nblocks; b += kAmaxUnroll * stride) {
    uint32_t w[kAmaxUnroll][8];
#pragma unroll
    for (int u = 0; u < kAmaxUnroll; ++u) {
      const int64_t bu = b + u * stride;
      if (bu < nblocks) ldg256_stream(amax_src<kContig>(x, bu, kblocks, ldx), w[u]);
      else
#pragma unroll
        for (int j = 0; j < 8; ++j) w[u][j] = 0u;
    }
#pragma unroll
    for (int u = 0; u < kAmaxUnroll; ++u)
#pragma unroll
      for (int j = 0; j < 8; ++j) m = __vmaxu2(m, w[u][j] & 0x7FFF7FFFu);
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
  // The quantize kernel that follows may start once every CTA got here.
  griddep_launch_dependents();
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
  int64_t grid = (nblocks + 256 * kAmaxUnroll - 1) / (256 * kAmaxUnroll);
  if (grid > num_sms() * 8) grid = num_sms() * 8;
  if (ldx == K) amax_kernel<true><<<(unsigned)grid, 256, 0, stream>>>(x, nblocks, kblocks, ldx, amax_word);
  else amax_kernel<false><<<(unsigned)grid, 256, 0, stream>>>(x, nblocks, kblocks, ldx, amax_word);
  return 0;
}

int launch_quantize(const uint16_t* x, int64_t rows, int64_t K, int64_t ldx, uint8_t* codes,
                    uint8_t* scales, float* tensor_scale, const uint32_t* amax_word, int mode,
                    int scale_given, cudaStream_t stream) {
  const int64_t kblocks = K / 16, nblocks = rows * kblocks;
  // Persistent grid: 4 CTAs per SM of the device, fewer for small tensors
  // (each thread takes at least two blocks).
  int64_t grid = (nblocks + 2 * kQuantThreads - 1) / (2 * kQuantThreads);
  if (grid > num_sms() * 4) grid = num_sms() * 4;
  if (grid == 0) return 0;
  // Launched as a programmatic dependent: it overlaps its launch with the tail
  // of the kernel before it (see the waits at the top of quantize_kernel).
  const int after_amax = !scale_given;
#define MIXFP4_LAUNCH_Q(MODE)                                                                           \
  do {                                                                                                  \
    if (ldx == K)                                                                                       \
      launch_pdl(quantize_kernel<MODE, true>, (unsigned)grid, kQuantThreads, 0, stream, x, nblocks,      \
                 kblocks, ldx, codes, scales, tensor_scale, amax_word, scale_given, after_amax);        \
    else                                                                                                \
      launch_pdl(quantize_kernel<MODE, false>, (unsigned)grid, kQuantThreads, 0, stream, x, nblocks,     \
                 kblocks, ldx, codes, scales, tensor_scale, amax_word, scale_given, after_amax);        \
  } while (0)
  switch (mode) {
    case MIXFP4_MODE_MIX: MIXFP4_LAUNCH_Q(MIXFP4_MODE_MIX); break;
    case MIXFP4_MODE_E2M1_ONLY: MIXFP4_LAUNCH_Q(MIXFP4_MODE_E2M1_ONLY); break;
    case MIXFP4_MODE_FOUR_SIX: MIXFP4_LAUNCH_Q(MIXFP4_MODE_FOUR_SIX); break;
    default: MIXFP4_LAUNCH_Q(MIXFP4_MODE_E1M2_ONLY); break;
  }
#undef MIXFP4_LAUNCH_Q
  return 0;
}

int launch_rht_amax(const uint16_t* x, int64_t rows, int64_t K, int64_t ldx, const uint8_t* signs,
                    uint32_t* amax_word, cudaStream_t stream) {
  const int64_t kblocks = K / 16, nblocks = rows * kblocks;
  if (nblocks == 0) return 0;
  int64_t grid = (nblocks + 255) / 256;
  if (grid > num_sms() * 8) grid = num_sms() * 8;
  if (ldx == K) rht_amax_kernel<true><<<(unsigned)grid, 256, 0, stream>>>(x, nblocks, kblocks, ldx, signs, amax_word);
  else rht_amax_kernel<false><<<(unsigned)grid, 256, 0, stream>>>(x, nblocks, kblocks, ldx, signs, amax_word);
  return 0;
}

int launch_rht_quantize(const uint16_t* x, int64_t rows, int64_t K, int64_t ldx, const uint8_t* signs,
                        uint8_t* codes, uint8_t* scales, float* tensor_scale, const uint32_t* amax_word, int mode,
                        int scale_given, cudaStream_t stream) {
  const int64_t kblocks = K / 16, nblocks = rows * kblocks;
  int64_t grid = (nblocks + kQuantThreads - 1) / kQuantThreads;
  if (grid > num_sms() * 2) grid = num_sms() * 2;
  if (grid == 0) return 0;
  const int after_amax = !scale_given;
#define MIXFP4_LAUNCH_R(MODE)                                                                            \
  do {                                                                                                   \
    if (ldx == K)                                                                                        \
      launch_pdl(rht_quantize_kernel<MODE, true>, (unsigned)grid, kQuantThreads, 0, stream, x, nblocks,   \
                 kblocks, ldx, signs, codes, scales, tensor_scale, amax_word, scale_given, after_amax);  \
    else                                                                                                 \
      launch_pdl(rht_quantize_kernel<MODE, false>, (unsigned)grid, kQuantThreads, 0, stream, x, nblocks,  \
                 kblocks, ldx, signs, codes, scales, tensor_scale, amax_word, scale_given, after_amax);  \
  } while (0)
  switch (mode) {
    case MIXFP4_MODE_MIX: MIXFP4_LAUNCH_R(MIXFP4_MODE_MIX); break;
    case MIXFP4_MODE_E2M1_ONLY: MIXFP4_LAUNCH_R(MIXFP4_MODE_E2M1_ONLY); break;
    default: MIXFP4_LAUNCH_R(MIXFP4_MODE_E1M2_ONLY); break;
  }
#undef MIXFP4_LAUNCH_R
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
