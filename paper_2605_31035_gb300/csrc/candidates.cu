// Candidate-set and block-size quantize-dequantize (reading R14): Algorithm 1
// with the per-block MSE choice taken over any subset of four FP4 candidates
// -- E2M1 with largest value 6 (Algorithm 1's E2M1), E1M2 in x2 units, E2M1
// with the block max mapped to 4, and E3M0 (Eq. 1-2 with W_E = 3, W_M = 0:
// {0, 1/4, ..., 16}) -- and blocks of g = 8, 16, 32 or 64 elements.  These are
// the paper's ablations (Sec. 2.3 candidate sets, Sec. 5 Table 5 block
// sizes).  The stored MixFP4 format holds one type bit, so the kernel returns
// what the ablations measure: the dequantized tensor (fp32 or bf16) and each
// block's chosen candidate.
//
// One thread holds 16 consecutive elements of a row (one 32-byte load).  A
// g = 8 thread carries two blocks; a g = 32 / 64 block spans 2 / 4 adjacent
// lanes, which combine the block max and each candidate's error sum with xor
// shuffles (lane i with i ^ 1, then i ^ 2: the pairwise tree of the 16-element
// sums, the same on every lane because fp32 addition is commutative).  Every
// division is the correctly rounded one (__fdiv_rn); the E4M3 scale and the
// E2M1 codes come from the hardware conversions (round to nearest even,
// saturating), E1M2 from rint, E3M0 from the exponent and mantissa bits.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "kernels.cuh"
#include "ptx.cuh"

namespace mixfp4 {
namespace {

constexpr int kFqThreads = 256;

// E4M3 value nearest to v >= 0 (ties to even, saturating at 448, subnormals).
__device__ __forceinline__ float e4m3_round(float v) {
  const uint32_t h2 = cvt_f16x2_from_e4m3x2(cvt_e4m3x2(0.0f, v));
  float lo, hi;
  f16x2_to_f32(h2, lo, hi);
  return lo;
}

// E2M1 magnitude nearest to y >= 0 (ties to the even payload, saturating at 6).
__device__ __forceinline__ float e2m1_round(float y) {
  float lo, hi;
  f16x2_to_f32(cvt_f16x2_from_e2m1x2(cvt_e2m1x2(0.0f, y)), lo, hi);
  return lo;
}

// E3M0 magnitude nearest to y >= 0: 0 or 2^e, e = -2..4, ties to the even
// payload (payload of 2^e is e + 3, so of the two neighbours the one whose
// biased fp32 exponent is even).
__device__ __forceinline__ float e3m0_round(float y) {
  if (y >= 16.0f) return 16.0f;
  if (y < 0.25f) return y > 0.125f ? 0.25f : 0.0f;  // 1/8 is a tie between payloads 0 and 1
  const uint32_t u = __float_as_uint(y);
  const uint32_t ebits = u & 0x7F800000u, m = u & 0x007FFFFFu;
  const float lo = __uint_as_float(ebits);
  const bool up = m > 0x00400000u || (m == 0x00400000u && ((ebits >> 23) & 1u));
  return up ? 2.0f * lo : lo;
}

__device__ __forceinline__ float cand_round(int c, float y) {
  if (c == 1) return fminf(rintf(y), 7.0f);
  if (c == 3) return e3m0_round(y);
  return e2m1_round(y);  // c = 0, 2
}

template <int kG>
__global__ void __launch_bounds__(kFqThreads)
fake_quantize_kernel(const uint16_t* __restrict__ x, int64_t rows, int64_t K, int64_t ldx, int mask,
                     float* tensor_scale, const uint32_t* amax_word, int scale_given, void* __restrict__ out,
                     int out_bf16, int64_t ldo, uint8_t* __restrict__ choice) {
  constexpr int kParts = kG == 8 ? 2 : 1;  // blocks per thread
  constexpr int kLen = 16 / kParts;       // elements of a block held by one thread
  griddep_wait();
  griddep_launch_dependents();
  float s32;
  if (scale_given) {
    s32 = *tensor_scale;
  } else {
    s32 = __fdiv_rn(__uint_as_float(*amax_word), 2688.0f);  // 6 * 448
    if (blockIdx.x == 0 && threadIdx.x == 0) *tensor_scale = s32;
  }
  const int lane = threadIdx.x & 31;
  const int64_t kb = K / 16, nsub = rows * kb;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  // Warp-uniform loop: the lanes of a g > 16 block shuffle together.
  for (int64_t base = warp * 32; base < nsub; base += nwarps * 32) {
    const int64_t b = base + lane;
    const bool live = b < nsub;
    const int64_t r = live ? b / kb : 0, j = live ? b % kb : 0;
    uint32_t w[8];
    if (live) {
      ldg256_stream(x + r * ldx + j * 16, w);
    } else {
#pragma unroll
      for (int i = 0; i < 8; ++i) w[i] = 0u;
    }
    float a[16];
    uint32_t neg = 0u;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float lo = __uint_as_float(w[i] << 16), hi = __uint_as_float(w[i] & 0xFFFF0000u);
      neg |= ((w[i] >> 15) & 1u) << (2 * i);
      neg |= (w[i] >> 31) << (2 * i + 1);
      a[2 * i] = s32 > 0.0f ? __fdiv_rn(fabsf(lo), s32) : 0.0f;      // R1, R7
      a[2 * i + 1] = s32 > 0.0f ? __fdiv_rn(fabsf(hi), s32) : 0.0f;
    }
    float B[kParts];
#pragma unroll
    for (int p = 0; p < kParts; ++p) {
      B[p] = 0.0f;
#pragma unroll
      for (int i = 0; i < kLen; ++i) B[p] = fmaxf(B[p], a[p * kLen + i]);
      if (kG >= 32) B[p] = fmaxf(B[p], __shfl_xor_sync(0xffffffffu, B[p], 1));
      if (kG == 64) B[p] = fmaxf(B[p], __shfl_xor_sync(0xffffffffu, B[p], 2));
    }
    float best_S[kParts], best_s8[kParts], q_best[16];
    int best_c[kParts];
#pragma unroll
    for (int p = 0; p < kParts; ++p) {
      best_S[p] = 0.0f;
      best_s8[p] = 0.0f;
      best_c[p] = -1;
    }
#pragma unroll
    for (int i = 0; i < 16; ++i) q_best[i] = 0.0f;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      if (!((mask >> c) & 1)) continue;  // uniform over the launch
      const float div = c == 0 ? 6.0f : c == 1 ? 7.0f : c == 2 ? 4.0f : 16.0f;
#pragma unroll
      for (int p = 0; p < kParts; ++p) {
        const float s8 = e4m3_round(__fdiv_rn(B[p], div));  // R2
        float q[kLen], se = 0.0f, so = 0.0f;
#pragma unroll
        for (int i = 0; i < kLen; ++i) {
          const float y = s8 > 0.0f ? __fdiv_rn(a[p * kLen + i], s8) : 0.0f;
          q[i] = cand_round(c, y);
          const float d = __fmaf_rn(q[i], s8, -a[p * kLen + i]);  // q s8 is exact
          if (i & 1) so = __fmaf_rn(d, d, so);
          else se = __fmaf_rn(d, d, se);
        }
        float S = __fadd_rn(se, so);
        if (kG >= 32) S = __fadd_rn(S, __shfl_xor_sync(0xffffffffu, S, 1));
        if (kG == 64) S = __fadd_rn(S, __shfl_xor_sync(0xffffffffu, S, 2));
        if (best_c[p] < 0 || S <= best_S[p]) {  // a later candidate wins a tie
          best_c[p] = c;
          best_S[p] = S;
          best_s8[p] = s8;
#pragma unroll
          for (int i = 0; i < kLen; ++i) q_best[p * kLen + i] = q[i];
        }
      }
    }
    if (live) {
      float o[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const float v = __fmul_rn(__fmul_rn(q_best[i], best_s8[i / kLen]), s32);
        o[i] = ((neg >> i) & 1u) ? -v : v;
      }
      if (out_bf16) {
        uint32_t ow[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const uint32_t lo = __bfloat16_as_ushort(__float2bfloat16_rn(o[2 * i]));
          const uint32_t hi = __bfloat16_as_ushort(__float2bfloat16_rn(o[2 * i + 1]));
          ow[i] = lo | (hi << 16);
        }
        stg256(static_cast<uint16_t*>(out) + r * ldo + j * 16, ow);
      } else {
        float* dst = static_cast<float*>(out) + r * ldo + j * 16;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          uint32_t ow[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) ow[i] = __float_as_uint(o[8 * h + i]);
          stg256(dst + 8 * h, ow);
        }
      }
      if (choice) {
        if (kG == 8) {
          *reinterpret_cast<uint16_t*>(choice + r * (K / 8) + 2 * j) =
              (uint16_t)(best_c[0] | (best_c[kParts - 1] << 8));
        } else if (kG == 16) {
          choice[r * kb + j] = (uint8_t)best_c[0];
        } else if ((lane & (kG / 16 - 1)) == 0) {
          choice[r * (K / kG) + j / (kG / 16)] = (uint8_t)best_c[0];
        }
      }
    }
  }
}

}  // namespace

int launch_fake_quantize(const uint16_t* x, int64_t rows, int64_t K, int64_t ldx, int candidates, int block,
                         float* tensor_scale, const uint32_t* amax_word, int scale_given, void* out, int out_bf16,
                         int64_t ldo, uint8_t* choice, cudaStream_t stream) {
  const int64_t nsub = rows * (K / 16);
  if (nsub == 0) return 0;
  int64_t grid = (nsub + kFqThreads - 1) / kFqThreads;
  if (grid > 152 * 8) grid = 152 * 8;
  cudaError_t e;
#define MIXFP4_LAUNCH_FQ(G)                                                                                  \
  e = launch_pdl(fake_quantize_kernel<G>, (unsigned)grid, kFqThreads, 0, stream, x, rows, K, ldx, candidates, \
                 tensor_scale, amax_word, scale_given, out, out_bf16, ldo, choice)
  switch (block) {
    case 8: MIXFP4_LAUNCH_FQ(8); break;
    case 16: MIXFP4_LAUNCH_FQ(16); break;
    case 32: MIXFP4_LAUNCH_FQ(32); break;
    default: MIXFP4_LAUNCH_FQ(64); break;
  }
#undef MIXFP4_LAUNCH_FQ
  return e == cudaSuccess ? 0 : -1;
}

}  // namespace mixfp4
