// Candidate-set and block-size quantize-dequantize (reading R14): Algorithm 1
// with the per-block MSE choice taken over any subset of four FP4 candidates
// -- E2M1 with largest value 6 (Algorithm 1's E2M1), E1M2 in x2 units, E2M1
// with the block max mapped to 4, and E3M0 (Eq. 1-2 with W_E = 3, W_M = 0:
// {0, 1/4, ..., 16}) -- and blocks of g = 8, 16, 32 or 64 elements.  These are
// the paper's ablations (Sec. 2.4 candidate sets, Sec. 4.3 Table 5 block
// sizes).  The stored MixFP4 format holds one type bit, so the kernel returns
// what the ablations measure: the dequantized tensor (fp32 or bf16) and each
// block's chosen candidate.
//
// One thread holds 16 consecutive elements of a row (one 32-byte load).  A
// g = 8 thread carries two blocks; a g = 32 / 64 block spans 2 / 4 adjacent
// lanes, which combine the block max and each candidate's error sum with xor
// shuffles (lane i with i ^ 1, then i ^ 2: the pairwise tree of the 16-element
// sums, the same on every lane because fp32 addition is commutative).  The
// divisions are the quantizer's (quant_core.cuh): x / s32, B / 6, B / 7 and
// |a| / s8 in the checked two-instruction form on packed pairs (x / s32 with
// Markstein's correction where the run-time check asks for it); B / 4 and
// B / 16 are exact scalings.  The E4M3 scale and the E2M1 codes come from the
// hardware conversions (round to nearest even, saturating), E1M2 from rint,
// E3M0 from the exponent and mantissa bits.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "host_util.cuh"
#include "kernels.cuh"
#include "ptx.cuh"
#include "quant_core.cuh"

namespace mixfp4 {
namespace {

constexpr int kFqThreads = 256;

// E3M0 magnitude nearest to y >= 0: 0 or 2^e, e = -2..4, ties to the even
// payload.  The payload of 2^e is e + 3, so between 2^e and 2^(e+1) a tie
// (mantissa exactly 1.5) goes up iff the biased fp32 exponent of 2^e is odd:
// round up iff mantissa + (exponent bit 0) > 2^22.  Then 16 caps the top;
// below 1/4 the neighbours are 0 and 1/4, with the tie 1/8 going to 0.
__device__ __forceinline__ float e3m0_round(float y) {
  const uint32_t u = __float_as_uint(y);
  const bool up = (u & 0x007FFFFFu) + ((u >> 23) & 1u) > 0x00400000u;
  const float p2 = fminf(__uint_as_float((u & 0x7F800000u) + (up ? 0x00800000u : 0u)), 16.0f);
  return y > 0.125f ? fmaxf(p2, 0.25f) : 0.0f;
}

// One candidate of a block part: s8 from the block max, codes of the pairs
// a[j0 .. j0 + kPairs - 1], their values q (packed, in candidate units) and
// the error sum (even elements in the low lane chain, odd in the high).
template <int kPairs>
__device__ __forceinline__ void candidate_part(int c, const u64* a, float B, const TensorConsts& tc,
                                               const float4* __restrict__ tab, u64* q, float& s8, float& se,
                                               float& so) {
  float bd;  // fl32(B / divisor): 6 and 7 by the checked two-instruction form, 4 and 16 exactly
  if (c == 0) bd = __fmaf_rn(B, tc.kd6.x, __fmul_rn(B, tc.kd6.y));
  else if (c == 1) bd = __fmaf_rn(B, tc.kd7.x, __fmul_rn(B, tc.kd7.y));
  else if (c == 2) bd = __fmul_rn(B, 0.25f);
  else bd = __fmul_rn(B, 0.0625f);
  const float4 t = tab[cvt_e4m3x2(0.0f, bd) & 0x7Fu];  // R2: E4M3 RNE, saturating
  s8 = t.x;
  const u64 zh8 = pack2(t.y, t.y), zl8 = pack2(t.z, t.z), ns8 = pack2(-t.x, -t.x);
  u64 acc = 0;
#pragma unroll
  for (int j = 0; j < kPairs; ++j) {
    float ylo, yhi, qlo, qhi;
    unpack2(div_kd2(a[j], zh8, zl8), ylo, yhi);  // fl32(|a| / s8); s8 = 0 gives 0
    if (c == 1) {
      qlo = fminf(rintf(ylo), 7.0f);
      qhi = fminf(rintf(yhi), 7.0f);
    } else if (c == 3) {
      qlo = e3m0_round(ylo);
      qhi = e3m0_round(yhi);
    } else {
      f16x2_to_f32(cvt_f16x2_from_e2m1x2(cvt_e2m1x2(yhi, ylo)), qlo, qhi);
    }
    q[j] = pack2(qlo, qhi);
    const u64 d = fma2(q[j], ns8, a[j]);  // |a| - q s8, the product exact
    acc = fma2(d, d, acc);
  }
  unpack2(acc, se, so);
}

template <int kG>
__device__ __forceinline__ void fake_quantize_unit(const u64 a[8], const TensorConsts& tc, float s32,
                                                   const float4* __restrict__ tab, int mask, float o[16],
                                                   int best_c[2]) {
  constexpr int kParts = kG == 8 ? 2 : 1;  // blocks per thread
  constexpr int kPairs = 8 / kParts;      // element pairs of a block held by one thread
#pragma unroll
  for (int p = 0; p < kParts; ++p) {
    float v[2 * kPairs];
#pragma unroll
    for (int j = 0; j < kPairs; ++j) unpack2(a[p * kPairs + j], v[2 * j], v[2 * j + 1]);
    float B = 0.0f;
#pragma unroll
    for (int i = 0; i < 2 * kPairs; ++i) B = fmaxf(B, v[i]);
    if (kG >= 32) B = fmaxf(B, __shfl_xor_sync(0xffffffffu, B, 1));
    if (kG == 64) B = fmaxf(B, __shfl_xor_sync(0xffffffffu, B, 2));
    float best_S = 0.0f, best_s8 = 0.0f;
    u64 qb[kPairs];
    best_c[p] = -1;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      if (!((mask >> c) & 1)) continue;  // uniform over the launch
      u64 q[kPairs];
      float s8, se, so;
      candidate_part<kPairs>(c, a + p * kPairs, B, tc, tab, q, s8, se, so);
      float S = __fadd_rn(se, so);
      if (kG >= 32) S = __fadd_rn(S, __shfl_xor_sync(0xffffffffu, S, 1));
      if (kG == 64) S = __fadd_rn(S, __shfl_xor_sync(0xffffffffu, S, 2));
      if (best_c[p] < 0 || S <= best_S) {  // a later candidate wins a tie
        best_c[p] = c;
        best_S = S;
        best_s8 = s8;
#pragma unroll
        for (int j = 0; j < kPairs; ++j) qb[j] = q[j];
      }
    }
    const u64 s8s = pack2(best_s8, best_s8), s32s = pack2(s32, s32);
#pragma unroll
    for (int j = 0; j < kPairs; ++j) unpack2(mul2(mul2(qb[j], s8s), s32s), o[2 * (p * kPairs + j)],
                                             o[2 * (p * kPairs + j) + 1]);
  }
}

template <int kG>
__global__ void __launch_bounds__(kFqThreads)
fake_quantize_kernel(const uint16_t* __restrict__ x, int64_t rows, int64_t K, int64_t ldx, int mask,
                     float* tensor_scale, const uint32_t* amax_word, int scale_given, void* __restrict__ out,
                     int out_bf16, int64_t ldo, uint8_t* __restrict__ choice) {
  __shared__ float4 tab[128];  // E4M3 code -> {s8, zh, zl, 0}
  griddep_wait();
  griddep_launch_dependents();
  fill_scale_table(tab);
  const TensorConsts tc = tensor_consts(tensor_scale, amax_word, scale_given);
  const bool markstein = markstein_needed(tc);  // ends with a CTA barrier (tab is ready)
  const float s32 = tc.scaled ? scalbnf(tc.s32, -tc.k) : tc.s32;  // the tensor's own s32 (exact)
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
    float o[16];
    int best_c[2] = {0, 0};
    u64 a[8];  // |X_FP8| pairs (R1, R7)
    if (tc.scaled) x_fp8_magnitudes<true, true>(w, tc, a);
    else if (markstein) x_fp8_magnitudes<false, true>(w, tc, a);
    else x_fp8_magnitudes<false, false>(w, tc, a);
    fake_quantize_unit<kG>(a, tc, s32, tab, mask, o, best_c);
    if (live) {
      uint32_t ow[16];
#pragma unroll
      for (int i = 0; i < 8; ++i) {  // sign(x) on the magnitudes
        ow[2 * i] = __float_as_uint(o[2 * i]) | ((w[i] & 0x8000u) << 16);
        ow[2 * i + 1] = __float_as_uint(o[2 * i + 1]) | (w[i] & 0x80000000u);
      }
      if (out_bf16) {
        uint32_t hw[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const __nv_bfloat162 h = __floats2bfloat162_rn(__uint_as_float(ow[2 * i]), __uint_as_float(ow[2 * i + 1]));
          hw[i] = *reinterpret_cast<const uint32_t*>(&h);  // low half: element 2i
        }
        stg256(static_cast<uint16_t*>(out) + r * ldo + j * 16, hw);
      } else {
        float* dst = static_cast<float*>(out) + r * ldo + j * 16;
        stg256(dst, ow);
        stg256(dst + 8, ow + 8);
      }
      if (choice) {
        constexpr int kLanes = kG >= 16 ? kG / 16 : 1;  // lanes sharing one block
        if constexpr (kG == 8) {
          *reinterpret_cast<uint16_t*>(choice + r * (K / 8) + 2 * j) = (uint16_t)(best_c[0] | (best_c[1] << 8));
        } else if ((lane & (kLanes - 1)) == 0) {
          choice[r * (K / kG) + j / kLanes] = (uint8_t)best_c[0];
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
  if (grid > num_sms() * 8) grid = num_sms() * 8;
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
