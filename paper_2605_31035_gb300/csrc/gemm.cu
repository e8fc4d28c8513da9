// MixFP4 x MixFP4 GEMM for sm_103a: C = A_deq . B_deq^T (App. B.1 Eq. (factor)).
//
// Per 16-element block the MixFP4 codes are decoded to the unified E2M2 value
// (Sec. 3.3, App. B.5) times the block's E4M3 scale.  Written as 2*v*s8 that
// product has at most 7 significant bits and lies in [2^-9, 2*7*448], so it is
// exact in bf16; the tensor cores then contract bf16 x bf16 with fp32
// accumulation (tcgen05.mma kind::f16, K = 16 = one block per instruction) and
// the epilogue applies s32A * s32B / 4.
//
// One CTA computes a 128 x 256 tile of C:
//   warp 0      TMA producer: packed codes [rows][128 B] (128-byte swizzle) and
//               scales [rows][16 B] for a 256-wide K slice, into a 2-deep ring;
//   warp 1      TMEM allocator and single-thread MMA issuer (accumulator
//               128 lanes x 256 fp32 columns in tensor memory);
//   warps 2-13  decoders, one thread per tile row (128 A rows + 256 B rows):
//               each turns 64 K of its row per sub-stage into bf16 in the
//               canonical K-major no-swizzle UMMA layout, in a 2-deep ring;
//   warps 2-9   after the K loop: epilogue, tcgen05.ld -> scale -> global fp32.
// All pipeline waits are bounded; a wait that gives up records a nonzero
// status word and the CTA drains and exits without touching C.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "kernels.cuh"
#include "ptx.cuh"
#include "sm100.cuh"

namespace mixfp4 {
namespace {

using namespace sm100;

constexpr int BM = 128;            // tile rows of A (MMA M)
constexpr int BN = 256;            // tile rows of B (MMA N)
constexpr int BKC = 256;           // K per TMA code stage
constexpr int BKD = 64;            // K per decoded sub-stage
constexpr int kSub = BKC / BKD;    // sub-stages per code stage
constexpr int kCodeStages = 2;
constexpr int kDecStages = 2;
constexpr int kDecodeWarps = (BM + BN) / 32;   // 12
constexpr int kThreads = 32 * (2 + kDecodeWarps);
constexpr uint32_t kTmemCols = 256;

constexpr int A_CODE_BYTES = BM * BKC / 2;
constexpr int B_CODE_BYTES = BN * BKC / 2;
constexpr int A_SCALE_BYTES = BM * BKC / 16;
constexpr int B_SCALE_BYTES = BN * BKC / 16;
constexpr int CODE_STAGE_BYTES = A_CODE_BYTES + B_CODE_BYTES + A_SCALE_BYTES + B_SCALE_BYTES;
constexpr int A_DEC_BYTES = BM * BKD * 2;
constexpr int B_DEC_BYTES = BN * BKD * 2;
constexpr int DEC_STAGE_BYTES = A_DEC_BYTES + B_DEC_BYTES;
constexpr int OFF_DEC = kCodeStages * CODE_STAGE_BYTES;
constexpr int OFF_BAR = OFF_DEC + kDecStages * DEC_STAGE_BYTES;
constexpr int SMEM_BYTES = OFF_BAR + 256;
constexpr int SMEM_ALLOC = SMEM_BYTES + 1024;  // slack to align the base to 1024 B

static_assert(CODE_STAGE_BYTES % 1024 == 0, "code stages must keep 1024-byte alignment");
static_assert(SMEM_ALLOC <= 232448, "shared memory budget");

// Decoded-operand layout: core matrix (8 rows x 16 B) at
//   (row / 8) * SBO + kchunk * LBO + (row % 8) * 16
constexpr uint32_t kLBO = 128;                  // next 8 K-elements
constexpr uint32_t kSBO = (BKD / 8) * 128;      // next 8 rows (1024 B)
constexpr uint32_t kIdesc = idesc_bf16_f32(BM, BN);

constexpr uint64_t kWaitLimitNs = 1000000000ull;  // 1 s per pipeline wait

struct Bars {
  uint64_t code_full[kCodeStages];
  uint64_t code_empty[kCodeStages];
  uint64_t dec_full[kDecStages];
  uint64_t dec_empty[kDecStages];
  uint64_t acc_full;
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
};
static_assert(sizeof(Bars) <= 256, "barrier block");

__device__ __forceinline__ void sts128(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" :: "r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}
__device__ __forceinline__ uint4 lds128(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.b32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr) : "memory");
  return v;
}
__device__ __forceinline__ uint32_t fma_bf16x2(uint32_t a, uint32_t b, uint32_t c) {
  uint32_t d;
  asm("fma.rn.bf16x2 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}
__device__ __forceinline__ uint32_t bf16x2_splat(float v) {
  uint32_t d;
  asm("cvt.rn.bf16x2.f32 %0, %1, %1;" : "=r"(d) : "f"(v));
  return d;
}
__device__ __forceinline__ uint32_t lop_xor_and(uint32_t a, uint32_t b, uint32_t mask) {
  return a ^ (b & mask);
}

// Decode 8 consecutive codes (one 32-bit word, element 2j in the low nibble of
// byte j) of a block to 8 bf16 values 2*v*s8 = u*s8, u = 2v:
//   E2M1 u in {0,1,2,3,4,6,8,12}, E1M2 u in {0,2,...,14} (selected by the LUT).
// u is looked up with prmt, turned into the bf16 128+u, and
//   fma(128+u, s8, -128*s8) = u*s8 exactly; the nibble sign is then XORed in.
__device__ __forceinline__ void decode8(uint32_t w, uint32_t lut_lo, uint32_t lut_hi, uint32_t s2,
                                        uint32_t c2, uint32_t out[4]) {
  const uint32_t wp = w & 0x77777777u;
  const uint32_t u0 = prmt(lut_lo, lut_hi, wp);
  const uint32_t u1 = prmt(lut_lo, lut_hi, wp >> 16);
  const uint32_t ws = w << 4;
  const uint32_t k43 = 0x43434343u;
  const uint32_t m0 = prmt(u0, k43, 0x4140u), m1 = prmt(u0, k43, 0x4342u);
  const uint32_t m2 = prmt(u1, k43, 0x4140u), m3 = prmt(u1, k43, 0x4342u);
  out[0] = lop_xor_and(fma_bf16x2(m0, s2, c2), prmt(w, ws, 0x0040u), 0x80008000u);
  out[1] = lop_xor_and(fma_bf16x2(m1, s2, c2), prmt(w, ws, 0x1050u), 0x80008000u);
  out[2] = lop_xor_and(fma_bf16x2(m2, s2, c2), prmt(w, ws, 0x2060u), 0x80008000u);
  out[3] = lop_xor_and(fma_bf16x2(m3, s2, c2), prmt(w, ws, 0x3070u), 0x80008000u);
}

__global__ void __launch_bounds__(kThreads, 1)
mixfp4_gemm_kernel(const __grid_constant__ CUtensorMap tm_ac, const __grid_constant__ CUtensorMap tm_bc,
                   const __grid_constant__ CUtensorMap tm_as, const __grid_constant__ CUtensorMap tm_bs,
                   const float* __restrict__ a_ts, const float* __restrict__ b_ts,
                   int M, int N, int K, float* __restrict__ C, long long ldc,
                   uint32_t* status_word) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  Bars* bars = reinterpret_cast<Bars*>(smem + OFF_BAR);
  volatile int* abort_flag = &bars->abort;
  const uint32_t sbase = smem_u32(smem);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN;
  const int num_kc = K / BKC;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kCodeStages; ++s) {
      mbar_init(smem_u32(&bars->code_full[s]), 1);
      mbar_init(smem_u32(&bars->code_empty[s]), kDecodeWarps);
    }
    for (int s = 0; s < kDecStages; ++s) {
      mbar_init(smem_u32(&bars->dec_full[s]), kDecodeWarps);
      mbar_init(smem_u32(&bars->dec_empty[s]), 1);
    }
    mbar_init(smem_u32(&bars->acc_full), 1);
    mbar_init(smem_u32(&bars->drain), 1);
    bars->abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&bars->tmem_base), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_acc = bars->tmem_base;

  auto fail = [&](uint32_t code) {
    *abort_flag = 1;
    if (status_word) atomicOr(status_word, code);
  };

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      tma_prefetch(&tm_ac);
      tma_prefetch(&tm_bc);
      tma_prefetch(&tm_as);
      tma_prefetch(&tm_bs);
      int last_phase[kCodeStages];
      for (int s = 0; s < kCodeStages; ++s) last_phase[s] = -1;
      for (int kc = 0; kc < num_kc; ++kc) {
        const int s = kc % kCodeStages;
        const uint32_t ph = (kc / kCodeStages) & 1;
        if (!mbar_wait(smem_u32(&bars->code_empty[s]), ph ^ 1, abort_flag, kWaitLimitNs)) {
          fail(1u);
          break;
        }
        const uint32_t st = sbase + s * CODE_STAGE_BYTES;
        const uint32_t fb = smem_u32(&bars->code_full[s]);
        mbar_arrive_expect_tx(fb, CODE_STAGE_BYTES);
        const int xk = kc * (BKC / 2), xs = kc * (BKC / 16);
        tma_load_2d(st, &tm_ac, xk, m0, fb);
        tma_load_2d(st + A_CODE_BYTES, &tm_bc, xk, n0, fb);
        tma_load_2d(st + A_CODE_BYTES + B_CODE_BYTES, &tm_as, xs, m0, fb);
        tma_load_2d(st + A_CODE_BYTES + B_CODE_BYTES + A_SCALE_BYTES, &tm_bs, xs, n0, fb);
        last_phase[s] = (int)ph;
      }
      if (*abort_flag) {
        // Let the copies this thread started land before the CTA may exit.
        for (int s = 0; s < kCodeStages; ++s)
          if (last_phase[s] >= 0)
            mbar_wait(smem_u32(&bars->code_full[s]), (uint32_t)last_phase[s], nullptr, kWaitLimitNs);
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      int d = 0;
      uint32_t dph = 0;
      bool ok = true;
      for (int kc = 0; kc < num_kc && ok; ++kc) {
        for (int sub = 0; sub < kSub; ++sub) {
          if (!mbar_wait(smem_u32(&bars->dec_full[d]), dph, abort_flag, kWaitLimitNs)) {
            fail(2u);
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t abase = sbase + OFF_DEC + d * DEC_STAGE_BYTES;
          const uint32_t bbase = abase + A_DEC_BYTES;
#pragma unroll
          for (int j = 0; j < BKD / 16; ++j) {
            const uint64_t ad = smem_desc_noswizzle(abase + j * 256, kLBO, kSBO);
            const uint64_t bd = smem_desc_noswizzle(bbase + j * 256, kLBO, kSBO);
            mma_bf16(tmem_acc, ad, bd, kIdesc, (kc | sub | j) != 0 ? 1u : 0u);
          }
          mma_commit(smem_u32(&bars->dec_empty[d]));
          if (++d == kDecStages) { d = 0; dph ^= 1; }
        }
      }
      // acc_full fires when every MMA issued above has completed.  The issuer
      // also waits for it (ignoring the abort flag), so tensor memory is never
      // freed under a running MMA.
      mma_commit(smem_u32(&bars->acc_full));
      if (!mbar_wait(smem_u32(&bars->acc_full), 0, nullptr, kWaitLimitNs)) fail(32u);
    }
  } else {
    // ---------------- decoders (one thread per tile row) ----------------
    const int row = threadIdx.x - 64;  // 0..383
    const bool is_a = row < BM;
    const int rl = is_a ? row : row - BM;
    const uint32_t code_off = (is_a ? 0 : A_CODE_BYTES) + rl * (BKC / 2);
    const uint32_t scale_off = A_CODE_BYTES + B_CODE_BYTES + (is_a ? 0 : A_SCALE_BYTES) + rl * (BKC / 16);
    const uint32_t dec_off = OFF_DEC + (is_a ? 0 : A_DEC_BYTES) + (rl >> 3) * kSBO + (rl & 7) * 16;
    const uint32_t swz = rl & 7;
    int d = 0;
    uint32_t dph = 0;
    bool ok = true;
    for (int kc = 0; kc < num_kc && ok; ++kc) {
      const int s = kc % kCodeStages;
      const uint32_t ph = (kc / kCodeStages) & 1;
      if (!mbar_wait(smem_u32(&bars->code_full[s]), ph, abort_flag, kWaitLimitNs)) {
        fail(4u);
        break;
      }
      const uint32_t st = sbase + s * CODE_STAGE_BYTES;
      const uint4 sc = lds128(st + scale_off);
      const uint32_t scw[4] = {sc.x, sc.y, sc.z, sc.w};
#pragma unroll
      for (int sub = 0; sub < kSub; ++sub) {
        // this row's 64 codes of the sub-stage: logical 16-byte chunks 2*sub, 2*sub+1
        const uint4 c0 = lds128(st + code_off + (((2 * sub) ^ swz) << 4));
        const uint4 c1 = lds128(st + code_off + (((2 * sub + 1) ^ swz) << 4));
        if (sub == kSub - 1) {
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&bars->code_empty[s]));
        }
        if (!mbar_wait(smem_u32(&bars->dec_empty[d]), dph ^ 1, abort_flag, kWaitLimitNs)) {
          fail(8u);
          ok = false;
          break;
        }
        const uint32_t w[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
        const uint32_t s4 = scw[sub];
        const uint32_t mag = s4 & 0x7F7F7F7Fu;
        float sv[4];
        f16x2_to_f32(cvt_f16x2_from_e4m3x2((uint16_t)(mag & 0xFFFFu)), sv[0], sv[1]);
        f16x2_to_f32(cvt_f16x2_from_e4m3x2((uint16_t)(mag >> 16)), sv[2], sv[3]);
        const uint32_t dst = sbase + dec_off + d * DEC_STAGE_BYTES;
#pragma unroll
        for (int b = 0; b < 4; ++b) {
          const bool e1m2 = (s4 >> (8 * b + 7)) & 1u;
          const uint32_t lut_lo = e1m2 ? 0x06040200u : 0x03020100u;
          const uint32_t lut_hi = e1m2 ? 0x0E0C0A08u : 0x0C080604u;
          const uint32_t s2 = bf16x2_splat(sv[b]);
          const uint32_t c2 = bf16x2_splat(-128.0f * sv[b]);
#pragma unroll
          for (int i = 0; i < 2; ++i) {
            uint32_t o[4];
            decode8(w[2 * b + i], lut_lo, lut_hi, s2, c2, o);
            sts128(dst + (2 * b + i) * kLBO, o[0], o[1], o[2], o[3]);
          }
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&bars->dec_full[d]));
        if (++d == kDecStages) { d = 0; dph ^= 1; }
      }
    }

    // ---------------- epilogue (warps 2-9) ----------------
    if (warp < 10) {
      const bool acc_ok = mbar_wait(smem_u32(&bars->acc_full), 0, abort_flag, kWaitLimitNs);
      tc_fence_after();
      // tcgen05.ld is warp-collective: decide for the whole warp.
      const bool go = __all_sync(0xffffffffu, acc_ok && !*abort_flag);
      if (!acc_ok && !*abort_flag) fail(16u);
      if (go) {
        const int q = warp & 3;                 // TMEM lane quarter of this warp
        const int half = (warp - 2) >> 2;       // column half
        const int r = m0 + q * 32 + lane;
        const float sa = 0.25f * __ldg(a_ts), sb = __ldg(b_ts);
        const bool vec_ok = ((ldc & 3) == 0) && ((reinterpret_cast<uintptr_t>(C) & 15) == 0);
        for (int cc = 0; cc < BN / 2; cc += 16) {
          const int col = half * (BN / 2) + cc;
          uint32_t v[16];
          tmem_ld_32x32b_x16(tmem_acc + ((uint32_t)(q * 32) << 16) + (uint32_t)col, v);
          tmem_ld_wait();
          if (r < M) {
            float* crow = C + (long long)r * ldc + n0 + col;
            float o[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) o[i] = __fmul_rn(__fmul_rn(__uint_as_float(v[i]), sa), sb);
            if (vec_ok && n0 + col + 16 <= N) {
#pragma unroll
              for (int i = 0; i < 16; i += 4)
                *reinterpret_cast<float4*>(crow + i) = make_float4(o[i], o[i + 1], o[i + 2], o[i + 3]);
            } else {
              for (int i = 0; i < 16; ++i)
                if (n0 + col + i < N) crow[i] = o[i];
            }
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_acc, kTmemCols);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// 2D uint8 tensor [rows][row_bytes] (dense), box [box_rows][box_bytes].
bool make_map(CUtensorMap* m, const void* base, uint64_t row_bytes, uint64_t rows, uint32_t box_bytes,
              uint32_t box_rows, CUtensorMapSwizzle swz) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {row_bytes, rows};
  cuuint64_t strides[1] = {row_bytes};
  cuuint32_t box[2] = {box_bytes, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

int launch_gemm(const uint8_t* a_codes, const uint8_t* a_scales, const float* a_ts,
                const uint8_t* b_codes, const uint8_t* b_scales, const float* b_ts, int64_t M,
                int64_t N, int64_t K, float* C, int64_t ldc, uint32_t* status_word,
                cudaStream_t stream) {
  if (M > (int64_t)65535 * BM || N > (1 << 30) || K > (1 << 30)) return MIXFP4_ERR_SHAPE;
  CUtensorMap tac, tbc, tas, tbs;
  if (!make_map(&tac, a_codes, (uint64_t)K / 2, (uint64_t)M, BKC / 2, BM, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_map(&tbc, b_codes, (uint64_t)K / 2, (uint64_t)N, BKC / 2, BN, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_map(&tas, a_scales, (uint64_t)K / 16, (uint64_t)M, BKC / 16, BM, CU_TENSOR_MAP_SWIZZLE_NONE) ||
      !make_map(&tbs, b_scales, (uint64_t)K / 16, (uint64_t)N, BKC / 16, BN, CU_TENSOR_MAP_SWIZZLE_NONE))
    return MIXFP4_ERR_CUDA;
  static bool attr_set = false;
  if (!attr_set) {
    if (cudaFuncSetAttribute(mixfp4_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_ALLOC) !=
        cudaSuccess)
      return MIXFP4_ERR_CUDA;
    attr_set = true;
  }
  dim3 grid((unsigned)((N + BN - 1) / BN), (unsigned)((M + BM - 1) / BM));
  mixfp4_gemm_kernel<<<grid, kThreads, SMEM_ALLOC, stream>>>(tac, tbc, tas, tbs, a_ts, b_ts, (int)M, (int)N,
                                                               (int)K, C, (long long)ldc, status_word);
  return MIXFP4_OK;
}

}  // namespace mixfp4
