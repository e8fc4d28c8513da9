// Native block-scaled FP4 variant of the MixFP4 GEMM for sm_103a.
//
// A MixFP4 operand is the sum of two E2M1 operands that share its block
// scales.  An E2M1 block (type bit T = 0) is already an E2M1 block.  An E1M2
// block (T = 1) holds magnitudes v = p in {0..7} (Sec. 3.1 remap), and every
// such v is e + r with e the largest E2M1 value <= v and r = v - e in {0, 1}
// (5 = 4 + 1, 7 = 6 + 1, the rest have r = 0).  So
//   C = A . B^T = (A_main + A_res) . (B_main + B_res)^T
// is four products of E2M1 operands with the MixFP4 block scales (E4M3, block
// 16), which is exactly what tcgen05.mma kind::mxf4nvf4 (scale_vec::4X)
// contracts at the FP4 tensor rate; an operand without E1M2 blocks drops its
// residual and halves the products.  Every product term is exact; the tensor
// core accumulates in fp32 and the epilogue applies s32A * s32B.
//
// split_native_kernel writes, per operand, the main and residual codes (same
// [rows][K/2] layout as the MixFP4 codes, element 2j in the low nibble) and
// the ue4m3 block scales in the tensor core's tiled layout: tiles of 128 rows
// x 4 blocks (64 K) of 512 bytes, tile (rt, kt) at (rt * K/64 + kt) * 512,
// row r and block b at (r % 32) * 16 + (r / 32) * 4 + b, rows padded to a
// multiple of 256 with zero bytes.
//
// nvf4_gemm_kernel: persistent CTA pairs (cta_group::2), 256 x 256 output
// tiles, the stream-K split of the last wave as in the decoding kernel.  Per
// CTA:
//   warp 0      TMA producer: the main (and residual) code tiles of its 128
//               rows of A and 128 rows of B for a 256-wide K slice (128-byte
//               swizzle, the layout the MMA reads directly), and the scale
//               tiles of its A rows and of all 256 B rows (1D bulk copies);
//   warp 1      TMEM allocator; in the leader the MMA-issuing thread, which
//               also copies each K step's scale tiles from shared to tensor
//               memory (tcgen05.cp 32x128b.warpx4: the tiled layout puts row
//               32c + l's four scales of a K step in lane l's word c, and the
//               copy replicates the 32 lines to every lane quarter, so a K
//               step takes 4 (A) + 8 (B) scale columns) ahead of its MMAs in
//               the same tensor-core stream; in the peer the thread that
//               forwards "stage landed" to the leader;
//   warps 2-17  epilogue: 4 warps per lane quarter, 64 accumulator columns
//               each (two 32-column tcgen05.ld, then the accumulator is
//               released, then x s32A s32B -> fp32 stores or adds to C).
// TMEM per CTA: 256 fp32 accumulator columns, then 48 scale columns per stage.
// Every pipeline wait is bounded; a wait that gives up records a status bit
// and the CTA drains and exits without writing C.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "host_util.cuh"
#include "kernels.cuh"
#include "pipeline.cuh"
#include "ptx.cuh"
#include "sm100.cuh"

namespace mixfp4 {
namespace {

using namespace sm100;

// ---------------------------------------------------------------- operand split
// E2M1 codes of the split of an E1M2 payload p (nibble p of each constant).
constexpr uint32_t kMainOfE1M2 = 0x77665420u;  // e(p): 0,1,2,3,4,4,6,6 -> codes 0,2,4,5,6,6,7,7
constexpr uint32_t kResOfE1M2 = 0x20200000u;   // r(p): 1 for p = 5, 7 -> code 2

__device__ __forceinline__ void split_word(uint32_t w, bool e1m2, uint32_t& main, uint32_t& res) {
  if (!e1m2) {
    main = w;
    res = 0;
    return;
  }
  main = 0;
  res = 0;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const uint32_t n = (w >> (4 * i)) & 0xFu, p = n & 7u, s = n & 8u;
    main |= (s | ((kMainOfE1M2 >> (4 * p)) & 0xFu)) << (4 * i);
    res |= (s | ((kResOfE1M2 >> (4 * p)) & 0xFu)) << (4 * i);
  }
}

// Threads [0, n_code) split 32 elements (two blocks, 16 code bytes) each;
// threads [n_code, n_code + n_sf) write one 16-byte line of the scale tiles
// (tile (rt, kt), lane line l: rows 32j + l for j = 0..3, blocks 4kt..4kt+3).
__global__ void __launch_bounds__(256) split_native_kernel(const uint8_t* __restrict__ codes,
                                                           const uint8_t* __restrict__ scales, int64_t rows,
                                                           int64_t K, uint8_t* __restrict__ main_codes,
                                                           uint8_t* __restrict__ res_codes, uint8_t* __restrict__ sf,
                                                           int64_t n_code, int64_t n_sf) {
  const int64_t nb = K / 16;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n_code + n_sf;
       i += (int64_t)gridDim.x * blockDim.x) {
    if (i < n_code) {
      const int64_t r = i / (K / 32), c = i % (K / 32);  // row, 32-element chunk
      const uint4 w = *reinterpret_cast<const uint4*>(codes + r * (K / 2) + c * 16);
      const uint8_t s0 = scales[r * nb + 2 * c], s1 = scales[r * nb + 2 * c + 1];
      uint4 m, q;
      split_word(w.x, s0 >> 7, m.x, q.x);
      split_word(w.y, s0 >> 7, m.y, q.y);
      split_word(w.z, s1 >> 7, m.z, q.z);
      split_word(w.w, s1 >> 7, m.w, q.w);
      *reinterpret_cast<uint4*>(main_codes + r * (K / 2) + c * 16) = m;
      *reinterpret_cast<uint4*>(res_codes + r * (K / 2) + c * 16) = q;
    } else {
      const int64_t u = i - n_code;
      const int64_t line = u % 32, tile = u / 32, kt_n = K / 64;
      const int64_t rt = tile / kt_n, kt = tile % kt_n;
      uint32_t v[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int64_t r = rt * 128 + 32 * j + line;
        v[j] = r < rows ? (*reinterpret_cast<const uint32_t*>(scales + r * nb + 4 * kt) & 0x7F7F7F7Fu) : 0u;
      }
      *reinterpret_cast<uint4*>(sf + tile * 512 + line * 16) = make_uint4(v[0], v[1], v[2], v[3]);
    }
  }
}

// ---------------------------------------------------------------- GEMM
namespace nv {

constexpr int BM = 128, TILE_M = 256, TILE_N = 256;
constexpr int BKC = 256;                          // K per stage
constexpr int kKSteps = BKC / 64;                 // instructions per operand pair per stage (K = 64)
constexpr int ROW_BYTES = BKC / 2;                // 128 code bytes per row per stage
constexpr int TILE_BYTES = BM * ROW_BYTES;        // 16 KB: 128 rows of one operand
constexpr int SF_TILE = 512;                      // 128 rows x 4 blocks
constexpr int SFA_BYTES = kKSteps * SF_TILE;      // this CTA's 128 A rows
constexpr int SFB_BYTES = 2 * kKSteps * SF_TILE;  // all 256 B rows of the pair tile
constexpr uint32_t kSfCols = 12;                  // TMEM columns per K step: 4 (A) + 8 (B)
constexpr uint32_t kStageSfCols = kKSteps * kSfCols;
constexpr uint32_t kAccCols = TILE_N;
constexpr uint32_t kTmemCols = 512;
constexpr int kEpiWarps = 16;
constexpr int kFirstEpi = 2;
constexpr int kThreads = 32 * (kFirstEpi + kEpiWarps);  // 576
constexpr int kEpiCols = 64;                             // accumulator columns per epilogue warp
constexpr int kSmemBudget = 232448 - 1024 - 256;
constexpr uint64_t kWaitLimitNs = 1000000000ull;
constexpr int kMaxStages = 5;
static_assert(kAccCols + kMaxStages * kStageSfCols <= kTmemCols, "TMEM budget");
static_assert(kFirstEpi % 4 == 2, "epilogue warps cover every TMEM lane quarter");
static_assert(kEpiWarps * kEpiCols == 4 * TILE_N, "epilogue covers the accumulator");

template <bool kARes, bool kBRes>
struct Layout {
  static constexpr int kTiles = 2 + (kARes ? 1 : 0) + (kBRes ? 1 : 0);
  static constexpr int OFF_AM = 0;
  static constexpr int OFF_AR = TILE_BYTES;
  static constexpr int OFF_BM = (kARes ? 2 : 1) * TILE_BYTES;
  static constexpr int OFF_BR = OFF_BM + TILE_BYTES;
  static constexpr int OFF_SFA = kTiles * TILE_BYTES;
  static constexpr int OFF_SFB = OFF_SFA + SFA_BYTES;
  static constexpr int STAGE = OFF_SFB + SFB_BYTES;
  static constexpr int kStages = kSmemBudget / STAGE > kMaxStages ? kMaxStages : kSmemBudget / STAGE;
  static constexpr int OFF_BAR = kStages * STAGE;
  static constexpr int SMEM_ALLOC = OFF_BAR + 256 + 1024;
  static constexpr uint32_t kTx = kTiles * TILE_BYTES + SFA_BYTES + SFB_BYTES;
  static_assert(STAGE % 1024 == 0, "swizzled tiles need 1024-byte alignment");
  static_assert(kStages >= 2 && SMEM_ALLOC <= 232448, "shared memory budget");
};

struct Bars {
  uint64_t full[kMaxStages];        // TMA bytes of the stage landed (local)
  uint64_t ready[kMaxStages];       // leader: the peer's stage landed (forwarded)
  uint64_t empty[kMaxStages];       // MMA commit (multicast to both CTAs)
  uint64_t acc_full;                // MMA commit (multicast)
  uint64_t acc_empty;               // leader: 2 x kEpiWarps arrivals
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
};
static_assert(sizeof(Bars) <= 256, "barrier block");

template <bool kARes, bool kBRes>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
nvf4_gemm_kernel(const __grid_constant__ CUtensorMap tm_am, const __grid_constant__ CUtensorMap tm_ar,
                 const __grid_constant__ CUtensorMap tm_bm, const __grid_constant__ CUtensorMap tm_br,
                 const uint8_t* __restrict__ a_sf, const uint8_t* __restrict__ b_sf, const float* __restrict__ a_ts,
                 const float* __restrict__ b_ts, int M, int N, int K, float* __restrict__ C, long long ldc,
                 int dp_tiles, uint32_t* status_word) {
  using L = Layout<kARes, kBRes>;
  constexpr int S = L::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  Bars* bars = reinterpret_cast<Bars*>(smem + L::OFF_BAR);
  volatile int* abort_flag = &bars->abort;
  const uint32_t sbase = smem_u32(smem);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int num_kc = K / BKC, kt_n = K / 64;
  const int mtiles = (M + TILE_M - 1) / TILE_M, ntiles_n = (N + TILE_N - 1) / TILE_N;
  const int ntiles = mtiles * ntiles_n;
  const int cluster_id = blockIdx.x >> 1, nclusters = gridDim.x >> 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(smem_u32(&bars->full[s]), 1);
      mbar_init(smem_u32(&bars->ready[s]), 1);
      mbar_init(smem_u32(&bars->empty[s]), 1);
    }
    mbar_init(smem_u32(&bars->acc_full), 1);
    mbar_init(smem_u32(&bars->acc_empty), 2 * kEpiWarps);
    mbar_init(smem_u32(&bars->drain), 1);
    bars->abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc_pair(smem_u32(&bars->tmem_base), kTmemCols);
    tmem_relinquish_pair();
  }
  griddep_launch_dependents();
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem_base = bars->tmem_base;
  const uint32_t tmem_sf0 = tmem_base + kAccCols;

  auto fail = [&](uint32_t code) {
    *abort_flag = 1;
    if (status_word) atomicOr(status_word, code);
  };

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      tma_prefetch(&tm_am);
      tma_prefetch(&tm_bm);
      if (kARes) tma_prefetch(&tm_ar);
      if (kBRes) tma_prefetch(&tm_br);
      griddep_wait();
      int last_it = -1, it = 0;
      bool ok = true;
      Sched sched(cluster_id, nclusters, dp_tiles, ntiles, num_kc);
      int t, k0, k1;
      while (ok && sched.next(t, k0, k1)) {
        const int mt = t / ntiles_n, nt = t % ntiles_n;
        const int ma = mt * TILE_M + (int)rank * BM, nb = nt * TILE_N + (int)rank * BM;
        const uint8_t* sfa = a_sf + (size_t)(mt * 2 + (int)rank) * kt_n * SF_TILE;
        const uint8_t* sfb0 = b_sf + (size_t)(nt * 2) * kt_n * SF_TILE;
        const uint8_t* sfb1 = sfb0 + (size_t)kt_n * SF_TILE;
        for (int kc = k0; kc < k1; ++kc, ++it) {
          const int s = it % S;
          const uint32_t ph = (it / S) & 1;
          if (!mbar_wait(smem_u32(&bars->empty[s]), ph ^ 1, abort_flag, kWaitLimitNs)) {
            fail(1u);
            ok = false;
            break;
          }
          const uint32_t st = sbase + s * L::STAGE;
          const uint32_t fb = smem_u32(&bars->full[s]);
          mbar_arrive_expect_tx(fb, L::kTx);
          const int xk = kc * ROW_BYTES;
          tma_load_2d(st + L::OFF_AM, &tm_am, xk, ma, fb);
          if (kARes) tma_load_2d(st + L::OFF_AR, &tm_ar, xk, ma, fb);
          tma_load_2d(st + L::OFF_BM, &tm_bm, xk, nb, fb);
          if (kBRes) tma_load_2d(st + L::OFF_BR, &tm_br, xk, nb, fb);
          const size_t ko = (size_t)kc * kKSteps * SF_TILE;
          bulk_load(st + L::OFF_SFA, sfa + ko, SFA_BYTES, fb);
          bulk_load(st + L::OFF_SFB, sfb0 + ko, SFB_BYTES / 2, fb);
          bulk_load(st + L::OFF_SFB + SFB_BYTES / 2, sfb1 + ko, SFB_BYTES / 2, fb);
          last_it = it;
        }
      }
      if (*abort_flag) {
        for (int u = last_it - S + 1; u <= last_it; ++u)
          if (u >= 0)
            mbar_wait(smem_u32(&bars->full[u % S]), (uint32_t)((u / S) & 1), nullptr, kWaitLimitNs);
      }
    }
  } else if (warp == 1) {
    if (leader && lane == 0) {
      // ---------------- MMA issuer ----------------
      constexpr uint32_t kIdesc = idesc_nvf4_f32(TILE_M, TILE_N);
      int it = 0;
      bool ok = true;
      Sched sched(cluster_id, nclusters, dp_tiles, ntiles, num_kc);
      int t, k0, k1;
      for (int i = 0; ok && sched.next(t, k0, k1); ++i) {
        if (!mbar_wait_cluster(smem_u32(&bars->acc_empty), (i & 1) ^ 1, abort_flag, kWaitLimitNs)) {
          fail(2u);
          break;
        }
        tc_fence_after();
        for (int kc = k0; kc < k1; ++kc, ++it) {
          const int s = it % S;
          const uint32_t ph = (uint32_t)((it / S) & 1);
          if (!mbar_wait(smem_u32(&bars->full[s]), ph, abort_flag, kWaitLimitNs)) {
            fail(16u);
            ok = false;
            break;
          }
          if (!mbar_wait_cluster(smem_u32(&bars->ready[s]), ph, abort_flag, kWaitLimitNs)) {
            fail(4u);
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t st = sbase + s * L::STAGE;
#pragma unroll
          for (int j = 0; j < kKSteps; ++j) {
            const uint32_t sfa = tmem_sf0 + (uint32_t)s * kStageSfCols + (uint32_t)j * kSfCols;
            const uint32_t sfb = sfa + 4;
            // Scale tiles of this K step (32 lines of 16 bytes each, contiguous).
            tmem_cp_32x128b_x4_pair(sfa, smem_desc_noswizzle(st + L::OFF_SFA + j * SF_TILE, 128, 128));
            tmem_cp_32x128b_x4_pair(sfb, smem_desc_noswizzle(st + L::OFF_SFB + j * SF_TILE, 128, 128));
            tmem_cp_32x128b_x4_pair(sfb + 4,
                                    smem_desc_noswizzle(st + L::OFF_SFB + SFB_BYTES / 2 + j * SF_TILE, 128, 128));
            const uint64_t am = smem_desc_sw128(st + L::OFF_AM + j * 32);
            const uint64_t bm = smem_desc_sw128(st + L::OFF_BM + j * 32);
            mma_nvf4_pair(tmem_base, am, bm, kIdesc, sfa, sfb, (kc > k0 || j > 0) ? 1u : 0u);
            if (kBRes) mma_nvf4_pair(tmem_base, am, smem_desc_sw128(st + L::OFF_BR + j * 32), kIdesc, sfa, sfb, 1u);
            if (kARes) {
              const uint64_t ar = smem_desc_sw128(st + L::OFF_AR + j * 32);
              mma_nvf4_pair(tmem_base, ar, bm, kIdesc, sfa, sfb, 1u);
              if (kBRes)
                mma_nvf4_pair(tmem_base, ar, smem_desc_sw128(st + L::OFF_BR + j * 32), kIdesc, sfa, sfb, 1u);
            }
          }
          mma_commit_pair(smem_u32(&bars->empty[s]), 3);
        }
        if (ok) mma_commit_pair(smem_u32(&bars->acc_full), 3);
      }
      mma_commit_pair(smem_u32(&bars->drain), 1);
      if (!mbar_wait_cluster(smem_u32(&bars->drain), 0, nullptr, kWaitLimitNs)) fail(8u);
    } else if (!leader && lane == 0) {
      // ---------------- forwarder (peer CTA) ----------------
      // The leader's MMAs read this CTA's half of every stage: pass on each
      // landed stage as one remote arrival.
      const uint32_t ready_leader0 = mapa_shared(smem_u32(&bars->ready[0]), 0);
      int it = 0;
      bool ok = true;
      Sched sched(cluster_id, nclusters, dp_tiles, ntiles, num_kc);
      int t, k0, k1;
      while (ok && sched.next(t, k0, k1)) {
        for (int kc = k0; kc < k1; ++kc, ++it) {
          const int s = it % S;
          if (!mbar_wait(smem_u32(&bars->full[s]), (uint32_t)((it / S) & 1), abort_flag, kWaitLimitNs)) {
            fail(128u);
            ok = false;
            break;
          }
          mbar_arrive_cluster(ready_leader0 + s * 8);
        }
      }
    }
  } else {
    // ---------------- epilogue ----------------
    const int q = warp & 3;
    const int cg = (warp - kFirstEpi) >> 2;  // 64-column group
    griddep_wait();
    const float sa = __ldg(a_ts), sb = __ldg(b_ts);
    const bool vec_ok = ((ldc & 3) == 0) && ((reinterpret_cast<uintptr_t>(C) & 15) == 0);
    const uint32_t acc_empty_leader = mapa_shared(smem_u32(&bars->acc_empty), 0);
    const uint32_t tbase = tmem_base + (uint32_t)(cg * kEpiCols) + ((uint32_t)(q * 32) << 16);
    Sched sched(cluster_id, nclusters, dp_tiles, ntiles, num_kc);
    int t, k0, k1;
    for (int i = 0; sched.next(t, k0, k1); ++i) {
      const bool whole = k0 == 0 && k1 == num_kc;
      const bool acc_ok = mbar_wait_cluster(smem_u32(&bars->acc_full), i & 1, abort_flag, kWaitLimitNs);
      tc_fence_after();
      const bool go = __all_sync(0xffffffffu, acc_ok && !*abort_flag);
      if (!go) {
        if (!acc_ok && !*abort_flag) fail(64u);
        break;
      }
      const int mt = t / ntiles_n, nt = t % ntiles_n;
      const int row = mt * TILE_M + (int)rank * BM + q * 32 + lane;
      const int col0 = nt * TILE_N + cg * kEpiCols;
      float* crow = C + (long long)row * ldc + col0;
      uint32_t v[kEpiCols];
      tmem_ld_32x32b_x32(tbase, v);
      tmem_ld_32x32b_x32(tbase + 32, v + 32);
      tmem_ld_wait_x32(v);
      reg_fence16(v + 32);
      reg_fence16(v + 48);
      // The accumulator is free once all its columns sit in registers.
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(acc_empty_leader);
      if (row < M) {
#pragma unroll
        for (int c = 0; c < kEpiCols; c += 4) {
          float o[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) o[e] = __fmul_rn(__fmul_rn(__uint_as_float(v[c + e]), sa), sb);
          if (vec_ok && col0 + c + 4 <= N) {
            if (whole)
              *reinterpret_cast<float4*>(crow + c) = make_float4(o[0], o[1], o[2], o[3]);
            else
              red_add_v4(crow + c, o[0], o[1], o[2], o[3]);
          } else {
#pragma unroll
            for (int e = 0; e < 4; ++e)
              if (col0 + c + e < N) {
                if (whole) crow[c + e] = o[e];
                else atomicAdd(crow + c + e, o[e]);
              }
          }
        }
      }
    }
  }

  tc_fence_before();
  cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, kTmemCols);
  }
}

constexpr int kMinStreamKGainSlices = 8;

template <bool kARes, bool kBRes>
int launch(const uint8_t* a_main, const uint8_t* a_res, const uint8_t* a_sf, const float* a_ts,
           const uint8_t* b_main, const uint8_t* b_res, const uint8_t* b_sf, const float* b_ts, int64_t M, int64_t N,
           int64_t K, float* C, int64_t ldc, uint32_t* status_word, cudaStream_t stream) {
  using L = Layout<kARes, kBRes>;
  CUtensorMap tam, tar, tbm, tbr;
  const auto swz = CU_TENSOR_MAP_SWIZZLE_128B;
  if (!make_map(&tam, a_main, (uint64_t)K / 2, (uint64_t)M, ROW_BYTES, BM, swz) ||
      !make_map(&tbm, b_main, (uint64_t)K / 2, (uint64_t)N, ROW_BYTES, BM, swz) ||
      !make_map(&tar, kARes ? a_res : a_main, (uint64_t)K / 2, (uint64_t)M, ROW_BYTES, BM, swz) ||
      !make_map(&tbr, kBRes ? b_res : b_main, (uint64_t)K / 2, (uint64_t)N, ROW_BYTES, BM, swz))
    return MIXFP4_ERR_CUDA;
  static bool attr_set = false;
  if (!attr_set) {
    if (cudaFuncSetAttribute(nvf4_gemm_kernel<kARes, kBRes>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             L::SMEM_ALLOC) != cudaSuccess)
      return MIXFP4_ERR_CUDA;
    attr_set = true;
  }
  const int64_t mtiles = (M + TILE_M - 1) / TILE_M, ntiles_n = (N + TILE_N - 1) / TILE_N;
  const int64_t tiles = mtiles * ntiles_n, num_kc = K / BKC;
  int64_t clusters = num_sms() / 2;
  if (clusters > tiles) clusters = tiles;
  int64_t dp_tiles = tiles;
  const int64_t rem = tiles % clusters;
  if (tiles > clusters && rem != 0 && (clusters - rem) * num_kc >= kMinStreamKGainSlices * clusters)
    dp_tiles = tiles - rem;
  if (dp_tiles < tiles) {
    const int64_t r0 = (dp_tiles / ntiles_n) * TILE_M;
    cudaError_t e;
    if (ldc == N)
      e = cudaMemsetAsync(C + r0 * ldc, 0, (size_t)(M - r0) * (size_t)N * sizeof(float), stream);
    else
      e = cudaMemset2DAsync(C + r0 * ldc, (size_t)ldc * sizeof(float), 0, (size_t)N * sizeof(float),
                            (size_t)(M - r0), stream);
    if (e != cudaSuccess) return MIXFP4_ERR_CUDA;
  }
  if (launch_pdl(nvf4_gemm_kernel<kARes, kBRes>, (unsigned)(2 * clusters), kThreads, L::SMEM_ALLOC, stream, tam,
                 tar, tbm, tbr, a_sf, b_sf, a_ts, b_ts, (int)M, (int)N, (int)K, C, (long long)ldc, (int)dp_tiles,
                 status_word) != cudaSuccess)
    return MIXFP4_ERR_CUDA;
  return MIXFP4_OK;
}

}  // namespace nv
}  // namespace

int launch_split_native(const uint8_t* codes, const uint8_t* scales, int64_t rows, int64_t K, uint8_t* main_codes,
                        uint8_t* res_codes, uint8_t* sf, cudaStream_t stream) {
  const int64_t n_code = rows * (K / 32);
  const int64_t n_sf = ((rows + 255) / 256) * 2 * (K / 64) * 32;
  int64_t blocks = (n_code + n_sf + 255) / 256;
  const int64_t cap = (int64_t)num_sms() * 8;
  if (blocks > cap) blocks = cap;
  split_native_kernel<<<(unsigned)blocks, 256, 0, stream>>>(codes, scales, rows, K, main_codes, res_codes, sf, n_code,
                                                            n_sf);
  return cudaGetLastError() == cudaSuccess ? MIXFP4_OK : MIXFP4_ERR_CUDA;
}

int launch_gemm_native(const uint8_t* a_main, const uint8_t* a_res, const uint8_t* a_sf, const float* a_ts,
                       const uint8_t* b_main, const uint8_t* b_res, const uint8_t* b_sf, const float* b_ts, int64_t M,
                       int64_t N, int64_t K, float* C, int64_t ldc, uint32_t* status_word, cudaStream_t stream) {
  if (M > (1 << 30) || N > (1 << 30) || K > (1 << 30)) return MIXFP4_ERR_SHAPE;
  if (a_res && b_res)
    return nv::launch<true, true>(a_main, a_res, a_sf, a_ts, b_main, b_res, b_sf, b_ts, M, N, K, C, ldc, status_word,
                                  stream);
  if (a_res)
    return nv::launch<true, false>(a_main, a_res, a_sf, a_ts, b_main, b_res, b_sf, b_ts, M, N, K, C, ldc,
                                   status_word, stream);
  if (b_res)
    return nv::launch<false, true>(a_main, a_res, a_sf, a_ts, b_main, b_res, b_sf, b_ts, M, N, K, C, ldc,
                                   status_word, stream);
  return nv::launch<false, false>(a_main, a_res, a_sf, a_ts, b_main, b_res, b_sf, b_ts, M, N, K, C, ldc, status_word,
                                  stream);
}

}  // namespace mixfp4
