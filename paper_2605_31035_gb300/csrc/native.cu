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
// tiles, the stream-K split of the last wave and the accumulation chunks of
// at most 4096 K (later chunks added into C) as in the decoding kernel.  Per
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
// The E2M1 main and residual parts of eight E1M2 nibbles (sign in bit 3 of
// each, payload p in bits 0-2): main payload bits m0 = p1 (p0 | p2),
// m1 = p2 | (p0 ~p1), m2 = p2 | p1 (the codes of 0,1,2,3,4,4,6,6), residual
// payload 2 where p0 p2 (p = 5, 7); both keep the sign bit.  Each line is one
// three-input logic instruction (lop3; truth-table byte from a = 0xF0,
// b = 0xCC, c = 0xAA).
#define MIXFP4_LOP3(d, a, b, c, LUT) asm("lop3.b32 %0, %1, %2, %3, " #LUT ";" : "=r"(d) : "r"(a), "r"(b), "r"(c))
__device__ __forceinline__ void split_e1m2_word(uint32_t w, uint32_t tmask, uint32_t& main, uint32_t& res) {
  const uint32_t r1 = w >> 1, r2 = w >> 2, l1 = w << 1;
  uint32_t m0, m1, t, r;
  MIXFP4_LOP3(m0, r1, w, r2, 0xE0);                  // p1 & (p0 | p2)          at bit 4i
  MIXFP4_LOP3(m1, r1, l1, w, 0xF4);                  // p2 | (p0 & ~p1)         at bit 4i+1
  MIXFP4_LOP3(t, m0, m1, 0x22222222u, 0xD8);         // bit 4i+1 from m1
  MIXFP4_LOP3(t, t, w | l1, 0x44444444u, 0xD8);      // bit 4i+2: p2 | p1
  MIXFP4_LOP3(t, t, w, 0x88888888u, 0xD8);           // bit 4i+3: the sign
  MIXFP4_LOP3(r, l1, r1, 0x22222222u, 0x80);         // p0 & p2                 at bit 4i+1
  MIXFP4_LOP3(r, r, w, 0x88888888u, 0xF8);           // | the sign
  MIXFP4_LOP3(main, t, w, tmask, 0xE4);              // tmask ? main : w  (per bit: (a & c) | (b & ~c))
  res = r & tmask;                                    // E2M1 blocks have no residual
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
      const uint32_t k0 = (s0 & 0x80u) ? 0xFFFFFFFFu : 0u, k1 = (s1 & 0x80u) ? 0xFFFFFFFFu : 0u;
      uint4 m, q;
      split_e1m2_word(w.x, k0, m.x, q.x);
      split_e1m2_word(w.y, k0, m.y, q.y);
      split_e1m2_word(w.z, k1, m.z, q.z);
      split_e1m2_word(w.w, k1, m.w, q.w);
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
                 int dp_tiles, int chunk_kc, uint32_t* status_word) {
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
      Sched sched(cluster_id, nclusters, dp_tiles, ntiles, num_kc, chunk_kc);
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
      Sched sched(cluster_id, nclusters, dp_tiles, ntiles, num_kc, chunk_kc);
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
      Sched sched(cluster_id, nclusters, dp_tiles, ntiles, num_kc, chunk_kc);
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
    Sched sched(cluster_id, nclusters, dp_tiles, ntiles, num_kc, chunk_kc);
    int t, k0, k1;
    for (int i = 0; sched.next(t, k0, k1); ++i) {
      // The first chunk of a whole tile is stored; every other segment is
      // added into C (after that chunk, or into rows the host zeroed).
      const bool whole = sched.store;
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
  static std::atomic<uint64_t> smem_set{0};
  if (!set_dynamic_smem_once(reinterpret_cast<const void*>(nvf4_gemm_kernel<kARes, kBRes>), L::SMEM_ALLOC, smem_set))
    return MIXFP4_ERR_CUDA;
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
                 kAccumChunkK / BKC, status_word) != cudaSuccess)
    return MIXFP4_ERR_CUDA;
  return MIXFP4_OK;
}

}  // namespace nv

// ============================================================================
// Few-row native variant (M <= 64 activation rows, the decode shape).
//
// Decomposition used here (every product exact, same block scales):
//   main part     = the stored MixFP4 code itself read as an E2M1 code;
//   residual part = E2M1 code {0,1,2,3,4,4,4,2}[p] of the magnitude p (sign
//                   kept), scaled by the block's scale for an E1M2 block and
//                   by 0 for an E2M1 block.
// For an E2M1 block the main part is the block and the residual has scale 0.
// For an E1M2 block, E2M1 value e(p) + e(res(p)) = p for every p in 0..7
// (0, .5+.5, 1+1, 1.5+1.5, 2+2, 3+2, 4+2, 6+1), which is the E1M2 value of p
// under the same scale.  So the main codes need no rewriting: TMA lands them
// straight in the MMA operand tiles, and the splitters only write the
// residual rows (one bit-sliced function of the nibbles, no per-block type
// select) and the two scale tiles per operand (main: the scale with the type
// bit cleared; residual: the same where the type bit is set, else 0).
//
// Weight rows go on the MMA N side in units of 128 rows x one 256-wide K
// slice: rows 0-127 of the N = 256 operand tile hold the main codes, rows
// 128-255 the residual codes; the activation rows' main codes sit in rows
// 0..XR-1 of the M = 128 tile and their residual codes in rows XR..2XR-1
// (XR = 16, 32 or 64 by the row count; rows from 2XR on are never written,
// the MMA reads whatever follows in the stage there and the epilogue never
// loads those accumulator lanes).  ONE kind::mxf4nvf4 MMA per 64-K step forms
// all four products; C[m][n] = D[m][n] + D[m][128+n] + D[XR+m][n] +
// D[XR+m][128+n], the epilogue adding each accumulator lane's two column
// halves into C row (lane row mod XR).
// Per CTA (one per SM, units split evenly over all SMs, partial sums added
// into C which the host zeroed):
//   warp 0      TMA: weight codes (128 x 128 bytes, 128-byte swizzle) into
//               the operand tile, its 128 x 16-byte scale rows, the
//               activation rows' codes into the A tile and their scale rows,
//               into a ring of 3-5 stages (by the row count);
//   warp 1      TMEM allocation; lane 0 issues the MMAs (one per 64-K step)
//               and frees the stage with their commit;
//   warps 2-17  weight scale tiles (announced first, so their copies to
//               tensor memory overlap the rest), then the weight residual
//               rows (four threads per row, two 16-byte chunks each); warps
//               18-21 the same for the activation rows;
//   warps 22-25 epilogue, one TMEM lane quarter each;
//   warps 26-27 copy each stage's scale tiles into tensor memory
//               (tcgen05.cp, half of the K steps each) and commit.
// ============================================================================
namespace nvs {

constexpr int WR = 128;                    // weight rows per unit (MMA N = 2 x 128)
constexpr int BKC = 256;                   // K per unit
constexpr int ROWB = BKC / 2;              // 128 code bytes per row per unit
constexpr int kMaxStages = 5;
constexpr int SF_T = 4 * 512;              // tiled scales of 128 rows for the unit's four K steps
// Stage layout (offsets from the stage base): A tile (2 XR rows), weight main
// rows, weight residual rows, weight scale rows (TMA), activation scale rows
// (TMA, at most 64 x 16 bytes), then the tiled scales of the A tile, of the
// weight main rows and of the weight residual rows.
__host__ __device__ constexpr int xr_of(int nx) { return nx <= 16 ? 16 : (nx <= 32 ? 32 : 64); }
__host__ __device__ constexpr int off_b(int xr) { return 2 * xr * ROWB; }
__host__ __device__ constexpr int off_ws(int xr) { return off_b(xr) + 2 * WR * ROWB; }
__host__ __device__ constexpr int off_xs(int xr) { return off_ws(xr) + WR * 16; }
__host__ __device__ constexpr int off_sfa(int xr) { return off_xs(xr) + 64 * 16; }
__host__ __device__ constexpr int off_sfb(int xr) { return off_sfa(xr) + SF_T; }
__host__ __device__ constexpr int off_sfr(int xr) { return off_sfb(xr) + SF_T; }
__host__ __device__ constexpr int stage_bytes_of(int xr) { return ((off_sfr(xr) + SF_T + 1023) / 1024) * 1024; }
constexpr int OFF_RINGS = 1024;                                  // after the barrier block
constexpr int kSmemBudget = 232448 - 1024;                       // 1024 for the alignment of the base
__host__ __device__ constexpr int stages_of(int xr) {
  return (kSmemBudget - OFF_RINGS) / stage_bytes_of(xr) < kMaxStages ? (kSmemBudget - OFF_RINGS) / stage_bytes_of(xr)
                                                                     : kMaxStages;
}
static_assert(stages_of(16) == 5 && stages_of(32) == 4 && stages_of(64) == 3, "ring depths");
static_assert(off_b(16) % 1024 == 0 && stage_bytes_of(16) >= 128 * ROWB, "the M = 128 operand read stays in the stage");
constexpr int kWSplitWarps = 16, kXSplitWarps = 4;
constexpr int kFirstW = 2, kFirstX = kFirstW + kWSplitWarps, kFirstEpi = kFirstX + kXSplitWarps;  // 2, 18, 22
constexpr int kCopyWarp = kFirstEpi + 4, kCopyWarps = 2;                                          // 26, 27
constexpr int kThreads = 32 * (kCopyWarp + kCopyWarps);                                           // 896
static_assert(kFirstEpi % 4 == 2, "epilogue warps cover the four TMEM lane quarters");
constexpr uint32_t kAccCols = 2 * WR;                            // 256 fp32 columns
constexpr uint32_t kSfCols = 12;                                 // per K step: 4 (A) + 8 (B main, residual)
constexpr uint32_t kTmemCols = 512;
constexpr uint64_t kWaitLimitNs = 1000000000ull;
static_assert(kAccCols + kMaxStages * 4 * kSfCols <= kTmemCols, "TMEM budget");

struct Bars {
  uint64_t full[kMaxStages];        // TMA landed
  uint64_t split_full[kMaxStages];  // residual rows written
  uint64_t sf_full[kMaxStages];     // the stage's scales are in tensor memory (commit of the copy warps)
  uint64_t sf_ready[kMaxStages];    // the stage's scale tiles are written
  uint64_t empty[kMaxStages];       // the stage's MMAs completed
  uint64_t acc_full;
  uint64_t acc_empty;
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
};
static_assert(sizeof(Bars) <= 256, "barrier block");

// Residual E2M1 codes of eight nibbles (sign in bit 3, payload p in bits
// 0-2): payload {0,1,2,3,4,4,4,2}[p] = p & F with F's bit 0 = ~p2, bit 1 =
// ~p2 | p0, bit 2 = ~(p1 & p0), and the sign kept.  Checked exhaustively on
// the host against the table.
__device__ __forceinline__ uint32_t residual_word(uint32_t w) {
  const uint32_t r1 = w >> 1, r2 = w >> 2, l1 = w << 1, l2 = w << 2;
  uint32_t a, b, c, d;
  MIXFP4_LOP3(a, 0x22222222u, r1, l1, 0xBF);        // ~K | ~r1 | l1
  MIXFP4_LOP3(b, 0x44444444u, l1, l2, 0x7F);        // ~K | ~(l1 & l2)
  MIXFP4_LOP3(c, w, a, b, 0x80);                    // w & a & b
  MIXFP4_LOP3(d, c, r2, 0x11111111u, 0x70);         // c & (~r2 | ~K)
  return d;
}
// Scale bytes of a residual row: the scale (type bit cleared) where the type
// bit is set, else 0 (prmt with the sign-replicate selectors gives 0xFF per
// byte whose bit 7 is set).
__device__ __forceinline__ uint32_t residual_scales(uint32_t sw) {
  uint32_t m;
  asm("prmt.b32 %0, %1, %2, 0xBA98;" : "=r"(m) : "r"(sw), "r"(0u));
  return sw & m & 0x7F7F7F7Fu;
}

// Row r's four ue4m3 scales of K step j in the tiled layout of a 128-row tile.
__device__ __forceinline__ uint32_t sf_offset(int r) { return (uint32_t)((r & 31) * 16 + (r >> 5) * 4); }

__global__ void __launch_bounds__(kThreads, 1)
nvf4_fewrows_kernel(const __grid_constant__ CUtensorMap tm_wc, const __grid_constant__ CUtensorMap tm_ws,
                    const __grid_constant__ CUtensorMap tm_xc, const __grid_constant__ CUtensorMap tm_xs,
                    const float* __restrict__ a_ts, const float* __restrict__ b_ts, int Mx, int nx, int N, int K,
                    float* __restrict__ C, long long ldc, int chunk_units, uint32_t* status_word) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  Bars* bars = reinterpret_cast<Bars*>(smem);
  volatile int* abort_flag = &bars->abort;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int num_kc = K / BKC;
  const long long units = (long long)((N + WR - 1) / WR) * num_kc;
  const long long u_begin = units * blockIdx.x / gridDim.x, u_end = units * (blockIdx.x + 1) / gridDim.x;
  // End of the accumulation run that starts at unit u: the end of its weight
  // tile, of this CTA's units, or of its accumulation chunk (chunk_units K
  // slices), whichever is first.
  auto run_end_of = [&](long long u) {
    long long e = (u / num_kc + 1) * num_kc;
    if (e > u_end) e = u_end;
    if (e > u + chunk_units) e = u + chunk_units;
    return e;
  };
  const int XR = xr_of(nx);
  const uint32_t OB = (uint32_t)off_b(XR), OWS = (uint32_t)off_ws(XR), OXS = (uint32_t)off_xs(XR);
  const uint32_t OSFA = (uint32_t)off_sfa(XR), OSFB = (uint32_t)off_sfb(XR), OSFR = (uint32_t)off_sfr(XR);
  const uint32_t SB = (uint32_t)stage_bytes_of(XR);
  const int NST = stages_of(XR);
  const uint32_t tx_bytes = WR * ROWB + WR * 16 + (uint32_t)nx * (ROWB + 16);
  const uint32_t sbase = smem_u32(smem) + OFF_RINGS;

  if (threadIdx.x == 0) {
    for (int s = 0; s < NST; ++s) {
      mbar_init(smem_u32(&bars->full[s]), 1);
      mbar_init(smem_u32(&bars->split_full[s]), kWSplitWarps + kXSplitWarps);
      mbar_init(smem_u32(&bars->sf_full[s]), kCopyWarps);
      mbar_init(smem_u32(&bars->sf_ready[s]), kWSplitWarps + kXSplitWarps);
      mbar_init(smem_u32(&bars->empty[s]), 1);
    }
    mbar_init(smem_u32(&bars->acc_full), 1);
    mbar_init(smem_u32(&bars->acc_empty), 4);
    mbar_init(smem_u32(&bars->drain), 1);
    bars->abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&bars->tmem_base), kTmemCols);
    tmem_relinquish();
  }
  griddep_launch_dependents();
  tc_fence_before();
  __syncthreads();
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
      tma_prefetch(&tm_wc);
      tma_prefetch(&tm_ws);
      tma_prefetch(&tm_xc);
      tma_prefetch(&tm_xs);
      griddep_wait();
      int it = 0;
      long long last = -1;
      for (long long u = u_begin; u < u_end; ++u, ++it) {
        const int s = it % NST;
        if (!mbar_wait(smem_u32(&bars->empty[s]), ((it / NST) & 1) ^ 1, abort_flag, kWaitLimitNs)) {
          fail(1u);
          break;
        }
        const int g = (int)(u / num_kc), kc = (int)(u % num_kc);
        const uint32_t st = sbase + s * SB;
        const uint32_t fb = smem_u32(&bars->full[s]);
        mbar_arrive_expect_tx(fb, tx_bytes);
        tma_load_2d(st + OB, &tm_wc, kc * ROWB, g * WR, fb);
        tma_load_2d(st + OWS, &tm_ws, kc * 16, g * WR, fb);
        tma_load_2d(st, &tm_xc, kc * ROWB, 0, fb);
        tma_load_2d(st + OXS, &tm_xs, kc * 16, 0, fb);
        last = it;
      }
      if (*abort_flag)
        for (long long v = last - NST + 1; v <= last; ++v)
          if (v >= 0)
            mbar_wait(smem_u32(&bars->full[v % NST]), (uint32_t)((v / NST) & 1), nullptr, kWaitLimitNs);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      constexpr uint32_t kIdesc = idesc_nvf4_f32(128, 2 * WR);
      int it = 0, run = 0;
      bool ok = true;
      for (long long u = u_begin; u < u_end && ok; ++run) {
        const long long run_end = run_end_of(u);
        if (!mbar_wait(smem_u32(&bars->acc_empty), (run & 1) ^ 1, abort_flag, kWaitLimitNs)) {
          fail(2u);
          break;
        }
        tc_fence_after();
        bool first = true;
        for (; u < run_end; ++u, ++it) {
          const int s = it % NST;
          if (!mbar_wait(smem_u32(&bars->split_full[s]), (uint32_t)((it / NST) & 1), abort_flag, kWaitLimitNs) ||
              !mbar_wait(smem_u32(&bars->sf_full[s]), (uint32_t)((it / NST) & 1), abort_flag, kWaitLimitNs)) {
            fail(4u);
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sp = sbase + s * SB;
#pragma unroll
          for (int j = 0; j < BKC / 64; ++j) {
            const uint32_t sfa = tmem_sf0 + (uint32_t)(s * 4 + j) * kSfCols, sfb = sfa + 4;
            mma_nvf4(tmem_base, smem_desc_sw128(sp + j * 32), smem_desc_sw128(sp + OB + j * 32), kIdesc, sfa, sfb,
                     first ? 0u : 1u);
            first = false;
          }
          mma_commit(smem_u32(&bars->empty[s]));
        }
        if (ok) mma_commit(smem_u32(&bars->acc_full));
      }
      mma_commit(smem_u32(&bars->drain));
      if (!mbar_wait(smem_u32(&bars->drain), 0, nullptr, kWaitLimitNs)) fail(8u);
    }
  } else if (warp >= kCopyWarp) {
    // ---------------- scale copies ----------------
    // Once a stage's scale tiles are written (before its residual rows), the
    // A tile's scales, the weight main rows' scales and the weight residual
    // rows' scales go to tensor memory (tcgen05.cp, replicated to the four
    // lane quarters) and the commit tells the MMA thread, which also waits
    // for the residual rows; the two copy warps take K steps 0-1 and 2-3.  A
    // stage's columns are rewritten only after its next TMA landing, which
    // follows the MMAs that read them.
    const int j0 = 2 * (warp - kCopyWarp);
    if (lane == 0) {
      int it = 0;
      for (long long u = u_begin; u < u_end; ++u, ++it) {
        const int s = it % NST;
        if (!mbar_wait(smem_u32(&bars->sf_ready[s]), (uint32_t)((it / NST) & 1), abort_flag, kWaitLimitNs)) {
          fail(128u);
          break;
        }
        tc_fence_after();
        const uint32_t sp = sbase + s * SB;
#pragma unroll
        for (int j = j0; j < j0 + 2; ++j) {
          const uint32_t sfa = tmem_sf0 + (uint32_t)(s * 4 + j) * kSfCols, sfb = sfa + 4;
          tmem_cp_32x128b_x4(sfa, smem_desc_noswizzle(sp + OSFA + j * 512, 128, 128));
          tmem_cp_32x128b_x4(sfb, smem_desc_noswizzle(sp + OSFB + j * 512, 128, 128));
          tmem_cp_32x128b_x4(sfb + 4, smem_desc_noswizzle(sp + OSFR + j * 512, 128, 128));
        }
        mma_commit(smem_u32(&bars->sf_full[s]));
      }
    }
  } else if (warp < kFirstEpi) {
    // ---------------- residual rows and scale tiles ----------------
    // Weights: thread t of 512 takes row t / 4, chunks 2 (t % 4) and +1 and
    // scale word t % 4 (K step t % 4).  Activations: thread t of 128 takes
    // chunks q = t + 128 i (row q / 8, chunk q % 8) of rows < nx.
    const bool is_w = warp < kFirstX;
    const int t = is_w ? (warp - kFirstW) * 32 + lane : (warp - kFirstX) * 32 + lane;
    auto pick = [](const uint4& v, int i) {  // v[i] without dynamic indexing
      return (i & 2) ? ((i & 1) ? v.w : v.z) : ((i & 1) ? v.y : v.x);
    };
    int it = 0;
    for (long long u = u_begin; u < u_end; ++u, ++it) {
      const int s = it % NST;
      if (!mbar_wait(smem_u32(&bars->full[s]), (uint32_t)((it / NST) & 1), abort_flag, kWaitLimitNs)) {
        fail(16u);
        break;
      }
      const uint32_t sp = sbase + s * SB;
      if (is_w) {
        const int row = t >> 2, q4 = t & 3;
        const uint32_t swz = (uint32_t)(row & 7);
        {
          const uint32_t sw = lds32(sp + OWS + (uint32_t)row * 16 + (uint32_t)q4 * 4);
          sts32(sp + OSFB + q4 * 512 + sf_offset(row), sw & 0x7F7F7F7Fu);
          sts32(sp + OSFR + q4 * 512 + sf_offset(row), residual_scales(sw));
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&bars->sf_ready[s]));
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          const uint32_t a = sp + OB + (uint32_t)row * ROWB + ((((uint32_t)(2 * q4 + k)) ^ swz) << 4);
          const uint4 c = lds128(a);
          sts128(a + WR * ROWB, residual_word(c.x), residual_word(c.y), residual_word(c.z), residual_word(c.w));
        }
      } else {
        for (int q = t; q < nx * 4; q += kXSplitWarps * 32) {  // scale word q % 4 of row q / 4
          const int row = q >> 2, j = q & 3;
          const uint32_t sw = lds32(sp + OXS + (uint32_t)row * 16 + (uint32_t)j * 4);
          sts32(sp + OSFA + j * 512 + sf_offset(row), sw & 0x7F7F7F7Fu);
          sts32(sp + OSFA + j * 512 + sf_offset(row + XR), residual_scales(sw));
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&bars->sf_ready[s]));
#pragma unroll 1
        for (int q = t; q < nx * 8; q += kXSplitWarps * 32) {
          const int row = q >> 3, c8 = q & 7;
          const uint32_t a = sp + (uint32_t)row * ROWB + ((((uint32_t)c8) ^ (uint32_t)(row & 7)) << 4);
          const uint4 c = lds128(a);
          sts128(a + (uint32_t)XR * ROWB, residual_word(c.x), residual_word(c.y), residual_word(c.z),
                 residual_word(c.w));
        }
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&bars->split_full[s]));
    }
  } else {
    // ---------------- epilogue ----------------
    // Accumulator lane d (quarter q = warp % 4, d = 32 q + lane) holds
    // activation row d mod XR: main products for d < XR, residual products
    // for XR <= d < 2 XR; both add into C.
    const int q = warp & 3;
    const int d = q * 32 + lane;
    const int m = d % XR;
    griddep_wait();
    const float sa = __ldg(a_ts), sb = __ldg(b_ts);
    const bool vec_ok = ((ldc & 3) == 0) && ((reinterpret_cast<uintptr_t>(C) & 15) == 0);
    const bool mine = q * 32 < 2 * XR && (q * 32) % XR < Mx;
    const uint32_t tb = tmem_base + ((uint32_t)(q * 32) << 16);
    int run = 0;
    for (long long u = u_begin; u < u_end; ++run) {
      const int g = (int)(u / num_kc);
      u = run_end_of(u);
      const bool acc_ok = mbar_wait(smem_u32(&bars->acc_full), run & 1, abort_flag, kWaitLimitNs);
      tc_fence_after();
      const bool go = __all_sync(0xffffffffu, acc_ok && !*abort_flag);
      if (!go) {
        if (!acc_ok && !*abort_flag) fail(64u);
        break;
      }
#pragma unroll 1
      for (int cc = 0; cc < WR / 16; ++cc) {
        uint32_t v[16], w[16];
        if (mine) {
          tmem_ld_32x32b_x16(tb + (uint32_t)(cc * 16), v);
          tmem_ld_32x32b_x16(tb + (uint32_t)(WR + cc * 16), w);
          tmem_ld_wait_x16(v);
          reg_fence16(w);
        }
        if (cc == WR / 16 - 1) {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&bars->acc_empty));
        }
        const int n0 = g * WR + cc * 16;
        if (mine && d < 2 * XR && m < Mx) {
          float* crow = C + (long long)m * ldc + n0;
          float o[16];
#pragma unroll
          for (int k = 0; k < 16; ++k)
            o[k] = __fmul_rn(__fmul_rn(__fadd_rn(__uint_as_float(v[k]), __uint_as_float(w[k])), sa), sb);
          if (vec_ok && n0 + 16 <= N) {
#pragma unroll
            for (int k = 0; k < 16; k += 4) red_add_v4(crow + k, o[k], o[k + 1], o[k + 2], o[k + 3]);
          } else {
            for (int k = 0; k < 16; ++k)
              if (n0 + k < N) atomicAdd(crow + k, o[k]);
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

int launch(const uint8_t* a_codes, const uint8_t* a_scales, const float* a_ts, const uint8_t* b_codes,
           const uint8_t* b_scales, const float* b_ts, int64_t M, int64_t N, int64_t K, float* C, int64_t ldc,
           uint32_t* status_word, cudaStream_t stream) {
  const int nx = (int)((M + 15) & ~15);
  CUtensorMap twc, tws, txc, txs;
  if (!make_map(&twc, b_codes, (uint64_t)K / 2, (uint64_t)N, ROWB, WR, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_map(&tws, b_scales, (uint64_t)K / 16, (uint64_t)N, 16, WR, CU_TENSOR_MAP_SWIZZLE_NONE) ||
      !make_map(&txc, a_codes, (uint64_t)K / 2, (uint64_t)M, ROWB, (uint32_t)nx, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_map(&txs, a_scales, (uint64_t)K / 16, (uint64_t)M, 16, (uint32_t)nx, CU_TENSOR_MAP_SWIZZLE_NONE))
    return MIXFP4_ERR_CUDA;
  const int xr = xr_of(nx);
  const int smem = OFF_RINGS + stages_of(xr) * stage_bytes_of(xr) + 1024;
  static std::atomic<uint64_t> smem_set{0};
  if (!set_dynamic_smem_once(reinterpret_cast<const void*>(nvf4_fewrows_kernel), 232448, smem_set))
    return MIXFP4_ERR_CUDA;
  cudaError_t e;
  if (ldc == N)
    e = cudaMemsetAsync(C, 0, (size_t)M * (size_t)N * sizeof(float), stream);
  else
    e = cudaMemset2DAsync(C, (size_t)ldc * sizeof(float), 0, (size_t)N * sizeof(float), (size_t)M, stream);
  if (e != cudaSuccess) return MIXFP4_ERR_CUDA;
  const int64_t units = ((N + WR - 1) / WR) * (K / BKC);
  int64_t grid = num_sms();
  if (grid > units) grid = units;
  if (launch_pdl(nvf4_fewrows_kernel, (unsigned)grid, kThreads, smem, stream, twc, tws, txc, txs, a_ts, b_ts,
                 (int)M, nx, (int)N, (int)K, C, (long long)ldc, kAccumChunkK / BKC, status_word) != cudaSuccess)
    return MIXFP4_ERR_CUDA;
  return MIXFP4_OK;
}

}  // namespace nvs

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

namespace mixfp4 {
int launch_gemm_native_fewrows(const uint8_t* a_codes, const uint8_t* a_scales, const float* a_ts,
                               const uint8_t* b_codes, const uint8_t* b_scales, const float* b_ts, int64_t M,
                               int64_t N, int64_t K, float* C, int64_t ldc, uint32_t* status_word,
                               cudaStream_t stream) {
  return nvs::launch(a_codes, a_scales, a_ts, b_codes, b_scales, b_ts, M, N, K, C, ldc, status_word, stream);
}
}  // namespace mixfp4
