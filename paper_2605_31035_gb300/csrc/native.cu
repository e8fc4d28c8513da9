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
#undef MIXFP4_LOP3

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
// Few-row native variant (M <= 64 activation rows, the decode shape): the
// MixFP4 operands are split into E2M1 main + residual parts on the fly, in
// shared memory, instead of beforehand.  Weight rows go on the MMA N side in
// units of 128 rows x one 256-wide K slice: the split writes the 128 main rows
// to rows 0-127 and the 128 residual rows to rows 128-255 of one N = 256
// operand tile, and the activation rows' main and residual parts to rows
// 0-63 and 64-127 of the M = 128 operand tile, so ONE kind::mxf4nvf4 MMA per
// 64-K step forms all four products; the epilogue adds the accumulator's four
// quadrants: C[m][n] = D[m][n] + D[m][128+n] + D[64+m][n] + D[64+m][128+n].
// Per CTA (one per SM, units split evenly over all SMs, partial sums added
// into C which the host zeroed):
//   warp 0      TMA: 128 x 128-byte weight code tile (128-byte swizzle), its
//               128 x 16-byte scale tile, the activation rows' code and scale
//               tiles, into a ring of 2-4 stages (21-27 KB each, by the row
//               count), ahead of a 3-stage ring of split operand tiles;
//   warp 1      TMEM allocation; lane 0 issues the MMAs (one per 64-K step);
//   warps 2-17  split the weight codes (four threads per row, two 16-byte
//               chunks each: E2M1 blocks copied, E1M2 nibbles p -> main
//               {0,2,4,5,6,6,7,7}[p] and residual (p in {5,7} ? 2 : 0) by
//               bit logic on eight nibbles at a time) into the swizzled
//               operand tile, and the scale bytes into the tensor core's
//               tiled layout; warps 18-21 the same for the activation rows;
//   warps 22-25 epilogue, one TMEM lane quarter each;
//   warps 26-27 copy each split stage's scale tiles into tensor memory
//               (tcgen05.cp, half of the K steps each) and commit, so that
//               scale copies and MMAs are issued by three threads in parallel
//               (each tcgen05 instruction holds its issuing thread ~50 ns).
// ============================================================================
namespace nvs {

constexpr int WR = 128;                    // weight rows per unit (MMA N = 2 x 128)
constexpr int XR = 64;                     // activation rows (MMA M = 2 x 64)
constexpr int BKC = 256;                   // K per unit
constexpr int ROWB = BKC / 2;              // 128 code bytes per row per unit
constexpr int kMaxCodeStages = 4, kSplitStages = 3;
// Code stage (ring of TMA destinations): weight codes and scales, then the
// nx activation rows' codes and scales; its size depends on nx (host side).
constexpr int OFF_WC = 0, OFF_WS = WR * ROWB, OFF_XC = OFF_WS + WR * 16;
constexpr int S_B = 0, S_A = 2 * WR * ROWB, S_SFA = S_A + 2 * XR * ROWB, S_SFB = S_SFA + 4 * 512;
constexpr int SPLIT_STAGE = S_SFB + 4 * 512;                     // 52 KB
constexpr int OFF_RINGS = 1024;                                  // after the barrier block
constexpr int kSmemBudget = 232448 - 1024;                       // 1024 for the alignment of the base
static_assert(OFF_XC % 1024 == 0 && SPLIT_STAGE % 1024 == 0 && S_A % 1024 == 0,
              "swizzled tiles need 1024-byte alignment");
__host__ __device__ constexpr int code_stage_bytes(int nx) { return ((OFF_XC + nx * (ROWB + 16) + 1023) / 1024) * 1024; }
__host__ __device__ constexpr int code_stages(int nx) {
  return (kSmemBudget - OFF_RINGS - kSplitStages * SPLIT_STAGE) / code_stage_bytes(nx) < kMaxCodeStages
             ? (kSmemBudget - OFF_RINGS - kSplitStages * SPLIT_STAGE) / code_stage_bytes(nx)
             : kMaxCodeStages;
}
static_assert(code_stages(XR) >= 2, "shared memory budget");
constexpr int kWSplitWarps = 16, kXSplitWarps = 4;
constexpr int kFirstW = 2, kFirstX = kFirstW + kWSplitWarps, kFirstEpi = kFirstX + kXSplitWarps;  // 2, 18, 22
constexpr int kCopyWarp = kFirstEpi + 4, kCopyWarps = 2;                                          // 26, 27
constexpr int kThreads = 32 * (kCopyWarp + kCopyWarps);                                           // 896
static_assert(kFirstEpi % 4 == 2, "epilogue warps cover the four TMEM lane quarters");
constexpr uint32_t kAccCols = 2 * WR;                            // 256 fp32 columns
constexpr uint32_t kSfCols = 12;                                 // per K step: 4 (A) + 8 (B)
constexpr uint32_t kTmemCols = 512;
constexpr uint64_t kWaitLimitNs = 1000000000ull;
static_assert(kAccCols + kSplitStages * 4 * kSfCols <= kTmemCols, "TMEM budget");

struct Bars {
  uint64_t code_full[kMaxCodeStages];
  uint64_t code_empty[kMaxCodeStages];
  uint64_t split_full[kSplitStages];
  uint64_t sf_full[kSplitStages];   // the stage's scales are in tensor memory (commit of the copy warp)
  uint64_t split_empty[kSplitStages];
  uint64_t acc_full;
  uint64_t acc_empty;
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
};
static_assert(sizeof(Bars) <= 256, "barrier block");


// Split one 16-byte chunk (two blocks) given the blocks' type bits.
__device__ __forceinline__ void split_chunk(uint4 c, bool t0, bool t1, uint4& m, uint4& r) {
  const uint32_t k0 = t0 ? 0xFFFFFFFFu : 0u, k1 = t1 ? 0xFFFFFFFFu : 0u;
  split_e1m2_word(c.x, k0, m.x, r.x);
  split_e1m2_word(c.y, k0, m.y, r.y);
  split_e1m2_word(c.z, k1, m.z, r.z);
  split_e1m2_word(c.w, k1, m.w, r.w);
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
  const uint32_t stage_bytes = WR * ROWB + WR * 16 + (uint32_t)nx * (ROWB + 16);
  const int CS = code_stage_bytes(nx), NCS = code_stages(nx);
  const uint32_t OFF_XS = (uint32_t)(OFF_XC + nx * ROWB);
  const uint32_t sbase = smem_u32(smem) + OFF_RINGS;          // code ring, then the split ring
  const uint32_t OFF_SPLIT = (uint32_t)(NCS * CS);

  // Split stages start as zeros: activation rows >= nx (and their residual
  // rows and scales) are never written, so they stay zero.
  for (uint32_t i = threadIdx.x; i < (uint32_t)(kSplitStages * SPLIT_STAGE / 16); i += blockDim.x)
    sts128(sbase + OFF_SPLIT + i * 16, 0u, 0u, 0u, 0u);
  fence_proxy_async_smem();
  if (threadIdx.x == 0) {
    for (int s = 0; s < NCS; ++s) {
      mbar_init(smem_u32(&bars->code_full[s]), 1);
      mbar_init(smem_u32(&bars->code_empty[s]), kWSplitWarps + kXSplitWarps);
    }
    for (int s = 0; s < kSplitStages; ++s) {
      mbar_init(smem_u32(&bars->split_full[s]), kWSplitWarps + kXSplitWarps);
      mbar_init(smem_u32(&bars->sf_full[s]), kCopyWarps);
      mbar_init(smem_u32(&bars->split_empty[s]), 1);
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
        const int s = it % NCS;
        if (!mbar_wait(smem_u32(&bars->code_empty[s]), ((it / NCS) & 1) ^ 1, abort_flag, kWaitLimitNs)) {
          fail(1u);
          break;
        }
        const int g = (int)(u / num_kc), kc = (int)(u % num_kc);
        const uint32_t st = sbase + s * CS;
        const uint32_t fb = smem_u32(&bars->code_full[s]);
        mbar_arrive_expect_tx(fb, stage_bytes);
        tma_load_2d(st + OFF_WC, &tm_wc, kc * ROWB, g * WR, fb);
        tma_load_2d(st + OFF_WS, &tm_ws, kc * 16, g * WR, fb);
        tma_load_2d(st + OFF_XC, &tm_xc, kc * ROWB, 0, fb);
        tma_load_2d(st + OFF_XS, &tm_xs, kc * 16, 0, fb);
        last = it;
      }
      if (*abort_flag)
        for (long long v = last - NCS + 1; v <= last; ++v)
          if (v >= 0)
            mbar_wait(smem_u32(&bars->code_full[v % NCS]), (uint32_t)((v / NCS) & 1), nullptr,
                      kWaitLimitNs);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      constexpr uint32_t kIdesc = idesc_nvf4_f32(2 * XR, 2 * WR);
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
          const int s = it % kSplitStages;
          if (!mbar_wait(smem_u32(&bars->sf_full[s]), (uint32_t)((it / kSplitStages) & 1), abort_flag,
                         kWaitLimitNs)) {
            fail(4u);
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sp = sbase + OFF_SPLIT + s * SPLIT_STAGE;
#pragma unroll
          for (int j = 0; j < BKC / 64; ++j) {
            const uint32_t sfa = tmem_sf0 + (uint32_t)(s * 4 + j) * kSfCols, sfb = sfa + 4;
            mma_nvf4(tmem_base, smem_desc_sw128(sp + S_A + j * 32), smem_desc_sw128(sp + S_B + j * 32), kIdesc, sfa,
                     sfb, first ? 0u : 1u);
            first = false;
          }
          mma_commit(smem_u32(&bars->split_empty[s]));
        }
        if (ok) mma_commit(smem_u32(&bars->acc_full));
      }
      mma_commit(smem_u32(&bars->drain));
      if (!mbar_wait(smem_u32(&bars->drain), 0, nullptr, kWaitLimitNs)) fail(8u);
    }
  } else if (warp >= kCopyWarp) {
    // ---------------- scale copies ----------------
    // Once a stage is split, its A and B scale tiles go to tensor memory
    // (tcgen05.cp, replicated to the four lane quarters; the B tile twice, for
    // the main and residual halves of N) and the commits tell the MMA thread;
    // the two copy warps take K steps 0-1 and 2-3.  A stage's columns are
    // rewritten only after its next split, which waits for the MMAs that
    // read them.
    const int j0 = 2 * (warp - kCopyWarp);
    if (lane == 0) {
      int it = 0;
      for (long long u = u_begin; u < u_end; ++u, ++it) {
        const int s = it % kSplitStages;
        if (!mbar_wait(smem_u32(&bars->split_full[s]), (uint32_t)((it / kSplitStages) & 1), abort_flag,
                       kWaitLimitNs)) {
          fail(128u);
          break;
        }
        tc_fence_after();
        const uint32_t sp = sbase + OFF_SPLIT + s * SPLIT_STAGE;
#pragma unroll
        for (int j = j0; j < j0 + 2; ++j) {
          const uint32_t sfa = tmem_sf0 + (uint32_t)(s * 4 + j) * kSfCols, sfb = sfa + 4;
          tmem_cp_32x128b_x4(sfa, smem_desc_noswizzle(sp + S_SFA + j * 512, 128, 128));
          tmem_cp_32x128b_x4(sfb, smem_desc_noswizzle(sp + S_SFB + j * 512, 128, 128));
          tmem_cp_32x128b_x4(sfb + 4, smem_desc_noswizzle(sp + S_SFB + j * 512, 128, 128));
        }
        mma_commit(smem_u32(&bars->sf_full[s]));
      }
    }
  } else if (warp < kFirstEpi) {
    // ---------------- splitters ----------------
    // Weights: thread t of 512 splits row t / 4, chunks 2 (t % 4) and +1
    // (blocks 4 (t % 4) .. +3, scale word t % 4).  Activations: thread t of
    // 128 splits chunks q = t + 128 i (row q / 8, chunk q % 8) of rows < nx.
    const bool is_w = warp < kFirstX;
    const int t = is_w ? (warp - kFirstW) * 32 + lane : (warp - kFirstX) * 32 + lane;
    auto pick = [](const uint4& v, int i) {  // v[i] without dynamic indexing
      return (i & 2) ? ((i & 1) ? v.w : v.z) : ((i & 1) ? v.y : v.x);
    };
    int it = 0;
    for (long long u = u_begin; u < u_end; ++u, ++it) {
      const int s = it % NCS, sps = it % kSplitStages;
      if (!mbar_wait(smem_u32(&bars->code_full[s]), (uint32_t)((it / NCS) & 1), abort_flag,
                     kWaitLimitNs)) {
        fail(16u);
        break;
      }
      if (!mbar_wait(smem_u32(&bars->split_empty[sps]), (uint32_t)(((it / kSplitStages) & 1) ^ 1), abort_flag,
                     kWaitLimitNs)) {
        fail(32u);
        break;
      }
      const uint32_t st = sbase + s * CS, sp = sbase + OFF_SPLIT + sps * SPLIT_STAGE;
      if (is_w) {
        const int row = t >> 2, q4 = t & 3;
        const uint32_t swz = (uint32_t)(row & 7);
        const uint4 sc = lds128(st + OFF_WS + (uint32_t)row * 16);
        const uint32_t sw = pick(sc, q4);
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          const uint32_t pc = ((uint32_t)(2 * q4 + k) ^ swz) << 4;
          const uint32_t tb = sw >> (16 * k);
          uint4 m, r;
          split_chunk(lds128(st + OFF_WC + (uint32_t)row * ROWB + pc), (tb & 0x80u) != 0, (tb & 0x8000u) != 0, m, r);
          sts128(sp + S_B + (uint32_t)row * ROWB + pc, m.x, m.y, m.z, m.w);
          sts128(sp + S_B + (uint32_t)(row + WR) * ROWB + pc, r.x, r.y, r.z, r.w);
        }
        // Scales of K step q4 into the tiled layout (bit 7, the type, cleared).
        sts32(sp + S_SFB + q4 * 512 + sf_offset(row), sw & 0x7F7F7F7Fu);
      } else {
#pragma unroll 1
        for (int q = t; q < nx * 8; q += kXSplitWarps * 32) {
          const int row = q >> 3, c = q & 7;
          const uint32_t pc = ((uint32_t)c ^ (uint32_t)(row & 7)) << 4;
          const uint4 sc = lds128(st + OFF_XS + (uint32_t)row * 16);
          const uint32_t sw = pick(sc, c >> 1), tb = sw >> (16 * (c & 1));
          uint4 m, r;
          split_chunk(lds128(st + OFF_XC + (uint32_t)row * ROWB + pc), (tb & 0x80u) != 0, (tb & 0x8000u) != 0, m, r);
          sts128(sp + S_A + (uint32_t)row * ROWB + pc, m.x, m.y, m.z, m.w);
          sts128(sp + S_A + (uint32_t)(row + XR) * ROWB + pc, r.x, r.y, r.z, r.w);
          if ((c & 1) == 0) {  // scale word c / 2 = K step c / 2, for the main and residual rows
            sts32(sp + S_SFA + (c >> 1) * 512 + sf_offset(row), sw & 0x7F7F7F7Fu);
            sts32(sp + S_SFA + (c >> 1) * 512 + sf_offset(row + XR), sw & 0x7F7F7F7Fu);
          }
        }
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(smem_u32(&bars->split_full[sps]));
        mbar_arrive(smem_u32(&bars->code_empty[s]));
      }
    }
  } else {
    // ---------------- epilogue ----------------
    // Warps for lane quarters 0, 1 hold the activation rows' main products,
    // quarters 2, 3 their residual products (row m + 64); both add into C.
    const int q = warp & 3;
    const int m = (q & 1) * 32 + lane;
    griddep_wait();
    const float sa = __ldg(a_ts), sb = __ldg(b_ts);
    const bool vec_ok = ((ldc & 3) == 0) && ((reinterpret_cast<uintptr_t>(C) & 15) == 0);
    const bool mine = (q & 1) * 32 < Mx;
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
        if (mine && m < Mx) {
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
  const int smem = OFF_RINGS + code_stages(nx) * code_stage_bytes(nx) + kSplitStages * SPLIT_STAGE + 1024;
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
