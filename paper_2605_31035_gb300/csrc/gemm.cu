// MixFP4 x MixFP4 GEMM for sm_103a: C = A_deq . B_deq^T (App. B.1 Eq. (factor)).
//
// Per 16-element block the MixFP4 codes are decoded to the unified E2M2 value
// (Sec. 3.3, App. B.5) times the block's E4M3 scale.  Written as u * s8 with
// u = 2v (E2M1: {0,1,2,3,4,6,8,12}, E1M2: {0,2,...,14}) the product has at most
// 7 significant bits and lies in [2^-9, 14 * 448], so it is exact in f16; the
// tensor cores contract f16 x f16 with fp32 accumulation (tcgen05.mma
// kind::f16, K = 16 per instruction) and the epilogue applies s32A * s32B / 4.
//
// Accumulation length.  The tensor cores add each K step's products into the
// fp32 accumulator with an error that grows with the number of steps added
// into one accumulator (relative to |A|.|B|, about 1e-6 per 1024 of K on
// outlier-heavy operands whose outlier channels coincide).  So the work
// schedule cuts every tile's K into chunks of at most 16 K slices (4096 K):
// each chunk is accumulated from zero, and the epilogue stores the first
// chunk of a tile into C and adds the later ones (TMA add), so the
// bound no longer depends on K.
//
// Work decomposition: persistent CTA pairs (clusters of 2, cta_group::2).  A
// pair owns 256 x kTileN output tiles (kTileN = 256, 224 or 192); each CTA
// holds 128 rows of A and kTileN / 2 rows of B.  Tiles of the full waves are
// dealt whole (chunk by chunk);
// when the tile count leaves a partial last wave, that wave's (tile, K slice)
// units are split evenly over all pairs (stream-K) and their partial sums are
// added into C (TMA add) after the host zeroed those tiles.  Tiles are numbered
// row band by row band (t = mt * ntiles_n + nt).  Decoded A never touches
// shared memory: it is written to tensor memory (tcgen05.st) and the MMA reads
// it from there; decoded B goes through shared memory.  Per CTA:
//   warp 0        TMA producer: codes [rows][128 B] (128-byte swizzle) and
//                 scales [rows][16 B] of a 256-wide K slice into a 2-deep ring;
//   warp 1        TMEM allocator (both CTAs); in the leader CTA also the single
//                 MMA-issuing thread;
//   warps 2-9     A decoders, two groups of four (lane quarter = warp % 4): the
//                 first group decodes the first 128-K stage of every code
//                 stage, the second group the second, one thread per A row,
//                 128 K of the row -> f16 pairs in TMEM columns;
//   next 6-8      B decoders in the same two groups, one thread per B row of
//                 the tile (kTileN / 2 rows; a 224-wide tile puts the last 16
//                 rows of both groups in one shared warp), 128 K of the row ->
//                 f16 in the canonical K-major no-swizzle UMMA layout;
//   last 8 warps  epilogue: tcgen05.ld -> x s32A s32B / 4 -> a per-warp shared
//                 staging tile -> TMA store (or TMA add) of the 32 x 16 box.
// Each decoder warp synchronises once per code stage instead of once per
// decoded stage, so the decoders spend a smaller share of their time in
// barrier waits (their ALU work bounds the main loop).
// TMEM per CTA (512 columns): fp32 accumulator 128 lanes x 256 columns, then
// kDecStages A stages of 64 columns (128 K of f16 pairs).  The leader's MMA
// waits for both CTAs' decoders: every decoder warp of a stage arrives on the
// leader's barrier, the peer's through a remote arrival.
// All pipeline waits are bounded (1 s each, or the self-test's limit); a
// wait that gives up ORs its role's bit into the status word (1 producer,
// 2 MMA thread waiting for the accumulator, 4 MMA thread waiting for a
// decoded stage, 8 final drain, 16 / 32 decoders, 64 epilogue), raises the
// CTA's abort flag, and the CTA lets its issued copies
// and MMAs land, frees TMEM and exits without touching C.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <cstdint>
#include <cstring>

#include "host_util.cuh"
#include "kernels.cuh"
#include "pipeline.cuh"
#include "ptx.cuh"
#include "sm100.cuh"

namespace mixfp4 {
namespace {

using namespace sm100;

constexpr int BM = 128;                       // A rows per CTA (pair tile: 256)
constexpr int BNH = 128;                      // B rows per CTA (pair tile: 256)
constexpr int TILE_M = 2 * BM, TILE_N = 2 * BNH;
constexpr int BKC = 256;                      // K per TMA code stage
constexpr int BKD = 128;                      // K per decoded stage
constexpr int kSub = BKC / BKD;
constexpr int kCodeStages = 2;
constexpr int kDecStages = 4;
constexpr int kChunksPerSub = BKD / 32;       // 16-byte code chunks (32 codes) per row per stage
static_assert(kSub == 2 && kChunksPerSub == 4, "two decoder groups, one per 128-K stage of a code stage");
constexpr int kDecodeWarpsA = kSub * BM / 32;   // 8: one thread per A row in each group
constexpr int kEpiWarps = 8;
constexpr int kFirstDecA = 2;
constexpr int kFirstDecB = kFirstDecA + kDecodeWarpsA;   // 10
static_assert(kFirstDecA % 4 == 2 && kDecodeWarpsA % 4 == 0, "A decoders cover every TMEM lane quarter");

// Warp roles that depend on the tile width: one B decoder thread per B row of
// the CTA in each group; with kTileN / 2 = 32 f + 16 rows the last 16 rows of
// both groups share one warp (lanes 0-15 first group, 16-31 second).
template <int kTileN>
struct PairRoles {
  static constexpr int kBRows = kTileN / 2;
  static constexpr int kBFull = kBRows / 32;                  // B warps per group with 32 rows
  static constexpr int kBMixed = (kBRows % 32) ? 1 : 0;       // the shared warp
  static_assert(kBRows % 32 == 0 || kBRows % 32 == 16, "B rows per CTA: a multiple of 16");
  static constexpr int kBWarps = kSub * kBFull + kBMixed;
  static constexpr int kFirstEpi = kFirstDecB + kBWarps;
  static constexpr int kThreads = 32 * (kFirstEpi + kEpiWarps);
  static constexpr int kDecodeWarps = kDecodeWarpsA + kBWarps;  // arrivals per code stage
  // Arrivals on a decoded stage: its A group, its full B warps, the shared warp.
  static constexpr int kStageArrivals = kDecodeWarpsA / kSub + kBFull + kBMixed;
};

constexpr uint32_t kAccCols = TILE_N;                 // fp32 accumulator columns
constexpr uint32_t kAStageCols = BKD / 2;             // f16 pairs per A row per stage
constexpr uint32_t kTmemCols = 512;
static_assert(kAccCols + kDecStages * kAStageCols <= kTmemCols, "TMEM budget");

constexpr int A_CODE_BYTES = BM * BKC / 2;
constexpr int B_CODE_BYTES = BNH * BKC / 2;
constexpr int A_SCALE_BYTES = BM * BKC / 16;
constexpr int B_SCALE_BYTES = BNH * BKC / 16;
constexpr int CODE_STAGE_BYTES = A_CODE_BYTES + B_CODE_BYTES + A_SCALE_BYTES + B_SCALE_BYTES;
constexpr int B_DEC_BYTES = BNH * BKD * 2;
constexpr int OFF_DEC = kCodeStages * CODE_STAGE_BYTES;
constexpr int EPI_CHUNK = 16;                  // accumulator columns per epilogue step
constexpr int EPI_BYTES = 32 * EPI_CHUNK * 4;   // one warp's 32 rows x 16 fp32 staging tile
constexpr int OFF_EPI = OFF_DEC + kDecStages * B_DEC_BYTES;
constexpr int OFF_BAR = OFF_EPI + kEpiWarps * EPI_BYTES;
constexpr int SMEM_BYTES = OFF_BAR + 256;
constexpr int SMEM_ALLOC = SMEM_BYTES + 1024;  // slack to align the base to 1024 B

static_assert(CODE_STAGE_BYTES % 1024 == 0, "code stages must keep 1024-byte alignment");
static_assert(SMEM_ALLOC <= 232448, "shared memory budget");

// Decoded-B layout: core matrix (8 rows x 16 B) at
//   (row / 8) * SBO + kchunk * LBO + (row % 8) * 16
constexpr uint32_t kLBO = 128;                  // next 8 K-elements
constexpr uint32_t kSBO = (BKD / 8) * 128;      // next 8 rows

constexpr uint64_t kWaitLimitNs = 1000000000ull;  // 1 s per pipeline wait
constexpr int kMinStreamKGainSlices = 8;           // stream-K must save this many K slices per pair

struct Bars {
  uint64_t code_full[kCodeStages];
  uint64_t code_empty[kCodeStages];
  uint64_t dec_full[kDecStages];    // leader: the stage's decoder warps of both CTAs
  uint64_t dec_empty[kDecStages];   // MMA commit (multicast to both CTAs)
  uint64_t acc_full;                // MMA commit (multicast)
  uint64_t acc_empty;               // leader: 2 x kEpiWarps arrivals
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
};
static_assert(sizeof(Bars) <= 256, "barrier block");

__device__ __forceinline__ uint32_t hmul2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("mul.rn.f16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

// f16 high bytes of u = 2v by payload (the low byte of every such f16 is 0):
//   E2M1 u = {0,1,2,3,4,6,8,12} -> 00 3C 40 42 | 44 46 48 4A
//   E1M2 u = {0,2,4,...,14}     -> 00 40 44 46 | 48 49 4A 4B
constexpr uint32_t kLutE2M1Lo = 0x42403C00u, kLutE2M1Hi = 0x4A484644u;
constexpr uint32_t kLutE1M2Lo = 0x46444000u, kLutE1M2Hi = 0x4B4A4948u;

// Decode one 32-bit code word (8 elements, element 2j in the low nibble of
// byte j) of a block with f16x2 scale s2 into four f16x2 words, in the order
// (e0,e1) (e2,e3) (e4,e5) (e6,e7): byte LUT of the payloads (prmt), the
// nibble sign moved into bit 7 of each byte (prmt + lop3), bytes placed as f16
// high bytes (prmt), times s8 (exact).
__device__ __forceinline__ void decode8(uint32_t w, uint32_t lut_lo, uint32_t lut_hi, uint32_t s2,
                                        uint32_t* out) {
  const uint32_t wp = w & 0x77777777u;
  const uint32_t ws = w * 16u;
  const uint32_t u0 = prmt(lut_lo, lut_hi, wp);
  const uint32_t u1 = prmt(lut_lo, lut_hi, __umulhi(wp, 0x10000u));
  const uint32_t g0 = prmt(w, ws, 0x1504u);  // byte i bit 7 = sign of element i   (i = 0..3)
  const uint32_t g1 = prmt(w, ws, 0x3726u);  // byte i bit 7 = sign of element 4+i
  const uint32_t v0 = u0 | (g0 & 0x80808080u);
  const uint32_t v1 = u1 | (g1 & 0x80808080u);
  out[0] = hmul2(prmt(v0, 0u, 0x1404u), s2);
  out[1] = hmul2(prmt(v0, 0u, 0x3424u), s2);
  out[2] = hmul2(prmt(v1, 0u, 0x1404u), s2);
  out[3] = hmul2(prmt(v1, 0u, 0x3424u), s2);
}

// Decode 32 codes (one 16-byte chunk = two 16-element blocks) with their two
// scale bytes s2b into 16 f16x2 words in K order.
__device__ __forceinline__ void decode_chunk(const uint4& c, uint32_t s2b, uint32_t* out) {
  const uint32_t h01 = cvt_f16x2_from_e4m3x2((uint16_t)(s2b & 0x7F7Fu));
  const uint32_t sv[2] = {prmt(h01, 0u, 0x1010u), prmt(h01, 0u, 0x3232u)};
  const uint32_t w[4] = {c.x, c.y, c.z, c.w};
#pragma unroll
  for (int b = 0; b < 2; ++b) {
    const bool e1m2 = (s2b >> (8 * b + 7)) & 1u;
    const uint32_t lut_lo = e1m2 ? kLutE1M2Lo : kLutE2M1Lo;
    const uint32_t lut_hi = e1m2 ? kLutE1M2Hi : kLutE2M1Hi;
    decode8(w[2 * b], lut_lo, lut_hi, sv[b], out + 8 * b);
    decode8(w[2 * b + 1], lut_lo, lut_hi, sv[b], out + 8 * b + 4);
  }
}

__device__ __forceinline__ uint32_t scale_pair(const uint4& sc, int chunk) {
  const int sw = chunk >> 1;  // scale word holding blocks 2*chunk, 2*chunk+1
  const uint32_t s4 = sw == 0 ? sc.x : sw == 1 ? sc.y : sw == 2 ? sc.z : sc.w;
  return (s4 >> (16 * (chunk & 1))) & 0xFFFFu;
}

// kTileN: pair tile width (256, 224 or 192; each CTA holds kTileN / 2 rows of
// B).  Shared and tensor memory are laid out for 256; narrower tiles leave the
// tail of the B regions unused.
template <int kTileN>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(PairRoles<kTileN>::kThreads, 1)
mixfp4_gemm_kernel(const __grid_constant__ CUtensorMap tm_ac, const __grid_constant__ CUtensorMap tm_bc,
                   const __grid_constant__ CUtensorMap tm_as, const __grid_constant__ CUtensorMap tm_bs,
                   const __grid_constant__ CUtensorMap tm_c, int c_tma,
                   const float* __restrict__ a_ts, const float* __restrict__ b_ts,
                   int M, int N, int K, float* __restrict__ C, long long ldc, int dp_tiles, int chunk_kc,
                   uint32_t* status_word, uint64_t wait_ns, int skip_first_stage) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  Bars* bars = reinterpret_cast<Bars*>(smem + OFF_BAR);
  volatile int* abort_flag = &bars->abort;
  const uint32_t sbase = smem_u32(smem);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int num_kc = K / BKC;
  static_assert(kTileN % 32 == 0 && kTileN >= 64 && kTileN <= TILE_N, "tile width");
  using Roles = PairRoles<kTileN>;
  constexpr int kBRows = Roles::kBRows;  // B rows per CTA
  constexpr int kFirstEpi = Roles::kFirstEpi;
  constexpr uint32_t kStageTx = A_CODE_BYTES + A_SCALE_BYTES + kBRows * (BKC / 2 + BKC / 16);
  constexpr uint32_t kIdescT = idesc_f16_f32(TILE_M, kTileN);
  const int mtiles = (M + TILE_M - 1) / TILE_M, ntiles_n = (N + kTileN - 1) / kTileN;
  const int ntiles = mtiles * ntiles_n;
  const int cluster_id = blockIdx.x >> 1, nclusters = gridDim.x >> 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kCodeStages; ++s) {
      mbar_init(smem_u32(&bars->code_full[s]), 1);
      mbar_init(smem_u32(&bars->code_empty[s]), Roles::kDecodeWarps);
    }
    for (int s = 0; s < kDecStages; ++s) {
      mbar_init(smem_u32(&bars->dec_full[s]), 2 * Roles::kStageArrivals);
      mbar_init(smem_u32(&bars->dec_empty[s]), 1);
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
  cluster_sync();  // barriers of both CTAs initialised, TMEM allocated in both
  tc_fence_after();
  const uint32_t tmem_base = bars->tmem_base;
  const uint32_t tmem_a0 = tmem_base + kAccCols;  // first A stage column

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
      griddep_wait();  // the operands may come from the kernel before this one
      int last_it = -1;  // last code-stage use issued (its copies may be in flight)
      int it = 0;
      bool ok = true;
      Sched sched(cluster_id, nclusters, dp_tiles, ntiles, num_kc, chunk_kc);
      int t, k0, k1;
      while (ok && sched.next(t, k0, k1)) {
        const int mt = t / ntiles_n, nt = t % ntiles_n;
        const int ma = mt * TILE_M + (int)rank * BM, nb = nt * kTileN + (int)rank * kBRows;
        for (int kc = k0; kc < k1; ++kc, ++it) {
          // Self-test of the failure path: the first code stage is never
          // issued (no copy, no arrival), so the waits on it run out.
          if (skip_first_stage && it == 0) continue;
          const int s = it % kCodeStages;
          const uint32_t ph = (it / kCodeStages) & 1;
          if (!mbar_wait(smem_u32(&bars->code_empty[s]), ph ^ 1, abort_flag, wait_ns)) {
            fail(1u);
            ok = false;
            break;
          }
          const uint32_t st = sbase + s * CODE_STAGE_BYTES;
          const uint32_t fb = smem_u32(&bars->code_full[s]);
          mbar_arrive_expect_tx(fb, kStageTx);
          const int xk = kc * (BKC / 2), xs = kc * (BKC / 16);
          tma_load_2d(st, &tm_ac, xk, ma, fb);
          tma_load_2d(st + A_CODE_BYTES, &tm_bc, xk, nb, fb);
          tma_load_2d(st + A_CODE_BYTES + B_CODE_BYTES, &tm_as, xs, ma, fb);
          tma_load_2d(st + A_CODE_BYTES + B_CODE_BYTES + A_SCALE_BYTES, &tm_bs, xs, nb, fb);
          last_it = it;
        }
      }
      if (*abort_flag) {
        // Let the copies this thread started land before the CTA may exit.
        for (int u = last_it - kCodeStages + 1; u <= last_it; ++u)
          if (u >= 0 && !(skip_first_stage && u == 0))
            mbar_wait(smem_u32(&bars->code_full[u % kCodeStages]), (uint32_t)((u / kCodeStages) & 1), nullptr,
                      wait_ns);
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer (leader CTA) ----------------
    if (leader && lane == 0) {
      int d = 0;
      uint32_t dph = 0;
      bool ok = true;
      Sched sched(cluster_id, nclusters, dp_tiles, ntiles, num_kc, chunk_kc);
      int t, k0, k1;
      for (int i = 0; ok && sched.next(t, k0, k1); ++i) {
        if (!mbar_wait_cluster(smem_u32(&bars->acc_empty), (i & 1) ^ 1, abort_flag, wait_ns)) {
          fail(2u);
          break;
        }
        tc_fence_after();
        for (int kc = k0; kc < k1 && ok; ++kc) {
          for (int sub = 0; sub < kSub; ++sub) {
            if (!mbar_wait_cluster(smem_u32(&bars->dec_full[d]), dph, abort_flag, wait_ns)) {
              fail(4u);
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t bbase = sbase + OFF_DEC + d * B_DEC_BYTES;
            const uint32_t abase = tmem_a0 + (uint32_t)d * kAStageCols;
#pragma unroll
            for (int j = 0; j < BKD / 16; ++j) {
              const uint64_t bd = smem_desc_noswizzle(bbase + j * 256, kLBO, kSBO);
              mma_f16_pair_tmem_a(tmem_base, abase + j * 8, bd, kIdescT, ((kc - k0) | sub | j) != 0 ? 1u : 0u);
            }
            mma_commit_pair(smem_u32(&bars->dec_empty[d]), 3);
            if (++d == kDecStages) { d = 0; dph ^= 1; }
          }
        }
        if (ok) mma_commit_pair(smem_u32(&bars->acc_full), 3);
      }
      // Every MMA issued above completes before the drain barrier fires; wait
      // for it (ignoring the abort flag) so TMEM is never freed under an MMA.
      mma_commit_pair(smem_u32(&bars->drain), 1);
      if (!mbar_wait_cluster(smem_u32(&bars->drain), 0, nullptr, wait_ns)) fail(8u);
    }
  } else if (warp < kFirstEpi) {
    // ---------------- decoders ----------------
    // Group g decodes decoded stage g (K 128 g .. 128 g + 127) of every code
    // stage: A warps by warp index, B threads by warp and, in the shared
    // warp, by lane.
    const bool is_a = warp < kFirstDecB;
    const int dw = warp - (is_a ? kFirstDecA : kFirstDecB);
    int sub, rl;
    if (is_a) {
      sub = dw >> 2;
      rl = (warp & 3) * 32 + lane;  // rows follow the warp's TMEM lane quarter
    } else if (dw < kSub * Roles::kBFull) {
      sub = dw / Roles::kBFull;
      rl = (dw % Roles::kBFull) * 32 + lane;
    } else {
      sub = lane >> 4;
      rl = Roles::kBFull * 32 + (lane & 15);
    }
    const bool mixed = Roles::kBMixed && !is_a && dw >= kSub * Roles::kBFull;
    const uint32_t code_off = (is_a ? 0 : A_CODE_BYTES) + rl * (BKC / 2);
    const uint32_t scale_off =
        A_CODE_BYTES + B_CODE_BYTES + (is_a ? 0 : A_SCALE_BYTES) + rl * (BKC / 16) + sub * (BKD / 16);
    const uint32_t b_off = OFF_DEC + (rl >> 3) * kSBO + (rl & 7) * 16;
    const uint32_t a_lane = (uint32_t)((warp & 3) * 32) << 16;
    // 16-byte chunk c of the row sits at chunk c ^ (row % 8) (128-byte swizzle);
    // this thread's chunks are sub * 4 + j, j = 0..3.
    const uint32_t cswz = (uint32_t)(sub * kChunksPerSub) ^ (uint32_t)(rl & 7);
    int it = 0;
    bool ok = true;
    Sched sched(cluster_id, nclusters, dp_tiles, ntiles, num_kc, chunk_kc);
    int t, k0, k1;
    while (ok && sched.next(t, k0, k1)) {
      for (int kc = k0; kc < k1 && ok; ++kc, ++it) {
        const int s = it % kCodeStages;
        const uint32_t ph = (it / kCodeStages) & 1;
        if (!mbar_wait(smem_u32(&bars->code_full[s]), ph, abort_flag, wait_ns)) {
          fail(16u);
          ok = false;
          break;
        }
        const uint32_t st = sbase + s * CODE_STAGE_BYTES;
        const uint32_t crow = st + code_off;
        const uint2 sc = lds64(st + scale_off);  // this stage's 8 block scales of the row
        const int gstage = it * kSub + sub;
        const int d = gstage % kDecStages;
        const uint32_t dph = (uint32_t)(gstage / kDecStages) & 1u;
        uint4 c0 = lds128(crow + ((cswz ^ 0u) << 4)), c1 = lds128(crow + ((cswz ^ 1u) << 4));
        // The shared warp waits for both stages' slots (its lanes fill both).
        const int d_first = mixed ? (it * kSub) % kDecStages : d;
        const int d_last = mixed ? (it * kSub + kSub - 1) % kDecStages : d;
        const uint32_t ph_first = mixed ? (uint32_t)((it * kSub) / kDecStages) & 1u : dph;
        const uint32_t ph_last = mixed ? (uint32_t)((it * kSub + kSub - 1) / kDecStages) & 1u : dph;
        if (!mbar_wait_cluster(smem_u32(&bars->dec_empty[d_first]), ph_first ^ 1, abort_flag, wait_ns) ||
            (mixed && !mbar_wait_cluster(smem_u32(&bars->dec_empty[d_last]), ph_last ^ 1, abort_flag, wait_ns))) {
          fail(32u);
          ok = false;
          break;
        }
        if (is_a) {
          // 128 K of the row = 64 f16 pairs -> TMEM columns of stage d, 16
          // columns (one chunk) per store.
#pragma unroll
          for (int j = 0; j < kChunksPerSub; ++j) {
            const uint4 cj = j == 0 ? c0 : j == 1 ? c1 : lds128(crow + ((cswz ^ (uint32_t)j) << 4));
            const uint32_t sw = j < 2 ? sc.x : sc.y;
            uint32_t o[16];
            decode_chunk(cj, (j & 1) ? (sw >> 16) : (sw & 0xFFFFu), o);
            tmem_st_32x32b_x16(tmem_a0 + a_lane + (uint32_t)d * kAStageCols + (uint32_t)(16 * j), o);
          }
          tmem_st_wait();
          tc_fence_before();
        } else {
          const uint32_t dst = sbase + b_off + d * B_DEC_BYTES;
#pragma unroll
          for (int j = 0; j < kChunksPerSub; ++j) {
            const uint4 cj = j == 0 ? c0 : j == 1 ? c1 : lds128(crow + ((cswz ^ (uint32_t)j) << 4));
            const uint32_t sw = j < 2 ? sc.x : sc.y;
            uint32_t o[16];
            decode_chunk(cj, (j & 1) ? (sw >> 16) : (sw & 0xFFFFu), o);
#pragma unroll
            for (int q = 0; q < 4; ++q)
              sts128(dst + (j * 4 + q) * kLBO, o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]);
          }
          fence_proxy_async_smem();
        }
        __syncwarp();
        if (lane == 0) {
          // The leader's barrier, locally or through a remote arrival.
          const uint32_t full0 = mapa_shared(smem_u32(&bars->dec_full[0]), 0);
          mbar_arrive_cluster(full0 + 8u * (uint32_t)d_first);
          if (mixed) mbar_arrive_cluster(full0 + 8u * (uint32_t)d_last);
        }
        // Release the code stage only now: every value loaded from it has been
        // consumed (the decoded stores depend on it), so the TMA refill cannot
        // overtake a pending shared-memory load.
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&bars->code_empty[s]));
      }
    }
  } else {
    // ---------------- epilogue (two warps per TMEM lane quarter) ----------------
    // Each warp drains 32 rows x kTileN / 2 columns in 16-column steps:
    // tcgen05.ld (lane = row) -> scale -> its shared staging tile (row-major,
    // 64 bytes a row, 16-byte chunks XOR-swizzled by row: the 64-byte swizzle
    // of the tensor map of C) -> one TMA store (or TMA add) of the 32 x 16
    // box, which reads the tile and writes C asynchronously: the next step's
    // tcgen05.ld does not wait for the stores, so the accumulator is released
    // sooner and the C writes overlap the next tile's main loop.  Parts of a
    // box outside C are not written.  Without the tensor map (C or ldc not
    // 16-byte aligned) each lane stores its row's 16 values one by one.
    const int q = warp & 3;                  // TMEM lane quarter of this warp
    const int chalf = (warp - kFirstEpi) >> 2;  // column half
    griddep_wait();
    const float sa = 0.25f * __ldg(a_ts), sb = __ldg(b_ts);
    const u64 sa2 = pack2(sa, sa), sb2 = pack2(sb, sb);
    const uint32_t acc_empty_leader = mapa_shared(smem_u32(&bars->acc_empty), 0);
    // Staging tiles: the warp's own, and for tiles of at most 224 columns a
    // second one in the unused B rows 112-127 of a decoded-B stage (never
    // written by the decoders nor read by the MMA), so consecutive steps
    // alternate and a step's store need not finish reading before the next.
    constexpr bool kTwoStages = kBRows <= 112;
    const int ew = warp - kFirstEpi;
    const uint32_t stage0 = sbase + OFF_EPI + (uint32_t)ew * EPI_BYTES;
    const uint32_t stage1 = kTwoStages ? sbase + OFF_DEC + (uint32_t)(ew >> 1) * B_DEC_BYTES + 14u * kSBO +
                                             (uint32_t)(ew & 1) * EPI_BYTES
                                       : stage0;
    const uint32_t wr_off = (uint32_t)lane * 64u, wr_swz = (uint32_t)(lane >> 1) & 3u;
    Sched sched(cluster_id, nclusters, dp_tiles, ntiles, num_kc, chunk_kc);
    int t, k0, k1;
    for (int i = 0; sched.next(t, k0, k1); ++i) {
      // The first chunk of a whole tile is stored; every other segment is
      // added into C (after that chunk, or into rows the host zeroed).
      const bool whole = sched.store;
      // An add into C must follow the earlier segments' stores into the same
      // tile: bulk operations of different groups are not ordered, so wait
      // for their completion (issued a main loop ago, they are done).
      if (!whole && c_tma && lane == 0) bulk_wait_all();
      const bool acc_ok = mbar_wait_cluster(smem_u32(&bars->acc_full), i & 1, abort_flag, wait_ns);
      tc_fence_after();
      // tcgen05.ld is warp-collective: decide for the whole warp.
      const bool go = __all_sync(0xffffffffu, acc_ok && !*abort_flag);
      if (!go) {
        if (!acc_ok && !*abort_flag) fail(64u);
        break;
      }
      const int mt = t / ntiles_n, nt = t % ntiles_n;
      const int row0 = mt * TILE_M + (int)rank * BM + q * 32;
      const int n0 = nt * kTileN + chalf * kBRows;
      const uint32_t tbase = tmem_base + (uint32_t)(chalf * kBRows) + ((uint32_t)(q * 32) << 16);
#pragma unroll 1
      for (int cc = 0; cc < kBRows / EPI_CHUNK; ++cc) {
        uint32_t o[EPI_CHUNK];
        tmem_ld_32x32b_x16(tbase + (uint32_t)(cc * EPI_CHUNK), o);
        tmem_ld_wait_x16(o);
        if (cc == kBRows / EPI_CHUNK - 1) {
          // The accumulator is free once its last chunk sits in registers.
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_cluster(acc_empty_leader);
        }
#pragma unroll
        for (int k = 0; k < EPI_CHUNK; k += 2) {  // (acc x sa) x sb, two columns per instruction
          const u64 v = mul2(mul2(bits2(o[k], o[k + 1]), sa2), sb2);
          o[k] = (uint32_t)v;
          o[k + 1] = (uint32_t)(v >> 32);
        }
        const int col = n0 + cc * EPI_CHUNK;
        if (c_tma) {
          const uint32_t stage = (kTwoStages && (cc & 1)) ? stage1 : stage0;
          // The store that last used this staging tile must have read it.
          if (lane == 0) {
            if (kTwoStages) bulk_wait_read_one();
            else bulk_wait_read_all();
          }
          __syncwarp();
#pragma unroll
          for (int j = 0; j < 4; ++j)
            sts128(stage + wr_off + (((uint32_t)j ^ wr_swz) << 4), o[4 * j], o[4 * j + 1], o[4 * j + 2],
                   o[4 * j + 3]);
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            if (row0 < M && col < N) {  // boxes wholly outside C are skipped
              if (whole) tma_store_2d(&tm_c, stage, col, row0);
              else tma_reduce_add_2d(&tm_c, stage, col, row0);
            }
            bulk_commit_group();  // one group per step, empty or not: the waits count groups
          }
        } else if (row0 + lane < M) {
          float* crow = C + (long long)(row0 + lane) * ldc + col;
          for (int k = 0; k < EPI_CHUNK; ++k)
            if (col + k < N) {
              if (whole) crow[k] = __uint_as_float(o[k]);
              else atomicAdd(crow + k, __uint_as_float(o[k]));
            }
        }
      }
    }
    // The CTA's stores into C complete before it exits.
    if (c_tma && lane == 0) bulk_wait_all();
  }

  tc_fence_before();
  cluster_sync();  // both CTAs done with TMEM (and with each other's barriers)
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, kTmemCols);
  }
}

// ============================================================================
// Few-row path (M <= 64 activation rows, e.g. decoding).  A tcgen05.mma of
// M = 128, K = 16 costs a fixed ~65 ns whatever its N, so the weight rows go
// on the wide side: D[m][n] = sum_k X[m][k] W[n][k] with M_mma = 128 (the X
// rows, A operand decoded into TMEM; lanes past the X rows hold values that
// are never stored) and N_mma = 256 weight rows (B operand decoded into
// shared memory), cta_group::1.  Every weight element is decoded once.
// Work = (weight tile of 256 rows, 256-wide K slice) units split evenly over
// all CTAs (stream-K); each CTA adds its partial tiles into C (zeroed first)
// with red.global.add, so bits depend on the summation order but every result
// is within the fp32-accumulation bound.  A CTA's run of consecutive K slices
// of one weight tile is cut every `chunk_units` slices (2048 K), so no TMEM
// accumulation is longer than that (see the accumulation-length note at the
// top of this file).
// Per CTA: warp 0 TMA, warp 1 TMEM allocator + MMA thread, warps 2-17 weight
// decoders (two threads per weight row, one 32-code chunk each per stage),
// warps 18-25 X decoders (warp % 4 = TMEM lane quarter = 32 X rows; two warps
// per quarter, one chunk each per stage), warps 26-29 epilogue.
// ============================================================================
namespace skinny {

constexpr int BN = 256;                          // weight rows per tile (MMA N)
constexpr int MXMAX = 64;                        // max activation rows (MMA M is 128)
constexpr int BKC = 256, BKD = 64, kSub = BKC / BKD;
constexpr int kCodeStages = 2, kDecStages = 4;
constexpr int kWarpsW = 2 * BN / 32;             // 16
constexpr int kWarpsX = 8;                       // two per TMEM lane quarter: one chunk of a stage each
constexpr int kFirstW = 2, kFirstX = kFirstW + kWarpsW, kFirstEpi = kFirstX + kWarpsX;  // 2, 18, 26
constexpr int kEpiWarps = 4;
constexpr int kThreads = 32 * (kFirstEpi + kEpiWarps);  // 960
static_assert(kFirstX % 4 == 2 && kFirstEpi % 4 == 2, "warp w covers TMEM lane quarter w % 4");
constexpr int W_CODE = BN * BKC / 2, X_CODE = MXMAX * BKC / 2;
constexpr int W_SCALE = BN * BKC / 16, X_SCALE = MXMAX * BKC / 16;
constexpr int OFF_XC = W_CODE, OFF_WS = OFF_XC + X_CODE, OFF_XS = OFF_WS + W_SCALE;
constexpr int CODE_STAGE = OFF_XS + X_SCALE;
constexpr int W_DEC = BN * BKD * 2;
constexpr int OFF_DEC = kCodeStages * CODE_STAGE;
constexpr int OFF_BAR = OFF_DEC + kDecStages * W_DEC;
constexpr int SMEM_ALLOC = OFF_BAR + 256 + 1024;
static_assert(CODE_STAGE % 1024 == 0 && OFF_XC % 1024 == 0, "swizzled TMA tiles need 1024-byte alignment");
static_assert(SMEM_ALLOC <= 232448, "shared memory budget");
constexpr uint32_t kAccCols = BN;                // fp32 accumulator (lanes = X rows)
constexpr uint32_t kXStageCols = BKD / 2;        // f16 pairs per X row per stage
constexpr uint32_t kTmemCols = 512;
static_assert(kAccCols + kDecStages * kXStageCols <= kTmemCols, "TMEM budget");
constexpr uint32_t kLBO = 128, kSBO = (BKD / 8) * 128;  // decoded W: next 8 K / next 8 rows

struct Bars {
  uint64_t code_full[kCodeStages];
  uint64_t code_empty[kCodeStages];
  uint64_t dec_full[kDecStages];
  uint64_t dec_empty[kDecStages];
  uint64_t acc_full;
  uint64_t acc_empty;
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
};
static_assert(sizeof(Bars) <= 256, "barrier block");

__global__ void __launch_bounds__(kThreads, 1)
mixfp4_gemm_skinny_kernel(const __grid_constant__ CUtensorMap tm_wc, const __grid_constant__ CUtensorMap tm_xc,
                          const __grid_constant__ CUtensorMap tm_ws, const __grid_constant__ CUtensorMap tm_xs,
                          const float* __restrict__ a_ts, const float* __restrict__ b_ts, int Mx, int N, int K,
                          float* __restrict__ C, long long ldc, uint32_t idesc, int chunk_units,
                          uint32_t* status_word) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  Bars* bars = reinterpret_cast<Bars*>(smem + OFF_BAR);
  volatile int* abort_flag = &bars->abort;
  const uint32_t sbase = smem_u32(smem);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int num_kc = K / BKC;
  const int nx = (Mx + 15) & ~15;  // X rows fetched
  const long long units = (long long)((N + BN - 1) / BN) * num_kc;
  const long long u_begin = units * blockIdx.x / gridDim.x, u_end = units * (blockIdx.x + 1) / gridDim.x;
  const uint32_t stage_bytes = W_CODE + W_SCALE + (uint32_t)nx * (BKC / 2 + BKC / 16);
  // End of the accumulation run that starts at unit u: the end of its weight
  // tile, of this CTA's units, or of its accumulation chunk, whichever is first.
  auto run_end_of = [&](long long u) {
    long long e = (u / num_kc + 1) * num_kc;
    if (e > u_end) e = u_end;
    if (e > u + chunk_units) e = u + chunk_units;
    return e;
  };

  if (threadIdx.x == 0) {
    for (int s = 0; s < kCodeStages; ++s) {
      mbar_init(smem_u32(&bars->code_full[s]), 1);
      mbar_init(smem_u32(&bars->code_empty[s]), kWarpsW + kWarpsX);
    }
    for (int s = 0; s < kDecStages; ++s) {
      mbar_init(smem_u32(&bars->dec_full[s]), kWarpsW + kWarpsX);
      mbar_init(smem_u32(&bars->dec_empty[s]), 1);
    }
    mbar_init(smem_u32(&bars->acc_full), 1);
    mbar_init(smem_u32(&bars->acc_empty), kEpiWarps);
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
  const uint32_t tmem_base = bars->tmem_base;
  const uint32_t tmem_x0 = tmem_base + kAccCols;

  auto fail = [&](uint32_t code) {
    *abort_flag = 1;
    if (status_word) atomicOr(status_word, code);
  };

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      tma_prefetch(&tm_wc);
      tma_prefetch(&tm_xc);
      tma_prefetch(&tm_ws);
      tma_prefetch(&tm_xs);
      int it = 0;
      long long last = -1;
      for (long long u = u_begin; u < u_end; ++u, ++it) {
        const int s = it % kCodeStages;
        const uint32_t ph = (it / kCodeStages) & 1;
        if (!mbar_wait(smem_u32(&bars->code_empty[s]), ph ^ 1, abort_flag, kWaitLimitNs)) {
          fail(1u);
          break;
        }
        const int wt = (int)(u / num_kc), kc = (int)(u % num_kc);
        const uint32_t st = sbase + s * CODE_STAGE;
        const uint32_t fb = smem_u32(&bars->code_full[s]);
        mbar_arrive_expect_tx(fb, stage_bytes);
        const int xk = kc * (BKC / 2), xs = kc * (BKC / 16);
        tma_load_2d(st, &tm_wc, xk, wt * BN, fb);
        tma_load_2d(st + OFF_XC, &tm_xc, xk, 0, fb);
        tma_load_2d(st + OFF_WS, &tm_ws, xs, wt * BN, fb);
        tma_load_2d(st + OFF_XS, &tm_xs, xs, 0, fb);
        last = it;
      }
      if (*abort_flag)
        for (long long v = last - kCodeStages + 1; v <= last; ++v)
          if (v >= 0)
            mbar_wait(smem_u32(&bars->code_full[v % kCodeStages]), (uint32_t)((v / kCodeStages) & 1), nullptr,
                      kWaitLimitNs);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      int d = 0, ntile = 0;
      uint32_t dph = 0;
      bool ok = true;
      // Descriptor of decoded-W stage 0, first 16-K step; other stages and
      // steps only move the start address (14-bit field in 16-byte units, no
      // carry: shared addresses stay below 256 KiB).
      const uint64_t bdesc0 = smem_desc_noswizzle(sbase + OFF_DEC, kLBO, kSBO);
      for (long long u = u_begin; u < u_end && ok;) {
        const long long run_end = run_end_of(u);
        if (!mbar_wait(smem_u32(&bars->acc_empty), (ntile & 1) ^ 1, abort_flag, kWaitLimitNs)) {
          fail(2u);
          break;
        }
        tc_fence_after();
        bool first = true;
        for (; u < run_end && ok; ++u) {
          for (int sub = 0; sub < kSub; ++sub) {
            if (!mbar_wait(smem_u32(&bars->dec_full[d]), dph, abort_flag, kWaitLimitNs)) {
              fail(4u);
              ok = false;
              break;
            }
            tc_fence_after();
            const uint64_t bd = bdesc0 + (uint64_t)((d * W_DEC) >> 4);
            const uint32_t xa = tmem_x0 + (uint32_t)d * kXStageCols;
            mma_f16_tmem_a(tmem_base, xa, bd, idesc, first ? 0u : 1u);
            first = false;
#pragma unroll
            for (int j = 1; j < BKD / 16; ++j) mma_f16_tmem_a(tmem_base, xa + j * 8, bd + (uint64_t)(j * 16), idesc, 1u);
            mma_commit(smem_u32(&bars->dec_empty[d]));
            if (++d == kDecStages) { d = 0; dph ^= 1; }
          }
        }
        if (ok) mma_commit(smem_u32(&bars->acc_full));
        ++ntile;
      }
      mma_commit(smem_u32(&bars->drain));
      if (!mbar_wait(smem_u32(&bars->drain), 0, nullptr, kWaitLimitNs)) fail(8u);
    }
  } else if (warp < kFirstEpi) {
    // ---------------- decoders ----------------
    const bool is_w = warp < kFirstX;
    // W: row = (dw % 8) * 32 + lane, chunk part = dw / 8 of each 64-K stage.
    // X: row = (warp % 4) * 32 + lane = its TMEM lane, chunk part = (warp - 18) / 4.
    const int dw = warp - kFirstW;
    const int row = is_w ? ((dw & 7) * 32 + lane) : ((warp & 3) * 32 + lane);
    const int part = is_w ? (dw >> 3) : ((warp - kFirstX) >> 2);
    const bool active = is_w || (warp & 3) * 32 < nx;  // X warps past the fetched rows idle
    const uint32_t code_row = (is_w ? 0u : (uint32_t)OFF_XC) + (uint32_t)row * (BKC / 2);
    const uint32_t scale_row = (is_w ? (uint32_t)OFF_WS : (uint32_t)OFF_XS) + (uint32_t)row * (BKC / 16);
    const uint32_t w_dst = OFF_DEC + (uint32_t)(row >> 3) * kSBO + (uint32_t)(row & 7) * 16;
    const uint32_t x_lane = (uint32_t)((warp & 3) * 32) << 16;
    const uint32_t swz = (uint32_t)(row & 7);
    int d = 0, it = 0;
    uint32_t dph = 0;
    for (long long u = u_begin; u < u_end; ++u, ++it) {
      const int s = it % kCodeStages;
      const uint32_t ph = (it / kCodeStages) & 1;
      if (!mbar_wait(smem_u32(&bars->code_full[s]), ph, abort_flag, kWaitLimitNs)) {
        fail(16u);
        break;
      }
      const uint32_t st = sbase + s * CODE_STAGE;
      uint4 sc = make_uint4(0, 0, 0, 0);  // the row's 16 block scales of this K slice
      if (active) sc = lds128(st + scale_row);
      bool ok = true;
#pragma unroll
      for (int sub = 0; sub < kSub; ++sub) {
        uint4 c[2];
        if (active) {
          c[0] = lds128(st + code_row + ((((uint32_t)(sub * 2 + part)) ^ swz) << 4));
        }
        if (!mbar_wait(smem_u32(&bars->dec_empty[d]), dph ^ 1, abort_flag, kWaitLimitNs)) {
          fail(32u);
          ok = false;
          break;
        }
        if (is_w) {
          uint32_t o[16];
          decode_chunk(c[0], scale_pair(sc, sub * 2 + part), o);
          const uint32_t dst = sbase + w_dst + (uint32_t)d * W_DEC;
#pragma unroll
          for (int q = 0; q < 4; ++q)
            sts128(dst + (uint32_t)(part * 4 + q) * kLBO, o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]);
          fence_proxy_async_smem();
        } else if (active) {
          uint32_t o[16];
          decode_chunk(c[0], scale_pair(sc, sub * 2 + part), o);
          tmem_st_32x32b_x16(tmem_x0 + x_lane + (uint32_t)d * kXStageCols + (uint32_t)(16 * part), o);
          tmem_st_wait();
          tc_fence_before();
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&bars->dec_full[d]));
        if (++d == kDecStages) { d = 0; dph ^= 1; }
        if (sub == kSub - 1) {
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&bars->code_empty[s]));
        }
      }
      if (!ok) break;
    }
  } else {
    // ---------------- epilogue: lane = X row m, 256 weight columns -> red.add into C ----------------
    const int q = warp & 3;
    const int m = q * 32 + lane;
    const float sa = 0.25f * __ldg(a_ts), sb = __ldg(b_ts);
    const bool vec_ok = ((ldc & 3) == 0) && ((reinterpret_cast<uintptr_t>(C) & 15) == 0);
    const bool mine = q * 32 < Mx;  // warps whose lane quarter holds X rows
    int ntile = 0;
    for (long long u = u_begin; u < u_end; ++ntile) {
      const int wt = (int)(u / num_kc);
      u = run_end_of(u);
      const bool acc_ok = mbar_wait(smem_u32(&bars->acc_full), ntile & 1, abort_flag, kWaitLimitNs);
      tc_fence_after();
      const bool go = __all_sync(0xffffffffu, acc_ok && !*abort_flag);
      if (!go) {
        if (!acc_ok && !*abort_flag) fail(64u);
        break;
      }
      const uint32_t tb = tmem_base + ((uint32_t)(q * 32) << 16);
#pragma unroll 1
      for (int cc = 0; cc < BN / 32; ++cc) {
        uint32_t v[32];
        if (mine) {
          tmem_ld_32x32b_x32(tb + (uint32_t)(cc * 32), v);
          tmem_ld_wait_x32(v);
        }
        if (cc == BN / 32 - 1) {
          // The accumulator is free once its last chunk sits in registers.
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&bars->acc_empty));
        }
        const int n0 = wt * BN + cc * 32;
        if (mine && m < Mx) {
          float* crow = C + (long long)m * ldc + n0;
          if (vec_ok && n0 + 32 <= N) {
#pragma unroll
            for (int k = 0; k < 32; k += 4)
              red_add_v4(crow + k, __fmul_rn(__fmul_rn(__uint_as_float(v[k]), sa), sb),
                         __fmul_rn(__fmul_rn(__uint_as_float(v[k + 1]), sa), sb),
                         __fmul_rn(__fmul_rn(__uint_as_float(v[k + 2]), sa), sb),
                         __fmul_rn(__fmul_rn(__uint_as_float(v[k + 3]), sa), sb));
          } else {
            for (int k = 0; k < 32; ++k)
              if (n0 + k < N) atomicAdd(crow + k, __fmul_rn(__fmul_rn(__uint_as_float(v[k]), sa), sb));
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

}  // namespace skinny


}  // namespace

// Launch the pair kernel with tile width kTileN over `tiles` tiles, the first
// dp_tiles whole and the rest split into K slices (stream-K).
template <int kTileN>
int launch_pair(const uint8_t* a_codes, const uint8_t* a_scales, const float* a_ts, const uint8_t* b_codes,
                const uint8_t* b_scales, const float* b_ts, int64_t M, int64_t N, int64_t K, float* C, int64_t ldc,
                uint32_t* status_word, int64_t clusters, int64_t tiles, int64_t dp_tiles, cudaStream_t stream,
                uint64_t wait_ns = kWaitLimitNs, int skip_first_stage = 0) {
  CUtensorMap tac, tbc, tas, tbs;
  if (!make_map(&tac, a_codes, (uint64_t)K / 2, (uint64_t)M, BKC / 2, BM, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_map(&tbc, b_codes, (uint64_t)K / 2, (uint64_t)N, BKC / 2, kTileN / 2, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_map(&tas, a_scales, (uint64_t)K / 16, (uint64_t)M, BKC / 16, BM, CU_TENSOR_MAP_SWIZZLE_NONE) ||
      !make_map(&tbs, b_scales, (uint64_t)K / 16, (uint64_t)N, BKC / 16, kTileN / 2, CU_TENSOR_MAP_SWIZZLE_NONE))
    return MIXFP4_ERR_CUDA;
  // C by TMA stores: 32 x 16 fp32 boxes, 64-byte swizzle (the staging tiles'
  // layout), when C and its row stride are 16-byte aligned.
  CUtensorMap tmc;
  memset(&tmc, 0, sizeof(tmc));
  const int c_tma = ((ldc & 3) == 0) && ((reinterpret_cast<uintptr_t>(C) & 15) == 0);
  if (c_tma && !make_map_f32(&tmc, C, (uint64_t)N, (uint64_t)M, (uint64_t)ldc, EPI_CHUNK, 32,
                             CU_TENSOR_MAP_SWIZZLE_64B))
    return MIXFP4_ERR_CUDA;
  static std::atomic<uint64_t> smem_set{0};
  if (!set_dynamic_smem_once(reinterpret_cast<const void*>(mixfp4_gemm_kernel<kTileN>), SMEM_ALLOC, smem_set))
    return MIXFP4_ERR_CUDA;
  const int64_t ntiles_n = (N + kTileN - 1) / kTileN;
  if (dp_tiles < tiles) {
    // Zero C from the first stream-K tile's row band down (tile t: mt = t / ntiles_n,
    // nt = t % ntiles_n, so those rows hold every stream-K tile; whole tiles among
    // them are overwritten by plain stores after this).
    const int64_t r0 = (dp_tiles / ntiles_n) * TILE_M;
    cudaError_t e;
    if (ldc == N)
      e = cudaMemsetAsync(C + r0 * ldc, 0, (size_t)(M - r0) * (size_t)N * sizeof(float), stream);
    else
      e = cudaMemset2DAsync(C + r0 * ldc, (size_t)ldc * sizeof(float), 0, (size_t)N * sizeof(float),
                            (size_t)(M - r0), stream);
    if (e != cudaSuccess) return MIXFP4_ERR_CUDA;
  }
  // A programmatic dependent: barrier set-up and TMEM allocation overlap the
  // tail of the kernel before it; the TMA producer and the epilogue wait for
  // that kernel before they read the operands or the tensor scales.
  if (launch_pdl(mixfp4_gemm_kernel<kTileN>, (unsigned)(2 * clusters), PairRoles<kTileN>::kThreads, SMEM_ALLOC, stream,
                 tac, tbc, tas, tbs, tmc, c_tma, a_ts, b_ts, (int)M, (int)N, (int)K, C, (long long)ldc,
                 (int)dp_tiles, kAccumChunkK / BKC, status_word, wait_ns, skip_first_stage) != cudaSuccess)
    return MIXFP4_ERR_CUDA;
  return MIXFP4_OK;
}

// The pair kernel on 256-wide tiles with every pipeline wait limited to
// wait_ns and the first code stage of every CTA never issued: each CTA's
// waits on that stage run out, its status bits are set and it exits (the
// self-test of the failure path; C is not written).
int launch_gemm_missed_stage_selftest(const uint8_t* a_codes, const uint8_t* a_scales, const float* a_ts,
                                      const uint8_t* b_codes, const uint8_t* b_scales, const float* b_ts, int64_t M,
                                      int64_t N, int64_t K, float* C, int64_t ldc, uint32_t* status_word,
                                      uint64_t wait_ns, cudaStream_t stream) {
  const int64_t tiles = ((M + TILE_M - 1) / TILE_M) * ((N + 255) / 256);
  int64_t clusters = num_sms() / 2;
  if (clusters > tiles) clusters = tiles;
  return launch_pair<256>(a_codes, a_scales, a_ts, b_codes, b_scales, b_ts, M, N, K, C, ldc, status_word, clusters,
                          tiles, tiles, stream, wait_ns, 1);
}

int launch_gemm(const uint8_t* a_codes, const uint8_t* a_scales, const float* a_ts,
                const uint8_t* b_codes, const uint8_t* b_scales, const float* b_ts, int64_t M,
                int64_t N, int64_t K, float* C, int64_t ldc, uint32_t* status_word,
                cudaStream_t stream) {
  if (M > (1 << 30) || N > (1 << 30) || K > (1 << 30)) return MIXFP4_ERR_SHAPE;
  if (M <= skinny::MXMAX && N >= 2 * skinny::BN) {
    // Few activation rows: weight rows on the wide MMA N side, stream-K over all SMs.
    const int nx = (int)((M + 15) & ~15);
    CUtensorMap twc, txc, tws, txs;
    if (!make_map(&twc, b_codes, (uint64_t)K / 2, (uint64_t)N, BKC / 2, skinny::BN, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&txc, a_codes, (uint64_t)K / 2, (uint64_t)M, BKC / 2, nx, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&tws, b_scales, (uint64_t)K / 16, (uint64_t)N, BKC / 16, skinny::BN, CU_TENSOR_MAP_SWIZZLE_NONE) ||
        !make_map(&txs, a_scales, (uint64_t)K / 16, (uint64_t)M, BKC / 16, nx, CU_TENSOR_MAP_SWIZZLE_NONE))
      return MIXFP4_ERR_CUDA;
    static std::atomic<uint64_t> skinny_smem_set{0};
    if (!set_dynamic_smem_once(reinterpret_cast<const void*>(skinny::mixfp4_gemm_skinny_kernel), skinny::SMEM_ALLOC,
                               skinny_smem_set))
      return MIXFP4_ERR_CUDA;
    if (cudaMemset2DAsync(C, (size_t)ldc * sizeof(float), 0, (size_t)N * sizeof(float), (size_t)M, stream) !=
        cudaSuccess)
      return MIXFP4_ERR_CUDA;
    const int64_t units = ((N + skinny::BN - 1) / skinny::BN) * (K / BKC);
    int64_t grid = num_sms();
    if (grid > units) grid = units;
    skinny::mixfp4_gemm_skinny_kernel<<<(unsigned)grid, skinny::kThreads, skinny::SMEM_ALLOC, stream>>>(
        twc, txc, tws, txs, a_ts, b_ts, (int)M, (int)N, (int)K, C, (long long)ldc,
        idesc_f16_f32(128, skinny::BN), kAccumChunkK / skinny::BKC, status_word);
    return MIXFP4_OK;
  }
  // Tile width: the pair tiles are 256 rows of A by kTileN rows of B.  With
  // few tiles per pair a narrower tile can remove a partly idle last wave;
  // the main loop is bound by decoding A and B (256 + kTileN rows per K
  // step), so the cost of a width is waves * (256 + kTileN).  Stream-K (for
  // 256) is preferred when it applies.
  const int64_t mtiles = (M + TILE_M - 1) / TILE_M, num_kc = K / BKC;
  auto waves = [&](int64_t n, int64_t* tiles_out, int64_t* clusters_out) {
    const int64_t t = mtiles * ((N + n - 1) / n);
    int64_t c = num_sms() / 2;
    if (c > t) c = t;
    *tiles_out = t;
    *clusters_out = c;
    return (t + c - 1) / c;
  };
  int64_t tiles, clusters;
  const int64_t w256 = waves(256, &tiles, &clusters);
  // Whole tiles in full waves.  The last, partial wave's tiles are shared out
  // as K slices (stream-K) when the idle time that removes, (clusters - rem)
  // tiles' worth of K slices spread over all pairs, outweighs what stream-K
  // adds: zeroing those rows of C and one more accumulator drain per pair.
  int64_t dp_tiles = tiles;
  const int64_t rem = tiles % clusters;
  if (tiles > clusters && rem != 0 && (clusters - rem) * num_kc >= kMinStreamKGainSlices * clusters)
    dp_tiles = tiles - rem;
  int tile_n = 256;
  if (dp_tiles == tiles) {
    int64_t best = w256 * (256 + 256);
    for (int n : {224, 192}) {
      int64_t t, c;
      const int64_t cost = waves(n, &t, &c) * (256 + n);
      if (cost < best) {
        best = cost;
        tile_n = n;
        tiles = t;
        clusters = c;
        dp_tiles = t;
      }
    }
  }
  switch (tile_n) {
    case 224:
      return launch_pair<224>(a_codes, a_scales, a_ts, b_codes, b_scales, b_ts, M, N, K, C, ldc, status_word,
                              clusters, tiles, dp_tiles, stream);
    case 192:
      return launch_pair<192>(a_codes, a_scales, a_ts, b_codes, b_scales, b_ts, M, N, K, C, ldc, status_word,
                              clusters, tiles, dp_tiles, stream);
    default:
      return launch_pair<256>(a_codes, a_scales, a_ts, b_codes, b_scales, b_ts, M, N, K, C, ldc, status_word,
                              clusters, tiles, dp_tiles, stream);
  }
}

}  // namespace mixfp4
