// Quantizer orientations of the MixFP4 training flow (Sec. 3.2: FPROP, DGRAD
// and WGRAD all run on MixFP4 operands; weights use 2D blocks) for sm_103a.
//
//   quantize_colwise_kernel  Algorithm 1 with each 16-element block running
//       down a column of an [R][C] bf16 tensor: the operand of a GEMM that
//       reduces over R (WGRAD reduces over tokens).  Output as the row-wise
//       quantization of the transpose: codes [C][R/2], scales [C][R/16].
//       A CTA stages a 64-row x 256-column tile in shared memory with
//       coalesced 16-byte loads; thread t then owns column t, reads its four
//       16-row blocks (2-byte shared loads, consecutive threads on consecutive
//       columns, no bank conflicts) and writes 32 contiguous code bytes.
//   quantize_2d_kernel  Algorithm 1 with 16 x 16 blocks (reading R12): a
//       half-warp holds one tile, lane i one 16-element row of it, so the
//       tile max and the tree of the rows' error sums are warp shuffles
//       (block_core<kMode, true>); the two half-warps of a warp take
//       horizontally adjacent tiles (64 contiguous bytes per row).  Output in
//       the row-wise layout, every row of a tile repeating its scale byte, so
//       mixfp4_gemm consumes it unchanged.
//   quantize_sr_kernel  row-wise quantization with stochastic rounding of the
//       chosen format's codes (reading R13, the gradients of the training
//       flow); quantize_colwise_kernel<.., true> the same down the columns.
//   quantize_colwise_rht_kernel  the column-wise quantizer with the 128-point
//       rotation applied along the rows first (the WGRAD inputs).
//   transpose_2d_kernel  codes and tile scales of the transpose of a
//       2D-quantized tensor (the DGRAD operand of the weights): each lane
//       transposes a 16 x 16 nibble tile in registers.
// Every kernel shares quantize.cu's per-block arithmetic (quant_core.cuh), so
// its codes are those of Algorithm 1 on the same values bit for bit.
#include <cuda_runtime.h>
#include <cstdint>

#include "host_util.cuh"
#include "kernels.cuh"
#include "ptx.cuh"
#include "quant_core.cuh"

namespace mixfp4 {
namespace {

constexpr int kColThreads = 256;        // columns per tile
constexpr int kColRows = 64;            // rows per tile (four 16-row blocks)

template <int kMode, bool kSR>
__global__ void __launch_bounds__(kColThreads, kSR ? 3 : 4)
quantize_colwise_kernel(const uint16_t* __restrict__ x, int64_t R, int64_t C, int64_t ldx,
                        uint8_t* __restrict__ codes, uint8_t* __restrict__ scales, float* tensor_scale,
                        const uint32_t* amax_word, int scale_given, uint64_t seed, uint64_t offset) {
  __shared__ float4 tab[128];
  // Row pairs interleaved: pairs[p][c] = x[2p][c] | x[2p + 1][c] << 16, the
  // bf16 pair of column c that quantize_block takes as one word.
  __shared__ __align__(16) uint32_t pairs[kColRows / 2][kColThreads];
  griddep_wait();
  griddep_launch_dependents();
  fill_scale_table(tab);
  const TensorConsts tc = tensor_consts(tensor_scale, amax_word, scale_given);
  const bool markstein = markstein_needed(tc);
  const int tid = threadIdx.x;
  const int64_t ct_n = (C + kColThreads - 1) / kColThreads, rt_n = (R + kColRows - 1) / kColRows;
  const int64_t nblk_t = R / 16;  // blocks per output row
  // One 32-byte code store and one 4-byte scale store per full tile column
  // when every output row starts aligned for them (R a multiple of 64).
  const bool vec = (R % kColRows) == 0 && (reinterpret_cast<uintptr_t>(codes) & 31) == 0 &&
                   (reinterpret_cast<uintptr_t>(scales) & 3) == 0;
  for (int64_t t = blockIdx.x; t < ct_n * rt_n; t += gridDim.x) {
    const int64_t r0 = (t / ct_n) * kColRows, c0 = (t % ct_n) * kColThreads;
    // Stage the tile: 32 row pairs x 32 chunks of 8 columns; a thread loads
    // the chunk from both rows of a pair (two 16-byte loads) and stores the
    // eight interleaved words (two 16-byte stores).
#pragma unroll
    for (int k = 0; k < (kColRows / 2) * (kColThreads / 8) / kColThreads; ++k) {
      const int q = tid + k * kColThreads;
      const int pr = q / (kColThreads / 8), ch = q % (kColThreads / 8);
      uint4 a = make_uint4(0u, 0u, 0u, 0u), b = a;
      if (r0 + 2 * pr < R && c0 + ch * 8 < C) {
        a = __ldg(reinterpret_cast<const uint4*>(x + (r0 + 2 * pr) * ldx + c0 + ch * 8));
        b = __ldg(reinterpret_cast<const uint4*>(x + (r0 + 2 * pr + 1) * ldx + c0 + ch * 8));
      }
      uint4* dst = reinterpret_cast<uint4*>(&pairs[pr][ch * 8]);
      dst[0] = make_uint4(prmt(a.x, b.x, 0x5410u), prmt(a.x, b.x, 0x7632u), prmt(a.y, b.y, 0x5410u),
                          prmt(a.y, b.y, 0x7632u));
      dst[1] = make_uint4(prmt(a.z, b.z, 0x5410u), prmt(a.z, b.z, 0x7632u), prmt(a.w, b.w, 0x5410u),
                          prmt(a.w, b.w, 0x7632u));
    }
    __syncthreads();
    const int64_t c = c0 + tid;
    if (c < C) {
      // The four row blocks of column c are 32 contiguous code bytes (and 4
      // scale bytes) of output row c: gathered here, stored once.
      uint32_t out[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u}, sc4 = 0u;
      const int nrb = (int)((R - r0) / 16 < kColRows / 16 ? (R - r0) / 16 : kColRows / 16);
#pragma unroll
      for (int rb = 0; rb < kColRows / 16; ++rb) {
        if (rb >= nrb) break;
        uint32_t w[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) w[j] = pairs[rb * 8 + j][tid];
        uint32_t lo, hi, sb;
        const int64_t ob = r0 / 16 + rb;  // block index along R
        if (kSR) {
          const uint64_t e0 = (uint64_t)c * (uint64_t)R + (uint64_t)ob * 16;  // element index in X^T
          if (tc.scaled) quantize_block_sr<kMode, true, true>(w, tc, tab, seed, offset, e0, lo, hi, sb);
          else if (markstein) quantize_block_sr<kMode, false, true>(w, tc, tab, seed, offset, e0, lo, hi, sb);
          else quantize_block_sr<kMode, false, false>(w, tc, tab, seed, offset, e0, lo, hi, sb);
        } else {
          if (tc.scaled) quantize_block<kMode, true, true>(w, tc, tab, lo, hi, sb);
          else if (markstein) quantize_block<kMode, false, true>(w, tc, tab, lo, hi, sb);
          else quantize_block<kMode, false, false>(w, tc, tab, lo, hi, sb);
        }
        out[2 * rb] = lo;
        out[2 * rb + 1] = hi;
        sc4 |= sb << (8 * rb);
      }
      uint8_t* cdst = codes + c * (R / 2) + (r0 / 16) * 8;
      uint8_t* sdst = scales + c * nblk_t + r0 / 16;
      if (vec && nrb == kColRows / 16) {
        stg256(cdst, out);
        *reinterpret_cast<uint32_t*>(sdst) = sc4;
      } else {
#pragma unroll
        for (int rb = 0; rb < kColRows / 16; ++rb) {
          if (rb < nrb) {
            stg64(cdst + rb * 8, out[2 * rb], out[2 * rb + 1]);
            sdst[rb] = (uint8_t)(sc4 >> (8 * rb));
          }
        }
      }
    }
    __syncthreads();  // the tile is restaged next
  }
}

// Grid-stride loop of the stochastic-rounding quantizer with the division
// method fixed; the next block's load is in flight while a block is quantized.
template <int kMode, bool kContig, bool kScaled, bool kMarkstein>
__device__ __forceinline__ void sr_loop(const uint16_t* __restrict__ x, int64_t b, int64_t nthr, int64_t nblocks,
                                        int64_t kblocks, int64_t ldx, uint8_t* __restrict__ codes,
                                        uint8_t* __restrict__ scales, const TensorConsts& tc,
                                        const float4* __restrict__ tab, uint64_t seed, uint64_t offset) {
  uint32_t w[8];
  if (b < nblocks) ldg256_stream(block_src<kContig>(x, b, kblocks, ldx), w);
  for (; b < nblocks; b += nthr) {
    uint32_t wn[8];
    if (b + nthr < nblocks) ldg256_stream(block_src<kContig>(x, b + nthr, kblocks, ldx), wn);
    uint32_t lo, hi, sb;
    quantize_block_sr<kMode, kScaled, kMarkstein>(w, tc, tab, seed, offset, (uint64_t)b * 16, lo, hi, sb);
    stg64(codes + b * 8, lo, hi);
    scales[b] = (uint8_t)sb;
#pragma unroll
    for (int j = 0; j < 8; ++j) w[j] = wn[j];
  }
}

// Row-wise quantization with stochastic rounding (R13): one thread per
// 16-element block, grid-stride; the element index of block b's first element
// is 16 b (row-major over [rows][K]).
template <int kMode, bool kContig>
__global__ void __launch_bounds__(256, 3)
quantize_sr_kernel(const uint16_t* __restrict__ x, int64_t nblocks, int64_t kblocks, int64_t ldx,
                   uint8_t* __restrict__ codes, uint8_t* __restrict__ scales, float* tensor_scale,
                   const uint32_t* amax_word, int scale_given, uint64_t seed, uint64_t offset) {
  __shared__ float4 tab[128];
  griddep_wait();
  griddep_launch_dependents();
  fill_scale_table(tab);
  const TensorConsts tc = tensor_consts(tensor_scale, amax_word, scale_given);
  const bool markstein = markstein_needed(tc);
  const int64_t nthr = (int64_t)gridDim.x * blockDim.x;
  const int64_t b0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (tc.scaled) sr_loop<kMode, kContig, true, true>(x, b0, nthr, nblocks, kblocks, ldx, codes, scales, tc, tab, seed, offset);
  else if (markstein) sr_loop<kMode, kContig, false, true>(x, b0, nthr, nblocks, kblocks, ldx, codes, scales, tc, tab, seed, offset);
  else sr_loop<kMode, kContig, false, false>(x, b0, nthr, nblocks, kblocks, ldx, codes, scales, tc, tab, seed, offset);
}

constexpr int k2dThreads = 256;

template <int kMode>
__global__ void __launch_bounds__(k2dThreads, 4)
quantize_2d_kernel(const uint16_t* __restrict__ x, int64_t rows, int64_t K, int64_t ldx,
                   uint8_t* __restrict__ codes, uint8_t* __restrict__ scales, float* tensor_scale,
                   const uint32_t* amax_word, int scale_given) {
  __shared__ float4 tab[128];
  griddep_wait();
  griddep_launch_dependents();
  fill_scale_table(tab);
  const TensorConsts tc = tensor_consts(tensor_scale, amax_word, scale_given);
  const bool markstein = markstein_needed(tc);
  const int lane = threadIdx.x & 31, i = lane & 15, h = lane >> 4;
  const int64_t nb = K / 16, pairs = (nb + 1) / 2, rt_n = (rows + 15) / 16;
  const int64_t units = rt_n * pairs;  // (row tile, pair of block columns), one per warp
  const int64_t warp0 = ((int64_t)blockIdx.x * k2dThreads + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * k2dThreads) >> 5;
  for (int64_t u = warp0; u < units; u += nwarps) {
    const int64_t r = (u / pairs) * 16 + i, b = (u % pairs) * 2 + h;
    const bool live = r < rows && b < nb;
    uint32_t w[8];
    if (live) {
      ldg256_stream(x + r * ldx + b * 16, w);
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j) w[j] = 0u;  // missing rows of a ragged tile count as zeros (R12)
    }
    uint32_t lo, hi, sb;
    if (tc.scaled) quantize_block<kMode, true, true, true>(w, tc, tab, lo, hi, sb);
    else if (markstein) quantize_block<kMode, false, true, true>(w, tc, tab, lo, hi, sb);
    else quantize_block<kMode, false, false, true>(w, tc, tab, lo, hi, sb);
    if (live) {
      stg64(codes + r * (K / 2) + b * 8, lo, hi);
      scales[r * nb + b] = (uint8_t)sb;
    }
  }
}

// Column-wise quantization with the 128-point rotation along the rows (the
// weight-gradient inputs of the training recipe, Sec. 3.2 / Sec. 4.2: the RHT
// is applied to both WGRAD operands, whose reduction runs over tokens): every
// 128-row chunk of each column is rotated (reading R11: the caller's sign
// vector, the same butterfly order) and the rotated column is quantized down
// its rows -- bit for bit mixfp4_quantize_rht of X^T.  A CTA stages a
// 128-row x 64-column tile TRANSPOSED in shared memory (a column's 128 values
// contiguous, 272-byte pitch): each warp loads 8 columns of 32 consecutive
// rows (16-byte loads) and scatters them with 2-byte stores that are
// consecutive within the warp.  Then each 8-lane group holds one column chunk
// (lane b: rows 16b..16b+15, one 32-byte shared read) and rotates it with the
// row-wise kernel's shuffle butterfly.  kAmax: the pass that reduces max |y|
// of the rotated tensor into the workspace word instead of quantizing.
constexpr int kCrRows = 128, kCrCols = 64, kCrPitch = kCrRows + 8;  // staged column pitch (u16)

template <int kMode, bool kAmax>
__global__ void __launch_bounds__(256, 3)
quantize_colwise_rht_kernel(const uint16_t* __restrict__ x, int64_t R, int64_t C, int64_t ldx,
                            const uint8_t* __restrict__ signs, uint8_t* __restrict__ codes,
                            uint8_t* __restrict__ scales, float* tensor_scale, uint32_t* amax_word, int scale_given) {
  __shared__ float4 tab[128];
  __shared__ __align__(16) uint16_t tile[kCrCols][kCrPitch];
  griddep_wait();
  griddep_launch_dependents();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint32_t sw[8];
  rht_sign_words(signs, lane, sw);  // lane & 7 = the block of the chunk this lane holds
  TensorConsts tc{};
  if (!kAmax) {
    fill_scale_table(tab);
    tc = tensor_consts(tensor_scale, amax_word, scale_given);
  }
  uint32_t m = 0;
  const int64_t ct_n = (C + kCrCols - 1) / kCrCols, rt_n = R / kCrRows;
  for (int64_t t = blockIdx.x; t < ct_n * rt_n; t += gridDim.x) {
    const int64_t r0 = (t / ct_n) * kCrRows, c0 = (t % ct_n) * kCrCols;
    // Stage: chunk q = (8 columns from 8 cg, row q % 128).
#pragma unroll
    for (int k = 0; k < kCrRows * kCrCols / 8 / 256; ++k) {
      const int q = tid + 256 * k, row = q & (kCrRows - 1), cg = q >> 7;
      uint4 v = make_uint4(0u, 0u, 0u, 0u);
      if (c0 + cg * 8 < C) v = __ldg(reinterpret_cast<const uint4*>(x + (r0 + row) * ldx + c0 + cg * 8));
      const uint32_t e[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        tile[cg * 8 + 2 * i][row] = (uint16_t)(e[i] & 0xFFFFu);
        tile[cg * 8 + 2 * i + 1][row] = (uint16_t)(e[i] >> 16);
      }
    }
    __syncthreads();
#pragma unroll 1
    for (int pass = 0; pass < kCrCols / 32; ++pass) {
      const int cl = pass * 32 + warp * 4 + (lane >> 3), b = lane & 7;
      const int64_t c = c0 + cl;
      const uint4 lo4 = *reinterpret_cast<const uint4*>(&tile[cl][16 * b]);
      const uint4 hi4 = *reinterpret_cast<const uint4*>(&tile[cl][16 * b + 8]);
      const uint32_t w[8] = {lo4.x, lo4.y, lo4.z, lo4.w, hi4.x, hi4.y, hi4.z, hi4.w};
      u64 y[8];
      rht_rotate(w, sw, lane, y);  // all 32 lanes: shuffles within 8-lane groups
      if (kAmax) {
#pragma unroll
        for (int j = 0; j < 8; ++j) m = max(m, max(lo32(y[j]) & 0x7FFFFFFFu, hi32(y[j]) & 0x7FFFFFFFu));
      } else {
        uint32_t lo, hi, sb;
        if (tc.scaled) rht_block<kMode, true>(y, tc, tab, lo, hi, sb);
        else rht_block<kMode, false>(y, tc, tab, lo, hi, sb);
        if (c < C) {
          const int64_t ob = r0 / 16 + b;
          stg64(codes + c * (R / 2) + ob * 8, lo, hi);
          scales[c * (R / 16) + ob] = (uint8_t)sb;
        }
      }
    }
    __syncthreads();  // the tile is restaged next
  }
  if (kAmax) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = max(m, __shfl_xor_sync(0xffffffffu, m, o));
    __shared__ uint32_t red[8];
    if (lane == 0) red[warp] = m;
    __syncthreads();
    if (tid == 0) {
      for (int i = 1; i < 8; ++i) m = max(m, red[i]);
      if (m) atomicMax(amax_word, m);
    }
  }
}

// Transpose of a 16 x 16 nibble tile held in registers: row i of the tile is
// lo[i] (elements 0..7, element e at bits 4e) and hi[i] (elements 8..15); on
// return lo[c] / hi[c] hold column c (tile rows 0..7 / 8..15), packed the same
// way.  Block-recursive: swap the off-diagonal 8 x 8 blocks (register
// renaming), then within every 8 x 8 block the 4 x 4 blocks (16-bit fields),
// the 2 x 2 blocks (bytes) and the single nibbles.
__device__ __forceinline__ void transpose_nibbles16(uint32_t lo[16], uint32_t hi[16]) {
#pragma unroll
  for (int r = 0; r < 8; ++r) {
    const uint32_t t = lo[r + 8];
    lo[r + 8] = hi[r];
    hi[r] = t;
  }
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    uint32_t* w = h ? hi : lo;
#pragma unroll
    for (int r = 0; r < 16; ++r)
      if ((r & 7) < 4) {
        const uint32_t x = w[r], y = w[r + 4];
        w[r] = prmt(x, y, 0x5410u);
        w[r + 4] = prmt(x, y, 0x7632u);
      }
#pragma unroll
    for (int r = 0; r < 16; ++r)
      if ((r & 3) < 2) {
        const uint32_t x = w[r], y = w[r + 2];
        w[r] = prmt(x, y, 0x6240u);
        w[r + 2] = prmt(x, y, 0x7351u);
      }
#pragma unroll
    for (int r = 0; r < 16; r += 2) {
      const uint32_t x = w[r], y = w[r + 1];
      w[r] = (x & 0x0F0F0F0Fu) | ((y << 4) & 0xF0F0F0F0u);
      w[r + 1] = ((x >> 4) & 0x0F0F0F0Fu) | (y & 0xF0F0F0F0u);
    }
  }
}

// A warp moves 64 rows x 128 elements per unit; lane (rb = lane & 3,
// kc = lane >> 2) owns the 16 x 16 tile at rows 16 rb.., elements 16 kc..:
// sixteen 8-byte loads (8 lanes cover 64 contiguous bytes of a row), the
// register transpose, sixteen 8-byte stores (the 4 lanes of a kc write 32
// contiguous bytes of an output row).  No shared memory, no barriers.
constexpr int kTrUnitRows = 64, kTrUnitCols = 128;

__global__ void __launch_bounds__(256)
transpose_2d_kernel(const uint8_t* __restrict__ codes, const uint8_t* __restrict__ scales, int64_t rows, int64_t K,
                    uint8_t* __restrict__ codes_t, uint8_t* __restrict__ scales_t) {
  const int lane = threadIdx.x & 31, rb = lane & 3, kc = lane >> 2;
  const int64_t kt_n = (K + kTrUnitCols - 1) / kTrUnitCols, rt_n = (rows + kTrUnitRows - 1) / kTrUnitRows;
  const int64_t nbt = rows / 16, nb = K / 16;
  // The four row blocks of a unit write one 4-byte word of each transposed
  // scale row when those words are aligned (rows a multiple of 64).
  const bool vec = (rows % kTrUnitRows) == 0 && (reinterpret_cast<uintptr_t>(scales_t) & 3) == 0;
  const int64_t nwarps = (int64_t)gridDim.x * (blockDim.x / 32);
  for (int64_t u = (int64_t)blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5); u < kt_n * rt_n; u += nwarps) {
    const int64_t r0 = (u / kt_n) * kTrUnitRows + rb * 16, k0 = (u % kt_n) * kTrUnitCols + kc * 16;
    const bool live = r0 < rows && k0 < K;
    uint32_t lo[16], hi[16], s = 0u;
    if (live) {
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const uint2 v = __ldg(reinterpret_cast<const uint2*>(codes + (r0 + i) * (K / 2) + k0 / 2));
        lo[i] = v.x;
        hi[i] = v.y;
      }
      s = scales[r0 * nb + k0 / 16];  // tile (r0 / 16, k0 / 16): the same byte in all its 16 rows
    } else {
#pragma unroll
      for (int i = 0; i < 16; ++i) lo[i] = hi[i] = 0u;
    }
    transpose_nibbles16(lo, hi);
    // Scales of row blocks rb = 0..3 of this kc, byte rb of s4.
    const int base = lane & ~3;
    const uint32_t s4 = __shfl_sync(0xffffffffu, s, base) | (__shfl_sync(0xffffffffu, s, base + 1) << 8) |
                        (__shfl_sync(0xffffffffu, s, base + 2) << 16) | (__shfl_sync(0xffffffffu, s, base + 3) << 24);
    if (live) {
#pragma unroll
      for (int c = 0; c < 16; ++c) stg64(codes_t + (k0 + c) * (rows / 2) + r0 / 2, lo[c], hi[c]);
      if (vec) {
        // Lane rb writes output rows k0 + 4 rb .. k0 + 4 rb + 3, row blocks r0 / 16 - rb .. + 3.
#pragma unroll
        for (int j = 0; j < 4; ++j)
          *reinterpret_cast<uint32_t*>(scales_t + (k0 + 4 * rb + j) * nbt + r0 / 16 - rb) = s4;
      } else {
#pragma unroll
        for (int c = 0; c < 16; ++c) scales_t[(k0 + c) * nbt + r0 / 16] = (uint8_t)s;
      }
    }
  }
}

}  // namespace

int launch_quantize_colwise(const uint16_t* x, int64_t R, int64_t C, int64_t ldx, uint8_t* codes, uint8_t* scales,
                            float* tensor_scale, const uint32_t* amax_word, int mode, int scale_given, int sr,
                            uint64_t seed, uint64_t offset, cudaStream_t stream) {
  const int64_t tiles = ((C + kColThreads - 1) / kColThreads) * ((R + kColRows - 1) / kColRows);
  if (tiles == 0) return 0;
  int64_t grid = tiles < num_sms() * 4 ? tiles : num_sms() * 4;
  cudaError_t e;
#define MIXFP4_LAUNCH_C(MODE, SR)                                                                            \
  e = launch_pdl(quantize_colwise_kernel<MODE, SR>, (unsigned)grid, kColThreads, 0, stream, x, R, C, ldx, codes, \
                 scales, tensor_scale, amax_word, scale_given, seed, offset)
  switch (mode) {
    case MIXFP4_MODE_MIX:
      if (sr) MIXFP4_LAUNCH_C(MIXFP4_MODE_MIX, true); else MIXFP4_LAUNCH_C(MIXFP4_MODE_MIX, false);
      break;
    case MIXFP4_MODE_E2M1_ONLY:
      if (sr) MIXFP4_LAUNCH_C(MIXFP4_MODE_E2M1_ONLY, true); else MIXFP4_LAUNCH_C(MIXFP4_MODE_E2M1_ONLY, false);
      break;
    default:
      if (sr) MIXFP4_LAUNCH_C(MIXFP4_MODE_E1M2_ONLY, true); else MIXFP4_LAUNCH_C(MIXFP4_MODE_E1M2_ONLY, false);
      break;
  }
#undef MIXFP4_LAUNCH_C
  return e == cudaSuccess ? 0 : -1;
}

int launch_quantize_sr(const uint16_t* x, int64_t rows, int64_t K, int64_t ldx, uint8_t* codes, uint8_t* scales,
                       float* tensor_scale, const uint32_t* amax_word, int mode, int scale_given, uint64_t seed,
                       uint64_t offset, cudaStream_t stream) {
  const int64_t kblocks = K / 16, nblocks = rows * kblocks;
  if (nblocks == 0) return 0;
  int64_t grid = (nblocks + 255) / 256;
  if (grid > num_sms() * 3) grid = num_sms() * 3;
  cudaError_t e;
#define MIXFP4_LAUNCH_S(MODE)                                                                               \
  e = (ldx == K) ? launch_pdl(quantize_sr_kernel<MODE, true>, (unsigned)grid, 256, 0, stream, x, nblocks, kblocks, \
                              ldx, codes, scales, tensor_scale, amax_word, scale_given, seed, offset)          \
                 : launch_pdl(quantize_sr_kernel<MODE, false>, (unsigned)grid, 256, 0, stream, x, nblocks,       \
                              kblocks, ldx, codes, scales, tensor_scale, amax_word, scale_given, seed, offset)
  switch (mode) {
    case MIXFP4_MODE_MIX: MIXFP4_LAUNCH_S(MIXFP4_MODE_MIX); break;
    case MIXFP4_MODE_E2M1_ONLY: MIXFP4_LAUNCH_S(MIXFP4_MODE_E2M1_ONLY); break;
    default: MIXFP4_LAUNCH_S(MIXFP4_MODE_E1M2_ONLY); break;
  }
#undef MIXFP4_LAUNCH_S
  return e == cudaSuccess ? 0 : -1;
}

int launch_quantize_2d(const uint16_t* x, int64_t rows, int64_t K, int64_t ldx, uint8_t* codes, uint8_t* scales,
                       float* tensor_scale, const uint32_t* amax_word, int mode, int scale_given,
                       cudaStream_t stream) {
  const int64_t units = ((rows + 15) / 16) * ((K / 16 + 1) / 2);
  if (units == 0) return 0;
  int64_t grid = (units + k2dThreads / 32 - 1) / (k2dThreads / 32);
  if (grid > num_sms() * 4) grid = num_sms() * 4;
  cudaError_t e;
  switch (mode) {
    case MIXFP4_MODE_MIX:
      e = launch_pdl(quantize_2d_kernel<MIXFP4_MODE_MIX>, (unsigned)grid, k2dThreads, 0, stream, x, rows, K, ldx,
                     codes, scales, tensor_scale, amax_word, scale_given);
      break;
    case MIXFP4_MODE_E2M1_ONLY:
      e = launch_pdl(quantize_2d_kernel<MIXFP4_MODE_E2M1_ONLY>, (unsigned)grid, k2dThreads, 0, stream, x, rows, K,
                     ldx, codes, scales, tensor_scale, amax_word, scale_given);
      break;
    default:
      e = launch_pdl(quantize_2d_kernel<MIXFP4_MODE_E1M2_ONLY>, (unsigned)grid, k2dThreads, 0, stream, x, rows, K,
                     ldx, codes, scales, tensor_scale, amax_word, scale_given);
      break;
  }
  return e == cudaSuccess ? 0 : -1;
}

int launch_quantize_colwise_rht(const uint16_t* x, int64_t R, int64_t C, int64_t ldx, const uint8_t* signs,
                                uint8_t* codes, uint8_t* scales, float* tensor_scale, uint32_t* amax_word, int mode,
                                int scale_given, int amax_pass, cudaStream_t stream) {
  const int64_t tiles = ((C + kCrCols - 1) / kCrCols) * (R / kCrRows);
  if (tiles == 0) return 0;
  const int64_t grid = tiles < num_sms() * 3 ? tiles : num_sms() * 3;
  cudaError_t e;
#define MIXFP4_LAUNCH_CR(MODE, AMAX)                                                                           \
  e = launch_pdl(quantize_colwise_rht_kernel<MODE, AMAX>, (unsigned)grid, 256, 0, stream, x, R, C, ldx, signs, codes, \
                 scales, tensor_scale, amax_word, scale_given)
  if (amax_pass) {
    MIXFP4_LAUNCH_CR(MIXFP4_MODE_MIX, true);
  } else {
    switch (mode) {
      case MIXFP4_MODE_MIX: MIXFP4_LAUNCH_CR(MIXFP4_MODE_MIX, false); break;
      case MIXFP4_MODE_E2M1_ONLY: MIXFP4_LAUNCH_CR(MIXFP4_MODE_E2M1_ONLY, false); break;
      default: MIXFP4_LAUNCH_CR(MIXFP4_MODE_E1M2_ONLY, false); break;
    }
  }
#undef MIXFP4_LAUNCH_CR
  return e == cudaSuccess ? 0 : -1;
}

int launch_transpose_2d(const uint8_t* codes, const uint8_t* scales, int64_t rows, int64_t K, uint8_t* codes_t,
                        uint8_t* scales_t, cudaStream_t stream) {
  const int64_t units = ((K + kTrUnitCols - 1) / kTrUnitCols) * ((rows + kTrUnitRows - 1) / kTrUnitRows);
  if (units == 0) return 0;
  const int64_t blocks = (units + 7) / 8;  // 8 warps per CTA, one unit each per pass
  const int64_t grid = blocks < num_sms() * 8 ? blocks : num_sms() * 8;
  transpose_2d_kernel<<<(unsigned)grid, 256, 0, stream>>>(codes, scales, rows, K, codes_t, scales_t);
  return cudaGetLastError() == cudaSuccess ? 0 : -1;
}

}  // namespace mixfp4
