/*
 * mixfp4.h -- C ABI of libmixfp4.so, the GB300 (sm_103a) MixFP4 W4A4 linear
 * layer: an online MixFP4 quantizer, its decoder, and a MixFP4 x MixFP4 GEMM.
 *
 * MixFP4 (arXiv 2605.31035) extends NVFP4: every 16-element block along the
 * reduction dimension K stores sixteen 4-bit codes and one 8-bit block scale.
 * Each code is [s | p2 p1 p0] (App. B.2): a sign bit and a 3-bit payload read
 * as FP4 E2M1 {0,.5,1,1.5,2,3,4,6} or as FP4 E1M2 remapped x2 to {0,..,7}
 * (Table 1, Sec. 3.1).  The scale byte carries the block's format in bit 7
 * (T = 0 E2M1, T = 1 E1M2) and the unsigned E4M3 block scale s8 in bits 6:0
 * (App. B.3).  A tensor adds one fp32 per-tensor scale s32 (Alg. 1).
 * An element's value is  (-1)^s * v(T, p) * s8 * s32.
 *
 * Storage layout (the paper fixes none; this library's choice):
 *   codes  uint8 [rows][K/2]   element 2j of a row in the low nibble of byte j
 *   scales uint8 [rows][K/16]  one byte per block, blocks in K order
 *   both row-major with no padding (row pitch K/2 and K/16 bytes).
 *
 * Conventions for every entry point:
 *   - All tensor pointers are DEVICE pointers owned by the caller; the library
 *     allocates no device memory and keeps no per-call state.
 *   - Work is enqueued asynchronously on `stream` (a cudaStream_t; NULL = the
 *     legacy default stream).  The return value reports argument validation
 *     and launch errors only; results are ready once the stream is synchronised.
 *   - Invalid arguments return a negative mixfp4_status and enqueue nothing.
 *     No entry point traps or aborts.
 *   - Inputs must be finite; NaN or Inf input gives unspecified codes.
 */
#ifndef MIXFP4_H
#define MIXFP4_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  MIXFP4_OK = 0,
  MIXFP4_ERR_NULL = -1,    /* a required pointer is NULL */
  MIXFP4_ERR_SHAPE = -2,   /* a size is negative, or violates a multiple-of rule */
  MIXFP4_ERR_ALIGN = -3,   /* a pointer or leading dimension is misaligned */
  MIXFP4_ERR_DTYPE = -4,   /* unsupported input dtype */
  MIXFP4_ERR_CUDA = -5,    /* a CUDA runtime call or launch failed */
  MIXFP4_ERR_TIMEOUT = -6, /* a bounded device-side wait gave up (see status_word) */
  MIXFP4_ERR_ARG = -7      /* an enum argument is out of range */
} mixfp4_status;

enum { MIXFP4_MODE_MIX = 0,        /* Alg. 1: per-block E2M1/E1M2 by lower MSE */
       MIXFP4_MODE_E2M1_ONLY = 1,  /* every block E2M1, T = 0 (plain NVFP4 bits) */
       MIXFP4_MODE_E1M2_ONLY = 2,  /* every block E1M2, T = 1 (NVINT4 lattice) */
       MIXFP4_MODE_FOUR_SIX = 3    /* the {E2M1(6), E2M1(4)} candidate set of Sec. 2.4 ("4/6"):
                                      per block the lower-MSE of s8 from B/6 or B/4 (B/4 on a
                                      tie), E2M1 codes, T = 0 (plain NVFP4 bits, so both GEMMs
                                      take it); mixfp4_quantize and mixfp4_quantize_noalloc only */ };

enum { MIXFP4_SCALE_COMPUTE = 0,   /* compute s32 = fl32(max|x| / 2688), write *tensor_scale */
       MIXFP4_SCALE_GIVEN = 1      /* read s32 from *tensor_scale */ };

enum { MIXFP4_DTYPE_BF16 = 0, MIXFP4_DTYPE_F32 = 1 /* output of mixfp4_fake_quantize only */ };

/* Candidate formats of mixfp4_fake_quantize (bit c of `candidates`). */
enum { MIXFP4_CAND_E2M1_6 = 1,   /* E2M1, block max mapped to 6 (Algorithm 1's E2M1) */
       MIXFP4_CAND_E1M2 = 2,     /* E1M2 in x2 units {0..7}, block max mapped to 7 */
       MIXFP4_CAND_E2M1_4 = 4,   /* E2M1, block max mapped to 4 (the "4/6" candidate) */
       MIXFP4_CAND_E3M0 = 8      /* E3M0 {0, 1/4, ..., 16}, block max mapped to 16 */ };

/*
 * mixfp4_quantize -- Algorithm 1 (Sec. 3.2) with type-in-scale packing (App. B.3).
 *
 *   s32  = fl32(max|X| / 2688)              (2688 = 6*448 = 7*384)
 *   a_i  = fl32(x_i / s32)                   per element (0 when s32 == 0)
 *   per 16-element block with B = max|a_i|, for c in {E2M1 (max 6), E1M2 (max 7)}:
 *     s8_c = E4M3_RNE(fl32(B / max_c))       (subnormals, saturating at 448)
 *     q_i  = RNE_c(fl32(|a_i| / s8_c))       nearest codebook value, ties to the
 *                                            even payload, saturating (q = 0 if s8_c = 0)
 *     S_c  = S_even + S_odd, fma chains of d_i^2 over even / odd i, d_i = q_i*s8_c - |a_i|
 *   E2M1 iff S_E2M1 < S_E1M2 (strict), else E1M2 with T = 1.
 *
 * x            device, bf16 [rows][ldx]; 32-byte aligned; ldx % 16 == 0, ldx >= K.
 * dtype        MIXFP4_DTYPE_BF16.
 * rows, K      rows >= 0, K >= 0, K % 16 == 0.  rows*K == 0 is a valid no-op
 *              (with SCALE_COMPUTE, *tensor_scale is still set to 0).
 * codes        device, uint8 [rows][K/2], 8-byte aligned.            (output)
 * scales       device, uint8 [rows][K/16].                           (output)
 * tensor_scale device, one float: written (COMPUTE) or read (GIVEN).  A given
 *              s32 must be finite and >= 0, and max|x| / s32 must be finite.
 * workspace    device, one uint32 scratch word; required with SCALE_COMPUTE
 *              (it receives max|x|), ignored with SCALE_GIVEN.  Calls that share
 *              a workspace word must be ordered on the GPU.
 * mode         MIXFP4_MODE_*.   scale_flag  MIXFP4_SCALE_*.
 */
int mixfp4_quantize(const void* x, int dtype, int64_t rows, int64_t K, int64_t ldx,
                    uint8_t* codes, uint8_t* scales, float* tensor_scale,
                    uint32_t* workspace, int mode, int scale_flag, void* stream);

/*
 * mixfp4_quantize_rht -- the 128-point Walsh-Hadamard rotation applied before
 * quantization (the random Hadamard transform of Sec. 4.1 "+RHT" and the
 * Sec. 3.2 training flow), fused with Algorithm 1 (as mixfp4_quantize).
 *
 *   every 128-element chunk of a row along K, on its own:
 *     v_i = -x_i if bit i of `signs` is set, else x_i        (i = 0..127)
 *     v   = H_128 v   (Sylvester order) by the radix-2 butterfly in fp32,
 *                     strides 1, 2, 4, ..., 64 in that order, (a, b) -> (a+b, a-b)
 *     y_i = fl32(v_i * c),  c = RN(1/sqrt(128))
 *   then Algorithm 1 on the fp32 tensor y (s32 = fl32(max|y| / 2688) with
 *   SCALE_COMPUTE; x_i / s32 is the IEEE quotient of the fp32 y_i).
 * The paper fixes no arithmetic for the rotation; this order is the one used
 * (and checked bit for bit) here.
 *
 * signs        device, 16 bytes (bit i = byte i/8, bit i%8: negate chunk
 *              element i), the same for every chunk; NULL for no negation
 *              (the plain normalised Walsh-Hadamard transform).
 * rows, K      as mixfp4_quantize, and K % 128 == 0 (else MIXFP4_ERR_SHAPE).
 * Other arguments and the error behaviour are those of mixfp4_quantize.
 */
int mixfp4_quantize_rht(const void* x, int dtype, int64_t rows, int64_t K, int64_t ldx, const uint8_t* signs,
                        uint8_t* codes, uint8_t* scales, float* tensor_scale, uint32_t* workspace, int mode,
                        int scale_flag, void* stream);

/*
 * mixfp4_quantize_colwise -- Algorithm 1 with every 16-element block running
 * down a column: the operand orientation of a GEMM that reduces over the rows
 * of X, as in the weight-gradient GEMM of the training flow (Sec. 3.2, WGRAD
 * reduces over tokens; DGRAD over the weights' output dimension).  The
 * result is bit for bit mixfp4_quantize of the transpose X^T:
 *   codes  [C][R/2]   element r of column c in nibble r % 2 of byte r / 2
 *   scales [C][R/16]  one byte per 16 rows of a column
 * s32 = fl32(max|X| / 2688) as for mixfp4_quantize.
 *
 * x            device, bf16 [R][ldx]; 32-byte aligned; ldx % 16 == 0, ldx >= C.
 * R, C         R % 16 == 0, C % 16 == 0 (else MIXFP4_ERR_SHAPE); 0 is a no-op
 *              (with SCALE_COMPUTE *tensor_scale is set to 0).
 * codes        device, uint8 [C][R/2], 8-byte aligned.                  (output)
 * scales       device, uint8 [C][R/16].                                 (output)
 * tensor_scale, workspace, mode, scale_flag, stream: as mixfp4_quantize.
 */
int mixfp4_quantize_colwise(const void* x, int dtype, int64_t R, int64_t C, int64_t ldx, uint8_t* codes,
                            uint8_t* scales, float* tensor_scale, uint32_t* workspace, int mode, int scale_flag,
                            void* stream);

/*
 * mixfp4_quantize_colwise_rht -- mixfp4_quantize_colwise with the 128-point
 * Walsh-Hadamard rotation of mixfp4_quantize_rht applied along the rows first:
 * the weight-gradient inputs of the training recipe (Sec. 3.2, Sec. 4.2: the
 * RHT is applied to both WGRAD operands, whose reduction runs over R).  Every
 * 128-row chunk of each column is rotated (signs, butterfly order and scaling
 * as mixfp4_quantize_rht) and the rotated column is quantized down its rows:
 * bit for bit mixfp4_quantize_rht of X^T, codes [C][R/2], scales [C][R/16].
 * With SCALE_COMPUTE, s32 = fl32(max|rotated X| / 2688).
 * R, C         R % 128 == 0, C % 16 == 0 (else MIXFP4_ERR_SHAPE).
 * Other arguments and errors: as mixfp4_quantize_colwise and mixfp4_quantize_rht.
 */
int mixfp4_quantize_colwise_rht(const void* x, int dtype, int64_t R, int64_t C, int64_t ldx, const uint8_t* signs,
                                uint8_t* codes, uint8_t* scales, float* tensor_scale, uint32_t* workspace, int mode,
                                int scale_flag, void* stream);

/*
 * mixfp4_quantize_sr, mixfp4_quantize_colwise_sr -- mixfp4_quantize and
 * mixfp4_quantize_colwise with stochastic rounding of the codes, the
 * gradient quantization of the training flow (Sec. 4.2 pre-training recipe;
 * the paper's stochastic-rounding ablation).  Format and block scale are
 * chosen exactly as Algorithm 1 chooses them (round-to-nearest candidates, so
 * scale bytes and s32 equal those of the rounding-to-nearest entry point);
 * then each code of the chosen format is rounded stochastically: with
 * m = fl32(|x / s32| / s8) and l <= m < u its neighbours in the codebook,
 * the magnitude is u iff eps < (m - l) / (u - l), else l (m at or above the
 * largest value saturates), so the value rounds up with probability
 * (m - l) / (u - l).  The sign bit is signbit(x).
 *   eps = (w >> 8) * 2^-24, w = word e % 4 of Philox4x32-10 (Salmon et al.,
 *   SC'11) with key (seed & 0xFFFFFFFF, seed >> 32) and counter
 *   (e / 4 low word, e / 4 high word, offset low word, offset high word),
 *   e = the element's index in the output tensor's row-major order (r * K + k
 *   for mixfp4_quantize_sr; c * R + r, i.e. in X^T, for the column-wise one).
 * A fresh (seed, offset) per call gives independent draws; the same pair
 * reproduces the same codes.
 * Other arguments, layouts and errors: as mixfp4_quantize and
 * mixfp4_quantize_colwise.
 */
int mixfp4_quantize_sr(const void* x, int dtype, int64_t rows, int64_t K, int64_t ldx, uint8_t* codes,
                       uint8_t* scales, float* tensor_scale, uint32_t* workspace, int mode, int scale_flag,
                       uint64_t seed, uint64_t offset, void* stream);
int mixfp4_quantize_colwise_sr(const void* x, int dtype, int64_t R, int64_t C, int64_t ldx, uint8_t* codes,
                               uint8_t* scales, float* tensor_scale, uint32_t* workspace, int mode, int scale_flag,
                               uint64_t seed, uint64_t offset, void* stream);

/*
 * mixfp4_fake_quantize -- quantize-dequantize under a chosen candidate set
 * and block size: the paper's candidate-set ablation (Sec. 2.4, candidate
 * sets {E2M1(6), E2M1(4)} and {E2M1(6), E1M2, E3M0}) and block-size ablation
 * (Sec. 4.3, Table 5, g = 8..64).  A block is g consecutive elements of a row.
 * Every candidate c in `candidates` follows Algorithm 1 with its own divisor
 * d_c (6, 7, 4, 16): s8 = E4M3_RNE(fl32(B / d_c)) from the block max B of
 * |x / s32|, codes by round-to-nearest-even of fl32(|x / s32| / s8) onto its
 * codebook (saturating), error sum S in the order of mixfp4_quantize on each
 * 16-element chunk (for g = 8: the even and the odd elements of the 8) and,
 * for g > 16, the pairwise tree (S_0 + S_1) + (S_2 + S_3) of the chunks.
 * Candidates are visited in bit order and a later one wins a tie (S <= best),
 * so {E2M1_6, E1M2} at g = 16 is Algorithm 1.  s32 = fl32(max|X| / 2688).
 * The output is sign(x) fl32(v s8 s32) of the chosen candidate (v its code's
 * magnitude): for {E2M1_6, E1M2} at g = 16, bit for bit mixfp4_dequantize of
 * mixfp4_quantize.  Three or more formats, or other block sizes, cannot be
 * stored in the one type bit, so this entry point returns values, not codes.
 *
 * x            device, bf16 [rows][ldx]; 32-byte aligned; ldx % 16 == 0, ldx >= K.
 * rows, K      K % 16 == 0 and K % block == 0 (else MIXFP4_ERR_SHAPE); 0 is a
 *              no-op (with SCALE_COMPUTE *tensor_scale is set to 0).
 * candidates   nonzero mask of MIXFP4_CAND_* (else MIXFP4_ERR_ARG).
 * block        8, 16, 32 or 64 (else MIXFP4_ERR_ARG).
 * tensor_scale, workspace, scale_flag, stream: as mixfp4_quantize.
 * out          device, [rows][ldo] of out_dtype (MIXFP4_DTYPE_F32, or
 *              MIXFP4_DTYPE_BF16 = that fp32 value rounded to nearest even);
 *              32-byte aligned, ldo % 16 == 0, ldo >= K.             (output)
 * choice       device, uint8 [rows][K / block]: index (bit position) of each
 *              block's chosen candidate; 2-byte aligned; NULL to skip. (output)
 * Errors: as mixfp4_quantize; MIXFP4_ERR_DTYPE for another out_dtype.
 */
int mixfp4_fake_quantize(const void* x, int dtype, int64_t rows, int64_t K, int64_t ldx, int candidates, int block,
                         float* tensor_scale, uint32_t* workspace, int scale_flag, void* out, int out_dtype,
                         int64_t ldo, uint8_t* choice, void* stream);

/*
 * mixfp4_quantize_2d -- Algorithm 1 with 16 x 16 blocks, the weight
 * quantization of the training flow (Sec. 3.2: weights in 2D blocks).  The
 * tile of rows 16t..16t+15 and columns 16b..16b+15 has one block max (the
 * tile's), one E4M3 scale per candidate and one type bit; each candidate's
 * error is the per-row sum of mixfp4_quantize, combined over the tile's 16
 * rows by the pairwise tree ((S0+S1)+(S2+S3)) + ... in fp32 (rows past the
 * tensor count as zeros).  Output in the row-wise layout of mixfp4_quantize,
 * every row of a tile storing the tile's scale byte, so mixfp4_gemm takes it
 * as is and mixfp4_transpose_2d gives the transposed operand exactly.
 * Arguments, alignment and errors: as mixfp4_quantize (rows need not be a
 * multiple of 16).
 */
int mixfp4_quantize_2d(const void* x, int dtype, int64_t rows, int64_t K, int64_t ldx, uint8_t* codes,
                       uint8_t* scales, float* tensor_scale, uint32_t* workspace, int mode, int scale_flag,
                       void* stream);

/*
 * mixfp4_transpose_2d -- the MixFP4 tensor W^T of a tensor W quantized with
 * 2D blocks (mixfp4_quantize_2d): element (r, k) of W is element (k, r) of
 * the output, and each tile's shared scale byte becomes the scale of the
 * transposed tile's rows.  It needs no arithmetic: W^T decodes to the
 * transpose of W's decoded values exactly (the DGRAD operand of the weights).
 * The scale of a tile is read from its first row, so the input must come
 * from mixfp4_quantize_2d (or share one scale byte per tile otherwise).
 *
 * codes, scales      device, uint8 [rows][K/2] (8-byte aligned), [rows][K/16].
 * rows, K            rows % 16 == 0, K % 16 == 0 (else MIXFP4_ERR_SHAPE).
 * codes_t, scales_t  device, uint8 [K][rows/2] (8-byte aligned), [K][rows/16]. (output)
 * s32 is unchanged (the caller reuses the tensor scale).
 */
int mixfp4_transpose_2d(const uint8_t* codes, const uint8_t* scales, int64_t rows, int64_t K, uint8_t* codes_t,
                        uint8_t* scales_t, void* stream);

/*
 * mixfp4_dequantize -- App. B.2/B.3 decode:
 *   out[r][k] = fl32((-1)^s * v(T, p) * ue4m3(scale & 0x7F) * s32),
 * one rounding of the exact product.
 *
 * codes        device, uint8 [rows][K/2], 8-byte aligned.
 * scales       device, uint8 [rows][K/16].
 * tensor_scale device, one float s32.
 * rows, K      rows >= 0, K % 16 == 0.
 * out          device, float [rows][K], 32-byte aligned.                (output)
 */
int mixfp4_dequantize(const uint8_t* codes, const uint8_t* scales, const float* tensor_scale,
                      int64_t rows, int64_t K, float* out, void* stream);

/*
 * mixfp4_gemm -- MixFP4 x MixFP4 GEMM, C = A_deq . B_deq^T:
 *   C[m][n] = s32A * s32B * sum_blocks (sA * sB) * sum_i vA_i * vB_i
 * (App. B.1 Eq. (factor)), where each block's codes are decoded to the unified
 * E2M2 value (Sec. 3.3, App. B.5) times its E4M3 scale -- exact in f16 -- and
 * contracted on the tensor cores with fp32 accumulation.
 *
 * a_codes/a_scales/a_ts   A = activations, M x K, quantized by mixfp4_quantize.
 * b_codes/b_scales/b_ts   B = weights (nn.Linear layout), N x K.
 * M, N, K      M >= 0, N >= 0, K % 256 == 0; M and N need no padding.
 * C            device, float [M][ldc], ldc >= N, 4-byte aligned (16-byte alignment
 *              and ldc % 4 == 0 enable vector stores).                      (output)
 * status_word  device uint32 or NULL.  When given it is zeroed by the call and
 *              becomes nonzero if a bounded device-side pipeline wait gave up
 *              (C is then unspecified); the caller reads it after synchronising.
 * Code and scale pointers must be 16-byte aligned.
 */
int mixfp4_gemm(const uint8_t* a_codes, const uint8_t* a_scales, const float* a_ts,
                const uint8_t* b_codes, const uint8_t* b_scales, const float* b_ts,
                int64_t M, int64_t N, int64_t K, float* C, int64_t ldc,
                uint32_t* status_word, void* stream);

/*
 * mixfp4_split_native -- the operands of the native FP4 GEMM variant.  A
 * MixFP4 tensor is rewritten as the sum of two E2M1 tensors that share its
 * block scales (no counterpart in the paper; every value is exact):
 *   E2M1 block (T = 0): main = the stored codes, residual = 0;
 *   E1M2 block (T = 1): each magnitude v = p (Sec. 3.1 remap, v in 0..7) is
 *     e + r with e the largest E2M1 value <= v (0,1,2,3,4,4,6,6) and r = v - e
 *     (1 for v = 5 and 7, else 0); both parts carry the element's sign bit.
 * The block scales are written as ue4m3 (bits 6..0 of the scale byte) in the
 * tensor core's tiled block-16 layout: tiles of 128 rows x 4 blocks (64 K),
 * 512 bytes each; tile (rt, kt) starts at byte (rt * K/64 + kt) * 512; row r
 * of the tile, block b of the tile at (r % 32) * 16 + (r / 32) * 4 + b.  Rows
 * are padded to a multiple of 256 with zero bytes.
 *
 * codes, scales  device, a MixFP4 tensor [rows][K/2], [rows][K/16] (16- and
 *                4-byte aligned).
 * rows, K        rows >= 0, K % 64 == 0 (else MIXFP4_ERR_SHAPE).
 * main_codes, res_codes  device, uint8 [rows][K/2] each, 16-byte aligned.  (output)
 * sf_tiled       device, uint8 [ceil(rows/256) * 256 * K/16], 16-byte aligned.
 *                                                                         (output)
 */
int mixfp4_split_native(const uint8_t* codes, const uint8_t* scales, int64_t rows, int64_t K,
                        uint8_t* main_codes, uint8_t* res_codes, uint8_t* sf_tiled, void* stream);

/*
 * mixfp4_gemm_native -- the MixFP4 GEMM on the block-scaled FP4 tensor path:
 *   C = s32A * s32B * (A_main + A_res) . (B_main + B_res)^T,
 * the four products of E2M1 operands with ue4m3 block-16 scales contracted by
 * tcgen05.mma kind::mxf4nvf4 with fp32 accumulation.  It computes the same C
 * as mixfp4_gemm (App. B.1 Eq. (factor)) up to fp32 summation order.
 *
 * a_main/a_res/a_sf  A (activations, M x K) as written by mixfp4_split_native;
 *                    a_res may be NULL when A has no E1M2 block (an E2M1-only
 *                    tensor), which drops the products with it.
 * a_ts               device, one float s32A.
 * b_main/b_res/b_sf/b_ts  the same for B (weights, N x K).
 * M, N, K, C, ldc, status_word  as mixfp4_gemm (K % 256 == 0).
 * Code and scale pointers must be 16-byte aligned.
 */
int mixfp4_gemm_native(const uint8_t* a_main, const uint8_t* a_res, const uint8_t* a_sf, const float* a_ts,
                       const uint8_t* b_main, const uint8_t* b_res, const uint8_t* b_sf, const float* b_ts,
                       int64_t M, int64_t N, int64_t K, float* C, int64_t ldc, uint32_t* status_word,
                       void* stream);

/*
 * mixfp4_gemm_native_fewrows -- the native block-scaled FP4 variant for few
 * activation rows (decode-shaped GEMMs, M <= 64), taking the MixFP4 operands
 * as stored (the arguments of mixfp4_gemm).  Each operand is the sum of two
 * E2M1 parts with ue4m3 block-16 scales: the stored codes read as E2M1 codes
 * (scale: the block scale without its type bit), and a residual whose
 * payload is {0,1,2,3,4,4,4,2}[p] of the stored payload p (scale: the block
 * scale for an E1M2 block, 0 for an E2M1 block); for an E1M2 block the two
 * E2M1 values add up to the E1M2 value p, for an E2M1 block the residual
 * vanishes.  Each 128-row x 256-K unit of B and the matching slice of A are
 * loaded as stored, their residual rows and scale tiles are written in
 * shared memory, and tcgen05.mma kind::mxf4nvf4 contracts them, one
 * instruction per 64-K step covering all four products (main and residual
 * stacked on the M and N sides).  C is the same product as mixfp4_gemm's up
 * to fp32 summation order; the host zeroes C first and the partial sums of
 * the K slices are added into it.
 * M            0 <= M <= 64 (else MIXFP4_ERR_SHAPE).
 * Other arguments, alignment and errors: as mixfp4_gemm.
 */
int mixfp4_gemm_native_fewrows(const uint8_t* a_codes, const uint8_t* a_scales, const float* a_ts,
                               const uint8_t* b_codes, const uint8_t* b_scales, const float* b_ts, int64_t M,
                               int64_t N, int64_t K, float* C, int64_t ldc, uint32_t* status_word, void* stream);

/*
 * mixfp4_quantize_noalloc -- mixfp4_quantize with MIXFP4_SCALE_COMPUTE for
 * callers that cannot allocate device memory.  The paper has no counterpart;
 * this is a deployment convenience.
 *
 * mixfp4_quantize needs a caller-provided scratch word (`workspace`) to
 * compute the per-tensor scale.  Callers such as an inference runtime that
 * plans all device memory ahead of time and gives an operator only its input
 * and output buffers, or a plugin whose execute callback must not call
 * cudaMalloc, have no such word.  This entry point keeps it in a 256-byte
 * file-scope device array of the library instead and allocates nothing.
 *
 * Arguments and results are those of mixfp4_quantize with SCALE_COMPUTE:
 * x, dtype, rows, K, ldx, codes, scales, mode and stream as documented there;
 * tensor_scale (device, one float) receives s32.
 *
 * The first call on a device looks up the array's device address for that
 * device (make it before any stream capture); a call that finds a different
 * context current on the device (after cudaDeviceReset) looks it up again.  Every call shares the array,
 * and the array keeps the last call's contents (it is cleared before each
 * use); calls that overlap on the GPU race on it and must be ordered.  Any
 * shape needs one 32-bit word of the 64 the array holds; a larger need would
 * be rejected with MIXFP4_ERR_SHAPE.
 */
int mixfp4_quantize_noalloc(const void* x, int dtype, int64_t rows, int64_t K, int64_t ldx,
                            uint8_t* codes, uint8_t* scales, float* tensor_scale, int mode,
                            void* stream);

/* Human-readable name of a mixfp4_status value (static string). */
const char* mixfp4_status_string(int status);

/* ABI version of this library (major * 100 + minor). */
int mixfp4_version(void);

/*
 * mixfp4_selftest_bounded_wait -- check of the failure detection in the GEMM
 * pipelines (no counterpart in the paper): one CTA waits with the same
 * bounded mbarrier wait the GEMM kernels use on (a) a barrier whose phase
 * completes, (b) a barrier nothing arrives on (an injected missed arrival)
 * and (c) that barrier with its abort flag raised, and ORs into *status_word:
 * bit 0 if (a) failed, bit 1 if (b) gave up, bit 2 if (b) gave up only after
 * limit_ns, bit 3 if (c) gave up.  A healthy device reports 0xE.
 *
 * status_word  device, one uint32, 4-byte aligned (the caller zeroes it).
 * limit_ns     1 .. 2e9 (else MIXFP4_ERR_ARG).  The call occupies one SM for
 *              about limit_ns; it does not fault or trap.
 */
int mixfp4_selftest_bounded_wait(uint32_t* status_word, uint64_t limit_ns, void* stream);

/*
 * mixfp4_selftest_gemm_missed_stage -- check of the failure path of the
 * CTA-pair GEMM kernel itself (no counterpart in the paper): mixfp4_gemm's
 * pair kernel (256-wide tiles, any M) runs with every pipeline wait limited
 * to limit_ns and with the first code stage of every CTA never issued (no
 * copy, no arrival).  The waits on that stage run out, each role that gives
 * up ORs its bit into *status_word (1 producer, 2 / 4 MMA thread, 8 drain,
 * 16 / 32 decoders, 64 epilogue), raises its CTA's abort
 * flag, lets the copies and MMAs it issued complete, frees its tensor memory
 * and exits; C is not written.  Nothing faults or hangs, and the device stays
 * usable: a later mixfp4_gemm on it runs normally.
 *
 * Operands, M, N, K, C, ldc: as mixfp4_gemm (M, N >= 1, K >= 256).
 * status_word  device, one uint32, 4-byte aligned, required (zeroed first).
 * limit_ns     1 .. 2e9 (else MIXFP4_ERR_ARG); the call takes a few limit_ns.
 */
int mixfp4_selftest_gemm_missed_stage(const uint8_t* a_codes, const uint8_t* a_scales, const float* a_ts,
                                      const uint8_t* b_codes, const uint8_t* b_scales, const float* b_ts, int64_t M,
                                      int64_t N, int64_t K, float* C, int64_t ldc, uint32_t* status_word,
                                      uint64_t limit_ns, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* MIXFP4_H */
