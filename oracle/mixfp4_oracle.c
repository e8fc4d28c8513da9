/*
 * MixFP4 CPU oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, deliberately unoptimised restatement of the MixFP4 method
 * (arXiv 2605.31035).  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference legs of bench.py may load this library.  The CUDA
 * product path never links, imports or calls it, and the two share no code.
 *
 * Build: gcc -O2 -ffp-contract=off -fPIC -shared (no fast-math, no FMA
 * contraction) so every float operation below is one IEEE-754 binary32
 * operation rounded to nearest-even, with subnormals.
 *
 * What each function follows:
 *   fp_code_value      Eq. 1-2 (Sec. 2.1), the IEEE-like value of an S.E.M code
 *   e4m3_*             E4M3 block scale (Sec. 2.1; Alg. 1 scale steps)
 *   fp4_*              Table 1 (Sec. 3.1) and App. B.2 codebooks; the x2 E1M2
 *                      remap of Sec. 3.1 / App. B.2
 *   oracle_quantize    Algorithm 1 (MixFP4 quantization), with the type bit of
 *                      App. B.3 (type-in-scale packing); oracle_quantize_f32
 *                      is the same steps on an fp32 tensor
 *   oracle_rht         the random Hadamard transform applied before
 *                      quantization (Sec. 4.1 "+RHT", Sec. 3.2 training flow):
 *                      128-point Sylvester Walsh-Hadamard per chunk (reading
 *                      R11)
 *   oracle_dequantize  App. B.2/B.3 decode (scale_ue4m3 = scale with bit 7
 *                      cleared) times the per-tensor scale
 *   oracle_gemm_f64    C = A_deq . B_deq^T in float64 (plain definition)
 *   oracle_gemm_exact  App. B.1 Eq. (factor): per-block integer dot times the
 *                      scale product, accumulated exactly in __int128
 *   oracle_split_native  the MixFP4 operand as main + residual E2M1 operands
 *                      sharing its scales (Table 1 codebooks; 5 = 4 + 1,
 *                      7 = 6 + 1), scales in the tensor core's tiled layout
 *   oracle_quantize_2d Algorithm 1 with 2D 16 x 16 blocks, the weight
 *                      quantization of the training flow (Sec. 3.2, Sec. 4.2
 *                      pre-training recipe); reading R12
 *   oracle_transpose_2d  the transposed operand (DGRAD orientation) of a
 *                      2D-quantized tensor: codes and tile scales transposed
 *   oracle_philox4x32_10  the counter-based generator of J. K. Salmon et al.,
 *                      "Parallel random numbers: as easy as 1, 2, 3" (SC'11),
 *                      source of the stochastic-rounding uniforms
 *   oracle_quantize_sr Algorithm 1 with stochastic rounding of the codes
 *                      (App. D "Ablation Study of Stochastic Rounding", Sec. 4.2
 *                      pre-training recipe: SR on gradients); reading R13
 *   oracle_fake_quantize  Algorithm 1 with the per-block MSE choice taken over
 *                      a chosen candidate set and block size, returning the
 *                      quantized-then-dequantized tensor and each block's
 *                      choice: the candidate-set ablation (Sec. 2.4 "Format
 *                      Proliferation Has Diminishing Returns", E2M1(4) and
 *                      E3M0) and the block-size ablation (Sec. 4.3, Table 5);
 *                      reading R14
 *   oracle_f32_to_bf16 binary32 -> bfloat16, round to nearest even
 *
 * Readings where the paper is silent (binding on the CUDA path as well):
 *   R1 X_FP8 = fl32(X / s32) is an fp32 value (no FP8 cast).
 *   R2 s8 = E4M3_RNE(fl32(blockmax / c)), c = 6 (E2M1) or 7 (E1M2): two
 *      roundings, E4M3 with subnormals, saturating at 448.
 *   R3 E1M2 quantizes in x2 units: magnitudes {0..7}, payload = integer.
 *   R4 FP4 rounding is round-to-nearest of the fp32 quotient y = fl32(|a|/s8)
 *      onto the codebook, ties to the even payload, saturating at the maximum.
 *      The nibble sign bit is signbit(x).
 *   R5 block error: d_i = fl32(q_i*s8 - |a_i|) (the product is exact);
 *      S_even = fma chain over i = 0,2,..,14 from +0, S_odd over 1,3,..,15,
 *      S = fl32(S_even + S_odd); the division by 16 of the mean is omitted.
 *      The order is a definition (the paper names only the MSE); the sums
 *      are pinned to the exact rational sum of squares within 16 ulp-units
 *      by the tests, and the choice to the exact comparison beyond that.
 *   R6 E2M1 is chosen iff S_E2M1 < S_E1M2 (strict), otherwise E1M2 with T=1.
 *   R7 s8 == 0 gives all-zero magnitudes and d_i = -|a_i|; s32 == 0 gives a_i = 0.
 *   R9 element 2j in the low nibble of byte j; codes [rows][K/2], scales
 *      [rows][K/16], both K-major.
 *   R11 RHT: every 128-element chunk of a row along K is rotated on its own:
 *      v_i = -x_i where sign bit i (of a 128-bit vector shared by all chunks)
 *      is set, else x_i; the Sylvester Hadamard product H_128 v by the radix-2
 *      butterfly in fp32, strides h = 1, 2, 4, ..., 64 in that order, each
 *      pair (i, i+h) with i & h == 0 becoming (fl32(v_i + v_{i+h}),
 *      fl32(v_i - v_{i+h})); then y_i = fl32(v_i * c), c = RN(1/sqrt(128)).
 *      Algorithm 1 then runs on the fp32 y (X = y).
 *   R12 2D blocks: a block is the 16 x 16 tile of rows 16t..16t+15 and
 *      columns 16b..16b+15 (a ragged last tile has fewer rows; its missing
 *      rows count as zeros).  B is the tile max; each candidate has one s8
 *      from B; each row's 16 elements give the R5 sum S_r; the tile's S is
 *      the pairwise tree ((S_0+S_1)+(S_2+S_3))+((S_4+S_5)+(S_6+S_7)) + ...
 *      over the 16 row slots; T is chosen by R6 for the whole tile, and every
 *      row of the tile stores the tile's scale byte.
 *   R13 stochastic rounding: the format and block scale are chosen exactly as
 *      in Algorithm 1 (round-to-nearest candidates, R4-R6); the chosen
 *      format's codes are then rounded stochastically: with m = fl32(|a|/s8)
 *      and l <= m < u its two neighbours in the codebook (m at or above the
 *      largest value saturates), the code is u iff eps < (m - l) / (u - l)
 *      (both exact fp32 values), else l, so P(u) = (m - l) / (u - l): the
 *      probability falls with the distance, as the paper states; its integer
 *      formula clamp(round(q + eps - 0.5)) is the same distribution on the
 *      E1M2 grid.  eps = (w >> 8) * 2^-24 for the word w of Philox4x32-10
 *      with key (seed low, seed high) and counter (e / 4 low, e / 4 high,
 *      offset low, offset high), word e % 4, e = the element's row-major index
 *      (r * K + k).  The sign bit stays signbit(x).
 *   R14 candidate sets and block sizes (the ablations; the stored format
 *      holds one type bit, so these exist only as quantize-dequantize):
 *      candidate c = 0 E2M1 with largest value 6 (Algorithm 1's E2M1),
 *      1 E1M2 in x2 units (R3), 2 E2M1 with largest value 4 (block scale
 *      from B / 4, the same E2M1 codebook and rounding, saturating at 6),
 *      3 E3M0 (Eq. 1-2 with W_E = 3, W_M = 0, bias 3: {0, 1/4, 1/2, 1, 2, 4,
 *      8, 16}, block scale from B / 16).  Each candidate follows Algorithm 1
 *      (R1, R2, R4, R7) with its own divisor; the tensor scale stays
 *      max|X| / 2688.  A block is g consecutive elements of a row, g in
 *      {8, 16, 32, 64}; its error sum is R5 on each 16-element chunk (for
 *      g = 8: the even and the odd elements of the 8), combined for g > 16
 *      by the pairwise tree (S_0 + S_1) + (S_2 + S_3).  Candidates are taken
 *      in index order and a later one wins a tie (S <= best), which for
 *      {E2M1(6), E1M2} is R6.  The output element is
 *      sign(x) fl32(v s8 s32) (v s8 is exact), the value the dequantizer
 *      returns; a bf16 output is that fp32 rounded to nearest even.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ---------------------------------------------------------------------------
 * Eq. 1-2: value of a non-negative code with exponent field e, mantissa field
 * m, W_M mantissa bits and bias B:  2^(e-B) (1 + m/2^W_M) for e >= 1,
 * 2^(1-B) (m/2^W_M) for e == 0.
 * ------------------------------------------------------------------------- */
static double fp_code_value(int e, int m, int wm, int bias) {
  double frac = (double)m / (double)(1 << wm);
  if (e == 0) return ldexp(frac, 1 - bias);
  return ldexp(1.0 + frac, e - bias);
}

/* E4M3 ("fn" variant, as in NVFP4): W_E=4, W_M=3, B=7; code 0x7F is NaN and
 * is not a value.  Codes 0x00..0x7E are the 127 finite non-negative values. */
double oracle_e4m3_value(int code7) {
  int e = (code7 >> 3) & 0xF, m = code7 & 7;
  return fp_code_value(e, m, 3, 7);
}

/* Round-to-nearest-even onto the E4M3 grid by exhaustive search (R2):
 * the nearest finite value, ties to the code with an even mantissa LSB;
 * anything above 448 saturates to 448 (the nearest finite value). */
int oracle_e4m3_rne(float v) {
  if (v >= 448.0f) return 0x7E;                     /* saturate (R2) */
  int best = 0;
  double bestd = INFINITY;
  for (int c = 0; c <= 0x7E; ++c) {
    double d = fabs((double)v - oracle_e4m3_value(c));
    if (d < bestd || (d == bestd && (c & 1) == 0 && (best & 1) == 1)) {
      best = c;
      bestd = d;
    }
  }
  return best;
}

/* Table 1 / App. B.2 codebooks.  type 0 = E2M1 (W_E=2, W_M=1, bias 1),
 * type 1 = E1M2 (W_E=1, W_M=2, bias 0) followed by the fixed x2 remap of
 * Sec. 3.1.  The payload is [p2 p1 p0]: E2M1 e=[p2p1], m=[p0];
 * E1M2 e=[p2], m=[p1p0]. */
double oracle_fp4_value(int type, int payload) {
  if (type == 0) return fp_code_value((payload >> 1) & 3, payload & 1, 1, 1);
  return 2.0 * fp_code_value((payload >> 2) & 1, payload & 3, 2, 0);
}

/* Stored (pre-remap) E1M2 magnitude, for the Table 1 pin. */
double oracle_e1m2_stored_value(int payload) {
  return fp_code_value((payload >> 2) & 1, payload & 3, 2, 0);
}

/* R4: nearest codebook magnitude to y >= 0, ties to the even payload;
 * y above the maximum lands on the maximum (the nearest value). */
int oracle_fp4_rne(int type, float y) {
  if ((double)y >= oracle_fp4_value(type, 7)) return 7;  /* saturate (R4) */
  int best = 0;
  double bestd = INFINITY;
  for (int p = 0; p < 8; ++p) {
    double d = fabs((double)y - oracle_fp4_value(type, p));
    if (d < bestd || (d == bestd && (p & 1) == 0 && (best & 1) == 1)) {
      best = p;
      bestd = d;
    }
  }
  return best;
}

static float bf16_to_float(uint16_t h) {
  uint32_t u = (uint32_t)h << 16;
  float f;
  memcpy(&f, &u, 4);
  return f;
}

/* One candidate of Algorithm 1 for one 16-element block: scale, quantize,
 * dequantize, error.  a[] holds X_FP8 for the block, B its block max. */
static void candidate_div(int type, float cmax, const float a[16], float B, int* s8code,
                          int payload[16], float* S) {
  float ratio = B / cmax;                           /* fl32(B / c) */
  int code = oracle_e4m3_rne(ratio);                /* E4M3 RNE, R2 */
  float s8 = (float)oracle_e4m3_value(code);        /* exact in fp32 */
  float d[16];
  for (int i = 0; i < 16; ++i) {
    float mag = fabsf(a[i]);
    float y = (s8 > 0.0f) ? mag / s8 : 0.0f;        /* fl32(|a|/s8), R7 */
    int p = oracle_fp4_rne(type, y);                /* R4 */
    float q = (float)oracle_fp4_value(type, p);
    d[i] = q * s8 - mag;                            /* R5, product exact */
    payload[i] = p;
  }
  float se = 0.0f, so = 0.0f;                       /* R5 order */
  for (int i = 0; i < 16; i += 2) se = fmaf(d[i], d[i], se);
  for (int i = 1; i < 16; i += 2) so = fmaf(d[i], d[i], so);
  *S = se + so;
  *s8code = code;
}

/* Algorithm 1's candidates: E2M1 with the block max mapped to 6, E1M2 to 7. */
static void candidate(int type, const float a[16], float B, int* s8code,
                      int payload[16], float* S) {
  candidate_div(type, (type == 0) ? 6.0f : 7.0f, a, B, s8code, payload, S);
}

/* Algorithm 1 over a [rows][K] fp32 tensor (row stride ldx elements).
 *   mode 0 = MixFP4, 1 = E2M1 only (NVFP4), 2 = E1M2 only (NVINT4),
 *   3 = the {E2M1(6), E2M1(4)} set of R14 packed as E2M1 codes with T = 0
 *       (the error arrays then hold S of E2M1(6) and of E2M1(4))
 *   scale_given 0: s32 = fl32(max|X| / 2688) is computed and written to *s32;
 *   scale_given 1: *s32 is read.
 * Optional err_e2m1 / err_e1m2 ([rows][K/16]) receive each block's S.
 * Returns 0, or -1 on a non-finite input or K % 16 != 0. */
int oracle_quantize_f32(const float* x, int64_t rows, int64_t K, int64_t ldx,
                        int mode, int scale_given, float* s32, uint8_t* codes,
                        uint8_t* scales, float* err_e2m1, float* err_e1m2) {
  if (K % 16 != 0) return -1;
  float amax = 0.0f;
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t k = 0; k < K; ++k) {
      float v = x[r * ldx + k];
      if (!isfinite(v)) return -1;
      if (fabsf(v) > amax) amax = fabsf(v);
    }
  float s = scale_given ? *s32 : amax / 2688.0f;   /* 2688 = 6*448 = 7*384 */
  if (!scale_given) *s32 = s;

  int64_t nb = K / 16;
  for (int64_t r = 0; r < rows; ++r) {
    for (int64_t b = 0; b < nb; ++b) {
      float a[16], B = 0.0f;
      int sign[16];
      for (int i = 0; i < 16; ++i) {
        float v = x[r * ldx + b * 16 + i];
        sign[i] = signbit(v) ? 1 : 0;
        a[i] = (s > 0.0f) ? v / s : 0.0f;           /* X_FP8 = X / s32, R1, R7 */
        if (fabsf(a[i]) > B) B = fabsf(a[i]);       /* block-max(|X_FP8|) */
      }
      int c2 = 0, c1 = 0, p2[16], p1[16];
      float S2 = 0.0f, S1 = 0.0f;
      int T;
      const int* p;
      int code;
      if (mode == 3) {
        /* {E2M1(6), E2M1(4)} (R14): both E2M1, T = 0; E2M1(4) wins a tie */
        int c4 = 0, p4[16];
        float S4 = 0.0f;
        candidate(0, a, B, &c2, p2, &S2);
        candidate_div(0, 4.0f, a, B, &c4, p4, &S4);
        T = 0;
        p = (S4 <= S2) ? p4 : p2;
        code = (S4 <= S2) ? c4 : c2;
        if (err_e2m1) err_e2m1[r * nb + b] = S2;
        if (err_e1m2) err_e1m2[r * nb + b] = S4;
      } else {
        if (mode != 2) candidate(0, a, B, &c2, p2, &S2);
        if (mode != 1) candidate(1, a, B, &c1, p1, &S1);
        if (mode == 1) T = 0;
        else if (mode == 2) T = 1;
        else T = (S2 < S1) ? 0 : 1;                 /* R6: strict < */
        p = T ? p1 : p2;
        code = T ? c1 : c2;
      }
      uint8_t* crow = codes + r * (K / 2) + b * 8;
      for (int j = 0; j < 8; ++j) {
        int lo = (sign[2 * j] << 3) | p[2 * j];
        int hi = (sign[2 * j + 1] << 3) | p[2 * j + 1];
        crow[j] = (uint8_t)(lo | (hi << 4));        /* R9 */
      }
      scales[r * nb + b] = (uint8_t)((T << 7) | code);  /* App. B.3 */
      if (mode != 3) {
        if (err_e2m1) err_e2m1[r * nb + b] = S2;
        if (err_e1m2) err_e1m2[r * nb + b] = S1;
      }
    }
  }
  return 0;
}

/* Algorithm 1 over a [rows][K] bf16 tensor (row stride ldx elements): the
 * bf16 values are exact in fp32, so this is oracle_quantize_f32 on them. */
int oracle_quantize(const uint16_t* x, int64_t rows, int64_t K, int64_t ldx,
                    int mode, int scale_given, float* s32, uint8_t* codes,
                    uint8_t* scales, float* err_e2m1, float* err_e1m2) {
  if (K % 16 != 0) return -1;
  float* xf = (float*)malloc((size_t)(rows > 0 ? rows : 1) * (size_t)(K > 0 ? K : 1) * sizeof(float));
  if (!xf) return -1;
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t k = 0; k < K; ++k) xf[r * K + k] = bf16_to_float(x[r * ldx + k]);
  int rc = oracle_quantize_f32(xf, rows, K, K, mode, scale_given, s32, codes, scales, err_e2m1, err_e1m2);
  free(xf);
  return rc;
}

/* R11: the 128-point rotation of every chunk of a bf16 [rows][K] tensor
 * (K % 128 == 0) into fp32 y [rows][K].  signs: 16 bytes, bit i (byte i/8,
 * bit i%8) negates element i of every chunk; NULL for none. */
int oracle_rht(const uint16_t* x, int64_t rows, int64_t K, int64_t ldx, const uint8_t* signs, float* y) {
  if (K % 128 != 0) return -1;
  const float c = (float)(1.0 / sqrt(128.0));     /* RN(1/sqrt(128)) = 0x3DB504F3 */
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t k0 = 0; k0 < K; k0 += 128) {
      float v[128];
      for (int i = 0; i < 128; ++i) {
        float xi = bf16_to_float(x[r * ldx + k0 + i]);
        v[i] = (signs && ((signs[i >> 3] >> (i & 7)) & 1)) ? -xi : xi;
      }
      for (int h = 1; h < 128; h <<= 1)
        for (int i = 0; i < 128; ++i)
          if ((i & h) == 0) {
            float a = v[i], b = v[i + h];
            v[i] = a + b;
            v[i + h] = a - b;
          }
      for (int i = 0; i < 128; ++i) y[r * K + k0 + i] = v[i] * c;
    }
  return 0;
}

/* Decode one element to its value in units of the block scale:
 * sign * v(T, payload) (App. B.2, Sec. 3.1 remap). */
static double decode_unit(uint8_t codebyte, int hi, int T) {
  int nib = hi ? (codebyte >> 4) : (codebyte & 0xF);
  double v = oracle_fp4_value(T, nib & 7);
  return (nib & 8) ? -v : v;
}

/* App. B.3: the block scale is the scale byte with bit 7 forced to 0, and the
 * type bit T = bit 7 selects the payload interpretation. */
static double block_scale(uint8_t s) { return oracle_e4m3_value(s & 0x7F); }

/* out = fl32(sign * v * s8 * s32); the product is exact in double. */
void oracle_dequantize(const uint8_t* codes, const uint8_t* scales, float s32,
                       int64_t rows, int64_t K, float* out) {
  int64_t nb = K / 16;
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t k = 0; k < K; ++k) {
      uint8_t s = scales[r * nb + k / 16];
      double v = decode_unit(codes[r * (K / 2) + k / 2], (int)(k & 1), s >> 7);
      out[r * K + k] = (float)(v * block_scale(s) * (double)s32);
    }
}

/* Plain definition: C[m][n] = sum_k A_deq[m][k] * B_deq[n][k] in float64,
 * with A_deq = v * s8 * s32 exact in double. */
void oracle_gemm_f64(const uint8_t* ac, const uint8_t* as, float as32,
                     const uint8_t* bc, const uint8_t* bs, float bs32,
                     int64_t M, int64_t N, int64_t K, double* C) {
  int64_t nb = K / 16;
  for (int64_t m = 0; m < M; ++m)
    for (int64_t n = 0; n < N; ++n) {
      double acc = 0.0;
      for (int64_t k = 0; k < K; ++k) {
        uint8_t sa = as[m * nb + k / 16], sb = bs[n * nb + k / 16];
        double va = decode_unit(ac[m * (K / 2) + k / 2], (int)(k & 1), sa >> 7) *
                    block_scale(sa) * (double)as32;
        double vb = decode_unit(bc[n * (K / 2) + k / 2], (int)(k & 1), sb >> 7) *
                    block_scale(sb) * (double)bs32;
        acc += va * vb;
      }
      C[m * N + n] = acc;
    }
}

/* Row m of A_deq (float64), for sampled checks at large sizes. */
void oracle_dequant_row_f64(const uint8_t* codes, const uint8_t* scales,
                            float s32, int64_t K, int64_t r, double* out) {
  int64_t nb = K / 16;
  for (int64_t k = 0; k < K; ++k) {
    uint8_t s = scales[r * nb + k / 16];
    out[k] = decode_unit(codes[r * (K / 2) + k / 2], (int)(k & 1), s >> 7) *
             block_scale(s) * (double)s32;
  }
}

/* Integer form of a block scale: s8 = mant * 2^(ex - 10), mant in [0, 15],
 * ex in [1, 15] (Eq. 1 with the subnormal exponent 1 - B). */
static void scale_int(uint8_t s, int* mant, int* ex) {
  int e = (s >> 3) & 0xF, m = s & 7;
  if (e == 0) { *mant = m; *ex = 1; }
  else { *mant = 8 + m; *ex = e; }
}

/* Twice the decoded magnitude as an integer: E2M1 {0,1,2,3,4,6,8,12},
 * E1M2 {0,2,...,14}. */
static int unit2(uint8_t codebyte, int hi, int T) {
  double v = decode_unit(codebyte, hi, T);
  return (int)lrint(2.0 * v);
}

/* App. B.1 Eq. (factor): sum_b (sA_b sB_b) sum_i a_i b_i, with every term an
 * integer times a power of two, accumulated exactly.  The element values are
 * u/2 and the scales mant * 2^(ex-10), so each block contributes
 * mantA*mantB*2^(exA+exB) * sum(uA*uB) in units of 2^-22.  The final value is
 * total * 2^-22 * s32A * s32B, formed in long double. */
void oracle_gemm_exact(const uint8_t* ac, const uint8_t* as, float as32,
                       const uint8_t* bc, const uint8_t* bs, float bs32,
                       int64_t M, int64_t N, int64_t K, long double* C) {
  int64_t nb = K / 16;
  for (int64_t m = 0; m < M; ++m)
    for (int64_t n = 0; n < N; ++n) {
      __int128 total = 0;
      for (int64_t b = 0; b < nb; ++b) {
        uint8_t sa = as[m * nb + b], sb = bs[n * nb + b];
        int ma, ea, mb, eb;
        scale_int(sa, &ma, &ea);
        scale_int(sb, &mb, &eb);
        int64_t dot = 0;
        for (int i = 0; i < 16; ++i) {
          int64_t k = b * 16 + i;
          dot += (int64_t)unit2(ac[m * (K / 2) + k / 2], (int)(k & 1), sa >> 7) *
                 unit2(bc[n * (K / 2) + k / 2], (int)(k & 1), sb >> 7);
        }
        total += (__int128)dot * ma * mb * ((__int128)1 << (ea + eb));
      }
      long double t = (long double)total;
      C[m * N + n] = ldexpl(t, -22) * (long double)as32 * (long double)bs32;
    }
}

/* ---------------------------------------------------------------------------
 * Native block-scaled FP4 operands (the split behind the E2M1 x E2M1
 * tensor-core variant of the MixFP4 GEMM).  A MixFP4 operand is written as
 * the sum of two E2M1 operands that share its block scales:
 *   E2M1 block (T = 0): main = the stored nibble, residual = +0.
 *   E1M2 block (T = 1): the magnitude v = p (Sec. 3.1 remap) is split as
 *     v = e + r, e the largest E2M1 codebook value <= v, r = v - e (which is
 *     0 or 1, both E2M1 values); main = sign | code(e), residual = sign |
 *     code(r), sign = the stored sign bit.
 * Scales: the E4M3 magnitude (bits 6..0; the type bit is dropped because the
 * split codes carry the values) in the tensor core's block-16 scale layout:
 * tiles of 128 rows x 4 blocks (64 K), 512 bytes each, tile (rt, kt) at
 * ((rt * (K / 64)) + kt) * 512, row r of the tile and block b at
 * (r % 32) * 16 + (r / 32) * 4 + b.  Row tiles cover rows rounded up to a
 * multiple of 256; padding bytes are 0.
 * Parity of the value split is pinned on the CPU (the parts' decoded values
 * sum to the MixFP4 value for every nibble and type); the scale layout is a
 * hardware format, parity unpinned on the CPU and checked by the GPU product.
 * ------------------------------------------------------------------------- */
static int e2m1_code_of(double v) {
  for (int q = 0; q < 8; ++q)
    if (oracle_fp4_value(0, q) == v) return q;
  return -1;
}

static void split_nibble(int nib, int T, int* main_nib, int* res_nib) {
  if (!T) {
    *main_nib = nib;
    *res_nib = 0;
    return;
  }
  double v = oracle_fp4_value(1, nib & 7), e = 0.0;
  for (int q = 0; q < 8; ++q) {
    double c = oracle_fp4_value(0, q);
    if (c <= v && c > e) e = c;
  }
  *main_nib = (nib & 8) | e2m1_code_of(e);
  *res_nib = (nib & 8) | e2m1_code_of(v - e);
}

int oracle_split_native(const uint8_t* codes, const uint8_t* scales, int64_t rows, int64_t K,
                        uint8_t* main_codes, uint8_t* res_codes, uint8_t* sf) {
  if (K % 64 != 0) return -1;
  int64_t nb = K / 16, kt_n = K / 64, rt_n = 2 * ((rows + 255) / 256);
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t j = 0; j < K / 2; ++j) {
      int T = scales[r * nb + (2 * j) / 16] >> 7;
      int lo_m, lo_r, hi_m, hi_r;
      split_nibble(codes[r * (K / 2) + j] & 0xF, T, &lo_m, &lo_r);
      split_nibble(codes[r * (K / 2) + j] >> 4, T, &hi_m, &hi_r);
      if (lo_m < 0 || lo_r < 0 || hi_m < 0 || hi_r < 0) return -2;
      main_codes[r * (K / 2) + j] = (uint8_t)(lo_m | (hi_m << 4));
      res_codes[r * (K / 2) + j] = (uint8_t)(lo_r | (hi_r << 4));
    }
  memset(sf, 0, (size_t)(rt_n * kt_n * 512));
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t b = 0; b < nb; ++b) {
      int64_t rt = r / 128, rr = r % 128, kt = b / 4;
      sf[(rt * kt_n + kt) * 512 + (rr % 32) * 16 + (rr / 32) * 4 + (b % 4)] = scales[r * nb + b] & 0x7F;
    }
  return 0;
}

/* ---------------------------------------------------------------------------
 * 2D block quantization (Sec. 3.2: weights are quantized in 2D blocks in the
 * training flow; Sec. 4.2 pre-training recipe), reading R12: Algorithm 1 with
 * the block taken as a 16 x 16 tile.
 * ------------------------------------------------------------------------- */
static float tree16(const float s[16]) {
  float l1[8], l2[4], l3[2];
  for (int i = 0; i < 8; ++i) l1[i] = s[2 * i] + s[2 * i + 1];
  for (int i = 0; i < 4; ++i) l2[i] = l1[2 * i] + l1[2 * i + 1];
  for (int i = 0; i < 2; ++i) l3[i] = l2[2 * i] + l2[2 * i + 1];
  return l3[0] + l3[1];
}

int oracle_quantize_2d_f32(const float* x, int64_t rows, int64_t K, int64_t ldx, int mode, int scale_given,
                           float* s32, uint8_t* codes, uint8_t* scales) {
  if (K % 16 != 0) return -1;
  float amax = 0.0f;
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t k = 0; k < K; ++k) {
      float v = x[r * ldx + k];
      if (!isfinite(v)) return -1;
      if (fabsf(v) > amax) amax = fabsf(v);
    }
  float s = scale_given ? *s32 : amax / 2688.0f;   /* Alg. 1 tensor scale */
  if (!scale_given) *s32 = s;
  int64_t nb = K / 16;
  for (int64_t r0 = 0; r0 < rows; r0 += 16) {
    for (int64_t b = 0; b < nb; ++b) {
      float a[16][16], B = 0.0f;
      int sign[16][16];
      for (int i = 0; i < 16; ++i)
        for (int k = 0; k < 16; ++k) {
          float v = (r0 + i < rows) ? x[(r0 + i) * ldx + b * 16 + k] : 0.0f;  /* missing rows: zeros */
          sign[i][k] = signbit(v) ? 1 : 0;
          a[i][k] = (s > 0.0f) ? v / s : 0.0f;     /* X_FP8 = X / s32, R1, R7 */
          if (fabsf(a[i][k]) > B) B = fabsf(a[i][k]);  /* tile max */
        }
      int c2 = 0, c1 = 0, p2[16][16], p1[16][16];
      float S2r[16], S1r[16], S2 = 0.0f, S1 = 0.0f;
      for (int i = 0; i < 16; ++i) {
        S2r[i] = S1r[i] = 0.0f;
        if (mode != 2) candidate(0, a[i], B, &c2, p2[i], &S2r[i]);
        if (mode != 1) candidate(1, a[i], B, &c1, p1[i], &S1r[i]);
      }
      if (mode != 2) S2 = tree16(S2r);
      if (mode != 1) S1 = tree16(S1r);
      int T;
      if (mode == 1) T = 0;
      else if (mode == 2) T = 1;
      else T = (S2 < S1) ? 0 : 1;                   /* R6 on the tile */
      int code = T ? c1 : c2;
      for (int i = 0; i < 16 && r0 + i < rows; ++i) {
        const int* p = T ? p1[i] : p2[i];
        uint8_t* crow = codes + (r0 + i) * (K / 2) + b * 8;
        for (int j = 0; j < 8; ++j) {
          int lo = (sign[i][2 * j] << 3) | p[2 * j];
          int hi = (sign[i][2 * j + 1] << 3) | p[2 * j + 1];
          crow[j] = (uint8_t)(lo | (hi << 4));      /* R9 */
        }
        scales[(r0 + i) * nb + b] = (uint8_t)((T << 7) | code);
      }
    }
  }
  return 0;
}

int oracle_quantize_2d(const uint16_t* x, int64_t rows, int64_t K, int64_t ldx, int mode, int scale_given,
                       float* s32, uint8_t* codes, uint8_t* scales) {
  if (K % 16 != 0) return -1;
  float* xf = (float*)malloc((size_t)(rows > 0 ? rows : 1) * (size_t)(K > 0 ? K : 1) * sizeof(float));
  if (!xf) return -1;
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t k = 0; k < K; ++k) xf[r * K + k] = bf16_to_float(x[r * ldx + k]);
  int rc = oracle_quantize_2d_f32(xf, rows, K, K, mode, scale_given, s32, codes, scales);
  free(xf);
  return rc;
}

/* The transposed operand of a 2D-quantized [rows][K] tensor (rows % 16 == 0,
 * K % 16 == 0): element (r, k) of the input is element (k, r) of the output
 * (codes_t [K][rows/2], scales_t [K][rows/16]); the scale of output block
 * (k, r/16) is the scale byte shared by tile (r/16, k/16).  Returns -2 if a
 * tile's rows do not share one scale byte (not a 2D-quantized tensor). */
int oracle_transpose_2d(const uint8_t* codes, const uint8_t* scales, int64_t rows, int64_t K, uint8_t* codes_t,
                        uint8_t* scales_t) {
  if (rows % 16 != 0 || K % 16 != 0) return -1;
  int64_t nb = K / 16, nbt = rows / 16;
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t b = 0; b < nb; ++b)
      if (scales[r * nb + b] != scales[(r / 16) * 16 * nb + b]) return -2;
  for (int64_t k = 0; k < K; ++k) {
    for (int64_t j = 0; j < rows / 2; ++j) {
      int r = (int)(2 * j);
      int lo = (codes[r * (K / 2) + k / 2] >> (4 * (k % 2))) & 0xF;
      int hi = (codes[(r + 1) * (K / 2) + k / 2] >> (4 * (k % 2))) & 0xF;
      codes_t[k * (rows / 2) + j] = (uint8_t)(lo | (hi << 4));
    }
    for (int64_t t = 0; t < nbt; ++t) scales_t[k * nbt + t] = scales[(t * 16) * nb + k / 16];
  }
  return 0;
}

/* ---------------------------------------------------------------------------
 * Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11): ten rounds of two 32x32
 * -> 64-bit products with the multipliers 0xD2511F53 and 0xCD9E8D57, the key
 * bumped by (0x9E3779B9, 0xBB67AE85) between rounds.
 * ------------------------------------------------------------------------- */
void oracle_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
  uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3], k0 = key[0], k1 = key[1];
  for (int round = 0; round < 10; ++round) {
    if (round > 0) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    uint64_t p0 = (uint64_t)0xD2511F53u * c0;
    uint64_t p1 = (uint64_t)0xCD9E8D57u * c2;
    uint32_t n0 = (uint32_t)(p1 >> 32) ^ c1 ^ k0;
    uint32_t n1 = (uint32_t)p1;
    uint32_t n2 = (uint32_t)(p0 >> 32) ^ c3 ^ k1;
    uint32_t n3 = (uint32_t)p0;
    c0 = n0; c1 = n1; c2 = n2; c3 = n3;
  }
  out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

/* The R13 uniform of element e: a multiple of 2^-24 in [0, 1). */
float oracle_sr_uniform(uint64_t seed, uint64_t offset, uint64_t e) {
  uint32_t ctr[4] = {(uint32_t)(e / 4), (uint32_t)((e / 4) >> 32), (uint32_t)offset, (uint32_t)(offset >> 32)};
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  uint32_t w[4];
  oracle_philox4x32_10(ctr, key, w);
  return (float)(w[e % 4] >> 8) * 0x1p-24f;
}

/* R13: the stochastic payload of magnitude m in format `type`, by search over
 * the codebook for the neighbours l <= m < u. */
int oracle_sr_payload(int type, float m, float eps) {
  double lo = -1.0, hi = INFINITY;
  int plo = 0, phi = -1;
  for (int p = 0; p < 8; ++p) {
    double v = oracle_fp4_value(type, p);
    if (v <= m && v > lo) { lo = v; plo = p; }
    if (v > m && v < hi) { hi = v; phi = p; }
  }
  if (phi < 0) return plo;                          /* at or above the maximum */
  double f = ((double)m - lo) / (hi - lo);          /* exact: an fp32 value */
  return ((double)eps < f) ? phi : plo;
}

/* Algorithm 1 with stochastic rounding of the chosen format (R13) on a
 * [rows][K] bf16 tensor; arguments as oracle_quantize plus seed and offset. */
int oracle_quantize_sr(const uint16_t* x, int64_t rows, int64_t K, int64_t ldx, int mode, int scale_given,
                       float* s32, uint64_t seed, uint64_t offset, uint8_t* codes, uint8_t* scales) {
  if (K % 16 != 0) return -1;
  int rc = oracle_quantize(x, rows, K, ldx, mode, scale_given, s32, codes, scales, NULL, NULL);
  if (rc != 0) return rc;
  float s = *s32;
  int64_t nb = K / 16;
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t b = 0; b < nb; ++b) {
      int T = scales[r * nb + b] >> 7;
      float s8 = (float)oracle_e4m3_value(scales[r * nb + b] & 0x7F);
      for (int i = 0; i < 16; ++i) {
        int64_t k = b * 16 + i;
        float v = bf16_to_float(x[r * ldx + k]);
        float a = (s > 0.0f) ? v / s : 0.0f;                    /* R1, R7 */
        float m = (s8 > 0.0f) ? fabsf(a) / s8 : 0.0f;           /* R4's quotient */
        float eps = oracle_sr_uniform(seed, offset, (uint64_t)(r * K + k));
        int p = oracle_sr_payload(T, m, eps);
        int nib = ((signbit(v) ? 1 : 0) << 3) | p;
        uint8_t* byte = codes + r * (K / 2) + k / 2;
        *byte = (uint8_t)((k % 2) ? ((*byte & 0x0F) | (nib << 4)) : ((*byte & 0xF0) | nib));
      }
    }
  return 0;
}

/* ---------------------------------------------------------------------------
 * R14: candidate-set and block-size ablation (Sec. 2.4, Sec. 4.3 Table 5).
 * ------------------------------------------------------------------------- */

/* Magnitude of payload p (0..7) under candidate c (R14). */
double oracle_cand_value(int c, int p) {
  if (c == 0 || c == 2) return oracle_fp4_value(0, p);
  if (c == 1) return oracle_fp4_value(1, p);
  return fp_code_value(p, 0, 0, 3);                 /* E3M0: W_E=3, W_M=0, bias 3 */
}

/* Block-max divisor of candidate c: the value the block max is mapped to. */
float oracle_cand_divisor(int c) {
  return c == 0 ? 6.0f : c == 1 ? 7.0f : c == 2 ? 4.0f : 16.0f;
}

/* R4 on candidate c's codebook: the nearest magnitude, ties to the even
 * payload, saturating at the largest. */
int oracle_cand_rne(int c, float y) {
  if ((double)y >= oracle_cand_value(c, 7)) return 7;
  int best = 0;
  double bestd = INFINITY;
  for (int p = 0; p < 8; ++p) {
    double d = fabs((double)y - oracle_cand_value(c, p));
    if (d < bestd || (d == bestd && (p & 1) == 0 && (best & 1) == 1)) {
      best = p;
      bestd = d;
    }
  }
  return best;
}

/* Error sum of one block of g element errors (R5 per 16-element chunk, even
 * and odd chains; pairwise tree over the chunks for g > 16). */
static float block_error_sum(const float* d, int g) {
  if (g <= 16) {
    float se = 0.0f, so = 0.0f;
    for (int i = 0; i < g; i += 2) se = fmaf(d[i], d[i], se);
    for (int i = 1; i < g; i += 2) so = fmaf(d[i], d[i], so);
    return se + so;
  }
  float s[4];
  int n = g / 16;
  for (int j = 0; j < n; ++j) s[j] = block_error_sum(d + 16 * j, 16);
  for (; n > 1; n /= 2)
    for (int j = 0; j < n / 2; ++j) s[j] = s[2 * j] + s[2 * j + 1];
  return s[0];
}

/* Quantize-dequantize of a [rows][K] bf16 tensor (row stride ldx elements)
 * under the candidate set cand_mask (bit c = candidate c of R14) and block
 * size g.  scale_given / s32 as in oracle_quantize.  out: fp32 [rows][K];
 * choice: [rows][K/g] candidate index, or NULL.  Returns 0, or -1 on a bad
 * argument or a non-finite input. */
int oracle_fake_quantize(const uint16_t* x, int64_t rows, int64_t K, int64_t ldx, int cand_mask, int g,
                         int scale_given, float* s32, float* out, uint8_t* choice) {
  if (g != 8 && g != 16 && g != 32 && g != 64) return -1;
  if (K % 16 != 0 || K % g != 0 || (cand_mask & 15) == 0 || (cand_mask & ~15) != 0) return -1;
  float amax = 0.0f;
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t k = 0; k < K; ++k) {
      float v = bf16_to_float(x[r * ldx + k]);
      if (!isfinite(v)) return -1;
      if (fabsf(v) > amax) amax = fabsf(v);
    }
  float s = scale_given ? *s32 : amax / 2688.0f;
  if (!scale_given) *s32 = s;
  int64_t nb = K / g;
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t b = 0; b < nb; ++b) {
      float a[64], B = 0.0f;
      int neg[64];
      for (int i = 0; i < g; ++i) {
        float v = bf16_to_float(x[r * ldx + b * g + i]);
        neg[i] = signbit(v) ? 1 : 0;
        a[i] = (s > 0.0f) ? fabsf(v) / s : 0.0f;     /* R1, R7 */
        if (a[i] > B) B = a[i];
      }
      int best = -1;
      float best_S = 0.0f, best_s8 = 0.0f, best_q[64];
      for (int c = 0; c < 4; ++c) {
        if (!((cand_mask >> c) & 1)) continue;
        float s8 = (float)oracle_e4m3_value(oracle_e4m3_rne(B / oracle_cand_divisor(c)));  /* R2 */
        float q[64], d[64];
        for (int i = 0; i < g; ++i) {
          float y = (s8 > 0.0f) ? a[i] / s8 : 0.0f;
          q[i] = (float)oracle_cand_value(c, oracle_cand_rne(c, y));
          d[i] = q[i] * s8 - a[i];                    /* the product is exact */
        }
        float S = block_error_sum(d, g);
        if (best < 0 || S <= best_S) {                /* a later candidate wins a tie */
          best = c;
          best_S = S;
          best_s8 = s8;
          memcpy(best_q, q, sizeof(float) * (size_t)g);
        }
      }
      for (int i = 0; i < g; ++i) {
        float o = (float)((double)best_q[i] * (double)best_s8 * (double)s);
        out[r * K + b * g + i] = neg[i] ? -o : o;
      }
      if (choice) choice[r * nb + b] = (uint8_t)best;
    }
  return 0;
}

/* binary32 -> bfloat16 bits, round to nearest, ties to even (finite input). */
uint16_t oracle_f32_to_bf16(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  uint32_t keep = u >> 16, rest = u & 0xFFFFu;
  if (rest > 0x8000u || (rest == 0x8000u && (keep & 1u))) keep += 1u;
  return (uint16_t)keep;
}

/* oracle_f32_to_bf16 over an array of n values. */
void oracle_f32_to_bf16_array(const float* f, int64_t n, uint16_t* out) {
  for (int64_t i = 0; i < n; ++i) out[i] = oracle_f32_to_bf16(f[i]);
}
