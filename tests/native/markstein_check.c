/* Host check of the division method used by the CUDA quantizer: with
 * r = RN(1/b),  q0 = RN(a*r), e = RN(a - q0*b) (one fma), q = RN(q0 + e*r)
 * (one fma) must equal the IEEE quotient RN(a/b) (Markstein 1990).  The
 * checks enumerate every significand pair that the quantizer can present,
 * plus exponent edges.  Compiled with -ffp-contract=off; fmaf is the
 * correctly rounded C99 fused multiply-add.  Prints the number of mismatches
 * per check and exits nonzero on any. */
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

static float f_of(uint32_t u) { float f; memcpy(&f, &u, 4); return f; }
static uint32_t u_of(float f) { uint32_t u; memcpy(&u, &f, 4); return u; }

static float mdiv(float a, float b, float r) {
  float q0 = a * r;
  float e = fmaf(-q0, b, a);
  return fmaf(e, r, q0);
}

static long check_pair(float a, float b) {
  float r = 1.0f / b;
  float q = mdiv(a, b, r);
  float t = a / b;
  return u_of(q) != u_of(t);
}

int main(int argc, char** argv) {
  long bad;
  int rc = 0;
  /* (1) x / s32: every bf16 significand (128) x every fp32 significand of s32,
   * numerator exponents 0 and -90 (well above 2^-102), s32 exponents 0 and 30. */
  const int ea[2] = {0, -90}, eb[2] = {0, 30};
  for (int i = 0; i < 2; ++i)
    for (int j = 0; j < 2; ++j) {
      bad = 0;
#pragma omp parallel for reduction(+ : bad) schedule(static)
      for (uint32_t ma = 0; ma < 128; ++ma) {
        float a = ldexpf(f_of(0x3F800000u | (ma << 16)), ea[i]);
        for (uint32_t mb = 0; mb < (1u << 23); ++mb) {
          float b = ldexpf(f_of(0x3F800000u | mb), eb[j]);
          bad += check_pair(a, b);
        }
      }
      printf("x/s32 ea=%d eb=%d mismatches=%ld\n", ea[i], eb[j], bad);
      if (bad) rc = 1;
    }
  /* (2) |a| / s8: every fp32 significand of a x every E4M3 value's significand
   * (8 normal significands and the subnormal values m * 2^-9). */
  bad = 0;
#pragma omp parallel for reduction(+ : bad) schedule(static)
  for (uint32_t ma = 0; ma < (1u << 23); ++ma) {
    float a = f_of(0x3F800000u | ma);
    for (int m = 0; m < 8; ++m) {
      bad += check_pair(a, 1.0f + m / 8.0f);
      bad += check_pair(ldexpf(a, -20), ldexpf(1.0f + m / 8.0f, 8));
      if (m) bad += check_pair(ldexpf(a, -3), ldexpf((float)m, -9));
    }
  }
  printf("a/s8 mismatches=%ld\n", bad);
  if (bad) rc = 1;
  /* (3) B / 6 and B / 7 over every significand of B at several exponents. */
  bad = 0;
#pragma omp parallel for reduction(+ : bad) schedule(static)
  for (uint32_t ma = 0; ma < (1u << 23); ++ma)
    for (int e = -100; e <= 12; e += 16) {
      float a = ldexpf(f_of(0x3F800000u | ma), e);
      bad += check_pair(a, 6.0f) + check_pair(a, 7.0f);
    }
  printf("B/6,B/7 mismatches=%ld\n", bad);
  if (bad) rc = 1;
  /* (4) exponent edges: numerators down to 2^-102 with quotients >= 2^-125,
   * random significands. */
  bad = 0;
  srand(12345);
  for (int it = 0; it < 4000000; ++it) {
    uint32_t ma = ((uint32_t)rand() ^ ((uint32_t)rand() << 15)) & 0x7FFFFF;
    uint32_t mb = ((uint32_t)rand() ^ ((uint32_t)rand() << 15)) & 0x7FFFFF;
    int xe = -102 + rand() % 230;
    int be = -20 + rand() % 121;
    float a = ldexpf(f_of(0x3F800000u | ma), xe);
    float b = ldexpf(f_of(0x3F800000u | mb), be);
    if (!isfinite(a / b) || fabsf(a / b) < 0x1p-125f) continue;
    bad += check_pair(a, b);
  }
  printf("edges mismatches=%ld\n", bad);
  if (bad) rc = 1;
  return rc;
}
