/* Host check of the two-instruction division by a known divisor used by the
 * CUDA quantizer (Brisebarre, Muller, Raina, IEEE Trans. Computers 53(8),
 * 2004):  q = RN(a*zh + RN(a*zl)),  zh = RN(1/b),  zl = RN(RN(1 - b*zh)/b),
 * compared bit for bit with C's IEEE '/'.  Compiled with -ffp-contract=off;
 * fmaf is the correctly rounded C99 fused multiply-add.
 *
 *  (1) |a| / s8: every fp32 significand of a against every E4M3 significand,
 *      normal (exponents 0 and 8) and subnormal (m * 2^-9).
 *  (2) B / 6 and B / 7: every significand of B at exponents -100..12.
 *  (3) x / s32: the kernel accepts the method for a tensor when it returns
 *      the IEEE quotient for all 128 bf16 significands of x at exponent 0
 *      and the remainder 1 - s32*zh is 0 or at least 2^-44 in magnitude.
 *      For every s32 significand this check replays that rule, counts the
 *      rejected ones, and for the accepted ones requires the IEEE quotient at
 *      other exponents of x and s32 too (the scaling the rule relies on).
 * Prints one "mismatches=" line per check and exits nonzero on any mismatch. */
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <string.h>

static float f_of(uint32_t u) { float f; memcpy(&f, &u, 4); return f; }
static uint32_t u_of(float f) { uint32_t u; memcpy(&u, &f, 4); return u; }

static void consts(float b, float* zh, float* zl) {
  *zh = 1.0f / b;
  *zl = fmaf(-b, *zh, 1.0f) / b;
}
static float kdiv(float a, float zh, float zl) { return fmaf(a, zh, a * zl); }
static long bad_pair(float a, float b, float zh, float zl) { return u_of(kdiv(a, zh, zl)) != u_of(a / b); }

int main(void) {
  int rc = 0;
  long bad = 0;
  /* (1) */
#pragma omp parallel for reduction(+ : bad) schedule(static)
  for (uint32_t ma = 0; ma < (1u << 23); ++ma) {
    const float a = f_of(0x3F800000u | ma);
    for (int m = 0; m < 8; ++m) {
      float zh, zl, b = 1.0f + m / 8.0f;
      consts(b, &zh, &zl);
      bad += bad_pair(a, b, zh, zl);
      b = ldexpf(1.0f + m / 8.0f, 8);
      consts(b, &zh, &zl);
      bad += bad_pair(ldexpf(a, -20), b, zh, zl);
      if (m) {
        b = ldexpf((float)m, -9);
        consts(b, &zh, &zl);
        bad += bad_pair(ldexpf(a, -3), b, zh, zl);
      }
    }
  }
  printf("a/s8 mismatches=%ld\n", bad);
  if (bad) rc = 1;
  /* (2) */
  bad = 0;
  float zh6, zl6, zh7, zl7;
  consts(6.0f, &zh6, &zl6);
  consts(7.0f, &zh7, &zl7);
#pragma omp parallel for reduction(+ : bad) schedule(static)
  for (uint32_t ma = 0; ma < (1u << 23); ++ma)
    for (int e = -100; e <= 12; e += 16) {
      const float a = ldexpf(f_of(0x3F800000u | ma), e);
      bad += bad_pair(a, 6.0f, zh6, zl6) + bad_pair(a, 7.0f, zh7, zl7);
    }
  printf("B/6,B/7 mismatches=%ld\n", bad);
  if (bad) rc = 1;
  /* (3) */
  bad = 0;
  long rejected = 0;
  const int xe[3] = {-81, -40, 20}, se[3] = {-20, 7, 99};
#pragma omp parallel for reduction(+ : bad, rejected) schedule(dynamic, 4096)
  for (uint32_t mb = 0; mb < (1u << 23); ++mb) {
    const float s = f_of(0x3F800000u | mb);
    float zh, zl;
    consts(s, &zh, &zl);
    const float rem = fmaf(-s, zh, 1.0f);
    int ok = (rem == 0.0f || fabsf(rem) >= 0x1p-44f);
    for (uint32_t mx = 0; ok && mx < 128; ++mx)
      if (bad_pair(f_of(0x3F800000u | (mx << 16)), s, zh, zl)) ok = 0;
    if (!ok) {
      ++rejected;
      continue;
    }
    for (int i = 0; i < 3; ++i) {
      const float b = ldexpf(s, se[i]);
      float bh, bl;
      consts(b, &bh, &bl);
      for (uint32_t mx = 0; mx < 128; mx += 1) {
        const float x = ldexpf(f_of(0x3F800000u | (mx << 16)), xe[i] + se[i]);
        bad += bad_pair(x, b, bh, bl);
      }
    }
  }
  printf("x/s32 rejected=%ld accepted mismatches=%ld\n", rejected, bad);
  if (bad) rc = 1;
  return rc;
}
