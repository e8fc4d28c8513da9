// Inline-PTX helpers for sm_103a: packed fp32 arithmetic, FP8/FP4 conversions
// and wide global memory access.  Every helper maps to one PTX instruction.
#pragma once
#include <cstdint>

namespace mixfp4 {

typedef unsigned long long u64;

// ---- packed fp32 pairs (lo = first element, hi = second) ------------------
__device__ __forceinline__ u64 pack2(float lo, float hi) {
  u64 r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void unpack2(u64 v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ u64 bits2(uint32_t lo, uint32_t hi) {
  return (u64)lo | ((u64)hi << 32);
}
// Each lane is an IEEE fma / mul / add, rounded to nearest-even.
__device__ __forceinline__ u64 fma2(u64 a, u64 b, u64 c) {
  u64 d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ u64 mul2(u64 a, u64 b) {
  u64 d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ u64 add2(u64 a, u64 b) {
  u64 d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ u64 sub2(u64 a, u64 b) {
  u64 d;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

// ---- programmatic dependent launch ----------------------------------------
// Let the next kernel on the stream, if launched as a programmatic dependent,
// start its prologue now.
__device__ __forceinline__ void griddep_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
// Wait until the preceding kernel on the stream has completed and its memory
// operations are visible (returns at once when this kernel was not launched
// as a programmatic dependent).
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

__device__ __forceinline__ float max3f(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// ---- FP8 / FP4 conversions ---------------------------------------------------
// Two fp32 -> two E4M3 bytes, round-to-nearest-even, saturating to +-448.
// The first operand lands in the HIGH byte.
__device__ __forceinline__ uint16_t cvt_e4m3x2(float hi, float lo) {
  uint16_t d;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(d) : "f"(hi), "f"(lo));
  return d;
}
// Two E4M3 bytes -> f16x2 (exact); high byte -> high half.
__device__ __forceinline__ uint32_t cvt_f16x2_from_e4m3x2(uint16_t v) {
  uint32_t d;
  asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(d) : "h"(v));
  return d;
}
// Two fp32 -> two E2M1 nibbles in one byte, RNE, saturating to +-6.
// The first operand lands in the HIGH nibble.
__device__ __forceinline__ uint32_t cvt_e2m1x2(float hi, float lo) {
  uint32_t d;
  asm("{ .reg .b8 t; cvt.rn.satfinite.e2m1x2.f32 t, %1, %2; cvt.u32.u8 %0, t; }"
      : "=r"(d) : "f"(hi), "f"(lo));
  return d;
}
// One byte of two E2M1 nibbles -> f16x2 (exact); high nibble -> high half.
__device__ __forceinline__ uint32_t cvt_f16x2_from_e2m1x2(uint32_t byte) {
  uint32_t d;
  asm("{ .reg .b8 t; cvt.u8.u32 t, %1; cvt.rn.f16x2.e2m1x2 %0, t; }" : "=r"(d) : "r"(byte));
  return d;
}
__device__ __forceinline__ void f16x2_to_f32(uint32_t h2, float& lo, float& hi) {
  asm("{ .reg .f16 a, b; mov.b32 {a, b}, %2; cvt.f32.f16 %0, a; cvt.f32.f16 %1, b; }"
      : "=f"(lo), "=f"(hi) : "r"(h2));
}

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
  uint32_t d;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
  return d;
}

// ---- wide global memory access ------------------------------------------------
// 32-byte streaming load (read once, do not keep in L1).
__device__ __forceinline__ void ldg256_stream(const void* p, uint32_t v[8]) {
  asm volatile("ld.global.nc.L1::no_allocate.v8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
               : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]),
                 "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7])
               : "l"(p));
}
__device__ __forceinline__ void stg256(void* p, const uint32_t v[8]) {
  asm volatile("st.global.v8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};"
               :: "l"(p), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]),
                  "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]) : "memory");
}
__device__ __forceinline__ void stg64(void* p, uint32_t lo, uint32_t hi) {
  asm volatile("st.global.v2.b32 [%0], {%1,%2};" :: "l"(p), "r"(lo), "r"(hi) : "memory");
}

}  // namespace mixfp4
