// Device pieces shared by the GEMM kernels: 16-byte shared-memory moves, the
// vector fp32 reduction into global memory, and the persistent work schedule
// of a CTA pair (whole tiles, then stream-K slices).
#pragma once
#include <cstdint>

namespace mixfp4 {

// Longest run of K accumulated into one TMEM accumulator by any GEMM kernel.
// The tensor cores' fp32 accumulation drifts from the exact sum by an amount
// that grows with the number of K steps added into one accumulator (on
// operands whose outlier channels coincide, about 1e-6 of |A|.|B| per 1024 of
// K, measured on this part); runs are cut at this length and their partial
// sums added into C in fp32, which keeps the GEMMs within 1e-5 of |A|.|B|
// for any K.
constexpr int kAccumChunkK = 4096;

__device__ __forceinline__ void sts128(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" :: "r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}
__device__ __forceinline__ void sts32(uint32_t addr, uint32_t a) {
  asm volatile("st.shared.b32 [%0], %1;" :: "r"(addr), "r"(a) : "memory");
}
__device__ __forceinline__ uint32_t lds32(uint32_t addr) {
  uint32_t v;
  asm volatile("ld.shared.b32 %0, [%1];" : "=r"(v) : "r"(addr) : "memory");
  return v;
}
__device__ __forceinline__ uint4 lds128(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.b32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr) : "memory");
  return v;
}
__device__ __forceinline__ uint2 lds64(uint32_t addr) {
  uint2 v;
  asm volatile("ld.shared.v2.b32 {%0,%1}, [%2];" : "=r"(v.x), "=r"(v.y) : "r"(addr) : "memory");
  return v;
}
__device__ __forceinline__ void red_add_v4(float* p, float a, float b, float c, float d) {
  asm volatile("red.global.add.v4.f32 [%0], {%1,%2,%3,%4};" :: "l"(p), "f"(a), "f"(b), "f"(c), "f"(d)
               : "memory");
}

// Work schedule of one CTA pair, walked identically by every role.  Tiles
// below dp_tiles are whole-tile work, dealt round-robin (tile = cluster,
// cluster + nclusters, ...).  The (tile, 256-wide K slice) units of the
// remaining tiles are split evenly over all pairs (stream-K).  Every segment
// is also cut where the K slice index crosses a multiple of `chunk`, so no
// accumulation runs longer than chunk slices.  The first segment of a whole
// tile is stored into C (`store`); every other segment is added into C
// (after the first segment of its tile, or into rows the host zeroed).
struct Sched {
  int t, dp_tiles, nclusters, num_kc, chunk, kd;
  long long u, u_end;
  bool store;
  __device__ Sched(int cluster, int ncl, int dp, int ntiles, int nkc, int chunk_kc)
      : t(cluster), dp_tiles(dp), nclusters(ncl), num_kc(nkc), chunk(chunk_kc > 0 ? chunk_kc : nkc), kd(0),
        store(false) {
    const long long sk_units = (long long)(ntiles - dp) * nkc;
    u = sk_units * cluster / ncl;
    u_end = sk_units * (cluster + 1) / ncl;
  }
  // Next segment: tile, K slices [k0, k1).  False when the pair is done.
  __device__ bool next(int& tile, int& k0, int& k1) {
    if (t < dp_tiles) {
      tile = t;
      k0 = kd;
      k1 = (kd / chunk + 1) * chunk < num_kc ? (kd / chunk + 1) * chunk : num_kc;
      store = kd == 0;
      kd = k1;
      if (kd >= num_kc) {
        kd = 0;
        t += nclusters;
      }
      return true;
    }
    if (u >= u_end) return false;
    const long long tt = u / num_kc;
    long long end = (tt + 1) * num_kc < u_end ? (tt + 1) * num_kc : u_end;
    const int kb = (int)(u - tt * num_kc);
    const long long cend = tt * num_kc + (long long)(kb / chunk + 1) * chunk;
    if (cend < end) end = cend;
    tile = dp_tiles + (int)tt;
    k0 = kb;
    k1 = k0 + (int)(end - u);
    store = false;
    u = end;
    return true;
  }
};

}  // namespace mixfp4
