// Device pieces shared by the GEMM kernels: 16-byte shared-memory moves, the
// vector fp32 reduction into global memory, and the persistent work schedule
// of a CTA pair (whole tiles, then stream-K slices).
#pragma once
#include <cstdint>

namespace mixfp4 {

__device__ __forceinline__ void sts128(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" :: "r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}
__device__ __forceinline__ void sts32(uint32_t addr, uint32_t a) {
  asm volatile("st.shared.b32 [%0], %1;" :: "r"(addr), "r"(a) : "memory");
}
__device__ __forceinline__ uint4 lds128(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.b32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr) : "memory");
  return v;
}
__device__ __forceinline__ void red_add_v4(float* p, float a, float b, float c, float d) {
  asm volatile("red.global.add.v4.f32 [%0], {%1,%2,%3,%4};" :: "l"(p), "f"(a), "f"(b), "f"(c), "f"(d)
               : "memory");
}

// Work schedule of one CTA pair, walked identically by every role.  Tiles
// below dp_tiles are whole-tile work, dealt round-robin (tile = cluster,
// cluster + nclusters, ...).  The (tile, 256-wide K slice) units of the
// remaining tiles are split evenly over all pairs (stream-K) and cut into
// segments at tile edges; a segment that is not a whole tile is added into C
// (which the host zeroed over those tiles).
struct Sched {
  int t, dp_tiles, nclusters, num_kc;
  long long u, u_end;
  __device__ Sched(int cluster, int ncl, int dp, int ntiles, int nkc)
      : t(cluster), dp_tiles(dp), nclusters(ncl), num_kc(nkc) {
    const long long sk_units = (long long)(ntiles - dp) * nkc;
    u = sk_units * cluster / ncl;
    u_end = sk_units * (cluster + 1) / ncl;
  }
  // Next segment: tile, K slices [k0, k1).  False when the pair is done.
  __device__ bool next(int& tile, int& k0, int& k1) {
    if (t < dp_tiles) {
      tile = t;
      k0 = 0;
      k1 = num_kc;
      t += nclusters;
      return true;
    }
    if (u >= u_end) return false;
    const long long tt = u / num_kc;
    const long long end = (tt + 1) * num_kc < u_end ? (tt + 1) * num_kc : u_end;
    tile = dp_tiles + (int)tt;
    k0 = (int)(u - tt * num_kc);
    k1 = k0 + (int)(end - u);
    u = end;
    return true;
  }
};

}  // namespace mixfp4
