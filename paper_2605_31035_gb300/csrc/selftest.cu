// Self-test of the bounded pipeline waits used by the GEMM kernels: one CTA
// waits (a) on an mbarrier whose phase completes, (b) on one that nothing
// ever arrives on (an injected missed arrival), and (c) on the latter with
// its abort flag raised.  (a) must succeed; (b) must give up after the time
// limit and (c) at once, each recording a status bit, so a lost arrival in a
// real pipeline ends in an error the host can read instead of a hang.
#include <cuda_runtime.h>
#include <cstdint>

#include "kernels.cuh"
#include "sm100.cuh"

namespace mixfp4 {
namespace {

using namespace sm100;

__global__ void bounded_wait_selftest_kernel(uint32_t* status, uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bars[2];
  __shared__ int abort_flag;
  if (threadIdx.x != 0) return;
  const uint32_t done = smem_u32(&bars[0]), lost = smem_u32(&bars[1]);
  mbar_init(done, 1);
  mbar_init(lost, 1);
  abort_flag = 0;
  fence_mbar_init();
  mbar_arrive(done);  // completes phase 0 of `done`
  uint32_t bits = 0;
  if (!mbar_wait(done, 0, &abort_flag, limit_ns)) bits |= 1u;           // must not be set
  const uint64_t t0 = globaltimer();
  if (!mbar_wait(lost, 0, &abort_flag, limit_ns)) bits |= 2u;           // must be set: timed out
  if (globaltimer() - t0 >= limit_ns) bits |= 4u;                       // and only after the limit
  abort_flag = 1;
  if (!mbar_wait(lost, 0, &abort_flag, limit_ns)) bits |= 8u;           // must be set: aborted
  atomicOr(status, bits);
}

}  // namespace

int launch_bounded_wait_selftest(uint32_t* status, uint64_t limit_ns, cudaStream_t stream) {
  bounded_wait_selftest_kernel<<<1, 32, 0, stream>>>(status, limit_ns);
  return 0;
}

}  // namespace mixfp4
