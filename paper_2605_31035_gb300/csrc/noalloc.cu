// mixfp4_quantize_noalloc: the quantizer with a computed per-tensor scale,
// for callers that cannot allocate device memory.
//
// mixfp4_quantize with MIXFP4_SCALE_COMPUTE needs one scratch word of device
// memory (the amax accumulator), which its caller passes in.  Some callers
// cannot provide it: an inference runtime that plans every device buffer up
// front and hands an operator only its input and output tensors, or a plugin
// interface whose execute callback must not call cudaMalloc (an allocation
// can synchronise the device, stall other streams, or fail under memory
// pressure in the middle of a step).  This variant keeps that scratch word in
// a file-scope __device__ array instead, so the call allocates nothing.
//
// Properties a caller must know:
//   * The array is kNoAllocScratchWords 32-bit words (256 bytes).  It is
//     created when the library is loaded and every GPU that loads the library
//     holds it until the process exits.  This entry point needs one word for
//     any input shape; a requirement above the array's size is rejected with
//     MIXFP4_ERR_SHAPE.
//   * In host code the array's name is only a host-side stand-in; the device
//     address is obtained with cudaGetSymbolAddress once per device, with that
//     device current, on the first call made on it.  Make that first call
//     before any stream capture begins.  The address is cached together with
//     the unique id of the context it was looked up in: after a
//     cudaDeviceReset the library's module is loaded again in a new context,
//     possibly at another address, so a call that finds a different current
//     context looks the address up again (as a first call does).
//   * All calls share the one array and it keeps the last call's contents; the
//     word is cleared on the stream before each use.  Calls that overlap on the
//     GPU (different streams without ordering, or several host threads) race
//     on it and may produce a wrong scale: order them.
//   * No cudaMalloc, cudaFree or other allocating routine is called.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cstdint>
#include <mutex>

#include "kernels.cuh"

namespace {

constexpr int kNoAllocScratchWords = 64;
constexpr int kAmaxWords = 1;  // the amax accumulator of the SCALE_COMPUTE pass
constexpr int kMaxDevices = 64;

static __device__ __align__(256) uint32_t g_noalloc_scratch[kNoAllocScratchWords];

std::mutex g_setup_mutex;
uint32_t* g_scratch_ptr[kMaxDevices] = {};
unsigned long long g_scratch_ctx[kMaxDevices] = {};  // context id the address belongs to (0: none)

using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

// Unique id of the current context (ids are never reused within a process);
// 0 when there is no current context or the driver does not report ids.
unsigned long long current_context_id() {
  static CtxGetCurrentFn get_current = nullptr;
  static CtxGetIdFn get_id = nullptr;
  static bool resolved = false;
  if (!resolved) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<CtxGetCurrentFn>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<CtxGetIdFn>(p);
    resolved = true;
  }
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (!get_current || !get_id || get_current(&ctx) != CUDA_SUCCESS || !ctx || get_id(ctx, &id) != CUDA_SUCCESS)
    return 0;
  return id;
}

// Device address of the scratch array on the current device, looked up on
// the first call on each device (and again when the device's context has
// changed since, e.g. after cudaDeviceReset); nullptr on failure.
uint32_t* scratch_for_current_device() {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  const unsigned long long ctx = current_context_id();
  if (!g_scratch_ptr[dev] || ctx == 0 || ctx != g_scratch_ctx[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return nullptr;
    g_scratch_ptr[dev] = static_cast<uint32_t*>(p);
    g_scratch_ctx[dev] = current_context_id();  // the lookup above made the context current if it was not
  }
  return g_scratch_ptr[dev];
}

inline bool aligned_to(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

}  // namespace

extern "C" int mixfp4_quantize_noalloc(const void* x, int dtype, int64_t rows, int64_t K,
                                       int64_t ldx, uint8_t* codes, uint8_t* scales,
                                       float* tensor_scale, int mode, void* stream) {
  if (dtype != MIXFP4_DTYPE_BF16) return MIXFP4_ERR_DTYPE;
  if (mode < MIXFP4_MODE_MIX || mode > MIXFP4_MODE_FOUR_SIX) return MIXFP4_ERR_ARG;
  if (rows < 0 || K < 0 || K % 16 != 0 || ldx < K) return MIXFP4_ERR_SHAPE;
  if (kAmaxWords > kNoAllocScratchWords) return MIXFP4_ERR_SHAPE;
  if (!tensor_scale) return MIXFP4_ERR_NULL;
  const bool empty = (rows == 0 || K == 0);
  if (!empty && (!x || !codes || !scales)) return MIXFP4_ERR_NULL;
  if (!empty && (!aligned_to(x, 32) || ldx % 16 != 0 || !aligned_to(codes, 8))) return MIXFP4_ERR_ALIGN;
  if (!aligned_to(tensor_scale, 4)) return MIXFP4_ERR_ALIGN;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (empty) {
    if (cudaMemsetAsync(tensor_scale, 0, sizeof(float), s) != cudaSuccess) return MIXFP4_ERR_CUDA;
    return MIXFP4_OK;
  }
  uint32_t* amax_word = scratch_for_current_device();
  if (!amax_word) return MIXFP4_ERR_CUDA;
  if (cudaMemsetAsync(amax_word, 0, kAmaxWords * sizeof(uint32_t), s) != cudaSuccess) return MIXFP4_ERR_CUDA;
  const uint16_t* xb = static_cast<const uint16_t*>(x);
  mixfp4::launch_amax(xb, rows, K, ldx, amax_word, s);
  if (cudaGetLastError() != cudaSuccess) return MIXFP4_ERR_CUDA;
  mixfp4::launch_quantize(xb, rows, K, ldx, codes, scales, tensor_scale, amax_word, mode,
                          /*scale_given=*/0, s);
  return cudaGetLastError() == cudaSuccess ? MIXFP4_OK : MIXFP4_ERR_CUDA;
}
