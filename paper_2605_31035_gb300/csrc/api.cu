// C ABI of libmixfp4.so (declared in include/mixfp4.h): argument validation,
// status codes, and kernel launches.  No entry point allocates device memory.
#include <cuda_runtime.h>
#include <cstdint>

#include "kernels.cuh"

namespace {

inline bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

inline int launch_status() {
  return cudaGetLastError() == cudaSuccess ? MIXFP4_OK : MIXFP4_ERR_CUDA;
}

}  // namespace

extern "C" {

int mixfp4_version(void) { return 100; }

const char* mixfp4_status_string(int status) {
  switch (status) {
    case MIXFP4_OK: return "ok";
    case MIXFP4_ERR_NULL: return "null pointer";
    case MIXFP4_ERR_SHAPE: return "invalid shape";
    case MIXFP4_ERR_ALIGN: return "misaligned pointer or leading dimension";
    case MIXFP4_ERR_DTYPE: return "unsupported dtype";
    case MIXFP4_ERR_CUDA: return "CUDA error";
    case MIXFP4_ERR_TIMEOUT: return "device-side wait timed out";
    case MIXFP4_ERR_ARG: return "argument out of range";
    default: return "unknown status";
  }
}

int mixfp4_quantize(const void* x, int dtype, int64_t rows, int64_t K, int64_t ldx,
                    uint8_t* codes, uint8_t* scales, float* tensor_scale, uint32_t* workspace,
                    int mode, int scale_flag, void* stream) {
  if (dtype != MIXFP4_DTYPE_BF16) return MIXFP4_ERR_DTYPE;
  if (mode < MIXFP4_MODE_MIX || mode > MIXFP4_MODE_FOUR_SIX) return MIXFP4_ERR_ARG;
  if (scale_flag != MIXFP4_SCALE_COMPUTE && scale_flag != MIXFP4_SCALE_GIVEN) return MIXFP4_ERR_ARG;
  if (rows < 0 || K < 0 || K % 16 != 0 || ldx < K) return MIXFP4_ERR_SHAPE;
  if (!tensor_scale) return MIXFP4_ERR_NULL;
  if (scale_flag == MIXFP4_SCALE_COMPUTE && !workspace) return MIXFP4_ERR_NULL;
  const bool empty = (rows == 0 || K == 0);
  if (!empty && (!x || !codes || !scales)) return MIXFP4_ERR_NULL;
  if (!empty && (!aligned(x, 32) || ldx % 16 != 0 || !aligned(codes, 8))) return MIXFP4_ERR_ALIGN;
  if (!aligned(tensor_scale, 4) || (workspace && !aligned(workspace, 4))) return MIXFP4_ERR_ALIGN;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int given = scale_flag == MIXFP4_SCALE_GIVEN;
  if (empty) {
    if (!given && cudaMemsetAsync(tensor_scale, 0, sizeof(float), s) != cudaSuccess)
      return MIXFP4_ERR_CUDA;
    return MIXFP4_OK;
  }
  const uint16_t* xb = static_cast<const uint16_t*>(x);
  if (!given) {
    if (cudaMemsetAsync(workspace, 0, sizeof(uint32_t), s) != cudaSuccess) return MIXFP4_ERR_CUDA;
    mixfp4::launch_amax(xb, rows, K, ldx, workspace, s);
    if (int st = launch_status()) return st;
  }
  mixfp4::launch_quantize(xb, rows, K, ldx, codes, scales, tensor_scale, workspace, mode, given, s);
  return launch_status();
}

int mixfp4_quantize_rht(const void* x, int dtype, int64_t rows, int64_t K, int64_t ldx, const uint8_t* signs,
                        uint8_t* codes, uint8_t* scales, float* tensor_scale, uint32_t* workspace, int mode,
                        int scale_flag, void* stream) {
  if (dtype != MIXFP4_DTYPE_BF16) return MIXFP4_ERR_DTYPE;
  if (mode < MIXFP4_MODE_MIX || mode > MIXFP4_MODE_E1M2_ONLY) return MIXFP4_ERR_ARG;
  if (scale_flag != MIXFP4_SCALE_COMPUTE && scale_flag != MIXFP4_SCALE_GIVEN) return MIXFP4_ERR_ARG;
  if (rows < 0 || K < 0 || K % 128 != 0 || ldx < K) return MIXFP4_ERR_SHAPE;
  if (!tensor_scale) return MIXFP4_ERR_NULL;
  if (scale_flag == MIXFP4_SCALE_COMPUTE && !workspace) return MIXFP4_ERR_NULL;
  const bool empty = (rows == 0 || K == 0);
  if (!empty && (!x || !codes || !scales)) return MIXFP4_ERR_NULL;
  if (!empty && (!aligned(x, 32) || ldx % 16 != 0 || !aligned(codes, 8))) return MIXFP4_ERR_ALIGN;
  if (!aligned(tensor_scale, 4) || (workspace && !aligned(workspace, 4))) return MIXFP4_ERR_ALIGN;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int given = scale_flag == MIXFP4_SCALE_GIVEN;
  if (empty) {
    if (!given && cudaMemsetAsync(tensor_scale, 0, sizeof(float), s) != cudaSuccess)
      return MIXFP4_ERR_CUDA;
    return MIXFP4_OK;
  }
  const uint16_t* xb = static_cast<const uint16_t*>(x);
  if (!given) {
    if (cudaMemsetAsync(workspace, 0, sizeof(uint32_t), s) != cudaSuccess) return MIXFP4_ERR_CUDA;
    mixfp4::launch_rht_amax(xb, rows, K, ldx, signs, workspace, s);
    if (int st = launch_status()) return st;
  }
  mixfp4::launch_rht_quantize(xb, rows, K, ldx, signs, codes, scales, tensor_scale, workspace, mode, given, s);
  return launch_status();
}

namespace {

// Shared body of the column-wise entry points (sr = 0: round to nearest).
int quantize_colwise_impl(const void* x, int dtype, int64_t R, int64_t C, int64_t ldx, uint8_t* codes,
                          uint8_t* scales, float* tensor_scale, uint32_t* workspace, int mode, int scale_flag,
                          int sr, uint64_t seed, uint64_t offset, void* stream) {
  if (dtype != MIXFP4_DTYPE_BF16) return MIXFP4_ERR_DTYPE;
  if (mode < MIXFP4_MODE_MIX || mode > MIXFP4_MODE_E1M2_ONLY) return MIXFP4_ERR_ARG;
  if (scale_flag != MIXFP4_SCALE_COMPUTE && scale_flag != MIXFP4_SCALE_GIVEN) return MIXFP4_ERR_ARG;
  if (R < 0 || C < 0 || R % 16 != 0 || C % 16 != 0 || ldx < C) return MIXFP4_ERR_SHAPE;
  if (!tensor_scale) return MIXFP4_ERR_NULL;
  if (scale_flag == MIXFP4_SCALE_COMPUTE && !workspace) return MIXFP4_ERR_NULL;
  const bool empty = (R == 0 || C == 0);
  if (!empty && (!x || !codes || !scales)) return MIXFP4_ERR_NULL;
  if (!empty && (!aligned(x, 32) || ldx % 16 != 0 || !aligned(codes, 8))) return MIXFP4_ERR_ALIGN;
  if (!aligned(tensor_scale, 4) || (workspace && !aligned(workspace, 4))) return MIXFP4_ERR_ALIGN;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int given = scale_flag == MIXFP4_SCALE_GIVEN;
  if (empty) {
    if (!given && cudaMemsetAsync(tensor_scale, 0, sizeof(float), s) != cudaSuccess) return MIXFP4_ERR_CUDA;
    return MIXFP4_OK;
  }
  const uint16_t* xb = static_cast<const uint16_t*>(x);
  if (!given) {
    if (cudaMemsetAsync(workspace, 0, sizeof(uint32_t), s) != cudaSuccess) return MIXFP4_ERR_CUDA;
    mixfp4::launch_amax(xb, R, C, ldx, workspace, s);  // max |x| does not depend on the orientation
    if (int st = launch_status()) return st;
  }
  if (mixfp4::launch_quantize_colwise(xb, R, C, ldx, codes, scales, tensor_scale, workspace, mode, given, sr, seed,
                                      offset, s) != 0)
    return MIXFP4_ERR_CUDA;
  return launch_status();
}

}  // namespace

int mixfp4_quantize_colwise(const void* x, int dtype, int64_t R, int64_t C, int64_t ldx, uint8_t* codes,
                            uint8_t* scales, float* tensor_scale, uint32_t* workspace, int mode, int scale_flag,
                            void* stream) {
  return quantize_colwise_impl(x, dtype, R, C, ldx, codes, scales, tensor_scale, workspace, mode, scale_flag, 0, 0, 0,
                               stream);
}

int mixfp4_quantize_colwise_sr(const void* x, int dtype, int64_t R, int64_t C, int64_t ldx, uint8_t* codes,
                               uint8_t* scales, float* tensor_scale, uint32_t* workspace, int mode, int scale_flag,
                               uint64_t seed, uint64_t offset, void* stream) {
  return quantize_colwise_impl(x, dtype, R, C, ldx, codes, scales, tensor_scale, workspace, mode, scale_flag, 1, seed,
                               offset, stream);
}

int mixfp4_quantize_sr(const void* x, int dtype, int64_t rows, int64_t K, int64_t ldx, uint8_t* codes,
                       uint8_t* scales, float* tensor_scale, uint32_t* workspace, int mode, int scale_flag,
                       uint64_t seed, uint64_t offset, void* stream) {
  if (dtype != MIXFP4_DTYPE_BF16) return MIXFP4_ERR_DTYPE;
  if (mode < MIXFP4_MODE_MIX || mode > MIXFP4_MODE_E1M2_ONLY) return MIXFP4_ERR_ARG;
  if (scale_flag != MIXFP4_SCALE_COMPUTE && scale_flag != MIXFP4_SCALE_GIVEN) return MIXFP4_ERR_ARG;
  if (rows < 0 || K < 0 || K % 16 != 0 || ldx < K) return MIXFP4_ERR_SHAPE;
  if (!tensor_scale) return MIXFP4_ERR_NULL;
  if (scale_flag == MIXFP4_SCALE_COMPUTE && !workspace) return MIXFP4_ERR_NULL;
  const bool empty = (rows == 0 || K == 0);
  if (!empty && (!x || !codes || !scales)) return MIXFP4_ERR_NULL;
  if (!empty && (!aligned(x, 32) || ldx % 16 != 0 || !aligned(codes, 8))) return MIXFP4_ERR_ALIGN;
  if (!aligned(tensor_scale, 4) || (workspace && !aligned(workspace, 4))) return MIXFP4_ERR_ALIGN;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int given = scale_flag == MIXFP4_SCALE_GIVEN;
  if (empty) {
    if (!given && cudaMemsetAsync(tensor_scale, 0, sizeof(float), s) != cudaSuccess) return MIXFP4_ERR_CUDA;
    return MIXFP4_OK;
  }
  const uint16_t* xb = static_cast<const uint16_t*>(x);
  if (!given) {
    if (cudaMemsetAsync(workspace, 0, sizeof(uint32_t), s) != cudaSuccess) return MIXFP4_ERR_CUDA;
    mixfp4::launch_amax(xb, rows, K, ldx, workspace, s);
    if (int st = launch_status()) return st;
  }
  if (mixfp4::launch_quantize_sr(xb, rows, K, ldx, codes, scales, tensor_scale, workspace, mode, given, seed, offset,
                                 s) != 0)
    return MIXFP4_ERR_CUDA;
  return launch_status();
}

int mixfp4_quantize_colwise_rht(const void* x, int dtype, int64_t R, int64_t C, int64_t ldx, const uint8_t* signs,
                                uint8_t* codes, uint8_t* scales, float* tensor_scale, uint32_t* workspace, int mode,
                                int scale_flag, void* stream) {
  if (dtype != MIXFP4_DTYPE_BF16) return MIXFP4_ERR_DTYPE;
  if (mode < MIXFP4_MODE_MIX || mode > MIXFP4_MODE_E1M2_ONLY) return MIXFP4_ERR_ARG;
  if (scale_flag != MIXFP4_SCALE_COMPUTE && scale_flag != MIXFP4_SCALE_GIVEN) return MIXFP4_ERR_ARG;
  if (R < 0 || C < 0 || R % 128 != 0 || C % 16 != 0 || ldx < C) return MIXFP4_ERR_SHAPE;
  if (!tensor_scale) return MIXFP4_ERR_NULL;
  if (scale_flag == MIXFP4_SCALE_COMPUTE && !workspace) return MIXFP4_ERR_NULL;
  const bool empty = (R == 0 || C == 0);
  if (!empty && (!x || !codes || !scales)) return MIXFP4_ERR_NULL;
  if (!empty && (!aligned(x, 32) || ldx % 16 != 0 || !aligned(codes, 8))) return MIXFP4_ERR_ALIGN;
  if (!aligned(tensor_scale, 4) || (workspace && !aligned(workspace, 4))) return MIXFP4_ERR_ALIGN;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int given = scale_flag == MIXFP4_SCALE_GIVEN;
  if (empty) {
    if (!given && cudaMemsetAsync(tensor_scale, 0, sizeof(float), s) != cudaSuccess) return MIXFP4_ERR_CUDA;
    return MIXFP4_OK;
  }
  const uint16_t* xb = static_cast<const uint16_t*>(x);
  if (!given) {
    if (cudaMemsetAsync(workspace, 0, sizeof(uint32_t), s) != cudaSuccess) return MIXFP4_ERR_CUDA;
    if (mixfp4::launch_quantize_colwise_rht(xb, R, C, ldx, signs, codes, scales, tensor_scale, workspace, mode, 0, 1,
                                            s) != 0)
      return MIXFP4_ERR_CUDA;
  }
  if (mixfp4::launch_quantize_colwise_rht(xb, R, C, ldx, signs, codes, scales, tensor_scale, workspace, mode, given, 0,
                                          s) != 0)
    return MIXFP4_ERR_CUDA;
  return launch_status();
}

int mixfp4_quantize_2d(const void* x, int dtype, int64_t rows, int64_t K, int64_t ldx, uint8_t* codes,
                       uint8_t* scales, float* tensor_scale, uint32_t* workspace, int mode, int scale_flag,
                       void* stream) {
  if (dtype != MIXFP4_DTYPE_BF16) return MIXFP4_ERR_DTYPE;
  if (mode < MIXFP4_MODE_MIX || mode > MIXFP4_MODE_E1M2_ONLY) return MIXFP4_ERR_ARG;
  if (scale_flag != MIXFP4_SCALE_COMPUTE && scale_flag != MIXFP4_SCALE_GIVEN) return MIXFP4_ERR_ARG;
  if (rows < 0 || K < 0 || K % 16 != 0 || ldx < K) return MIXFP4_ERR_SHAPE;
  if (!tensor_scale) return MIXFP4_ERR_NULL;
  if (scale_flag == MIXFP4_SCALE_COMPUTE && !workspace) return MIXFP4_ERR_NULL;
  const bool empty = (rows == 0 || K == 0);
  if (!empty && (!x || !codes || !scales)) return MIXFP4_ERR_NULL;
  if (!empty && (!aligned(x, 32) || ldx % 16 != 0 || !aligned(codes, 8))) return MIXFP4_ERR_ALIGN;
  if (!aligned(tensor_scale, 4) || (workspace && !aligned(workspace, 4))) return MIXFP4_ERR_ALIGN;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int given = scale_flag == MIXFP4_SCALE_GIVEN;
  if (empty) {
    if (!given && cudaMemsetAsync(tensor_scale, 0, sizeof(float), s) != cudaSuccess) return MIXFP4_ERR_CUDA;
    return MIXFP4_OK;
  }
  const uint16_t* xb = static_cast<const uint16_t*>(x);
  if (!given) {
    if (cudaMemsetAsync(workspace, 0, sizeof(uint32_t), s) != cudaSuccess) return MIXFP4_ERR_CUDA;
    mixfp4::launch_amax(xb, rows, K, ldx, workspace, s);
    if (int st = launch_status()) return st;
  }
  if (mixfp4::launch_quantize_2d(xb, rows, K, ldx, codes, scales, tensor_scale, workspace, mode, given, s) != 0)
    return MIXFP4_ERR_CUDA;
  return launch_status();
}

int mixfp4_fake_quantize(const void* x, int dtype, int64_t rows, int64_t K, int64_t ldx, int candidates, int block,
                         float* tensor_scale, uint32_t* workspace, int scale_flag, void* out, int out_dtype,
                         int64_t ldo, uint8_t* choice, void* stream) {
  if (dtype != MIXFP4_DTYPE_BF16) return MIXFP4_ERR_DTYPE;
  if (out_dtype != MIXFP4_DTYPE_BF16 && out_dtype != MIXFP4_DTYPE_F32) return MIXFP4_ERR_DTYPE;
  if (candidates <= 0 || candidates > 15) return MIXFP4_ERR_ARG;
  if (block != 8 && block != 16 && block != 32 && block != 64) return MIXFP4_ERR_ARG;
  if (scale_flag != MIXFP4_SCALE_COMPUTE && scale_flag != MIXFP4_SCALE_GIVEN) return MIXFP4_ERR_ARG;
  if (rows < 0 || K < 0 || K % 16 != 0 || K % block != 0 || ldx < K || ldo < K) return MIXFP4_ERR_SHAPE;
  if (!tensor_scale) return MIXFP4_ERR_NULL;
  if (scale_flag == MIXFP4_SCALE_COMPUTE && !workspace) return MIXFP4_ERR_NULL;
  const bool empty = (rows == 0 || K == 0);
  if (!empty && (!x || !out)) return MIXFP4_ERR_NULL;
  if (!empty && (!aligned(x, 32) || ldx % 16 != 0 || !aligned(out, 32) || ldo % 16 != 0)) return MIXFP4_ERR_ALIGN;
  if (choice && !aligned(choice, 2)) return MIXFP4_ERR_ALIGN;
  if (!aligned(tensor_scale, 4) || (workspace && !aligned(workspace, 4))) return MIXFP4_ERR_ALIGN;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int given = scale_flag == MIXFP4_SCALE_GIVEN;
  if (empty) {
    if (!given && cudaMemsetAsync(tensor_scale, 0, sizeof(float), s) != cudaSuccess) return MIXFP4_ERR_CUDA;
    return MIXFP4_OK;
  }
  const uint16_t* xb = static_cast<const uint16_t*>(x);
  if (!given) {
    if (cudaMemsetAsync(workspace, 0, sizeof(uint32_t), s) != cudaSuccess) return MIXFP4_ERR_CUDA;
    mixfp4::launch_amax(xb, rows, K, ldx, workspace, s);
    if (int st = launch_status()) return st;
  }
  if (mixfp4::launch_fake_quantize(xb, rows, K, ldx, candidates, block, tensor_scale, workspace, given, out,
                                   out_dtype == MIXFP4_DTYPE_BF16, ldo, choice, s) != 0)
    return MIXFP4_ERR_CUDA;
  return launch_status();
}

int mixfp4_transpose_2d(const uint8_t* codes, const uint8_t* scales, int64_t rows, int64_t K, uint8_t* codes_t,
                        uint8_t* scales_t, void* stream) {
  if (rows < 0 || K < 0 || rows % 16 != 0 || K % 16 != 0) return MIXFP4_ERR_SHAPE;
  if (rows == 0 || K == 0) return MIXFP4_OK;
  if (!codes || !scales || !codes_t || !scales_t) return MIXFP4_ERR_NULL;
  if (!aligned(codes, 8) || !aligned(codes_t, 8)) return MIXFP4_ERR_ALIGN;
  if (mixfp4::launch_transpose_2d(codes, scales, rows, K, codes_t, scales_t, static_cast<cudaStream_t>(stream)) != 0)
    return MIXFP4_ERR_CUDA;
  return MIXFP4_OK;
}

int mixfp4_dequantize(const uint8_t* codes, const uint8_t* scales, const float* tensor_scale,
                      int64_t rows, int64_t K, float* out, void* stream) {
  if (rows < 0 || K < 0 || K % 16 != 0) return MIXFP4_ERR_SHAPE;
  if (rows == 0 || K == 0) return MIXFP4_OK;
  if (!codes || !scales || !tensor_scale || !out) return MIXFP4_ERR_NULL;
  if (!aligned(codes, 8) || !aligned(out, 32) || !aligned(tensor_scale, 4)) return MIXFP4_ERR_ALIGN;
  mixfp4::launch_dequantize(codes, scales, tensor_scale, rows, K, out, static_cast<cudaStream_t>(stream));
  return launch_status();
}

int mixfp4_gemm(const uint8_t* a_codes, const uint8_t* a_scales, const float* a_ts,
                const uint8_t* b_codes, const uint8_t* b_scales, const float* b_ts,
                int64_t M, int64_t N, int64_t K, float* C, int64_t ldc,
                uint32_t* status_word, void* stream) {
  if (M < 0 || N < 0 || K < 0 || K % 256 != 0 || ldc < N) return MIXFP4_ERR_SHAPE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (status_word) {
    if (!aligned(status_word, 4)) return MIXFP4_ERR_ALIGN;
    if (cudaMemsetAsync(status_word, 0, sizeof(uint32_t), s) != cudaSuccess) return MIXFP4_ERR_CUDA;
  }
  if (M == 0 || N == 0) return MIXFP4_OK;
  if (!C) return MIXFP4_ERR_NULL;
  if (!aligned(C, 4)) return MIXFP4_ERR_ALIGN;
  if (K == 0) {  // empty reduction: C = 0
    if (cudaMemset2DAsync(C, (size_t)ldc * sizeof(float), 0, (size_t)N * sizeof(float), (size_t)M, s) != cudaSuccess)
      return MIXFP4_ERR_CUDA;
    return MIXFP4_OK;
  }
  if (!a_codes || !a_scales || !a_ts || !b_codes || !b_scales || !b_ts) return MIXFP4_ERR_NULL;
  if (!aligned(a_codes, 16) || !aligned(a_scales, 16) || !aligned(b_codes, 16) ||
      !aligned(b_scales, 16) || !aligned(a_ts, 4) || !aligned(b_ts, 4))
    return MIXFP4_ERR_ALIGN;
  int st = mixfp4::launch_gemm(a_codes, a_scales, a_ts, b_codes, b_scales, b_ts, M, N, K, C, ldc,
                               status_word, s);
  if (st) return st;
  return launch_status();
}

int mixfp4_gemm_native_fewrows(const uint8_t* a_codes, const uint8_t* a_scales, const float* a_ts,
                               const uint8_t* b_codes, const uint8_t* b_scales, const float* b_ts, int64_t M,
                               int64_t N, int64_t K, float* C, int64_t ldc, uint32_t* status_word, void* stream) {
  if (M < 0 || M > 64 || N < 0 || K < 0 || K % 256 != 0 || ldc < N) return MIXFP4_ERR_SHAPE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (status_word) {
    if (!aligned(status_word, 4)) return MIXFP4_ERR_ALIGN;
    if (cudaMemsetAsync(status_word, 0, sizeof(uint32_t), s) != cudaSuccess) return MIXFP4_ERR_CUDA;
  }
  if (M == 0 || N == 0) return MIXFP4_OK;
  if (!C) return MIXFP4_ERR_NULL;
  if (!aligned(C, 4)) return MIXFP4_ERR_ALIGN;
  if (K == 0) {
    if (cudaMemset2DAsync(C, (size_t)ldc * sizeof(float), 0, (size_t)N * sizeof(float), (size_t)M, s) != cudaSuccess)
      return MIXFP4_ERR_CUDA;
    return MIXFP4_OK;
  }
  if (!a_codes || !a_scales || !a_ts || !b_codes || !b_scales || !b_ts) return MIXFP4_ERR_NULL;
  if (!aligned(a_codes, 16) || !aligned(a_scales, 16) || !aligned(b_codes, 16) || !aligned(b_scales, 16) ||
      !aligned(a_ts, 4) || !aligned(b_ts, 4))
    return MIXFP4_ERR_ALIGN;
  int st = mixfp4::launch_gemm_native_fewrows(a_codes, a_scales, a_ts, b_codes, b_scales, b_ts, M, N, K, C, ldc,
                                              status_word, s);
  if (st) return st;
  return launch_status();
}

int mixfp4_split_native(const uint8_t* codes, const uint8_t* scales, int64_t rows, int64_t K,
                        uint8_t* main_codes, uint8_t* res_codes, uint8_t* sf_tiled, void* stream) {
  if (rows < 0 || K < 0 || K % 64 != 0) return MIXFP4_ERR_SHAPE;
  if (rows == 0 || K == 0) return MIXFP4_OK;
  if (!codes || !scales || !main_codes || !res_codes || !sf_tiled) return MIXFP4_ERR_NULL;
  if (!aligned(codes, 16) || !aligned(scales, 4) || !aligned(main_codes, 16) || !aligned(res_codes, 16) ||
      !aligned(sf_tiled, 16))
    return MIXFP4_ERR_ALIGN;
  int st = mixfp4::launch_split_native(codes, scales, rows, K, main_codes, res_codes, sf_tiled,
                                       static_cast<cudaStream_t>(stream));
  if (st) return st;
  return launch_status();
}

int mixfp4_gemm_native(const uint8_t* a_main, const uint8_t* a_res, const uint8_t* a_sf, const float* a_ts,
                       const uint8_t* b_main, const uint8_t* b_res, const uint8_t* b_sf, const float* b_ts,
                       int64_t M, int64_t N, int64_t K, float* C, int64_t ldc, uint32_t* status_word,
                       void* stream) {
  if (M < 0 || N < 0 || K < 0 || K % 256 != 0 || ldc < N) return MIXFP4_ERR_SHAPE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (status_word) {
    if (!aligned(status_word, 4)) return MIXFP4_ERR_ALIGN;
    if (cudaMemsetAsync(status_word, 0, sizeof(uint32_t), s) != cudaSuccess) return MIXFP4_ERR_CUDA;
  }
  if (M == 0 || N == 0) return MIXFP4_OK;
  if (!C) return MIXFP4_ERR_NULL;
  if (!aligned(C, 4)) return MIXFP4_ERR_ALIGN;
  if (K == 0) {
    if (cudaMemset2DAsync(C, (size_t)ldc * sizeof(float), 0, (size_t)N * sizeof(float), (size_t)M, s) != cudaSuccess)
      return MIXFP4_ERR_CUDA;
    return MIXFP4_OK;
  }
  if (!a_main || !a_sf || !a_ts || !b_main || !b_sf || !b_ts) return MIXFP4_ERR_NULL;
  if (!aligned(a_main, 16) || !aligned(a_sf, 16) || !aligned(b_main, 16) || !aligned(b_sf, 16) ||
      (a_res && !aligned(a_res, 16)) || (b_res && !aligned(b_res, 16)) || !aligned(a_ts, 4) || !aligned(b_ts, 4))
    return MIXFP4_ERR_ALIGN;
  int st = mixfp4::launch_gemm_native(a_main, a_res, a_sf, a_ts, b_main, b_res, b_sf, b_ts, M, N, K, C, ldc,
                                      status_word, s);
  if (st) return st;
  return launch_status();
}

}  // extern "C"

int mixfp4_selftest_gemm_missed_stage(const uint8_t* a_codes, const uint8_t* a_scales, const float* a_ts,
                                      const uint8_t* b_codes, const uint8_t* b_scales, const float* b_ts, int64_t M,
                                      int64_t N, int64_t K, float* C, int64_t ldc, uint32_t* status_word,
                                      uint64_t limit_ns, void* stream) {
  if (M < 1 || N < 1 || K < 256 || K % 256 != 0 || ldc < N) return MIXFP4_ERR_SHAPE;
  if (M > (1 << 30) || N > (1 << 30) || K > (1 << 30)) return MIXFP4_ERR_SHAPE;
  if (limit_ns == 0 || limit_ns > 2000000000ull) return MIXFP4_ERR_ARG;
  if (!a_codes || !a_scales || !a_ts || !b_codes || !b_scales || !b_ts || !C || !status_word) return MIXFP4_ERR_NULL;
  if (!aligned(a_codes, 16) || !aligned(a_scales, 16) || !aligned(b_codes, 16) || !aligned(b_scales, 16) ||
      !aligned(a_ts, 4) || !aligned(b_ts, 4) || !aligned(C, 4) || !aligned(status_word, 4))
    return MIXFP4_ERR_ALIGN;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(status_word, 0, sizeof(uint32_t), s) != cudaSuccess) return MIXFP4_ERR_CUDA;
  int st = mixfp4::launch_gemm_missed_stage_selftest(a_codes, a_scales, a_ts, b_codes, b_scales, b_ts, M, N, K, C,
                                                     ldc, status_word, limit_ns, s);
  if (st) return st;
  return launch_status();
}

int mixfp4_selftest_bounded_wait(uint32_t* status_word, uint64_t limit_ns, void* stream) {
  if (!status_word) return MIXFP4_ERR_NULL;
  if (!aligned(status_word, 4)) return MIXFP4_ERR_ALIGN;
  if (limit_ns == 0 || limit_ns > 2000000000ull) return MIXFP4_ERR_ARG;
  mixfp4::launch_bounded_wait_selftest(status_word, limit_ns, static_cast<cudaStream_t>(stream));
  return launch_status();
}
