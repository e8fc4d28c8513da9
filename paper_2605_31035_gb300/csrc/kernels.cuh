// Kernel launchers behind the C ABI (include/mixfp4.h).  Arguments are
// validated by the caller (api.cu); these only enqueue work on `stream`.
#pragma once
#include <cuda_runtime.h>
#include <cstdint>

#include "mixfp4.h"

namespace mixfp4 {

int launch_amax(const uint16_t* x, int64_t rows, int64_t K, int64_t ldx, uint32_t* amax_word,
                cudaStream_t stream);
int launch_quantize(const uint16_t* x, int64_t rows, int64_t K, int64_t ldx, uint8_t* codes,
                    uint8_t* scales, float* tensor_scale, const uint32_t* amax_word, int mode,
                    int scale_given, cudaStream_t stream);
int launch_rht_amax(const uint16_t* x, int64_t rows, int64_t K, int64_t ldx, const uint8_t* signs,
                    uint32_t* amax_word, cudaStream_t stream);
int launch_rht_quantize(const uint16_t* x, int64_t rows, int64_t K, int64_t ldx, const uint8_t* signs,
                        uint8_t* codes, uint8_t* scales, float* tensor_scale, const uint32_t* amax_word, int mode,
                        int scale_given, cudaStream_t stream);
int launch_quantize_colwise(const uint16_t* x, int64_t R, int64_t C, int64_t ldx, uint8_t* codes, uint8_t* scales,
                            float* tensor_scale, const uint32_t* amax_word, int mode, int scale_given, int sr,
                            uint64_t seed, uint64_t offset, cudaStream_t stream);
int launch_quantize_sr(const uint16_t* x, int64_t rows, int64_t K, int64_t ldx, uint8_t* codes, uint8_t* scales,
                       float* tensor_scale, const uint32_t* amax_word, int mode, int scale_given, uint64_t seed,
                       uint64_t offset, cudaStream_t stream);
int launch_quantize_colwise_rht(const uint16_t* x, int64_t R, int64_t C, int64_t ldx, const uint8_t* signs,
                                uint8_t* codes, uint8_t* scales, float* tensor_scale, uint32_t* amax_word, int mode,
                                int scale_given, int amax_pass, cudaStream_t stream);
int launch_quantize_2d(const uint16_t* x, int64_t rows, int64_t K, int64_t ldx, uint8_t* codes, uint8_t* scales,
                       float* tensor_scale, const uint32_t* amax_word, int mode, int scale_given,
                       cudaStream_t stream);
int launch_transpose_2d(const uint8_t* codes, const uint8_t* scales, int64_t rows, int64_t K, uint8_t* codes_t,
                        uint8_t* scales_t, cudaStream_t stream);
int launch_fake_quantize(const uint16_t* x, int64_t rows, int64_t K, int64_t ldx, int candidates, int block,
                         float* tensor_scale, const uint32_t* amax_word, int scale_given, void* out, int out_bf16,
                         int64_t ldo, uint8_t* choice, cudaStream_t stream);
int launch_bounded_wait_selftest(uint32_t* status, uint64_t limit_ns, cudaStream_t stream);
int launch_gemm_missed_stage_selftest(const uint8_t* a_codes, const uint8_t* a_scales, const float* a_ts,
                                      const uint8_t* b_codes, const uint8_t* b_scales, const float* b_ts, int64_t M,
                                      int64_t N, int64_t K, float* C, int64_t ldc, uint32_t* status_word,
                                      uint64_t wait_ns, cudaStream_t stream);
int launch_dequantize(const uint8_t* codes, const uint8_t* scales, const float* tensor_scale,
                      int64_t rows, int64_t K, float* out, cudaStream_t stream);
int launch_gemm(const uint8_t* a_codes, const uint8_t* a_scales, const float* a_ts,
                const uint8_t* b_codes, const uint8_t* b_scales, const float* b_ts,
                int64_t M, int64_t N, int64_t K, float* C, int64_t ldc, uint32_t* status_word,
                cudaStream_t stream);
int launch_gemm_native_fewrows(const uint8_t* a_codes, const uint8_t* a_scales, const float* a_ts,
                               const uint8_t* b_codes, const uint8_t* b_scales, const float* b_ts, int64_t M,
                               int64_t N, int64_t K, float* C, int64_t ldc, uint32_t* status_word,
                               cudaStream_t stream);
int launch_split_native(const uint8_t* codes, const uint8_t* scales, int64_t rows, int64_t K, uint8_t* main_codes,
                        uint8_t* res_codes, uint8_t* sf, cudaStream_t stream);
int launch_gemm_native(const uint8_t* a_main, const uint8_t* a_res, const uint8_t* a_sf, const float* a_ts,
                       const uint8_t* b_main, const uint8_t* b_res, const uint8_t* b_sf, const float* b_ts, int64_t M,
                       int64_t N, int64_t K, float* C, int64_t ldc, uint32_t* status_word, cudaStream_t stream);

// Launch `kernel` as a programmatic dependent of the previous kernel on the
// stream (it may start before that kernel completes; the kernel itself waits,
// with griddepcontrol.wait, before it reads anything that kernel may write).
template <typename... Params, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(Params...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t stream, Args... args) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Params>(args)...);
}

}  // namespace mixfp4
