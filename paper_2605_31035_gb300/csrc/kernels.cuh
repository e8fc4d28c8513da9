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
int launch_dequantize(const uint8_t* codes, const uint8_t* scales, const float* tensor_scale,
                      int64_t rows, int64_t K, float* out, cudaStream_t stream);
int launch_gemm(const uint8_t* a_codes, const uint8_t* a_scales, const float* a_ts,
                const uint8_t* b_codes, const uint8_t* b_scales, const float* b_ts,
                int64_t M, int64_t N, int64_t K, float* C, int64_t ldc, uint32_t* status_word,
                cudaStream_t stream);

}  // namespace mixfp4
