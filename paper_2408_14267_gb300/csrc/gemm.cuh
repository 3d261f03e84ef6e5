// Internal launchers of the integer GEMM kernels.
#pragma once
#include "common.cuh"

namespace fqt1 {

cudaError_t launch_xnor_gemm_simt(const uint32_t* A, const uint32_t* B, int64_t M, int64_t N, int64_t K,
                                  const float* gamma, int32_t* acc, float* y, cudaStream_t s);
cudaError_t launch_codes_gemm_simt(int bits, const uint8_t* Q, int64_t ldq, const int32_t* count,
                                   int64_t rows_per_count, int64_t max_rows, const uint32_t* S, int64_t n_s,
                                   int64_t L, int32_t* out, int64_t ldo, cudaStream_t s);

}  // namespace fqt1
