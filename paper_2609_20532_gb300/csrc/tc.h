// Tensor-core (tcgen05 / TMEM / TMA) kernels of the DP-SGD step, bf16 inputs.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

#include "internal.h"

namespace dpk {

// Gram-form per-example norms on tensor cores.
bool tc_ghost_supported(int T, int64_t d_in, int64_t d_out);
int tc_ghost_parts(int T);
cudaError_t tc_launch_ghost(const void* A, const void* D, int B, int T, int d_in, int d_out,
                            float* part, int NP, int row0, cudaStream_t s);

// Clipped sum S = A^T diag(c) D with the noise epilogue, and the materialised
// per-example norm that shares its main loop.
bool tc_gemm_supported(int T, int64_t d_in, int64_t d_out);
int tc_mat_parts(int64_t d_in, int64_t d_out);
cudaError_t tc_launch_mat_norm(const void* A, const void* D, int B, int T, int d_in, int d_out,
                               float* part, int NP, int row0, cudaStream_t s);
cudaError_t tc_launch_clipsum(const void* A, const void* D, const float* c, int B, int T,
                              int d_in, int d_out, float* out, const Epilogue& ep,
                              cudaStream_t s);

}  // namespace dpk
