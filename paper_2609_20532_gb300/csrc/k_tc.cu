// Tensor-core kernels: not built yet; every shape takes the CUDA-core path.
#include "tc.h"

namespace dpk {

bool tc_ghost_supported(int, int64_t, int64_t) { return false; }
int tc_ghost_parts(int) { return 1; }
cudaError_t tc_launch_ghost(const void*, const void*, int, int, int, int, float*, int, int,
                            cudaStream_t) {
  return cudaErrorNotSupported;
}
bool tc_gemm_supported(int, int64_t, int64_t) { return false; }
int tc_mat_parts(int64_t, int64_t) { return 1; }
cudaError_t tc_launch_mat_norm(const void*, const void*, int, int, int, int, float*, int, int,
                               cudaStream_t) {
  return cudaErrorNotSupported;
}
cudaError_t tc_launch_clipsum(const void*, const void*, const float*, int, int, int, int, float*,
                              const Epilogue&, cudaStream_t) {
  return cudaErrorNotSupported;
}

}  // namespace dpk
