// Thin convolutions whose input per example fits in shared memory
// (csrc/k_conv.cu): the per-example gradient G_i = a_i^T d_i straight from the
// NHWC input, without patch rows, and one norm partial per example (partial
// slot 0 of row row0 + i).
#pragma once
#include <cuda_runtime.h>

#include <cstdint>

#include "internal.h"

namespace dpk {

constexpr int kConvThinMaxSmem = 200 * 1024;
bool conv_thin_norm_ok(const ConvGeom& g, int64_t c_out);
cudaError_t launch_conv_thin_norm(InType t, const void* x, const void* d, const ConvGeom& g,
                                  int c_out, int B, float* G, float* part, int NP, int row0,
                                  cudaStream_t s);

}  // namespace dpk
