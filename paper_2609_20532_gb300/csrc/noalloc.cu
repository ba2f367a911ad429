// dp_layer_sqnorms_noalloc: the per-example squared norms of one layer,
// computed without allocating any memory.
//
// Who needs it: callers that cannot call cudaMalloc (or anything that does)
// at the point where they need the norms -- code running inside a CUDA
// stream capture in global capture mode, where allocation calls are not
// permitted; processes that reserve their whole device-memory budget at
// start-up and must not grow it while serving; and callers that must not
// take the implicit device synchronisation cudaMalloc / cudaFree can cause.
// The step context (dp_step_init) allocates its scratch once, which those
// callers may not be able to do; this entry point needs no context.
//
// How: the Gram-form norm kernels write per-example partial sums to scratch
// memory.  Here that scratch is the file-scope device array g_noalloc_part
// below (kNoallocMaxPartials floats, 4 MiB, plus one error word), which
// every GPU that loads this library holds until the process exits.  Host
// code cannot use the array's name as a device address, so the first call
// on each device looks the address up with cudaGetSymbolAddress (with that
// device current) and caches it; that first call should therefore come
// before any stream capture.
//
// All calls share the one array and it keeps the last call's contents: the
// partial sums are fully overwritten by every call, and the error word is
// cleared at the start of every call.  Calls whose work overlaps on the GPU
// (two streams, or two host threads) race on the array; callers must order
// them (e.g. one stream).
#include <cuda_runtime.h>

#include <mutex>

#include "../../include/dp_step.h"
#include "internal.h"
#include "tc.h"

namespace {

constexpr int64_t kNoallocMaxPartials = int64_t(1) << 20;  // 4 MiB of fp32 partials
constexpr int kMaxDevices = 64;

// [0, kNoallocMaxPartials): partial sums; then 64 words for the error flag
// (only the first is used; the rest keep the array a multiple of 256 bytes).
static __device__ __align__(256) float g_noalloc_part[kNoallocMaxPartials + 64];

std::mutex g_setup_mu;
float* g_dev_ptr[kMaxDevices] = {};

// Sum the partials of each example in a fixed order; a tensor-core wait
// that gave up (error word != 0) turns every output into NaN.
__global__ void k_noalloc_reduce(const float* __restrict__ part, int B, int NP,
                                 const int* __restrict__ err, float* __restrict__ out) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= B) return;
  const float* p = part + static_cast<int64_t>(i) * NP;
  float n = 0.f;
  for (int q = 0; q < NP; ++q) n += p[q];
  out[i] = (*err != 0) ? __int_as_float(0x7fc00000) : n;
}

dp_status noalloc_fail(dp_status st, const char* msg) {
  dpk::set_last_error(msg);  // reported by dp_last_error()
  return st;
}

}  // namespace

extern "C" dp_status dp_layer_sqnorms_noalloc(const void* A, const void* D, int32_t B, int32_t T,
                                              int64_t d_in, int64_t d_out, dp_dtype dtype,
                                              float* d_sqnorm_out, void* cuda_stream) {
  if (!A || !D || !d_sqnorm_out) return noalloc_fail(DP_ERR_ARG, "NULL pointer argument");
  if ((reinterpret_cast<uintptr_t>(A) | reinterpret_cast<uintptr_t>(D)) & 15u)
    return noalloc_fail(DP_ERR_ARG, "A and D must be 16-byte aligned");
  if (dtype != DP_F32 && dtype != DP_BF16) return noalloc_fail(DP_ERR_DTYPE, "unknown dtype");
  if (B < 1 || T < 1 || int64_t(B) * T > 0x7fffffffLL)
    return noalloc_fail(DP_ERR_SHAPE, "need B >= 1, T >= 1, B*T <= 2^31-1");
  if (d_in < 1 || d_out < 1 || d_in > (1 << 20) || d_out > (1 << 20))
    return noalloc_fail(DP_ERR_SHAPE, "d_in, d_out must be in 1..2^20");
  if (dtype == DP_BF16 && ((d_in * 2) % 16 || (d_out * 2) % 16))
    return noalloc_fail(DP_ERR_SHAPE, "bf16 rows must be a multiple of 16 bytes");

  const bool tc = dtype == DP_BF16 && dpk::tc_ghost_supported(T, d_in, d_out);
  // partials per example, counted in 64 bits (about T^2 / 8192 of them)
  const int64_t parts = tc ? dpk::tc_ghost_parts(T) : dpk::ghost_simt_parts(T);
  if (parts < 1 || parts > kNoallocMaxPartials || int64_t(B) * parts > kNoallocMaxPartials)
    return noalloc_fail(DP_ERR_SHAPE,
                        "B x partials-per-example exceeds the 2^20-float scratch of "
                        "dp_layer_sqnorms_noalloc; use dp_layer_norms instead");
  const int NP = static_cast<int>(parts);

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
    return noalloc_fail(DP_ERR_CUDA, "cudaGetDevice failed or device index too large");
  float* part = nullptr;
  {
    std::lock_guard<std::mutex> lk(g_setup_mu);
    if (!g_dev_ptr[dev]) {
      void* p = nullptr;
      cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_part);
      if (e != cudaSuccess || !p) {
        cudaGetLastError();
        return noalloc_fail(DP_ERR_CUDA, "cudaGetSymbolAddress of the scratch array failed");
      }
      // the tensor-core kernels' per-device set-up happens here too, so that
      // calls after the first one make no set-up call of any kind
      if (dpk::tma_encode_available()) {
        e = dpk::tc_ghost_prepare();
        if (e != cudaSuccess) {
          cudaGetLastError();
          return noalloc_fail(DP_ERR_CUDA, "set-up of the Gram kernels failed");
        }
      }
      g_dev_ptr[dev] = static_cast<float*>(p);
    }
    part = g_dev_ptr[dev];
  }
  int* err = reinterpret_cast<int*>(part + kNoallocMaxPartials);
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  if (cudaMemsetAsync(err, 0, sizeof(int), s) != cudaSuccess)
    return noalloc_fail(DP_ERR_CUDA, "cudaMemsetAsync of the error word failed");
  const int din = static_cast<int>(d_in), dout = static_cast<int>(d_out);
  cudaError_t e = tc ? dpk::tc_launch_ghost(A, D, B, T, din, dout, part, NP, 0, err, s)
                     : dpk::launch_norm_ghost_simt(dtype == DP_BF16 ? dpk::IN_BF16 : dpk::IN_F32,
                                                   A, D, B, T, din, dout, part, NP, 0, s);
  if (e != cudaSuccess) return noalloc_fail(DP_ERR_CUDA, cudaGetErrorString(e));
  k_noalloc_reduce<<<(B + 127) / 128, 128, 0, s>>>(part, B, NP, err, d_sqnorm_out);
  e = cudaGetLastError();
  if (e != cudaSuccess) return noalloc_fail(DP_ERR_CUDA, cudaGetErrorString(e));
  return DP_OK;
}
