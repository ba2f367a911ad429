// Patch rows of a 2-D convolution (cross-correlation, zero padding, strides)
// over NHWC activations, so that the convolution's per-example weight
// gradient is the dense A_i^T D_i of the other kernels (the CIFAR-10
// WideResNet of App. B):
//   a[i][h*W_out + w][(ki*kw + kj)*C_in + c] = xp_i[h*sh + ki][w*sw + kj][c]
// with xp the input padded by zeros.  The kernel only copies values and
// writes zeros, so it is exact.  It is bound by HBM: the output (kh*kw times
// the input for a stride-1 3x3 kernel) is written once with streaming
// stores; the input is read about once from HBM, the taps of neighbouring
// rows finding it in L1/L2.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "internal.h"
#include "tc.h"

namespace dpk {

namespace {

constexpr int kConvThreads = 256;
constexpr int kConvRowElems = 4096;  // output units a block takes per row group

// One output unit = V consecutive elements of a row (V = 16 bytes' worth
// when C_in allows it, else 1).  U = units per row = kh*kw*C_in / V.
template <typename Unit>
__global__ void __launch_bounds__(kConvThreads)
    k_conv_unfold(const Unit* __restrict__ x, Unit* __restrict__ a, ConvGeom g, int64_t rows,
                  int cu /* units per pixel = C_in / V */) {
  const int U = g.kh * g.kw * cu;
  const int rpb = kConvRowElems / U > 0 ? kConvRowElems / U : 1;  // rows per group
  const int64_t groups = (rows + rpb - 1) / rpb;
  const int T = g.H_out * g.W_out;
  for (int64_t grp = blockIdx.x; grp < groups; grp += gridDim.x) {
    const int64_t r0 = grp * rpb;
    const int n = static_cast<int>((rows - r0 < rpb ? rows - r0 : rpb) * U);
    for (int e = threadIdx.x; e < n; e += kConvThreads) {
      const int dr = e / U, u = e - dr * U;
      const int64_t row = r0 + dr;
      const int i = static_cast<int>(row / T), t = static_cast<int>(row - static_cast<int64_t>(i) * T);
      const int ho = t / g.W_out, wo = t - ho * g.W_out;
      const int tap = u / cu, cc = u - tap * cu;
      const int ki = tap / g.kw, kj = tap - ki * g.kw;
      const int y = ho * g.stride_h + ki - g.pad_h;
      const int xx = wo * g.stride_w + kj - g.pad_w;
      Unit v{};
      if (y >= 0 && y < g.H && xx >= 0 && xx < g.W)
        v = x[((static_cast<int64_t>(i) * g.H + y) * g.W + xx) * cu + cc];
      __stcs(a + row * U + u, v);
    }
  }
}

template <typename Unit>
cudaError_t launch_unfold_t(const void* x, void* a, const ConvGeom& g, int B, int cu,
                            cudaStream_t s) {
  const int64_t rows = static_cast<int64_t>(B) * g.H_out * g.W_out;
  const int U = g.kh * g.kw * cu;
  const int rpb = kConvRowElems / U > 0 ? kConvRowElems / U : 1;
  const int64_t groups = (rows + rpb - 1) / rpb;
  const int64_t cap = static_cast<int64_t>(device_sm_count()) * 8;
  const int grid = static_cast<int>(groups < cap ? groups : cap);
  note_launch();
  k_conv_unfold<Unit><<<grid, kConvThreads, 0, s>>>(static_cast<const Unit*>(x),
                                                     static_cast<Unit*>(a), g, rows, cu);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_conv_unfold(InType t, const void* x, void* a, const ConvGeom& g, int B,
                               cudaStream_t s) {
  if (B < 1) return cudaSuccess;
  const int elem = t == IN_F32 ? 4 : 2;
  const int V = 16 / elem;
  if (g.C_in % V == 0)  // whole 16-byte vectors of channels (x and a are 16-byte aligned)
    return launch_unfold_t<uint4>(x, a, g, B, g.C_in / V, s);
  if (t == IN_F32) return launch_unfold_t<float>(x, a, g, B, g.C_in, s);
  return launch_unfold_t<__nv_bfloat16>(x, a, g, B, g.C_in, s);
}

}  // namespace dpk
