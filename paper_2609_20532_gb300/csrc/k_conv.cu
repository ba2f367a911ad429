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

#include "conv_thin.h"
#include "internal.h"
#include "tc.h"

namespace dpk {

namespace {

constexpr int kConvThreads = 256;
constexpr int kConvRowElems = 4096;  // output units a block takes per row group
constexpr int kConvUPT = 4;          // units a thread loads before it stores them

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
  // rows < 2^31 (checked on the host), so row and position indices are 32-bit
  for (int64_t grp = blockIdx.x; grp < groups; grp += gridDim.x) {
    const int r0 = static_cast<int>(grp * rpb);
    const int n = static_cast<int>((rows - r0 < rpb ? rows - r0 : rpb) * U);
    for (int e0 = threadIdx.x; e0 < n; e0 += kConvThreads * kConvUPT) {
      Unit v[kConvUPT];
      int64_t dst[kConvUPT];
#pragma unroll
      for (int j = 0; j < kConvUPT; ++j) {
        const int e = e0 + j * kConvThreads;
        dst[j] = -1;
        v[j] = Unit{};
        if (e >= n) continue;
        const int dr = e / U, u = e - dr * U;
        const int row = r0 + dr;
        const int i = row / T, t = row - i * T;
        const int ho = t / g.W_out, wo = t - ho * g.W_out;
        const int tap = u / cu, cc = u - tap * cu;
        const int ki = tap / g.kw, kj = tap - ki * g.kw;
        const int y = ho * g.stride_h + ki - g.pad_h;
        const int xx = wo * g.stride_w + kj - g.pad_w;
        dst[j] = static_cast<int64_t>(row) * U + u;
        if (y >= 0 && y < g.H && xx >= 0 && xx < g.W)
          v[j] = x[((static_cast<int64_t>(i) * g.H + y) * g.W + xx) * cu + cc];
      }
#pragma unroll
      for (int j = 0; j < kConvUPT; ++j)
        if (dst[j] >= 0) __stcs(a + dst[j], v[j]);
    }
  }
}

// Row-walking form for rows of at most kConvTab units: a table in shared
// memory gives every unit of a row its tap offsets and channel unit, and
// each warp copies a contiguous run of rows, lanes over the row's units, so
// the loop does no division; (example, h, w) advance by increments.
constexpr int kConvTab = 4096;
constexpr int kConvWarps = kConvThreads / 32;

template <typename Unit>
__global__ void __launch_bounds__(kConvThreads)
    k_conv_unfold_rows(const Unit* __restrict__ x, Unit* __restrict__ a, ConvGeom g, int rows,
                       int cu) {
  extern __shared__ int tab[];  // [3][U]: row offset, column offset, channel unit
  const int U = g.kh * g.kw * cu;
  for (int u = threadIdx.x; u < U; u += kConvThreads) {
    const int tap = u / cu, ki = tap / g.kw;
    tab[u] = ki - g.pad_h;
    tab[U + u] = tap - ki * g.kw - g.pad_w;
    tab[2 * U + u] = u - tap * cu;
  }
  __syncthreads();
  const int lane = static_cast<int>(threadIdx.x) & 31;
  const int64_t warp = static_cast<int64_t>(blockIdx.x) * kConvWarps + (threadIdx.x >> 5);
  const int64_t nwarps = static_cast<int64_t>(gridDim.x) * kConvWarps;
  int row = static_cast<int>(rows * warp / nwarps);
  const int row_end = static_cast<int>(rows * (warp + 1) / nwarps);
  if (row >= row_end) return;
  const int T = g.H_out * g.W_out;
  int i = row / T;
  const int t = row - i * T;
  int ho = t / g.W_out, wo = t - ho * g.W_out;
  for (; row < row_end; ++row) {
    const int y0 = ho * g.stride_h, x0 = wo * g.stride_w;
    const Unit* xi = x + static_cast<int64_t>(i) * g.H * g.W * cu;
    Unit* ar = a + static_cast<int64_t>(row) * U;
    for (int u0 = lane; u0 < U; u0 += 32 * kConvUPT) {
      Unit v[kConvUPT];
#pragma unroll
      for (int j = 0; j < kConvUPT; ++j) {
        const int u = u0 + 32 * j;
        v[j] = Unit{};
        if (u < U) {
          const int y = y0 + tab[u], xx = x0 + tab[U + u];
          if (y >= 0 && y < g.H && xx >= 0 && xx < g.W)
            v[j] = xi[(static_cast<int64_t>(y) * g.W + xx) * cu + tab[2 * U + u]];
        }
      }
#pragma unroll
      for (int j = 0; j < kConvUPT; ++j)
        if (u0 + 32 * j < U) __stcs(ar + u0 + 32 * j, v[j]);
    }
    if (++wo == g.W_out) {
      wo = 0;
      if (++ho == g.H_out) {
        ho = 0;
        ++i;
      }
    }
  }
}

template <typename Unit>
cudaError_t launch_unfold_t(const void* x, void* a, const ConvGeom& g, int B, int cu,
                            cudaStream_t s) {
  const int64_t rows = static_cast<int64_t>(B) * g.H_out * g.W_out;
  const int U = g.kh * g.kw * cu;
  if (U <= kConvTab) {
    const int smem = 3 * U * static_cast<int>(sizeof(int));
    if (smem > 48 * 1024) {
      cudaError_t e = setup_once_per_device(
          reinterpret_cast<const void*>(&k_conv_unfold_rows<Unit>), [] {
            return cudaFuncSetAttribute(k_conv_unfold_rows<Unit>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        3 * kConvTab * static_cast<int>(sizeof(int)));
          });
      if (e != cudaSuccess) return e;
    }
    const int64_t warps_needed = rows;  // at least one row per warp
    const int64_t cap = static_cast<int64_t>(device_sm_count()) * 8;
    int64_t grid = (warps_needed + kConvWarps - 1) / kConvWarps;
    if (grid > cap) grid = cap;
    note_launch();
    k_conv_unfold_rows<Unit><<<static_cast<int>(grid), kConvThreads, smem, s>>>(
        static_cast<const Unit*>(x), static_cast<Unit*>(a), g, static_cast<int>(rows), cu);
    return cudaGetLastError();
  }
  const int rpb = kConvRowElems / U > 0 ? kConvRowElems / U : 1;
  const int64_t groups = (rows + rpb - 1) / rpb;
  const int64_t cap = static_cast<int64_t>(device_sm_count()) * 8;
  const int grid = static_cast<int>(groups < cap ? groups : cap);
  note_launch();
  k_conv_unfold<Unit><<<grid, kConvThreads, 0, s>>>(static_cast<const Unit*>(x),
                                                     static_cast<Unit*>(a), g, rows, cu);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Thin convolution, per-example gradient from the input in shared memory:
//   G_i[j][k] = sum_t a_i[t][j] d_i[t][k]
// with a the patch rows above, for a layer whose per-example gradient the
// step stores (few output channels) and whose input per example fits in
// shared memory.  One block per example holds x_i [H][W][C_in] (fp32) and
// walks the output positions in chunks of kThinChunk, the chunk's output
// gradients [chunk][C_out] staged in shared memory.  Thread (j, q) owns
// gradient row j (tap (ki, kj), channel c) for the positions q, q + Q, ... of
// every chunk and all C_out columns (thread q K + j); the Q partial rows are
// then added in q order, the row is written to G_i, and the squares of the
// example's rows are summed in a fixed order into its single norm partial.
// No patch row is formed in memory; the result differs from the unfolded
// path's only in the order of the fp32 additions.
// ---------------------------------------------------------------------------
constexpr int kThinThreads = 256;
constexpr int kThinChunk = 256;  // positions per staged chunk of d_i

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(__nv_bfloat16 v) { return __bfloat162float(v); }

// Sum over the block's threads: warp butterflies, then the warps' sums in
// warp order (a fixed order).
__device__ __forceinline__ float block_sum(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) red[w] = v;
  __syncthreads();
  float t = lane < static_cast<int>(blockDim.x >> 5) ? red[lane] : 0.f;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
  return t;
}

template <typename TIn, int CO>
__global__ void __launch_bounds__(kThinThreads)
    k_conv_thin_norm(const TIn* __restrict__ x, const TIn* __restrict__ d, ConvGeom g,
                     int c_out, float* __restrict__ G, float* __restrict__ part, int NP,
                     int row0) {
  extern __shared__ __align__(16) float sm[];
  __shared__ float red[32];
  const int HWC = g.H * g.W * g.C_in;
  float* img = sm;                         // [H][W][C_in]
  float* buf = sm + ((HWC + 3) & ~3);      // chunk [kThinChunk][C_out], then [Q][K][C_out]
  const int i = blockIdx.x;
  const int K = g.kh * g.kw * g.C_in;      // <= kThinThreads (host check)
  const int T = g.H_out * g.W_out;
  const int Q = kThinThreads / K;
  const int tid = threadIdx.x;
  const TIn* xi = x + static_cast<int64_t>(i) * HWC;
  const TIn* di = d + static_cast<int64_t>(i) * T * c_out;
  for (int e = tid; e < HWC; e += kThinThreads) img[e] = to_f(xi[e]);
  // consecutive threads take consecutive rows j at the same positions, so a
  // warp's reads of a staged output-gradient row are one broadcast
  const int q = tid / K, j = tid - q * K;
  const bool own = q < Q;
  int ki = 0, kj = 0, ch = 0;
  if (own) {
    const int tap = j / g.C_in;
    ch = j - tap * g.C_in;
    ki = tap / g.kw;
    kj = tap - ki * g.kw;
  }
  float acc[CO];
#pragma unroll
  for (int k = 0; k < CO; ++k) acc[k] = 0.f;
  const bool vec4 = (c_out & 3) == 0;  // staged rows 16-byte aligned
  for (int t0 = 0; t0 < T; t0 += kThinChunk) {
    const int nt = T - t0 < kThinChunk ? T - t0 : kThinChunk;
    __syncthreads();  // the image is in place; the previous chunk is used up
    for (int e = tid; e < nt * c_out; e += kThinThreads)
      buf[e] = to_f(di[static_cast<int64_t>(t0) * c_out + e]);
    __syncthreads();
    if (own) {
      for (int tt = q; tt < nt; tt += Q) {
        const int t = t0 + tt;
        const int ho = t / g.W_out, wo = t - ho * g.W_out;
        const int y = ho * g.stride_h + ki - g.pad_h, xx = wo * g.stride_w + kj - g.pad_w;
        if (y < 0 || y >= g.H || xx < 0 || xx >= g.W) continue;  // zero padding
        const float v = img[(y * g.W + xx) * g.C_in + ch];
        const float* dr = buf + tt * c_out;
        if (vec4) {  // the row as float4 broadcasts: a quarter of the shared loads
#pragma unroll
          for (int k4 = 0; k4 < CO / 4; ++k4) {
            if (4 * k4 >= c_out) break;
            const float4 d4 = *reinterpret_cast<const float4*>(dr + 4 * k4);
            acc[4 * k4 + 0] = fmaf(v, d4.x, acc[4 * k4 + 0]);
            acc[4 * k4 + 1] = fmaf(v, d4.y, acc[4 * k4 + 1]);
            acc[4 * k4 + 2] = fmaf(v, d4.z, acc[4 * k4 + 2]);
            acc[4 * k4 + 3] = fmaf(v, d4.w, acc[4 * k4 + 3]);
          }
        } else {
#pragma unroll
          for (int k = 0; k < CO; ++k)
            if (k < c_out) acc[k] = fmaf(v, dr[k], acc[k]);
        }
      }
    }
  }
  __syncthreads();
  if (own) {
#pragma unroll
    for (int k = 0; k < CO; ++k)
      if (k < c_out) buf[(q * K + j) * c_out + k] = acc[k];
  }
  __syncthreads();
  float sq = 0.f;
  if (tid < K) {
    float* gi = G + (static_cast<int64_t>(i) * K + tid) * c_out;
    for (int k = 0; k < c_out; ++k) {
      float s = 0.f;
      for (int r = 0; r < Q; ++r) s += buf[(r * K + tid) * c_out + k];
      gi[k] = s;
      sq = fmaf(s, s, sq);
    }
  }
  sq = block_sum(sq, red);
  if (tid == 0) part[static_cast<int64_t>(row0 + i) * NP] = sq;
}

int64_t thin_smem_bytes(const ConvGeom& g, int64_t c_out) {
  const int64_t hwc = static_cast<int64_t>(g.H) * g.W * g.C_in;
  return (((hwc + 3) & ~int64_t(3)) + int64_t(kThinChunk) * c_out) * 4;
}

template <typename TIn, int CO>
cudaError_t launch_thin_t(const void* x, const void* d, const ConvGeom& g, int c_out, int B,
                          float* G, float* part, int NP, int row0, cudaStream_t s) {
  const int smem = static_cast<int>(thin_smem_bytes(g, c_out));  // <= kConvThinMaxSmem
  if (smem > 48 * 1024) {
    cudaError_t e = setup_once_per_device(
        reinterpret_cast<const void*>(&k_conv_thin_norm<TIn, CO>), [] {
          return cudaFuncSetAttribute(k_conv_thin_norm<TIn, CO>,
                                      cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      kConvThinMaxSmem);
        });
    if (e != cudaSuccess) return e;
  }
  note_launch();
  k_conv_thin_norm<TIn, CO><<<B, kThinThreads, smem, s>>>(
      static_cast<const TIn*>(x), static_cast<const TIn*>(d), g, c_out, G, part, NP, row0);
  return cudaGetLastError();
}

template <typename TIn>
cudaError_t launch_thin_co(const void* x, const void* d, const ConvGeom& g, int c_out, int B,
                           float* G, float* part, int NP, int row0, cudaStream_t s) {
  if (c_out <= 16) return launch_thin_t<TIn, 16>(x, d, g, c_out, B, G, part, NP, row0, s);
  if (c_out <= 32) return launch_thin_t<TIn, 32>(x, d, g, c_out, B, G, part, NP, row0, s);
  return launch_thin_t<TIn, 64>(x, d, g, c_out, B, G, part, NP, row0, s);
}

}  // namespace

bool conv_thin_norm_ok(const ConvGeom& g, int64_t c_out) {
  const int64_t K = static_cast<int64_t>(g.kh) * g.kw * g.C_in;
  return K >= 1 && K <= kThinThreads && c_out >= 1 && c_out <= 64 && g.H >= 1 && g.W >= 1 &&
         thin_smem_bytes(g, c_out) <= kConvThinMaxSmem;
}

cudaError_t launch_conv_thin_norm(InType t, const void* x, const void* d, const ConvGeom& g,
                                  int c_out, int B, float* G, float* part, int NP, int row0,
                                  cudaStream_t s) {
  if (B < 1) return cudaSuccess;
  if (!conv_thin_norm_ok(g, c_out)) return cudaErrorInvalidValue;
  if (t == IN_F32) return launch_thin_co<float>(x, d, g, c_out, B, G, part, NP, row0, s);
  return launch_thin_co<__nv_bfloat16>(x, d, g, c_out, B, G, part, NP, row0, s);
}

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
