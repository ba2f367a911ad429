// The GPU's update after the trusted side releases the step's noise seed
// (Algorithm 2): g~ = committed average + out_scale * sigma * C * z, then
// OptStep = AdamW as the paper writes its one-step map (App. A):
//   m = b1 m + (1 - b1) g,  v = b2 v + (1 - b2) g^2,
//   theta <- theta - lr (m / (1 - b1^t) / (sqrt(v / (1 - b2^t)) + eps) + wd theta).
// One pass over the parameters: the noise is generated in registers (the
// same Philox quads and global indices as every other noise path), so the
// kernel moves 28 bytes per parameter (32 when it also writes g~ back).
#include <cuda_runtime.h>

#include "internal.h"
#include "philox.cuh"

namespace dpk {

namespace {

__device__ __forceinline__ void adamw1(float g, float& th, float& m, float& v, const AdamWArgs& h) {
  m = fmaf(h.beta1, m, (1.f - h.beta1) * g);
  v = fmaf(h.beta2, v, (1.f - h.beta2) * g * g);
  const float mh = m * h.bc1;
  const float vh = v * h.bc2;
  th = th - h.lr * (mh / (sqrtf(vh) + h.eps) + h.weight_decay * th);
}

__global__ void __launch_bounds__(256) k_noise_adamw(float* __restrict__ grad, float* __restrict__ theta,
                                                     float* __restrict__ m, float* __restrict__ v,
                                                     int64_t n, uint64_t p_base,
                                                     const uint64_t* __restrict__ key,
                                                     float noise_scale, int add_noise, int write_grad,
                                                     AdamWArgs h) {
  const PhiloxKeys keys = philox_keys(key[0]);  // round keys formed once per thread
  const uint64_t step = key[1];
  const uint64_t q_first = p_base >> 2;
  const int64_t nq = static_cast<int64_t>(((p_base + n - 1) >> 2) - q_first + 1);
  const bool vec = ((p_base & 3) == 0) &&
                   (((reinterpret_cast<uintptr_t>(grad) | reinterpret_cast<uintptr_t>(theta) |
                      reinterpret_cast<uintptr_t>(m) | reinterpret_cast<uintptr_t>(v)) & 15) == 0);
  for (int64_t gq = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; gq < nq;
       gq += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const uint64_t q = q_first + gq;
    float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
    if (add_noise) z = gauss_quad(keys, step, q);
    const int64_t e0 = static_cast<int64_t>(4 * q) - static_cast<int64_t>(p_base);
    if (vec && e0 + 3 < n) {
      float4 g = *reinterpret_cast<const float4*>(grad + e0);
      float4 th = *reinterpret_cast<const float4*>(theta + e0);
      float4 mm = *reinterpret_cast<const float4*>(m + e0);
      float4 vv = *reinterpret_cast<const float4*>(v + e0);
      g.x = fmaf(noise_scale, z.x, g.x);
      g.y = fmaf(noise_scale, z.y, g.y);
      g.z = fmaf(noise_scale, z.z, g.z);
      g.w = fmaf(noise_scale, z.w, g.w);
      adamw1(g.x, th.x, mm.x, vv.x, h);
      adamw1(g.y, th.y, mm.y, vv.y, h);
      adamw1(g.z, th.z, mm.z, vv.z, h);
      adamw1(g.w, th.w, mm.w, vv.w, h);
      *reinterpret_cast<float4*>(theta + e0) = th;
      *reinterpret_cast<float4*>(m + e0) = mm;
      *reinterpret_cast<float4*>(v + e0) = vv;
      if (write_grad) *reinterpret_cast<float4*>(grad + e0) = g;
    } else {
      const float zv[4] = {z.x, z.y, z.z, z.w};
#pragma unroll
      for (int w = 0; w < 4; ++w) {
        const int64_t e = e0 + w;
        if (e < 0 || e >= n) continue;
        const float g = fmaf(noise_scale, zv[w], grad[e]);
        float th = theta[e], mm = m[e], vv = v[e];
        adamw1(g, th, mm, vv, h);
        theta[e] = th;
        m[e] = mm;
        v[e] = vv;
        if (write_grad) grad[e] = g;
      }
    }
  }
}

}  // namespace

cudaError_t launch_noise_adamw(float* grad, float* theta, float* m, float* v, int64_t n,
                               uint64_t p_base, const uint64_t* key, float noise_scale,
                               int add_noise, int write_grad, const AdamWArgs& h, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  const int64_t nq = static_cast<int64_t>(((p_base + n - 1) >> 2) - (p_base >> 2) + 1);
  int64_t blocks = (nq + 255) / 256;
  const int64_t cap = 152 * 8;
  note_launch();
  if (blocks > cap) blocks = cap;
  k_noise_adamw<<<static_cast<int>(blocks), 256, 0, s>>>(grad, theta, m, v, n, p_base, key,
                                                         noise_scale, add_noise, write_grad, h);
  return cudaGetLastError();
}

}  // namespace dpk
