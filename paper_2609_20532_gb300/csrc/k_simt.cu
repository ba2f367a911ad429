// CUDA-core kernels of the DP-SGD step: per-example norms (rank-1, Gram and
// materialised forms), the cross-layer clip-factor kernel, the fp32 clipped
// sum with its fused noise epilogue, the standalone noise add, the audit
// gather and the generator exports.
//
// The clipped sum here is the fp32 path (an FFMA GEMM, exact in the inputs'
// precision); bf16 layers whose T is a multiple of the tensor-core K-block
// go through the tcgen05 kernels instead.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "internal.h"
#include "philox.cuh"
#include "tc_util.cuh"

namespace dpk {

namespace {

__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(__nv_bfloat16 x) { return __bfloat162float(x); }

// Sum of v over the block (blockDim.x a multiple of 32, <= 1024); result in
// every thread.  Fixed reduction order, so results are reproducible.
__device__ __forceinline__ float block_sum(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) red[w] = v;
  __syncthreads();
  const int nw = blockDim.x >> 5;
  float t = lane < nw ? red[lane] : 0.f;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
  return t;
}

// ---------------------------------------------------------------------------
// Rank-1 norm (T = 1): n_i = ||a_i||^2 ||d_i||^2
// ---------------------------------------------------------------------------
template <typename TIn>
__global__ void __launch_bounds__(256) k_norm_rank1(const TIn* __restrict__ A,
                                                    const TIn* __restrict__ D, int d_in, int d_out,
                                                    float* __restrict__ part, int NP, int row0) {
  __shared__ float red[32];
  const int i = blockIdx.x;
  const TIn* a = A + static_cast<int64_t>(i) * d_in;
  const TIn* d = D + static_cast<int64_t>(i) * d_out;
  float sa = 0.f, sd = 0.f;
  for (int j = threadIdx.x; j < d_in; j += blockDim.x) {
    const float v = to_f(a[j]);
    sa = fmaf(v, v, sa);
  }
  for (int k = threadIdx.x; k < d_out; k += blockDim.x) {
    const float v = to_f(d[k]);
    sd = fmaf(v, v, sd);
  }
  sa = block_sum(sa, red);
  sd = block_sum(sd, red);
  if (threadIdx.x == 0) part[static_cast<int64_t>(row0 + i) * NP] = sa * sd;
}

// ---------------------------------------------------------------------------
// Gram ("ghost") norm: n_i = sum_{t,s} (a_t . a_s)(d_t . d_s).
// One block per (example, 64x64 tile pair (bt <= bs) of the T x T Grams);
// off-diagonal tiles count twice, the upper and lower halves being equal.
// ---------------------------------------------------------------------------
constexpr int GT = 64;   // Gram tile edge
constexpr int GF = 32;   // features per staged chunk

__device__ __forceinline__ void pair_of(int pid, int nb, int& bt, int& bs) {
  // enumerate (bt, bs), bt <= bs, row by row
  int r = 0, left = pid;
  while (left >= nb - r) {
    left -= nb - r;
    ++r;
  }
  bt = r;
  bs = r + left;
}

template <typename TIn>
__device__ __forceinline__ void gram_tile(const TIn* __restrict__ X, int T, int d, int t0, int s0,
                                          float (&g)[4][4], float (*Xt)[GT + 4],
                                          float (*Xs)[GT + 4]) {
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  for (int f0 = 0; f0 < d; f0 += GF) {
#pragma unroll
    for (int r = 0; r < (GT * GF) / 256; ++r) {
      const int e = tid + 256 * r;
      const int row = e / GF, f = e % GF;
      const int t = t0 + row, s = s0 + row, ff = f0 + f;
      Xt[f][row] = (t < T && ff < d) ? to_f(X[static_cast<int64_t>(t) * d + ff]) : 0.f;
      Xs[f][row] = (s < T && ff < d) ? to_f(X[static_cast<int64_t>(s) * d + ff]) : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int f = 0; f < GF; ++f) {
      const float4 a = *reinterpret_cast<const float4*>(&Xt[f][ty * 4]);
      const float4 b = *reinterpret_cast<const float4*>(&Xs[f][tx * 4]);
      const float av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) g[u][v] = fmaf(av[u], bv[v], g[u][v]);
    }
    __syncthreads();
  }
}

template <typename TIn>
__global__ void __launch_bounds__(256) k_norm_ghost_simt(const TIn* __restrict__ A,
                                                         const TIn* __restrict__ D, int T, int d_in,
                                                         int d_out, float* __restrict__ part,
                                                         int NP, int row0) {
  __shared__ __align__(16) float Xt[GF][GT + 4];
  __shared__ __align__(16) float Xs[GF][GT + 4];
  __shared__ float red[32];
  const int nb = (T + GT - 1) / GT;
  int bt, bs;
  pair_of(blockIdx.x, nb, bt, bs);
  const int i = blockIdx.y;
  const int t0 = bt * GT, s0 = bs * GT;
  float ga[4][4] = {}, gd[4][4] = {};
  gram_tile(A + static_cast<int64_t>(i) * T * d_in, T, d_in, t0, s0, ga, Xt, Xs);
  gram_tile(D + static_cast<int64_t>(i) * T * d_out, T, d_out, t0, s0, gd, Xt, Xs);
  float acc = 0.f;
#pragma unroll
  for (int u = 0; u < 4; ++u)
#pragma unroll
    for (int v = 0; v < 4; ++v) acc = fmaf(ga[u][v], gd[u][v], acc);
  acc = block_sum(acc, red);
  if (threadIdx.x == 0)
    part[static_cast<int64_t>(row0 + i) * NP + blockIdx.x] = (bt == bs ? 1.f : 2.f) * acc;
}

// ---------------------------------------------------------------------------
// FFMA GEMM over positions: tile TB (d_in) x TB (d_out), K-chunks of SK rows,
// 256 threads with 8 x 8 outputs each.
// CLIPSUM: S = sum_k c[k / T] A[k, :]^T D[k, :] over all B*T rows, + epilogue.
// NORM:    per example (blockIdx.z), G tile = A_i^T D_i, writes sum of squares.
// TB = 128: one group of 256 threads walks all chunks.  TB = 64 (grids too
// small to fill the GPU twice with 128-wide tiles): four groups of 64
// threads each walk every fourth chunk, so a block keeps four chains of
// loads and multiply-adds in flight, and the groups' tiles are added in
// shared memory in a fixed order, ((g0 + g2) + (g1 + g3)).
// ---------------------------------------------------------------------------
constexpr int SB = 128, SK = 16;

template <typename TIn, bool NORM, int TB>
__global__ void __launch_bounds__(256) k_gemm_simt(const TIn* __restrict__ A,
                                                   const TIn* __restrict__ D,
                                                   const float* __restrict__ cvec, int T, int B,
                                                   int d_in, int d_out, float* __restrict__ out,
                                                   Epilogue ep, float* __restrict__ part, int NP,
                                                   int row0) {
  constexpr int KG = TB == 128 ? 1 : 4;  // K groups
  constexpr int GTH = 256 / KG;          // threads per group
  constexpr int TD = TB / 8;             // a group's threads per tile row
  constexpr int HALF = TB / 2;
  constexpr int LPT = (SK * TB) / GTH;   // A (and D) elements per thread and chunk
  static_assert(TD * TD == GTH && TB % 64 == 0, "8 x 8 outputs per thread");
  static_assert(KG == 1 || KG * SK * TB == TB * TB, "a group's tile fits one operand buffer");
  __shared__ __align__(16) float As[KG][SK][TB];
  __shared__ __align__(16) float Ds[KG][SK][TB];
  __shared__ float red[32];
  const int tid = threadIdx.x, grp = tid / GTH, gt = tid % GTH, tx = gt % TD, ty = gt / TD;
  const int j0 = blockIdx.y * TB, k0 = blockIdx.x * TB;
  int64_t K;
  if (NORM) {
    const int64_t i = blockIdx.z;
    A += i * T * d_in;
    D += i * T * d_out;
    K = T;
  } else {
    K = static_cast<int64_t>(B) * T;
  }
  const int64_t nch = (K + SK - 1) / SK;
  float acc[8][8] = {};
  // The group's next chunk is loaded into registers while the current one is
  // multiplied out of shared memory; the loads only load (the clip factor is
  // applied when the chunk is stored to shared memory), so all of a chunk's
  // loads are in flight together.  Rows stay below B T <= 2^31 - 1, so a
  // row's example index is a 32-bit division.
  float ra[LPT], rc[LPT], rd[LPT];
  auto load = [&](int64_t ch) {
    const int64_t kk = ch * SK;
#pragma unroll
    for (int r = 0; r < LPT; ++r) {
      const int e = gt + GTH * r;
      const int row = e / TB, col = e % TB;
      const int64_t kr = kk + row;
      const int j = j0 + col, k = k0 + col;
      const bool in_k = kr < K;
      ra[r] = in_k && j < d_in ? to_f(A[kr * d_in + j]) : 0.f;
      rc[r] = !NORM && in_k ? cvec[static_cast<uint32_t>(kr) / static_cast<uint32_t>(T)] : 1.f;
      rd[r] = in_k && k < d_out ? to_f(D[kr * d_out + k]) : 0.f;
    }
  };
  if (grp < nch) load(grp);
  const int64_t rounds = (nch + KG - 1) / KG;
  for (int64_t rnd = 0; rnd < rounds; ++rnd) {
    const int64_t ch = rnd * KG + grp;
    const bool have = ch < nch;
    if (have) {
#pragma unroll
      for (int r = 0; r < LPT; ++r) {
        const int e = gt + GTH * r;
        As[grp][e / TB][e % TB] = NORM ? ra[r] : ra[r] * rc[r];
        Ds[grp][e / TB][e % TB] = rd[r];
      }
    }
    __syncthreads();
    if (ch + KG < nch) load(ch + KG);
    if (have) {
#pragma unroll
      for (int q = 0; q < SK; ++q) {
        float av[8], bv[8];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const float4 a = *reinterpret_cast<const float4*>(&As[grp][q][h * HALF + ty * 4]);
          const float4 b = *reinterpret_cast<const float4*>(&Ds[grp][q][h * HALF + tx * 4]);
          av[4 * h + 0] = a.x; av[4 * h + 1] = a.y; av[4 * h + 2] = a.z; av[4 * h + 3] = a.w;
          bv[4 * h + 0] = b.x; bv[4 * h + 1] = b.y; bv[4 * h + 2] = b.z; bv[4 * h + 3] = b.w;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u)
#pragma unroll
          for (int v = 0; v < 8; ++v) acc[u][v] = fmaf(av[u], bv[v], acc[u][v]);
      }
    }
    __syncthreads();
  }
  // tile row and column of this thread's output (u, v)
  auto trow = [&](int u) { return (u / 4) * HALF + ty * 4 + (u % 4); };
  auto tcol = [&](int v) { return (v / 4) * HALF + tx * 4 + (v % 4); };

  if constexpr (KG > 1) {
    // ((g0 + g2) + (g1 + g3)) through the two operand buffers, one tile each
    auto slot = [&](int i) { return i ? &Ds[0][0][0] : &As[0][0][0]; };
    auto put = [&](float* t) {
#pragma unroll
      for (int u = 0; u < 8; ++u)
#pragma unroll
        for (int v = 0; v < 8; ++v) t[trow(u) * TB + tcol(v)] = acc[u][v];
    };
    auto add = [&](const float* t) {
#pragma unroll
      for (int u = 0; u < 8; ++u)
#pragma unroll
        for (int v = 0; v < 8; ++v) acc[u][v] += t[trow(u) * TB + tcol(v)];
    };
    if (grp >= 2) put(slot(grp - 2));
    __syncthreads();
    if (grp < 2) add(slot(grp));
    __syncthreads();
    if (grp == 1) put(slot(0));
    __syncthreads();
    if (grp == 0) {
      add(slot(0));
      put(slot(0));
    }
    __syncthreads();
    // the block's tile is in slot 0; every thread takes 4 quads of it
    const float* tile = slot(0);
    if constexpr (NORM) {
      float sq = 0.f;
#pragma unroll
      for (int m = 0; m < (TB * TB) / 256; ++m) {
        const float x = tile[tid + 256 * m];
        sq = fmaf(x, x, sq);  // padding is zero
      }
      sq = block_sum(sq, red);
      if (tid == 0) {
        const int t_ = blockIdx.y * gridDim.x + blockIdx.x;
        part[static_cast<int64_t>(row0 + blockIdx.z) * NP + t_] = sq;
      }
    } else {
#pragma unroll
      for (int m = 0; m < (TB * TB) / (4 * 256); ++m) {
        const int qd = tid + 256 * m;
        const int r = qd / (TB / 4), c4 = (qd % (TB / 4)) * 4;
        const int j = j0 + r, kb = k0 + c4;
        if (j >= d_in || kb >= d_out) continue;
        float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
        if (ep.add_noise) z = gauss4_at(ep.key[0], ep.key[1], ep.p_base + static_cast<uint64_t>(j) * d_out + kb);
        const float zv[4] = {z.x, z.y, z.z, z.w};
        float* o = out + static_cast<int64_t>(j) * d_out;
#pragma unroll
        for (int v = 0; v < 4; ++v) {
          const int k = kb + v;
          if (k < d_out) {
            const float val = ep.out_scale * fmaf(ep.sigmaC, zv[v], tile[r * TB + c4 + v]);
            o[k] = ep.accumulate ? o[k] + val : val;
          }
        }
      }
    }
  } else if constexpr (NORM) {
    float sq = 0.f;
#pragma unroll
    for (int u = 0; u < 8; ++u)
#pragma unroll
      for (int v = 0; v < 8; ++v) sq = fmaf(acc[u][v], acc[u][v], sq);  // padding is zero
    sq = block_sum(sq, red);
    if (tid == 0) {
      const int t_ = blockIdx.y * gridDim.x + blockIdx.x;
      part[static_cast<int64_t>(row0 + blockIdx.z) * NP + t_] = sq;
    }
  } else {
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int j = j0 + trow(u);
      if (j >= d_in) continue;
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int kb = k0 + h * HALF + tx * 4;
        if (kb >= d_out) continue;
        float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
        const uint64_t p0 = ep.p_base + static_cast<uint64_t>(j) * d_out + kb;
        if (ep.add_noise) z = gauss4_at(ep.key[0], ep.key[1], p0);
        const float zv[4] = {z.x, z.y, z.z, z.w};
        float* o = out + static_cast<int64_t>(j) * d_out;
#pragma unroll
        for (int v = 0; v < 4; ++v) {
          const int k = kb + v;
          if (k < d_out) {
            const float val = ep.out_scale * fmaf(ep.sigmaC, zv[v], acc[u][h * 4 + v]);
            o[k] = ep.accumulate ? o[k] + val : val;
          }
        }
      }
    }
  }
}

// ---------------------------------------------------------------------------
// Cross-layer sum and clip factors, in one of three arrangements chosen by
// the partials per example of a layer (NP); the order of the additions
// never depends on timing.
//   WARPS = 0 (NP < 64: few partials, maybe many layers, e.g. LoRA factors):
//     one warp per example, lane j adds the layers j, j + 32, ... (each
//     layer's partials in slot order), then a fixed butterfly adds the 32
//     lane sums;
//   WARPS = 1 or 8 (thousands of partials per layer: one per tile and
//     epilogue warp of the materialised form): a group of WARPS warps per
//     example; for each layer in turn, thread j of the group adds the
//     partials j, j + G, ... (G = 32 WARPS threads; coalesced), a fixed
//     butterfly adds each warp's 32 sums and the warps' sums are added in
//     warp order; thread 0 adds the layer sums in layer order.
// ---------------------------------------------------------------------------
// mode kClipLocal: only the layers' norms and their sum (into user_s); no
// clip factor, no flag.  mode kClipGiven: s_i = s_given[i] (the squared norm
// summed over every rank's layers) instead of this context's sum.
template <int WARPS>
__global__ void k_clip(const float* __restrict__ part, int L, int B, int NP,
                       const int* __restrict__ nparts, float C, float* __restrict__ layer_sq,
                       float* __restrict__ s_out, float* __restrict__ c_out,
                       float* __restrict__ user_s, float* __restrict__ user_c, int* flag,
                       int mode, const float* __restrict__ s_given) {
  constexpr int G = WARPS > 0 ? 32 * WARPS : 32;  // threads per example
  __shared__ float red[WARPS > 0 ? WARPS : 1];
  const int64_t gid = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  const int64_t w = gid / G;
  const int t = static_cast<int>(gid - w * G);
  const int lane = t & 31;
  if (w >= B) return;  // a whole group leaves together (WARPS > 1: one group per block)
  const int i = static_cast<int>(w);
  float s = 0.f;
  if constexpr (WARPS == 0) {
    for (int l = lane; l < L; l += 32) {
      const float* p = part + (static_cast<int64_t>(l) * B + i) * NP;
      const int np = nparts[l];
      float n = 0.f;
      for (int q = 0; q < np; ++q) n += p[q];
      layer_sq[static_cast<int64_t>(l) * B + i] = n;
      s += n;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  }
  for (int l = 0; l < (WARPS > 0 ? L : 0); ++l) {
    const float* p = part + (static_cast<int64_t>(l) * B + i) * NP;
    const int np = nparts[l];
    float n = 0.f;
    for (int q = t; q < np; q += G) n += p[q];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) n += __shfl_xor_sync(0xffffffffu, n, o);
    if constexpr (WARPS > 1) {
      if (lane == 0) red[t >> 5] = n;
      __syncthreads();
      n = 0.f;
#pragma unroll
      for (int k = 0; k < WARPS; ++k) n += red[k];
      __syncthreads();
    }
    if (t == 0) layer_sq[static_cast<int64_t>(l) * B + i] = n;
    s += n;
  }
  if (t != 0) return;
  if (mode == kClipLocal) {
    user_s[i] = s;
    return;
  }
  if (mode == kClipGiven) s = s_given[i];
  float c;
  if (!isfinite(s)) {
    atomicOr(flag, 1);
    c = __int_as_float(0x7fc00000);  // NaN
  } else {
    c = (s <= C * C) ? 1.f : C / sqrtf(s);
  }
  s_out[i] = s;
  c_out[i] = c;
  if (user_s) user_s[i] = s;
  if (user_c) user_c[i] = c;
}

// ---------------------------------------------------------------------------
// Standalone noise add: out[e] += scale * z_{p_base + e}
// ---------------------------------------------------------------------------
// out[e] += scale * z for the four parameters of quad q (e0 = 4q - p_base,
// possibly negative for the first quad of an unaligned layer).
__device__ __forceinline__ void noise_store(float* __restrict__ out, int64_t e0, int64_t n,
                                            bool vec, float scale, float4 z) {
  if (vec && e0 + 3 < n) {
    float4* o = reinterpret_cast<float4*>(out + e0);
    float4 v = *o;
    v.x = fmaf(scale, z.x, v.x);
    v.y = fmaf(scale, z.y, v.y);
    v.z = fmaf(scale, z.z, v.z);
    v.w = fmaf(scale, z.w, v.w);
    *o = v;
  } else {
    const float zv[4] = {z.x, z.y, z.z, z.w};
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const int64_t e = e0 + w;
      if (e >= 0 && e < n) out[e] = fmaf(scale, zv[w], out[e]);
    }
  }
}

// Each block adds the noise of one contiguous chunk of kNoiseChunk quads of
// one layer (the quads that overlap [p_base, p_base + n)).  Threads take two
// quads 256 apart per iteration: two independent Philox / Box-Muller chains
// give the scheduler instruction-level parallelism, and the chunk keeps the
// index arithmetic in 32 bits.
__global__ void __launch_bounds__(256) k_noise_add(const __grid_constant__ NoiseAddBatch b) {
  int l = 0;
  while (l + 1 < b.L && static_cast<int64_t>(blockIdx.x) >= b.block0[l + 1]) ++l;
  const PhiloxKeys keys = philox_keys(b.key[0]);  // round keys formed once per thread
  const uint64_t step = b.key[1];
  float* __restrict__ out = b.out[l];
  const int64_t n = b.n[l];
  const uint64_t p_base = b.p_base[l];
  const uint64_t q_first = p_base >> 2;
  const int64_t nq = static_cast<int64_t>(((p_base + n - 1) >> 2) - q_first + 1);
  const int64_t c0 = (static_cast<int64_t>(blockIdx.x) - b.block0[l]) * kNoiseChunk;
  const int64_t rem = nq - c0;
  const int cnt = rem < kNoiseChunk ? static_cast<int>(rem) : kNoiseChunk;
  const uint64_t q0 = q_first + c0;
  const int64_t e_base = static_cast<int64_t>(4 * q0) - static_cast<int64_t>(p_base);
  const bool vec = (p_base & 3) == 0;
  for (int j = threadIdx.x; j < cnt; j += 512) {
    const bool has_b = j + 256 < cnt;
    const int jb = has_b ? j + 256 : j;
    const float4 za = gauss_quad(keys, step, q0 + j);
    const float4 zb = gauss_quad(keys, step, q0 + jb);
    noise_store(out, e_base + 4 * j, n, vec, b.scale, za);
    if (has_b) noise_store(out, e_base + 4 * jb, n, vec, b.scale, zb);
  }
}

// ---------------------------------------------------------------------------
// Audit gather: rec[r] = {idx, s, c, n_1..n_L}
// ---------------------------------------------------------------------------
// Gather the audit records of the n requested examples.  idx, rec and
// flag_out are device views of mapped pinned host memory: the indices are
// read and the records written over the host link by this kernel, so an
// audit uses no copy engine.  Thread 0 also reports the step's sticky flag.
__global__ void k_audit(const volatile int* idx, int n, int L, int B,
                        const float* __restrict__ layer_sq, const float* __restrict__ s_vec,
                        const float* __restrict__ c_vec, const int* __restrict__ flag,
                        volatile float* rec, volatile int* flag_out) {
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r == 0) *flag_out = *flag;
  if (r >= n) return;
  const int i = idx[r];
  volatile float* o = rec + static_cast<int64_t>(r) * (3 + L);
  reinterpret_cast<volatile int*>(o)[0] = i;
  o[1] = s_vec[i];
  o[2] = c_vec[i];
  for (int l = 0; l < L; ++l) o[3 + l] = layer_sq[l * B + i];
}

// Start of a step: copy the noise key from mapped pinned host memory to
// device memory and clear the step's sticky flag word.  A kernel instead of
// a DMA copy and a memset: it runs on the SMs, so it never queues behind
// large host<->device copies on the copy engines, and inside a CUDA graph it
// reads the host words current at replay time.
__global__ void k_load_key(const volatile uint64_t* host_key, uint64_t* __restrict__ key,
                           int* __restrict__ flag) {
  key[0] = host_key[0];
  key[1] = host_key[1];
  *flag = 0;
}

// The same for eager launches: the key travels as a kernel argument, fixed
// when the launch is enqueued, so a later re-key cannot reach a step that
// is still queued.
__global__ void k_set_key(uint64_t seed, uint64_t step, uint64_t* __restrict__ key,
                          int* __restrict__ flag) {
  key[0] = seed;
  key[1] = step;
  *flag = 0;
}

// A wait that runs out: one thread waits, with the pipelines' bounded-wait
// helper, for phase 0 of an mbarrier that nothing ever arrives on; after
// limit_ns it records the timeout in *err and the kernel returns.  No TMA
// copy, no MMA and no TMEM are involved, so nothing is left in flight.
__global__ void k_debug_wait(uint64_t limit_ns, int* err) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    tc::mbar_init(&bar, 1);
    abort_flag = 0;
    tc::fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) tc::mbar_wait_for(&bar, 0, &abort_flag, err, limit_ns);
}

__global__ void k_debug_philox(uint64_t seed, uint64_t step, uint64_t q0, int64_t nq,
                               uint32_t* __restrict__ out) {
  for (int64_t r = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; r < nq;
       r += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const uint64_t q = q0 + r;
    const uint4 w = philox4x32_10(philox_counter(q, step), static_cast<uint32_t>(seed),
                                  static_cast<uint32_t>(seed >> 32));
    out[4 * r + 0] = w.x;
    out[4 * r + 1] = w.y;
    out[4 * r + 2] = w.z;
    out[4 * r + 3] = w.w;
  }
}

__global__ void k_debug_gauss(uint64_t seed, uint64_t step, uint64_t p0, int64_t n,
                              float* __restrict__ out) {
  for (int64_t r = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; r < n;
       r += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const uint64_t p = p0 + r;
    const float4 z = gauss_quad(seed, step, p >> 2);
    const float zv[4] = {z.x, z.y, z.z, z.w};
    out[r] = zv[p & 3];
  }
}

int grid_for(int64_t work, int threads) {
  const int64_t g = (work + threads - 1) / threads;
  const int64_t cap = 152 * 16;
  return static_cast<int>(g < 1 ? 1 : (g > cap ? cap : g));
}

}  // namespace

int64_t rank1_parts() { return 1; }
int64_t ghost_simt_parts(int T) {
  const int64_t nb = (static_cast<int64_t>(T) + GT - 1) / GT;
  return nb * (nb + 1) / 2;
}
int64_t mat_simt_parts(int64_t d_in, int64_t d_out) {
  return ((d_in + SB - 1) / SB) * ((d_out + SB - 1) / SB);
}

// The per-example norm kernels below index examples with blockIdx.y / .z,
// which stop at 65535: larger batches launch once per 65535 examples, each
// launch on its slice of A, D and the partial-sum rows.
constexpr int kMaxGridYZ = 65535;

template <typename F>
cudaError_t per_example_slices(InType t, const void* A, const void* D, int B, int T, int d_in,
                               int d_out, int row0, F&& launch) {
  const int64_t es = t == IN_F32 ? 4 : 2;
  for (int b0 = 0; b0 < B; b0 += kMaxGridYZ) {
    const int nb = B - b0 < kMaxGridYZ ? B - b0 : kMaxGridYZ;
    const char* a = static_cast<const char*>(A) + static_cast<int64_t>(b0) * T * d_in * es;
    const char* d = static_cast<const char*>(D) + static_cast<int64_t>(b0) * T * d_out * es;
    launch(static_cast<const void*>(a), static_cast<const void*>(d), nb, row0 + b0);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t launch_norm_rank1(InType t, const void* A, const void* D, int B, int d_in, int d_out,
                              float* part, int NP, int row0, cudaStream_t s) {
  note_launch();
  if (t == IN_F32)
    k_norm_rank1<float><<<B, 256, 0, s>>>(static_cast<const float*>(A),
                                           static_cast<const float*>(D), d_in, d_out, part, NP,
                                           row0);
  else
    k_norm_rank1<__nv_bfloat16><<<B, 256, 0, s>>>(static_cast<const __nv_bfloat16*>(A),
                                                   static_cast<const __nv_bfloat16*>(D), d_in,
                                                   d_out, part, NP, row0);
  return cudaGetLastError();
}

cudaError_t launch_norm_ghost_simt(InType t, const void* A, const void* D, int B, int T, int d_in,
                                   int d_out, float* part, int NP, int row0, cudaStream_t s) {
  const int64_t parts = ghost_simt_parts(T);
  if (parts > NP || parts > 0x7fffffff) return cudaErrorInvalidValue;
  return per_example_slices(t, A, D, B, T, d_in, d_out, row0,
                            [&](const void* a, const void* d, int nb, int r0) {
    const dim3 grid(static_cast<unsigned>(parts), nb);
    note_launch();
    if (t == IN_F32)
      k_norm_ghost_simt<float><<<grid, 256, 0, s>>>(static_cast<const float*>(a),
                                                     static_cast<const float*>(d), T, d_in, d_out,
                                                     part, NP, r0);
    else
      k_norm_ghost_simt<__nv_bfloat16><<<grid, 256, 0, s>>>(
          static_cast<const __nv_bfloat16*>(a), static_cast<const __nv_bfloat16*>(d), T, d_in,
          d_out, part, NP, r0);
  });
}

cudaError_t launch_norm_mat_simt(InType t, const void* A, const void* D, int B, int T, int d_in,
                                 int d_out, float* part, int NP, int row0, cudaStream_t s) {
  if (mat_simt_parts(d_in, d_out) > NP || (d_in + SB - 1) / SB > kMaxGridYZ)
    return cudaErrorInvalidValue;
  return per_example_slices(t, A, D, B, T, d_in, d_out, row0,
                            [&](const void* a, const void* d, int nb, int r0) {
    const dim3 grid((d_out + SB - 1) / SB, (d_in + SB - 1) / SB, nb);
    Epilogue ep{};
    note_launch();
    if (t == IN_F32)
      k_gemm_simt<float, true, SB><<<grid, 256, 0, s>>>(static_cast<const float*>(a),
                                                         static_cast<const float*>(d), nullptr, T,
                                                         nb, d_in, d_out, nullptr, ep, part, NP,
                                                         r0);
    else
      k_gemm_simt<__nv_bfloat16, true, SB><<<grid, 256, 0, s>>>(
          static_cast<const __nv_bfloat16*>(a), static_cast<const __nv_bfloat16*>(d), nullptr, T,
          nb, d_in, d_out, nullptr, ep, part, NP, r0);
  });
}

cudaError_t launch_clip(const float* part, int L, int B, int NP, const int* d_nparts, float C,
                        float* layer_sq, float* s_out, float* c_out, float* user_s, float* user_c,
                        int* flag, cudaStream_t s, int mode, const float* s_given) {
  note_launch();
  if (NP >= 512)  // thousands of partials per example: a block of eight warps each
    k_clip<8><<<B, 256, 0, s>>>(part, L, B, NP, d_nparts, C, layer_sq, s_out, c_out, user_s,
                                user_c, flag, mode, s_given);
  else if (NP >= 64)
    k_clip<1><<<(B + 7) / 8, 256, 0, s>>>(part, L, B, NP, d_nparts, C, layer_sq, s_out, c_out,
                                          user_s, user_c, flag, mode, s_given);
  else  // few partials per layer: the layers in parallel over the lanes
    k_clip<0><<<(B + 7) / 8, 256, 0, s>>>(part, L, B, NP, d_nparts, C, layer_sq, s_out, c_out,
                                          user_s, user_c, flag, mode, s_given);
  return cudaGetLastError();
}

template <int TB>
void launch_gemm_simt_tb(InType t, const void* A, const void* D, const float* c, int B, int T,
                         int d_in, int d_out, float* out, const Epilogue& ep, cudaStream_t s) {
  const dim3 grid((d_out + TB - 1) / TB, (d_in + TB - 1) / TB, 1);
  note_launch();
  if (t == IN_F32)
    k_gemm_simt<float, false, TB><<<grid, 256, 0, s>>>(static_cast<const float*>(A),
                                                        static_cast<const float*>(D), c, T, B,
                                                        d_in, d_out, out, ep, nullptr, 0, 0);
  else
    k_gemm_simt<__nv_bfloat16, false, TB><<<grid, 256, 0, s>>>(
        static_cast<const __nv_bfloat16*>(A), static_cast<const __nv_bfloat16*>(D), c, T, B,
        d_in, d_out, out, ep, nullptr, 0, 0);
}

cudaError_t launch_gemm_simt(InType t, const void* A, const void* D, const float* c, int B, int T,
                             int d_in, int d_out, float* out, const Epilogue& ep, cudaStream_t s) {
  // 128 x 128 tiles when they alone fill the GPU twice, else 64 x 64 tiles
  const int64_t big = static_cast<int64_t>((d_out + SB - 1) / SB) * ((d_in + SB - 1) / SB);
  if (big >= 2 * 152)
    launch_gemm_simt_tb<SB>(t, A, D, c, B, T, d_in, d_out, out, ep, s);
  else
    launch_gemm_simt_tb<64>(t, A, D, c, B, T, d_in, d_out, out, ep, s);
  return cudaGetLastError();
}

cudaError_t launch_noise_add(NoiseAddBatch& b, cudaStream_t s) {
  int64_t blocks = 0;
  for (int l = 0; l < b.L; ++l) {
    b.block0[l] = blocks;
    if (b.n[l] <= 0) continue;
    const int64_t nq =
        static_cast<int64_t>(((b.p_base[l] + b.n[l] - 1) >> 2) - (b.p_base[l] >> 2) + 1);
    blocks += (nq + kNoiseChunk - 1) / kNoiseChunk;
  }
  b.block0[b.L] = blocks;
  if (blocks == 0) return cudaSuccess;
  if (blocks > 0x7FFFFFFF) return cudaErrorInvalidValue;
  note_launch();
  k_noise_add<<<static_cast<unsigned>(blocks), 256, 0, s>>>(b);
  return cudaGetLastError();
}

cudaError_t launch_audit(const int* idx, int n, int L, int B, const float* layer_sq,
                         const float* s_vec, const float* c_vec, const int* flag, float* rec,
                         int* flag_out, cudaStream_t s) {
  const int blocks = n > 0 ? (n + 127) / 128 : 1;
  note_launch();
  k_audit<<<blocks, 128, 0, s>>>(idx, n, L, B, layer_sq, s_vec, c_vec, flag, rec, flag_out);
  return cudaGetLastError();
}

cudaError_t launch_set_key(uint64_t seed, uint64_t step, uint64_t* key, int* flag,
                           cudaStream_t s) {
  note_launch();
  k_set_key<<<1, 1, 0, s>>>(seed, step, key, flag);
  return cudaGetLastError();
}

cudaError_t launch_load_key(const uint64_t* host_key_dev, uint64_t* key, int* flag,
                            cudaStream_t s) {
  note_launch();
  k_load_key<<<1, 1, 0, s>>>(host_key_dev, key, flag);
  return cudaGetLastError();
}

cudaError_t launch_debug_wait(uint64_t limit_ns, int* err, cudaStream_t s) {
  note_launch();
  k_debug_wait<<<1, 32, 0, s>>>(limit_ns, err);
  return cudaGetLastError();
}

cudaError_t launch_debug_philox(uint64_t seed, uint64_t step, uint64_t q0, int64_t nq,
                                uint32_t* out, cudaStream_t s) {
  note_launch();
  if (nq <= 0) return cudaSuccess;
  k_debug_philox<<<grid_for(nq, 256), 256, 0, s>>>(seed, step, q0, nq, out);
  return cudaGetLastError();
}

cudaError_t launch_debug_gauss(uint64_t seed, uint64_t step, uint64_t p0, int64_t n, float* out,
                               cudaStream_t s) {
  note_launch();
  if (n <= 0) return cudaSuccess;
  k_debug_gauss<<<grid_for(n, 256), 256, 0, s>>>(seed, step, p0, n, out);
  return cudaGetLastError();
}

}  // namespace dpk
