// Thin layers: one side of the weight at most kThinMax wide (LoRA factors of
// rank r, small classification heads, bias rows).  For them the per-example
// gradient g_i = A_i^T D_i of Sec. 2.2 is smaller than the example's inputs,
// so the norm pass materialises it once in context scratch and the clipped
// sum reads it back instead of reading A and D a second time:
//
//   norm pass   g_i = A_i^T D_i (fp32),  n_i = ||g_i||_F^2 (fixed-order
//               partials per 256-column slice of the wide side)
//   sum pass    out = out_scale (sum_i c_i g_i + sigma C z)   (examples in
//               order, so the result is the same on every run)
//
// The wide operand X ([B][T][n], n = the wide width) is read row by row,
// coalesced; the narrow operand Y ([B][T][r]) is staged in shared memory and
// broadcast.  Each thread owns VJ consecutive wide columns and all r narrow
// ones.  One launch serves up to kPerGradMaxLayers layers of the same
// narrow-width bucket and input type.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "internal.h"
#include "philox.cuh"
#include "tc.h"
#include "tc_util.cuh"

namespace dpk {

namespace {

constexpr int kThreads = 256;
constexpr int TT = 64;  // positions staged per round

__device__ __forceinline__ float to_float(float x) { return x; }
__device__ __forceinline__ float to_float(__nv_bfloat16 x) { return __bfloat162float(x); }

// VJ consecutive wide-side values of one row, read once and not kept in L1.
template <typename TIn, int VJ>
__device__ __forceinline__ void load_row(const TIn* p, float (&x)[VJ]);
template <>
__device__ __forceinline__ void load_row<__nv_bfloat16, 4>(const __nv_bfloat16* p, float (&x)[4]) {
  const uint2 u = __ldcs(reinterpret_cast<const uint2*>(p));
  x[0] = __uint_as_float(u.x << 16);
  x[1] = __uint_as_float(u.x & 0xffff0000u);
  x[2] = __uint_as_float(u.y << 16);
  x[3] = __uint_as_float(u.y & 0xffff0000u);
}
template <>
__device__ __forceinline__ void load_row<__nv_bfloat16, 2>(const __nv_bfloat16* p, float (&x)[2]) {
  const unsigned u = __ldcs(reinterpret_cast<const unsigned*>(p));
  x[0] = __uint_as_float(u << 16);
  x[1] = __uint_as_float(u & 0xffff0000u);
}
template <>
__device__ __forceinline__ void load_row<__nv_bfloat16, 1>(const __nv_bfloat16* p, float (&x)[1]) {
  x[0] = __bfloat162float(p[0]);
}
template <>
__device__ __forceinline__ void load_row<float, 4>(const float* p, float (&x)[4]) {
  const float4 v = __ldcs(reinterpret_cast<const float4*>(p));
  x[0] = v.x;
  x[1] = v.y;
  x[2] = v.z;
  x[3] = v.w;
}
template <>
__device__ __forceinline__ void load_row<float, 2>(const float* p, float (&x)[2]) {
  const float2 v = __ldcs(reinterpret_cast<const float2*>(p));
  x[0] = v.x;
  x[1] = v.y;
}
template <>
__device__ __forceinline__ void load_row<float, 1>(const float* p, float (&x)[1]) {
  x[0] = __ldcs(p);
}

template <int R>
struct Vj {
  static constexpr int value = R <= 8 ? 4 : (R <= 16 ? 2 : 1);
};

__device__ __forceinline__ int find_layer(const PerGradBatch& g, int item) {
  int l = 0;
  while (l + 1 < g.L && item >= g.l[l + 1].item0) ++l;
  return l;
}

// VJ consecutive values from shared memory.
template <typename TIn, int VJ>
__device__ __forceinline__ void load_smem(const TIn* p, float (&x)[VJ]);
template <>
__device__ __forceinline__ void load_smem<__nv_bfloat16, 4>(const __nv_bfloat16* p, float (&x)[4]) {
  const uint2 u = *reinterpret_cast<const uint2*>(p);
  x[0] = __uint_as_float(u.x << 16);
  x[1] = __uint_as_float(u.x & 0xffff0000u);
  x[2] = __uint_as_float(u.y << 16);
  x[3] = __uint_as_float(u.y & 0xffff0000u);
}
template <>
__device__ __forceinline__ void load_smem<__nv_bfloat16, 2>(const __nv_bfloat16* p, float (&x)[2]) {
  const unsigned u = *reinterpret_cast<const unsigned*>(p);
  x[0] = __uint_as_float(u << 16);
  x[1] = __uint_as_float(u & 0xffff0000u);
}
template <>
__device__ __forceinline__ void load_smem<__nv_bfloat16, 1>(const __nv_bfloat16* p, float (&x)[1]) {
  x[0] = __bfloat162float(p[0]);
}
template <>
__device__ __forceinline__ void load_smem<float, 4>(const float* p, float (&x)[4]) {
  const float4 v = *reinterpret_cast<const float4*>(p);
  x[0] = v.x;
  x[1] = v.y;
  x[2] = v.z;
  x[3] = v.w;
}
template <>
__device__ __forceinline__ void load_smem<float, 2>(const float* p, float (&x)[2]) {
  const float2 v = *reinterpret_cast<const float2*>(p);
  x[0] = v.x;
  x[1] = v.y;
}
template <>
__device__ __forceinline__ void load_smem<float, 1>(const float* p, float (&x)[1]) {
  x[0] = p[0];
}

template <typename TIn, int R, int VJ>
__device__ __forceinline__ void fma_row(const float (&x)[VJ], const float* y, float (&acc)[VJ][R]) {
#pragma unroll
  for (int k = 0; k < R; ++k) {
    const float yk = y[k];
#pragma unroll
    for (int v = 0; v < VJ; ++v) acc[v][k] = fmaf(x[v], yk, acc[v][k]);
  }
}

// Bulk-staged rows: NS ring stages of STAGE_BYTES in dynamic shared memory.
constexpr int NS = 4;
constexpr int STAGE_BYTES = 16384;
constexpr int kPerGradSmem = NS * STAGE_BYTES;

template <typename TIn, int R>
__global__ void __launch_bounds__(kThreads) k_pergrad_norm(const __grid_constant__ PerGradBatch g) {
  constexpr int VJ = Vj<R>::value;
  constexpr int SR = STAGE_BYTES / (kThreads * VJ * static_cast<int>(sizeof(TIn)));  // rows / stage
  static_assert(TT % SR == 0, "stages must tile the staged positions");
  extern __shared__ __align__(128) uint8_t stage_mem[];
  __shared__ __align__(16) float ys[TT][R];
  __shared__ uint64_t full[NS];
  __shared__ float red[kThreads / 32];
  __shared__ int abort_flag;
  volatile int* abrt = &abort_flag;
  const int l = find_layer(g, blockIdx.x);
  const PerGradLayer& P = g.l[l];
  const int local = static_cast<int>(blockIdx.x) - P.item0;
  const int i = local / P.chunks, chunk = local - i * P.chunks;
  const int n = P.n, r = P.r, T = g.T;
  const TIn* X = static_cast<const TIn*>(P.X) + static_cast<int64_t>(i) * T * n;
  const TIn* Y = static_cast<const TIn*>(P.Y) + static_cast<int64_t>(i) * T * r;
  const int c0 = chunk * kThreads * VJ;
  const int W = n - c0 < kThreads * VJ ? n - c0 : kThreads * VJ;  // columns of this block
  const int j0 = c0 + static_cast<int>(threadIdx.x) * VJ;
  float acc[VJ][R];
#pragma unroll
  for (int v = 0; v < VJ; ++v)
#pragma unroll
    for (int k = 0; k < R; ++k) acc[v][k] = 0.f;

  auto fill_ys = [&](int tb) {
    const int tt = T - tb < TT ? T - tb : TT;
    for (int e = threadIdx.x; e < TT * R; e += kThreads) {
      const int t = e / R, k = e - (e / R) * R;
      ys[t][k] = (t < tt && k < r) ? to_float(Y[static_cast<int64_t>(tb + t) * r + k]) : 0.f;
    }
  };

  if (P.bulk) {
    // One thread streams the block's rows of X (W contiguous columns per row,
    // one copy per stage when the block spans the whole row) into the ring;
    // every thread waits on the stage's barrier, then reads its VJ columns.
    const uint32_t row_bytes = static_cast<uint32_t>(W) * sizeof(TIn);
    const int nst = (T + SR - 1) / SR;
    if (threadIdx.x == 0) {
      for (int q = 0; q < NS; ++q) tc::mbar_init(&full[q], 1);
      abort_flag = 0;
      tc::fence_mbar_init();
    }
    __syncthreads();
    int issued = 0;  // meaningful in thread 0
    auto issue = [&](int st) {
      const int q = st % NS, r0 = st * SR;
      const int nr = T - r0 < SR ? T - r0 : SR;
      uint8_t* dst = stage_mem + q * STAGE_BYTES;
      tc::mbar_arrive_expect_tx(&full[q], static_cast<uint32_t>(nr) * row_bytes);
      if (W == n) {
        tc::bulk_load(dst, X + static_cast<int64_t>(r0) * n, static_cast<uint32_t>(nr) * row_bytes,
                      &full[q]);
      } else {
        for (int rr = 0; rr < nr; ++rr)
          tc::bulk_load(dst + rr * row_bytes, X + static_cast<int64_t>(r0 + rr) * n + c0,
                        row_bytes, &full[q]);
      }
    };
    if (threadIdx.x == 0)
      for (; issued < NS && issued < nst; ++issued) issue(issued);
    int st = 0;
    for (; st < nst; ++st) {
      const int r0 = st * SR;
      if (r0 % TT == 0) {
        fill_ys(r0);
        __syncthreads();
      }
      const int q = st % NS;
      tc::mbar_wait(&full[q], static_cast<uint32_t>(st / NS) & 1u, abrt, g.err);
      __syncthreads();
      if (*abrt) break;  // uniform: read after the barrier by every thread
      const TIn* xs = reinterpret_cast<const TIn*>(stage_mem + q * STAGE_BYTES);
      const int nr = T - r0 < SR ? T - r0 : SR;
      const int yb = r0 % TT;
      if (static_cast<int>(threadIdx.x) * VJ < W) {
        const TIn* xp = xs + threadIdx.x * VJ;
#pragma unroll 4
        for (int rr = 0; rr < nr; ++rr, xp += W) {
          float x[VJ];
          load_smem<TIn, VJ>(xp, x);
          fma_row<TIn, R, VJ>(x, &ys[yb + rr][0], acc);
        }
      }
      __syncthreads();  // the stage is free again
      if (threadIdx.x == 0 && issued < nst) issue(issued++);
    }
    if (st < nst) {
      // gave up: let every copy issued into the ring land before leaving
      if (threadIdx.x == 0) {
        for (int k = st; k < issued; ++k) {
          const uint64_t t0 = tc::globaltimer_ns();
          while (!tc::mbar_try_wait(&full[k % NS], static_cast<uint32_t>(k / NS) & 1u))
            if (tc::globaltimer_ns() - t0 > tc::kWaitLimitNs) break;
        }
      }
      return;
    }
  } else {
    // Rows read straight into registers (widths whose rows are not 16-byte
    // multiples).  A block narrower than its threads splits the positions
    // over S groups of tpr threads (group s takes t = s, s + S, ...) and adds
    // the groups' sums in order at the end.
    const int tpr = (W + VJ - 1) / VJ;
    const int S = tpr < kThreads ? kThreads / tpr : 1;
    const int s = static_cast<int>(threadIdx.x) / tpr;
    const int jj0 = c0 + (static_cast<int>(threadIdx.x) - s * tpr) * VJ;
    const bool active = s < S && jj0 < n;
    const bool vec = jj0 + VJ <= n && n % VJ == 0 &&
                     (reinterpret_cast<uintptr_t>(P.X) % (VJ * sizeof(TIn))) == 0;
    for (int t0 = 0; t0 < T; t0 += TT) {
      const int tt = T - t0 < TT ? T - t0 : TT;
      fill_ys(t0);
      __syncthreads();
      const TIn* xrow = X + static_cast<int64_t>(t0 + s) * n + jj0;
      const int64_t step = static_cast<int64_t>(S) * n;
      if (active && vec) {
#pragma unroll 8
        for (int t = s; t < tt; t += S, xrow += step) {
          float x[VJ];
          load_row<TIn, VJ>(xrow, x);
          fma_row<TIn, R, VJ>(x, &ys[t][0], acc);
        }
      } else if (active) {
#pragma unroll 4
        for (int t = s; t < tt; t += S, xrow += step) {
          float x[VJ];
#pragma unroll
          for (int v = 0; v < VJ; ++v) x[v] = (jj0 + v < n) ? to_float(xrow[v]) : 0.f;
          fma_row<TIn, R, VJ>(x, &ys[t][0], acc);
        }
      }
      __syncthreads();
    }
    if (S > 1) {
      // groups 1.. hand their sums to group 0 through the (unused) staging
      // memory: S * tpr <= kThreads slots of VJ * R floats (at most 32 KB)
      float* part = reinterpret_cast<float*>(stage_mem);
      float* mine = part + static_cast<int64_t>(threadIdx.x) * VJ * R;
      if (s > 0 && s < S) {
#pragma unroll
        for (int v = 0; v < VJ; ++v)
#pragma unroll
          for (int k = 0; k < R; ++k) mine[v * R + k] = acc[v][k];
      }
      __syncthreads();
      if (s == 0) {
        for (int q = 1; q < S; ++q) {
          const float* o = part + static_cast<int64_t>(q * tpr + threadIdx.x) * VJ * R;
#pragma unroll
          for (int v = 0; v < VJ; ++v)
#pragma unroll
            for (int k = 0; k < R; ++k) acc[v][k] += o[v * R + k];
        }
      } else {
        // the sums now live in group 0 (and these threads' columns j0 are
        // past the layer's width, so they store nothing)
#pragma unroll
        for (int v = 0; v < VJ; ++v)
#pragma unroll
          for (int k = 0; k < R; ++k) acc[v][k] = 0.f;
      }
    }
  }

  // g_i rows are [d_in][d_out]: X = A gives G[j][k], X = D gives G[k][j]
  float* G = P.G + static_cast<int64_t>(i) * n * r;
  float sq = 0.f;
#pragma unroll
  for (int v = 0; v < VJ; ++v)
#pragma unroll
    for (int k = 0; k < R; ++k) sq = fmaf(acc[v][k], acc[v][k], sq);  // padding is zero
  const bool g16 = (reinterpret_cast<uintptr_t>(G) & 15) == 0;
  if (P.wide_is_in && R % 4 == 0 && r == R && g16) {
#pragma unroll
    for (int v = 0; v < VJ; ++v) {
      const int j = j0 + v;
      if (j >= n) continue;
      float4* dst = reinterpret_cast<float4*>(G + static_cast<int64_t>(j) * r);
#pragma unroll
      for (int k4 = 0; k4 < R / 4; ++k4)
        dst[k4] = make_float4(acc[v][4 * k4], acc[v][4 * k4 + 1], acc[v][4 * k4 + 2],
                              acc[v][4 * k4 + 3]);
    }
  } else if (!P.wide_is_in && VJ == 4 && n % 4 == 0 && g16 && j0 + 3 < n) {
#pragma unroll
    for (int k = 0; k < R; ++k) {
      if (k >= r) continue;
      *reinterpret_cast<float4*>(G + static_cast<int64_t>(k) * n + j0) =
          make_float4(acc[0][k], acc[VJ > 1 ? 1 : 0][k], acc[VJ > 2 ? 2 : 0][k],
                      acc[VJ > 3 ? 3 : 0][k]);
    }
  } else {
#pragma unroll
    for (int v = 0; v < VJ; ++v) {
      const int j = j0 + v;
      if (j >= n) continue;
#pragma unroll
      for (int k = 0; k < R; ++k) {
        if (k >= r) continue;
        if (P.wide_is_in)
          G[static_cast<int64_t>(j) * r + k] = acc[v][k];
        else
          G[static_cast<int64_t>(k) * n + j] = acc[v][k];
      }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = sq;
  __syncthreads();
  if (threadIdx.x == 0) {
    float s2 = 0.f;
    for (int w = 0; w < kThreads / 32; ++w) s2 += red[w];
    g.part[static_cast<int64_t>(P.row0 + i) * g.NP + chunk] = s2;
  }
}

// ---------------------------------------------------------------------------
// bf16 thin layers on warp tensor-core MMAs.  Per example the contraction is
// tiny (N = r <= 32, K = T) and the pass is bound by HBM, but on CUDA cores
// the multiply-adds and bf16 unpacking spend more issue slots than the bytes
// take to arrive; one m16n8k16 MMA does 2048 multiply-adds in one
// instruction.  A block covers one example and kMmaCols wide columns; each
// of its 8 warps owns 4 m-tiles of 16 wide columns against all NT n-tiles of
// 8 narrow columns.  A stage is one k16 step: 16 rows of the wide operand at
// a padded stride (the 8 rows one ldmatrix reads fall in distinct banks) and
// the same 16 rows of the narrow operand, zero-padded to 8 NT columns.
// ---------------------------------------------------------------------------
constexpr int kMmaCols = 512;
constexpr int kMmaSR = 16;  // rows per stage, a multiple of 16 (one k16 step each)
constexpr int kMmaNS = 2;   // stages in the ring
constexpr int kMmaThreads = kMmaCols / 64 * 32;  // a warp owns 64 wide columns
constexpr int kMmaXStride = kMmaCols * 2 + 16;  // bytes per staged wide row

template <int NT>
struct MmaCfg {
  static constexpr int YW = 8 * NT;            // staged narrow width
  static constexpr int Y_STRIDE = YW * 2;      // bytes per staged narrow row
  static constexpr int X_BYTES = kMmaSR * kMmaXStride;
  static constexpr int Y_BYTES = kMmaSR * Y_STRIDE;
  static constexpr int STAGE = ((X_BYTES + Y_BYTES + 127) / 128) * 128;
  static constexpr int SMEM = kMmaNS * STAGE;
  static_assert(kMmaSR % 16 == 0, "a stage is whole k16 steps");
  static_assert(SMEM <= 227 * 1024, "stage ring exceeds shared memory");
};

__device__ __forceinline__ void ldsm_x4_trans(uint32_t addr, uint32_t (&a)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(a[0]), "=r"(a[1]), "=r"(a[2]), "=r"(a[3])
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x2_trans(uint32_t addr, uint32_t (&b)[2]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.trans.shared.b16 {%0, %1}, [%2];"
               : "=r"(b[0]), "=r"(b[1])
               : "r"(addr));
}
__device__ __forceinline__ void mma_16816(float (&c)[4], const uint32_t (&a)[4],
                                          const uint32_t (&b)[2]) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, "
      "{%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

// One (layer, example, column slice) work item of a launch.
struct MmaItem {
  const __nv_bfloat16* X;  // the example's wide rows, at this slice's first column
  const __nv_bfloat16* Y;  // the example's narrow rows
  float* G;                // the example's gradient
  int n, r, W, wide_is_in, row, slot;
};

__device__ __forceinline__ MmaItem mma_item(const PerGradBatch& g, int item) {
  const int l = find_layer(g, item);
  const PerGradLayer& P = g.l[l];
  const int local = item - P.item0;
  const int i = local / P.chunks, chunk = local - i * P.chunks;
  MmaItem it;
  it.n = P.n;
  it.r = P.r;
  const int c0 = chunk * kMmaCols;
  it.W = P.n - c0 < kMmaCols ? P.n - c0 : kMmaCols;
  it.X = static_cast<const __nv_bfloat16*>(P.X) + static_cast<int64_t>(i) * g.T * P.n + c0;
  it.Y = static_cast<const __nv_bfloat16*>(P.Y) + static_cast<int64_t>(i) * g.T * P.r;
  it.G = P.G + static_cast<int64_t>(i) * P.n * P.r;
  it.wide_is_in = P.wide_is_in;
  it.row = P.row0 + i;
  it.slot = chunk;
  return it;
}

// One block per item; its stage ring runs over the item's T rows.
template <int NT>
__global__ void __launch_bounds__(kMmaThreads) k_pergrad_norm_mma(const __grid_constant__ PerGradBatch g) {
  using Cf = MmaCfg<NT>;
  extern __shared__ __align__(128) uint8_t stage_mem[];
  __shared__ uint64_t full[kMmaNS];
  __shared__ float red[kMmaThreads / 32];
  __shared__ int abort_flag;
  volatile int* abrt = &abort_flag;
  const int warp = static_cast<int>(threadIdx.x) >> 5, lane = static_cast<int>(threadIdx.x) & 31;
  const int T = g.T;
  const int nst = (T + kMmaSR - 1) / kMmaSR;
  const MmaItem it = mma_item(g, static_cast<int>(blockIdx.x));
  const bool yb = it.r == Cf::YW;  // narrow rows arrive by copy (no padding needed)
  float acc[4][NT][4];
#pragma unroll
  for (int mt = 0; mt < 4; ++mt)
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[mt][nt][e] = 0.f;

  if (threadIdx.x == 0) {
    for (int q = 0; q < kMmaNS; ++q) tc::mbar_init(&full[q], 1);
    abort_flag = 0;
    tc::fence_mbar_init();
  }
  __syncthreads();
  int issued = 0;  // thread 0
  const uint32_t row_bytes = static_cast<uint32_t>(it.W) * 2;
  auto issue = [&](int st) {
    const int q = st % kMmaNS, r0 = st * kMmaSR;
    const int nr = T - r0 < kMmaSR ? T - r0 : kMmaSR;
    uint8_t* xs = stage_mem + q * Cf::STAGE;
    tc::mbar_arrive_expect_tx(&full[q], static_cast<uint32_t>(nr) * row_bytes +
                                            (yb ? static_cast<uint32_t>(nr * it.r * 2) : 0u));
    for (int rr = 0; rr < nr; ++rr)
      tc::bulk_load(xs + rr * kMmaXStride, it.X + static_cast<int64_t>(r0 + rr) * it.n, row_bytes,
                    &full[q]);
    if (yb)
      tc::bulk_load(xs + Cf::X_BYTES, it.Y + static_cast<int64_t>(r0) * it.r, nr * it.r * 2,
                    &full[q]);
  };
  if (threadIdx.x == 0)
    for (; issued < kMmaNS && issued < nst; ++issued) issue(issued);

  // narrow rows that no copy brings (padded widths): each thread holds its
  // elements of the next stage in registers, loaded a stage ahead
  constexpr int YPT = (kMmaSR * Cf::YW + kMmaThreads - 1) / kMmaThreads;
  __nv_bfloat16 ypre[YPT];
  auto load_y = [&](int st) {
    if (yb || st >= nst) return;
    const int rn0 = st * kMmaSR;
#pragma unroll
    for (int u = 0; u < YPT; ++u) {
      const int e = static_cast<int>(threadIdx.x) + u * kMmaThreads;
      const int t = e / Cf::YW, k = e - (e / Cf::YW) * Cf::YW;
      ypre[u] = (e < kMmaSR * Cf::YW && rn0 + t < T && k < it.r)
                    ? it.Y[static_cast<int64_t>(rn0 + t) * it.r + k]
                    : __float2bfloat16_rn(0.f);
    }
  };
  load_y(0);

  const uint32_t sbase = tc::smem_u32(stage_mem);
  const int mat = lane >> 3, mrow = lane & 7;
  const int gq = lane >> 2, tq = lane & 3;
  int st = 0;
  for (; st < nst; ++st) {
    const int q = st % kMmaNS, r0 = st * kMmaSR;
    const int nr = T - r0 < kMmaSR ? T - r0 : kMmaSR;
    uint8_t* xs = stage_mem + q * Cf::STAGE;
    __nv_bfloat16* ysm = reinterpret_cast<__nv_bfloat16*>(xs + Cf::X_BYTES);
    // parts no copy writes: rows past T, and narrow rows that need padding
    if (nr < kMmaSR) {
      const int words = (kMmaSR - nr) * (kMmaXStride / 4);
      uint32_t* z = reinterpret_cast<uint32_t*>(xs + nr * kMmaXStride);
      for (int e = threadIdx.x; e < words; e += kMmaThreads) z[e] = 0u;
    }
    if (!yb) {
#pragma unroll
      for (int u = 0; u < YPT; ++u) {
        const int e = static_cast<int>(threadIdx.x) + u * kMmaThreads;
        if (e < kMmaSR * Cf::YW) ysm[e] = ypre[u];
      }
    } else if (nr < kMmaSR) {
      for (int e = threadIdx.x; e < kMmaSR * Cf::YW; e += kMmaThreads)
        if (e / Cf::YW >= nr) ysm[e] = __float2bfloat16_rn(0.f);  // rows past T
    }
    load_y(st + 1);
    tc::mbar_wait(&full[q], static_cast<uint32_t>(st / kMmaNS) & 1u, abrt, g.err);
    __syncthreads();
    if (*abrt) break;
    const uint32_t xa = sbase + q * Cf::STAGE;
    const uint32_t ya = xa + Cf::X_BYTES;
#pragma unroll
    for (int kk = 0; kk < kMmaSR / 16; ++kk) {
      uint32_t b[NT][2];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
        ldsm_x2_trans(ya + (kk * 16 + (lane & 15)) * Cf::Y_STRIDE + nt * 16, b[nt]);
#pragma unroll
      for (int mt = 0; mt < 4; ++mt) {
        const int m0 = warp * 64 + mt * 16;
        if (m0 >= it.W) continue;
        uint32_t a[4];
        ldsm_x4_trans(xa + (kk * 16 + (mat >> 1) * 8 + mrow) * kMmaXStride +
                          (m0 + (mat & 1) * 8) * 2,
                      a);
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) mma_16816(acc[mt][nt], a, b[nt]);
      }
    }
    __syncthreads();  // the stage is free again
    if (threadIdx.x == 0 && issued < nst) {
      // rows this block wrote into the slot (padding, staged narrow rows)
      // may be overwritten by the copies: order them before the async proxy
      tc::fence_proxy_async_smem();
      issue(issued++);
    }
  }
  if (st < nst) {
    if (threadIdx.x == 0) {
      // gave up: let every copy issued into the ring land before leaving
      for (int k = st; k < issued; ++k) {
        const uint64_t t0 = tc::globaltimer_ns();
        while (!tc::mbar_try_wait(&full[k % kMmaNS], static_cast<uint32_t>(k / kMmaNS) & 1u))
          if (tc::globaltimer_ns() - t0 > tc::kWaitLimitNs) break;
      }
    }
    return;
  }

  // C fragment: c0, c1 at (row g, cols 2t, 2t+1), c2, c3 at row g + 8
  const int c0 = it.slot * kMmaCols;
  float sq = 0.f;
#pragma unroll
  for (int mt = 0; mt < 4; ++mt) {
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int mm = warp * 64 + mt * 16 + gq + (e >> 1) * 8;
        const int k = nt * 8 + 2 * tq + (e & 1);
        if (mm >= it.W || k >= it.r) continue;
        const int m = c0 + mm;
        const float v = acc[mt][nt][e];
        sq = fmaf(v, v, sq);
        if (it.wide_is_in)
          it.G[static_cast<int64_t>(m) * it.r + k] = v;
        else
          it.G[static_cast<int64_t>(k) * it.n + m] = v;
      }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
  if (lane == 0) red[warp] = sq;
  __syncthreads();
  if (threadIdx.x == 0) {
    float s2 = 0.f;
    for (int w = 0; w < kMmaThreads / 32; ++w) s2 += red[w];
    g.part[static_cast<int64_t>(it.row) * g.NP + it.slot] = s2;
  }
}

// out = out_scale (sum_i c_i g_i + sigma C z) over the global quads that
// overlap each layer's parameters.  A layer with few parameters splits its
// examples over `split` threads per quad (split from the layer's own size,
// so a batched launch rounds exactly like a single one): each thread sums a
// contiguous range of examples in order, and the ranges are added in order.
__global__ void __launch_bounds__(kThreads) k_pergrad_sum(const __grid_constant__ PerGradSumBatch g) {
  __shared__ float4 red[kThreads];
  int l = 0;
  while (l + 1 < g.L && static_cast<int64_t>(blockIdx.x) >= g.l[l + 1].item0) ++l;
  const PerGradSumLayer& P = g.l[l];
  const int split = P.split;
  const int qpb = kThreads / split;  // quads per block
  const int qi = static_cast<int>(threadIdx.x) % qpb, sp = static_cast<int>(threadIdx.x) / qpb;
  const int64_t local = (static_cast<int64_t>(blockIdx.x) - P.item0) * qpb + qi;
  const bool live = local < P.nq;
  const uint64_t q = (P.p_base >> 2) + static_cast<uint64_t>(live ? local : 0);
  const int64_t e0 = static_cast<int64_t>(4 * q) - static_cast<int64_t>(P.p_base);
  const int64_t n = P.count;
  const int i0 = static_cast<int>((static_cast<int64_t>(g.B) * sp) / split);
  const int i1 = static_cast<int>((static_cast<int64_t>(g.B) * (sp + 1)) / split);
  float s[4] = {0.f, 0.f, 0.f, 0.f};
  if (live) {
    const bool vec = P.vec && e0 >= 0 && e0 + 3 < n;
    if (vec) {
      const float* gp = P.G + static_cast<int64_t>(i0) * n + e0;
#pragma unroll 8
      for (int i = i0; i < i1; ++i, gp += n) {
        const float ci = g.c[i];
        const float4 v = __ldcs(reinterpret_cast<const float4*>(gp));
        s[0] = fmaf(ci, v.x, s[0]);
        s[1] = fmaf(ci, v.y, s[1]);
        s[2] = fmaf(ci, v.z, s[2]);
        s[3] = fmaf(ci, v.w, s[3]);
      }
    } else {
      for (int i = i0; i < i1; ++i) {
        const float ci = g.c[i];
#pragma unroll
        for (int w = 0; w < 4; ++w) {
          const int64_t e = e0 + w;
          if (e >= 0 && e < n) s[w] = fmaf(ci, P.G[static_cast<int64_t>(i) * n + e], s[w]);
        }
      }
    }
  }
  if (split > 1) {  // uniform per block
    red[threadIdx.x] = make_float4(s[0], s[1], s[2], s[3]);
    __syncthreads();
    if (sp != 0) return;
    for (int k = 1; k < split; ++k) {
      const float4 o = red[k * qpb + qi];
      s[0] += o.x;
      s[1] += o.y;
      s[2] += o.z;
      s[3] += o.w;
    }
  }
  if (!live) return;
  float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
  if (g.add_noise) z = gauss_quad(g.key[0], g.key[1], q);
  const float zv[4] = {z.x, z.y, z.z, z.w};
#pragma unroll
  for (int w = 0; w < 4; ++w) {
    const int64_t e = e0 + w;
    if (e < 0 || e >= n) continue;
    const float val = g.out_scale * fmaf(g.sigmaC, zv[w], s[w]);
    P.out[e] = g.accumulate ? P.out[e] + val : val;
  }
}

template <typename TIn, int R>
cudaError_t launch_norm_t(const PerGradBatch& g, int blocks, cudaStream_t s) {
  cudaError_t e = setup_once_per_device(reinterpret_cast<const void*>(&k_pergrad_norm<TIn, R>), [] {
    return cudaFuncSetAttribute(k_pergrad_norm<TIn, R>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, kPerGradSmem);
  });
  if (e != cudaSuccess) return e;
  note_launch();
  k_pergrad_norm<TIn, R><<<blocks, kThreads, kPerGradSmem, s>>>(g);
  return cudaGetLastError();
}

template <typename TIn>
cudaError_t launch_norm_r(const PerGradBatch& g, int R, int blocks, cudaStream_t s) {
  switch (R) {
    case 1: return launch_norm_t<TIn, 1>(g, blocks, s);
    case 2: return launch_norm_t<TIn, 2>(g, blocks, s);
    case 4: return launch_norm_t<TIn, 4>(g, blocks, s);
    case 8: return launch_norm_t<TIn, 8>(g, blocks, s);
    case 16: return launch_norm_t<TIn, 16>(g, blocks, s);
    case 32: return launch_norm_t<TIn, 32>(g, blocks, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

int pergrad_bucket(int r) {
  int R = 1;
  while (R < r) R <<= 1;
  return R <= kThinMax ? R : 0;
}

// bf16 layers whose wide rows are whole 16-byte vectors take the MMA kernel
// (narrow widths below 8 are zero-padded to one n-tile; the pass stays bound
// by the wide rows' bytes), as long as an example's T positions stay within
// the accumulation bound of the MMA's fp32 accumulators.
bool pergrad_mma(InType t, int64_t n, int r, int T) {
  return t == IN_BF16 && n % 8 == 0 && r > 0 && T <= kTcMaxAccum;
}

int64_t pergrad_parts(InType t, int64_t d_in, int64_t d_out, int T) {
  const int r = static_cast<int>(d_in < d_out ? d_in : d_out);
  const int64_t n = d_in < d_out ? d_out : d_in;
  const int R = pergrad_bucket(r);
  if (R == 0) return 0;
  if (pergrad_mma(t, n, r, T)) return (n + kMmaCols - 1) / kMmaCols;
  const int vj = R <= 8 ? 4 : (R <= 16 ? 2 : 1);
  return (n + kThreads * vj - 1) / (kThreads * vj);
}

template <int NT>
cudaError_t launch_mma_t(const PerGradBatch& g, int blocks, cudaStream_t s) {
  cudaError_t e = setup_once_per_device(reinterpret_cast<const void*>(&k_pergrad_norm_mma<NT>), [] {
    return cudaFuncSetAttribute(k_pergrad_norm_mma<NT>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, MmaCfg<NT>::SMEM);
  });
  if (e != cudaSuccess) return e;
  note_launch();
  k_pergrad_norm_mma<NT><<<blocks, kMmaThreads, MmaCfg<NT>::SMEM, s>>>(g);
  return cudaGetLastError();
}

// One launch of the layers of g that share a path (all on MMAs or none).
cudaError_t launch_norm_group(InType t, PerGradBatch& g, bool mma, cudaStream_t s) {
  int R = 0;
  for (int l = 0; l < g.L; ++l) {
    const int Rl = pergrad_bucket(g.l[l].r);
    if (Rl == 0) return cudaErrorInvalidValue;
    if (Rl > R) R = Rl;
  }
  const int vj = R <= 8 ? 4 : (R <= 16 ? 2 : 1);
  const int elem = t == IN_F32 ? 4 : 2;
  int64_t blocks = 0;
  for (int l = 0; l < g.L; ++l) {
    PerGradLayer& P = g.l[l];
    P.chunks = mma ? static_cast<int>((P.n + kMmaCols - 1) / kMmaCols)
                   : static_cast<int>((P.n + kThreads * vj - 1) / (kThreads * vj));
    // bulk copies need 16-byte aligned rows (the base is 16-byte aligned)
    P.bulk = (static_cast<int64_t>(P.n) * elem) % 16 == 0 &&
             (reinterpret_cast<uintptr_t>(P.X) & 15) == 0;
    P.item0 = static_cast<int>(blocks);
    blocks += static_cast<int64_t>(g.B) * P.chunks;
  }
  if (blocks > 0x7fffffffLL) return cudaErrorInvalidValue;
  const int nb = static_cast<int>(blocks);
  if (mma) {
    const int NT = R <= 8 ? 1 : (R <= 16 ? 2 : 4);
    return NT == 1 ? launch_mma_t<1>(g, nb, s) : NT == 2 ? launch_mma_t<2>(g, nb, s)
                                                         : launch_mma_t<4>(g, nb, s);
  }
  return t == IN_F32 ? launch_norm_r<float>(g, R, nb, s) : launch_norm_r<__nv_bfloat16>(g, R, nb, s);
}

cudaError_t launch_pergrad_norm(InType t, PerGradBatch& g, cudaStream_t s) {
  if (g.L < 1 || g.L > kPerGradMaxLayers) return cudaErrorInvalidValue;
  // split the batch by path, keeping each layer's partial rows and slots
  PerGradBatch part[2];
  for (int m = 0; m < 2; ++m) {
    part[m] = g;
    part[m].L = 0;
  }
  for (int l = 0; l < g.L; ++l) {
    const int m = pergrad_mma(t, g.l[l].n, g.l[l].r, g.T) ? 1 : 0;
    part[m].l[part[m].L++] = g.l[l];
  }
  for (int m = 0; m < 2; ++m) {
    if (part[m].L == 0) continue;
    cudaError_t e = launch_norm_group(t, part[m], m == 1, s);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t launch_pergrad_sum(PerGradSumBatch& g, cudaStream_t s) {
  if (g.L < 1 || g.L > kPerGradMaxLayers) return cudaErrorInvalidValue;
  const int64_t target = static_cast<int64_t>(device_sm_count()) * kThreads;  // ~one wave
  int64_t blocks = 0;
  for (int l = 0; l < g.L; ++l) {
    PerGradSumLayer& P = g.l[l];
    P.nq = static_cast<int64_t>(((P.p_base + P.count - 1) >> 2) - (P.p_base >> 2) + 1);
    P.vec = (P.p_base % 4 == 0) && (P.count % 4 == 0) &&
            (reinterpret_cast<uintptr_t>(P.G) % 16 == 0);
    // split the examples while the layer alone is short of a wave and every
    // range keeps at least 16 examples
    int split = 1;
    while (split < 8 && P.nq * split * 2 <= target && g.B / (split * 2) >= 16) split *= 2;
    P.split = split;
    P.item0 = blocks;  // in blocks
    const int qpb = kThreads / split;
    blocks += (P.nq + qpb - 1) / qpb;
  }
  note_launch();
  if (blocks > 0x7fffffffLL) return cudaErrorInvalidValue;
  k_pergrad_sum<<<static_cast<int>(blocks), kThreads, 0, s>>>(g);
  return cudaGetLastError();
}

}  // namespace dpk
