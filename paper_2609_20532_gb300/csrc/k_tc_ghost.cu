// tcgen05 Gram-form ("ghost") per-example squared norm of dense layers:
//   n_i = ||A_i^T D_i||_F^2 = sum_{t,s} (A_i A_i^T)_{ts} (D_i D_i^T)_{ts}
// (the expansion of the Frobenius norm of a sum of outer products), which
// never forms the d_in x d_out gradient.
//
// The T x T Grams are cut into 128-position blocks; only the upper triangle
// of block pairs is computed (off-diagonal pairs count twice, the Grams
// being symmetric).  A work item is a strip: one 128-row t-block against up
// to two consecutive s-blocks (N = 256 MMAs), for one example of one layer.
// For the strip the tensor core accumulates the A-Gram (K = d_in) and the
// D-Gram (K = d_out) into two 256-column TMEM accumulators; the epilogue
// multiplies them elementwise and reduces.  Strips that start on the
// diagonal load each 128-row tile once and use it for both operands.
// Operands are K-major rows of A_i / D_i read through 3-D tensor maps
// [B][T][d], so positions t >= T of an example read as zeros.
//
// One launch can serve up to kGhostMaxLayers layers of a step (they share B
// and T), so the few items of each layer balance across all SMs.
//
// Warp roles (384 threads, one CTA per SM):
//   warp 0 TMA producer, warp 1 TMEM allocator + MMA issuer, warps 2-3
//   idle, warps 4-11 epilogue (warp w reads TMEM lanes 32*(w%4)..+31,
//   column half (w-4)/4 of each 256-column accumulator).
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "internal.h"
#include "tc.h"
#include "tc_util.cuh"

namespace dpk {

namespace {

using namespace tc;

constexpr int GT = 128;                  // Gram block edge (positions)
constexpr int FK = 64;                   // features per stage (128 bytes of bf16)
constexpr int STAGES = 4;
constexpr int TILE_BYTES = GT * FK * 2;  // 16 KB: one 128-position tile
constexpr int A_OFF = 0;                 // t-tile (off-diagonal strips only)
constexpr int B_OFF = TILE_BYTES;        // two s-tiles, 256 rows
constexpr int STAGE_BYTES = 3 * TILE_BYTES;
constexpr int NUM_EPI_WARPS = 8;
constexpr int FIRST_EPI_WARP = 4;
constexpr int GHOST_THREADS = 128 + 32 * NUM_EPI_WARPS;
constexpr uint32_t TMEM_COLS = 512;      // A-Gram strip 256 + D-Gram strip 256
constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024;
// K-major, 128-byte swizzle: rows 128 B apart, 8-row groups 1024 B apart.
constexpr uint32_t LBO = 16, SBO = 1024;
constexpr uint32_t IDESC_N256 = idesc_bf16_f32(GT, 2 * GT, 0, 0);
constexpr uint32_t IDESC_N128 = idesc_bf16_f32(GT, GT, 0, 0);

struct GhostBatch {
  CUtensorMap mapA[kGhostMaxLayers];
  CUtensorMap mapD[kGhostMaxLayers];
  int d_in[kGhostMaxLayers];
  int d_out[kGhostMaxLayers];
  int row0[kGhostMaxLayers];   // partial-sum row of example 0 of the layer
  int L, B, T, nb;             // layers in this launch, examples, positions, blocks
  int n_full, n_half;          // strips per example
  float* part;
  int* err;
  int NP;
};

struct Strip {
  int layer, ex, tb, sb, ns, slot;
};

// Full strips of row tb: floor((nb - tb) / 2); a half strip ends every row
// with an odd number of blocks left.
__device__ __forceinline__ void full_strip(int k, int nb, int& tb, int& sb) {
  for (int t = 0; t < nb; ++t) {
    const int f = (nb - t) / 2;
    if (k < f) {
      tb = t;
      sb = t + 2 * k;
      return;
    }
    k -= f;
  }
  tb = sb = 0;
}
__device__ __forceinline__ void half_strip(int k, int nb, int& tb, int& sb) {
  for (int t = 0; t < nb; ++t) {
    if ((nb - t) & 1) {
      if (k == 0) {
        tb = t;
        sb = nb - 1;
        return;
      }
      --k;
    }
  }
  tb = sb = 0;
}

// Work list: layer-major, then example, then that example's strips (full
// strips first).  The strips of one example run at about the same time and
// share its rows in L2; with a few items per SM the largest makespan is the
// same as for a full-strips-first order.
__device__ __forceinline__ Strip decode(int item, const GhostBatch& g) {
  Strip s;
  const int per_ex = g.n_full + g.n_half;
  const int per_layer = g.B * per_ex;
  s.layer = item / per_layer;
  const int r = item - s.layer * per_layer;
  s.ex = r / per_ex;
  const int k = r - s.ex * per_ex;
  if (k < g.n_full) {
    full_strip(k, g.nb, s.tb, s.sb);
    s.ns = 2;
  } else {
    half_strip(k - g.n_full, g.nb, s.tb, s.sb);
    s.ns = 1;
  }
  s.slot = k;
  return s;
}

__global__ void __launch_bounds__(GHOST_THREADS, 1)
    k_ghost_tc(const __grid_constant__ GhostBatch g) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  __shared__ uint64_t full_bar[STAGES], empty_bar[STAGES], tfull_bar, tempty_bar, done_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_items = g.L * g.B * (g.n_full + g.n_half);
  volatile int* abrt = &abort_flag;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    mbar_init(&tfull_bar, 1);
    mbar_init(&tempty_bar, NUM_EPI_WARPS);
    mbar_init(&done_bar, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) tmem_alloc(&tmem_slot, TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      int stage = 0;
      uint32_t phase = 0;
      uint32_t uses[STAGES] = {};
      for (int item = blockIdx.x; item < n_items; item += gridDim.x) {
        const Strip st = decode(item, g);
        const bool diag = st.tb == st.sb;
        const CUtensorMap* mA = &g.mapA[st.layer];
        const CUtensorMap* mD = &g.mapD[st.layer];
        const int ka = (g.d_in[st.layer] + FK - 1) / FK, kd = (g.d_out[st.layer] + FK - 1) / FK;
        const uint32_t bytes = (diag ? 0 : TILE_BYTES) + st.ns * TILE_BYTES;
        for (int k = 0; k < ka + kd; ++k) {
          const CUtensorMap* map = k < ka ? mA : mD;
          const int f0 = (k < ka ? k : k - ka) * FK;
          if (!mbar_wait(&empty_bar[stage], phase ^ 1, abrt, g.err)) goto producer_done;
          uint8_t* sp = smem + stage * STAGE_BYTES;
          mbar_arrive_expect_tx(&full_bar[stage], bytes);
          if (!diag) tma_load_3d(map, &full_bar[stage], sp + A_OFF, f0, st.tb * GT, st.ex);
          tma_load_3d(map, &full_bar[stage], sp + B_OFF, f0, st.sb * GT, st.ex);
          if (st.ns == 2)
            tma_load_3d(map, &full_bar[stage], sp + B_OFF + TILE_BYTES, f0, (st.sb + 1) * GT,
                        st.ex);
          ++uses[stage];
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
    producer_done:
      for (int s = 0; s < STAGES; ++s) {
        if (uses[s] == 0) continue;
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_try_wait(&full_bar[s], (uses[s] - 1) & 1)) {
          if (globaltimer_ns() - t0 > kWaitLimitNs) {
            atomicOr(g.err, kErrTimeout);
            break;
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      for (int item = blockIdx.x; item < n_items; item += gridDim.x, ++it) {
        const Strip st = decode(item, g);
        const bool diag = st.tb == st.sb;
        const uint32_t idesc = st.ns == 2 ? IDESC_N256 : IDESC_N128;
        const int ka = (g.d_in[st.layer] + FK - 1) / FK, kd = (g.d_out[st.layer] + FK - 1) / FK;
        if (!mbar_wait(&tempty_bar, (it & 1) ^ 1, abrt, g.err)) goto mma_done;
        tc_fence_after();
        for (int k = 0; k < ka + kd; ++k) {
          const bool is_a = k < ka;
          const int kl = is_a ? k : k - ka;
          const uint32_t d_tmem = tmem_base + (is_a ? 0 : 2 * GT);
          if (!mbar_wait(&full_bar[stage], phase, abrt, g.err)) goto mma_done;
          tc_fence_after();
          const uint32_t sp = smem_u32(smem + stage * STAGE_BYTES);
          const uint32_t sb = sp + B_OFF;
          const uint32_t sa = diag ? sb : sp + A_OFF;
#pragma unroll
          for (int kk = 0; kk < FK / 16; ++kk) {
            const uint64_t ad = smem_desc_sw128(sa + kk * 32, LBO, SBO);
            const uint64_t bd = smem_desc_sw128(sb + kk * 32, LBO, SBO);
            mma_bf16(d_tmem, ad, bd, idesc, (kl | kk) != 0);
          }
          mma_commit(&empty_bar[stage]);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        mma_commit(&tfull_bar);
      }
    mma_done:
      mma_commit(&done_bar);
    }
  } else if (warp >= FIRST_EPI_WARP) {
    // ---------------- epilogue: weighted sum of GA * GD ----------------
    const int ew = warp - FIRST_EPI_WARP;
    const int quad = warp & 3;
    const int half = ew >> 2;  // which 128-column half of the strip
    const uint32_t t_lane = static_cast<uint32_t>(quad * 32) << 16;
    int it = 0;
    for (int item = blockIdx.x; item < n_items; item += gridDim.x, ++it) {
      const Strip st = decode(item, g);
      if (!mbar_wait(&tfull_bar, it & 1, abrt, g.err)) break;
      tc_fence_after();
      float acc = 0.f;
      if (half < st.ns) {
        const uint32_t ta = tmem_base + t_lane + half * GT;
#pragma unroll
        for (int ch = 0; ch < GT / 32; ++ch) {
          float va[32], vd[32];
          tmem_ld32(ta + ch * 32, va);
          tmem_ld32(ta + 2 * GT + ch * 32, vd);
#pragma unroll
          for (int i = 0; i < 32; ++i) acc = fmaf(va[i], vd[i], acc);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty_bar);
      // the diagonal block (first half of a diagonal strip) counts once,
      // every off-diagonal block twice
      const float wgt = (st.tb == st.sb && half == 0) ? 1.f : 2.f;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
      if (lane == 0)
        g.part[static_cast<int64_t>(g.row0[st.layer] + st.ex) * g.NP +
               st.slot * NUM_EPI_WARPS + ew] = wgt * acc;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    if (lane == 0) {
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(&done_bar, 0)) {
        if (globaltimer_ns() - t0 > kWaitLimitNs) {
          atomicOr(g.err, kErrTimeout);
          break;
        }
      }
    }
    __syncwarp();
    tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

bool make_map_3d(CUtensorMap* m, const void* base, int B, int T, int d) {
  const uint64_t dims[3] = {static_cast<uint64_t>(d), static_cast<uint64_t>(T),
                            static_cast<uint64_t>(B)};
  const uint64_t strides[2] = {static_cast<uint64_t>(d) * 2, static_cast<uint64_t>(T) * d * 2};
  const uint32_t box[3] = {FK, GT, 1};
  return make_tma_bf16(m, base, 3, dims, strides, box);
}

int blocks_of(int T) { return (T + GT - 1) / GT; }
int full_strips(int nb) {
  int f = 0;
  for (int t = 0; t < nb; ++t) f += (nb - t) / 2;
  return f;
}
int half_strips(int nb) { return (nb + 1) / 2; }

}  // namespace

bool tc_ghost_supported(int T, int64_t d_in, int64_t d_out) {
  (void)T;
  return d_in % 8 == 0 && d_out % 8 == 0 && d_in <= kTcMaxAccum && d_out <= kTcMaxAccum &&
         tma_encode_available();
}

int tc_ghost_parts(int T) {
  const int nb = blocks_of(T);
  return (full_strips(nb) + half_strips(nb)) * NUM_EPI_WARPS;
}

cudaError_t tc_launch_ghost_batch(int L, const void* const* A, const void* const* D,
                                  const int* d_in, const int* d_out, const int* row0, int B,
                                  int T, float* part, int NP, int* err, cudaStream_t s) {
  if (L < 1 || L > kGhostMaxLayers) return cudaErrorInvalidValue;
  GhostBatch g{};
  for (int l = 0; l < L; ++l) {
    if (!make_map_3d(&g.mapA[l], A[l], B, T, d_in[l]) ||
        !make_map_3d(&g.mapD[l], D[l], B, T, d_out[l]))
      return cudaErrorInvalidValue;
    g.d_in[l] = d_in[l];
    g.d_out[l] = d_out[l];
    g.row0[l] = row0[l];
  }
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e =
        cudaFuncSetAttribute(k_ghost_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  g.L = L;
  g.B = B;
  g.T = T;
  g.nb = blocks_of(T);
  g.n_full = full_strips(g.nb);
  g.n_half = half_strips(g.nb);
  g.part = part;
  g.err = err;
  g.NP = NP;
  const int items = L * B * (g.n_full + g.n_half);
  const int sms = device_sm_count();
  const int grid = items < sms ? items : sms;
  note_launch();
  k_ghost_tc<<<grid, GHOST_THREADS, SMEM_BYTES, s>>>(g);
  return cudaGetLastError();
}

cudaError_t tc_launch_ghost(const void* A, const void* D, int B, int T, int d_in, int d_out,
                            float* part, int NP, int row0, int* err, cudaStream_t s) {
  return tc_launch_ghost_batch(1, &A, &D, &d_in, &d_out, &row0, B, T, part, NP, err, s);
}

}  // namespace dpk
