// tcgen05 Gram-form ("ghost") per-example squared norm of a dense layer:
//   n_i = ||A_i^T D_i||_F^2 = sum_{t,s} (A_i A_i^T)_{ts} (D_i D_i^T)_{ts}
// (the expansion of the Frobenius norm of a sum of outer products), which
// never forms the d_in x d_out gradient.
//
// Work item = (example i, 128x128 tile pair (tb <= sb) of the T x T Grams).
// For an item the tensor core accumulates the A-Gram tile (K = d_in) and the
// D-Gram tile (K = d_out) into two TMEM accumulators; the epilogue multiplies
// them elementwise and reduces.  Off-diagonal tile pairs count twice, the
// Grams being symmetric, so only the upper triangle of tile pairs is
// computed.  Both operands are rows of A_i (or D_i): K-major, loaded by TMA
// through a 3-D tensor map [B][T][d] so positions t >= T of an example read
// as zeros.  Diagonal pairs load one tile and use it for both operands.
//
// Warp roles (192 threads, persistent, TMEM double-buffered across items):
//   warp 0 TMA producer, warp 1 TMEM allocator + MMA issuer,
//   warps 2-5 epilogue (warp w reads TMEM lanes 32*(w%4)..+31).
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "internal.h"
#include "tc.h"
#include "tc_util.cuh"

namespace dpk {

namespace {

using namespace tc;

constexpr int GT = 128;                 // Gram tile edge (positions)
constexpr int FK = 64;                  // features per stage (128 bytes of bf16)
constexpr int STAGES = 6;
constexpr int TILE_BYTES = GT * FK * 2;  // 16 KB
constexpr int STAGE_BYTES = 2 * TILE_BYTES;
constexpr int NUM_EPI_WARPS = 4;
constexpr int GHOST_THREADS = 64 + 32 * NUM_EPI_WARPS;
constexpr uint32_t TMEM_COLS = 512;     // 2 buffers x (A-Gram 128 + D-Gram 128)
constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024;
// K-major, 128-byte swizzle: rows 128 B apart, 8-row groups 1024 B apart.
constexpr uint32_t LBO = 16, SBO = 1024;
constexpr uint32_t IDESC = idesc_bf16_f32(GT, GT, /*a_mn=*/0, /*b_mn=*/0);

struct GhostArgs {
  float* part;
  int* err;
  int B, T, d_in, d_out;
  int nb, npairs;
  int NP, row0;
};

__device__ __forceinline__ void pair_of(int pid, int nb, int& tb, int& sb) {
  int r = 0, left = pid;
  while (left >= nb - r) {
    left -= nb - r;
    ++r;
  }
  tb = r;
  sb = r + left;
}

__global__ void __launch_bounds__(GHOST_THREADS, 1)
    k_ghost_tc(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapD,
               const GhostArgs g) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  __shared__ uint64_t full_bar[STAGES], empty_bar[STAGES], tfull_bar[2], tempty_bar[2], done_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_items = g.B * g.npairs;
  const int ka = (g.d_in + FK - 1) / FK, kd = (g.d_out + FK - 1) / FK;
  volatile int* abrt = &abort_flag;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull_bar[b], 1);
      mbar_init(&tempty_bar[b], NUM_EPI_WARPS);
    }
    mbar_init(&done_bar, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&mapA);
    tma_prefetch_desc(&mapD);
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
        const int ex = item / g.npairs;
        int tb, sb;
        pair_of(item % g.npairs, g.nb, tb, sb);
        const bool diag = tb == sb;
        for (int k = 0; k < ka + kd; ++k) {
          const CUtensorMap* map = k < ka ? &mapA : &mapD;
          const int f0 = (k < ka ? k : k - ka) * FK;
          if (!mbar_wait(&empty_bar[stage], phase ^ 1, abrt, g.err)) goto producer_done;
          uint8_t* st = smem + stage * STAGE_BYTES;
          mbar_arrive_expect_tx(&full_bar[stage], diag ? TILE_BYTES : 2 * TILE_BYTES);
          tma_load_3d(map, &full_bar[stage], st, f0, tb * GT, ex);
          if (!diag) tma_load_3d(map, &full_bar[stage], st + TILE_BYTES, f0, sb * GT, ex);
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
        int tb, sb;
        pair_of(item % g.npairs, g.nb, tb, sb);
        const bool diag = tb == sb;
        const int buf = it & 1;
        const uint32_t tph = (it >> 1) & 1;
        if (!mbar_wait(&tempty_bar[buf], tph ^ 1, abrt, g.err)) goto mma_done;
        tc_fence_after();
        for (int k = 0; k < ka + kd; ++k) {
          const bool is_a = k < ka;
          const int kl = is_a ? k : k - ka;
          const uint32_t d_tmem = tmem_base + buf * 2 * GT + (is_a ? 0 : GT);
          if (!mbar_wait(&full_bar[stage], phase, abrt, g.err)) goto mma_done;
          tc_fence_after();
          const uint32_t st = smem_u32(smem + stage * STAGE_BYTES);
          const uint32_t ss = diag ? st : st + TILE_BYTES;
#pragma unroll
          for (int kk = 0; kk < FK / 16; ++kk) {
            const uint64_t ad = smem_desc_sw128(st + kk * 32, LBO, SBO);
            const uint64_t bd = smem_desc_sw128(ss + kk * 32, LBO, SBO);
            mma_bf16(d_tmem, ad, bd, IDESC, (kl | kk) != 0);
          }
          mma_commit(&empty_bar[stage]);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        mma_commit(&tfull_bar[buf]);
      }
    mma_done:
      mma_commit(&done_bar);
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(&done_bar, 0)) {
        if (globaltimer_ns() - t0 > kWaitLimitNs) {
          atomicOr(g.err, kErrTimeout);
          break;
        }
      }
    }
  } else {
    // ---------------- epilogue: sum_{s} GA[t][s] * GD[t][s] ----------------
    const int ew = warp - 2;
    const int quad = warp & 3;
    const uint32_t t_lane = static_cast<uint32_t>(quad * 32) << 16;
    int it = 0;
    for (int item = blockIdx.x; item < n_items; item += gridDim.x, ++it) {
      const int ex = item / g.npairs;
      const int pid = item % g.npairs;
      int tb, sb;
      pair_of(pid, g.nb, tb, sb);
      const int buf = it & 1;
      const uint32_t tph = (it >> 1) & 1;
      if (!mbar_wait(&tfull_bar[buf], tph, abrt, g.err)) break;
      tc_fence_after();
      const uint32_t ta = tmem_base + t_lane + buf * 2 * GT;
      float acc = 0.f;
#pragma unroll
      for (int ch = 0; ch < GT / 32; ++ch) {
        float va[32], vd[32];
        tmem_ld32(ta + ch * 32, va);
        tmem_ld32(ta + GT + ch * 32, vd);
#pragma unroll
        for (int i = 0; i < 32; ++i) acc = fmaf(va[i], vd[i], acc);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty_bar[buf]);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
      if (lane == 0)
        g.part[static_cast<int64_t>(g.row0 + ex) * g.NP + pid * NUM_EPI_WARPS + ew] =
            (tb == sb ? 1.f : 2.f) * acc;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
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

}  // namespace

bool tc_ghost_supported(int T, int64_t d_in, int64_t d_out) {
  (void)T;
  return d_in % 8 == 0 && d_out % 8 == 0 && tma_encode_available();
}

int tc_ghost_parts(int T) {
  const int nb = (T + GT - 1) / GT;
  return nb * (nb + 1) / 2 * NUM_EPI_WARPS;
}

cudaError_t tc_launch_ghost(const void* A, const void* D, int B, int T, int d_in, int d_out,
                            float* part, int NP, int row0, int* err, cudaStream_t s) {
  CUtensorMap mA, mD;
  if (!make_map_3d(&mA, A, B, T, d_in) || !make_map_3d(&mD, D, B, T, d_out))
    return cudaErrorInvalidValue;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e =
        cudaFuncSetAttribute(k_ghost_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  GhostArgs g{};
  g.part = part;
  g.err = err;
  g.B = B;
  g.T = T;
  g.d_in = d_in;
  g.d_out = d_out;
  g.nb = (T + GT - 1) / GT;
  g.npairs = g.nb * (g.nb + 1) / 2;
  g.NP = NP;
  g.row0 = row0;
  const int items = B * g.npairs;
  const int sms = device_sm_count();
  const int grid = items < sms ? items : sms;
  k_ghost_tc<<<grid, GHOST_THREADS, SMEM_BYTES, s>>>(mA, mD, g);
  return cudaGetLastError();
}

}  // namespace dpk
