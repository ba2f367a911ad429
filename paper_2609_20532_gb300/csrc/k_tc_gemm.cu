// tcgen05 clipped-sum GEMM  S = A^T diag(c (x) 1_T) D  with the fused noise
// epilogue (Algorithm 2: sum of clipped per-example gradients, then
// out = out_scale * (S + sigma C z)), and the materialised per-example norm
// that shares its main loop (n_i = ||A_i^T D_i||_F^2 tile by tile).
//
// Operands: A is [B*T, d_in] and D is [B*T, d_out], both row-major, so as
// GEMM operands (M = d_in, N = d_out, K = B*T) both are MN-major; TMA loads
// 64-column x 64-row boxes with 128-byte swizzle straight into the canonical
// MN-major layout the tensor core reads.
//
// The clip factor varies along K (one value per example).  Instead of
// rescaling operand tiles in shared memory, the kernel folds it exactly:
// T is a multiple of the 64-row K block, so each example's contribution
// P_i = A_i^T D_i of the tile is accumulated in its own TMEM buffer (two
// buffers, 2 x 256 columns), and the epilogue warps add c_i * P_i into an
// fp32 register accumulator while the tensor core already works on the
// next example.  No extra rounding, no operand rewrite.
//
// Warp roles (3 warpgroups = 384 threads, one CTA per SM, persistent):
//   warpgroup 0: warp 0 TMA producer (one lane), warp 1 TMEM allocator +
//                MMA issuer (one lane), warps 2-3 idle; drops to 48 regs.
//   warpgroups 1-2 (warps 4-11): fold / epilogue, raised to 224 regs; warp w
//                reads TMEM lanes 32*(w%4)..+31, column half (w-4)/4.
// Register budget: launched at 168 x 384 = 64512; after the split
// 4*32*48 + 8*32*224 = 63488, and each SM sub-partition holds one warp of
// each warpgroup: 48 + 224 + 224 = 496 <= 512 registers per lane.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "internal.h"
#include "philox.cuh"
#include "tc.h"
#include "tc_util.cuh"

namespace dpk {

namespace {

using namespace tc;

constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr int A_STAGE = BM * BK * 2;           // 16 KB: two 64-col chunks of 64 rows x 128 B
constexpr int B_STAGE = BN * BK * 2;           // 32 KB: four chunks
constexpr int CHUNK = 64 * BK * 2;             // 8 KB: one 64-column chunk
constexpr int STAGE_BYTES = A_STAGE + B_STAGE;
constexpr int NUM_EPI_WARPS = 8;
constexpr int FIRST_EPI_WARP = 4;
constexpr int GEMM_THREADS = 128 + 32 * NUM_EPI_WARPS;
constexpr int REGS_CTRL = 48, REGS_EPI = 224;
constexpr uint32_t TMEM_COLS = 512;
constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024;
// MN-major, 128-byte swizzle: LBO = distance between 64-element MN chunks,
// SBO = distance between 8-row K groups.
constexpr uint32_t LBO = CHUNK, SBO = 1024;
constexpr uint32_t IDESC = idesc_bf16_f32(BM, BN, /*a_mn=*/1, /*b_mn=*/1);

struct GemmArgs {
  const float* c;
  float* out;
  float* part;
  int* err;
  int B, T, d_in, d_out;
  int n_m, n_n;
  int NP, row0;
  Epilogue ep;
};

template <bool NORM>
__global__ void __launch_bounds__(GEMM_THREADS, 1)
    k_gemm_tc(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapD,
              const GemmArgs g) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  __shared__ uint64_t full_bar[STAGES], empty_bar[STAGES], tfull_bar[2], tempty_bar[2], done_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int kpe = g.T / BK;
  const int n_tiles = g.n_m * g.n_n;
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

  if (warp < FIRST_EPI_WARP) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(REGS_CTRL));
  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      int stage = 0;
      uint32_t phase = 0;
      uint32_t uses[STAGES] = {};
      for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
        const int m0 = (tile % g.n_m) * BM, n0 = (tile / g.n_m) * BN;
        for (int ex = 0; ex < g.B; ++ex) {
          for (int kb = 0; kb < kpe; ++kb) {
            if (!mbar_wait(&empty_bar[stage], phase ^ 1, abrt, g.err)) goto producer_done;
            uint8_t* sa = smem + stage * STAGE_BYTES;
            uint8_t* sb = sa + A_STAGE;
            mbar_arrive_expect_tx(&full_bar[stage], STAGE_BYTES);
            const int krow = ex * g.T + kb * BK;
            tma_load_2d(&mapA, &full_bar[stage], sa, m0, krow);
            tma_load_2d(&mapA, &full_bar[stage], sa + CHUNK, m0 + 64, krow);
#pragma unroll
            for (int q = 0; q < 4; ++q)
              tma_load_2d(&mapD, &full_bar[stage], sb + q * CHUNK, n0 + 64 * q, krow);
            ++uses[stage];
            if (++stage == STAGES) {
              stage = 0;
              phase ^= 1;
            }
          }
        }
      }
    producer_done:
      // No TMA write may still be landing in shared memory when the CTA exits.
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
      for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
        for (int ex = 0; ex < g.B; ++ex, ++it) {
          const int buf = it & 1;
          const uint32_t tph = (it >> 1) & 1;
          if (!mbar_wait(&tempty_bar[buf], tph ^ 1, abrt, g.err)) goto mma_done;
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + buf * BN;
          for (int kb = 0; kb < kpe; ++kb) {
            if (!mbar_wait(&full_bar[stage], phase, abrt, g.err)) goto mma_done;
            tc_fence_after();
            const uint32_t sa = smem_u32(smem + stage * STAGE_BYTES);
            const uint32_t sb = sa + A_STAGE;
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk) {
              const uint64_t ad = smem_desc_sw128(sa + kk * 16 * 128, LBO, SBO);
              const uint64_t bd = smem_desc_sw128(sb + kk * 16 * 128, LBO, SBO);
              mma_bf16(d_tmem, ad, bd, IDESC, (kb | kk) != 0);
            }
            mma_commit(&empty_bar[stage]);
            if (++stage == STAGES) {
              stage = 0;
              phase ^= 1;
            }
          }
          mma_commit(&tfull_bar[buf]);
        }
      }
    mma_done:
      // all issued MMAs must complete before TMEM is released
      mma_commit(&done_bar);
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(&done_bar, 0)) {
        if (globaltimer_ns() - t0 > kWaitLimitNs) {
          atomicOr(g.err, kErrTimeout);
          break;
        }
      }
    }
  }
  } else {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(REGS_EPI));
    // ---------------- fold / epilogue warps ----------------
    const int ew = warp - FIRST_EPI_WARP;
    const int quad = warp & 3;         // TMEM lane quadrant this warp may access
    const int half = ew >> 2;          // column half of the tile
    const int row = quad * 32 + lane;  // tile row held by this thread
    const uint32_t t_lane = static_cast<uint32_t>(quad * 32) << 16;
    int it = 0;
    for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
      const int m0 = (tile % g.n_m) * BM, n0 = (tile / g.n_m) * BN;
      float S[128];
      if constexpr (!NORM) {
#pragma unroll
        for (int i = 0; i < 128; ++i) S[i] = 0.f;
      }
      for (int ex = 0; ex < g.B; ++ex, ++it) {
        const int buf = it & 1;
        const uint32_t tph = (it >> 1) & 1;
        if (!mbar_wait(&tfull_bar[buf], tph, abrt, g.err)) goto epi_done;
        tc_fence_after();
        const uint32_t tcol = t_lane + buf * BN + half * 128;
        float sq = 0.f;
        const float ci = NORM ? 0.f : g.c[ex];
#pragma unroll
        for (int ch = 0; ch < 4; ++ch) {
          float v[32];
          tmem_ld32(tmem_base + tcol + ch * 32, v);
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            if constexpr (NORM)
              sq = fmaf(v[i], v[i], sq);
            else
              S[ch * 32 + i] = fmaf(ci, v[i], S[ch * 32 + i]);
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty_bar[buf]);
        if constexpr (NORM) {
          // one partial per epilogue warp; the clip kernel sums them in order
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
          if (lane == 0)
            g.part[static_cast<int64_t>(g.row0 + ex) * g.NP + tile * NUM_EPI_WARPS + ew] = sq;
        }
      }
      if constexpr (!NORM) {
        const int j = m0 + row;
        if (j < g.d_in) {
          float* orow = g.out + static_cast<int64_t>(j) * g.d_out;
          const Epilogue& ep = g.ep;
          const uint64_t prow = ep.p_base + static_cast<uint64_t>(j) * g.d_out;
#pragma unroll
          for (int q = 0; q < 32; ++q) {
            const int k = n0 + half * 128 + 4 * q;
            if (k < g.d_out) {
              float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
              // p_base and d_out are multiples of 8 on this path, so the four
              // parameters prow+k .. +3 form exactly one Philox quad
              if (ep.add_noise) z = gauss_quad(ep.seed, ep.step, (prow + k) >> 2);
              float4 v;
              v.x = ep.out_scale * fmaf(ep.sigmaC, z.x, S[4 * q + 0]);
              v.y = ep.out_scale * fmaf(ep.sigmaC, z.y, S[4 * q + 1]);
              v.z = ep.out_scale * fmaf(ep.sigmaC, z.z, S[4 * q + 2]);
              v.w = ep.out_scale * fmaf(ep.sigmaC, z.w, S[4 * q + 3]);
              float4* o = reinterpret_cast<float4*>(orow + k);  // d_out % 8 == 0: aligned
              if (ep.accumulate) {
                const float4 p = *o;
                v.x += p.x;
                v.y += p.y;
                v.z += p.z;
                v.w += p.w;
              }
              *o = v;
            }
          }
        }
      }
    }
  epi_done:;
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
// 2D bf16 map over a row-major [rows, cols] array, box {64 cols, box_rows}.
bool make_map_2d(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows,
                 uint32_t box_rows) {
  const uint64_t dims[2] = {cols, rows};
  const uint64_t strides[1] = {cols * 2};
  const uint32_t box[2] = {64, box_rows};
  return make_tma_bf16(m, base, 2, dims, strides, box);
}

template <bool NORM>
cudaError_t launch_gemm(const void* A, const void* D, GemmArgs& g, cudaStream_t s) {
  CUtensorMap mA, mD;
  const uint64_t rows = static_cast<uint64_t>(g.B) * g.T;
  if (!make_map_2d(&mA, A, g.d_in, rows, BK) || !make_map_2d(&mD, D, g.d_out, rows, BK))
    return cudaErrorInvalidValue;
  static bool attr_set[2] = {false, false};
  if (!attr_set[NORM]) {
    cudaError_t e = cudaFuncSetAttribute(k_gemm_tc<NORM>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
    if (e != cudaSuccess) return e;
    attr_set[NORM] = true;
  }
  g.n_m = (g.d_in + BM - 1) / BM;
  g.n_n = (g.d_out + BN - 1) / BN;
  const int tiles = g.n_m * g.n_n;
  const int sms = device_sm_count();
  const int grid = tiles < sms ? tiles : sms;
  k_gemm_tc<NORM><<<grid, GEMM_THREADS, SMEM_BYTES, s>>>(mA, mD, g);
  return cudaGetLastError();
}

}  // namespace

bool tc_gemm_supported(int T, int64_t d_in, int64_t d_out) {
  return T % BK == 0 && d_in % 8 == 0 && d_out % 8 == 0 && tma_encode_available();
}

int tc_mat_parts(int64_t d_in, int64_t d_out) {
  return static_cast<int>(((d_in + BM - 1) / BM) * ((d_out + BN - 1) / BN)) * NUM_EPI_WARPS;
}

cudaError_t tc_launch_mat_norm(const void* A, const void* D, int B, int T, int d_in, int d_out,
                               float* part, int NP, int row0, int* err, cudaStream_t s) {
  GemmArgs g{};
  g.part = part;
  g.err = err;
  g.B = B;
  g.T = T;
  g.d_in = d_in;
  g.d_out = d_out;
  g.NP = NP;
  g.row0 = row0;
  return launch_gemm<true>(A, D, g, s);
}

cudaError_t tc_launch_clipsum(const void* A, const void* D, const float* c, int B, int T,
                              int d_in, int d_out, float* out, const Epilogue& ep, int* err,
                              cudaStream_t s) {
  GemmArgs g{};
  g.c = c;
  g.out = out;
  g.err = err;
  g.B = B;
  g.T = T;
  g.d_in = d_in;
  g.d_out = d_out;
  g.ep = ep;
  return launch_gemm<false>(A, D, g, s);
}

}  // namespace dpk
