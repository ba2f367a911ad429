// tcgen05 Gram-form ("ghost") per-example squared norm of dense layers:
//   n_i = ||A_i^T D_i||_F^2 = sum_{t,s} (A_i A_i^T)_{ts} (D_i D_i^T)_{ts}
// (the expansion of the Frobenius norm of a sum of outer products), which
// never forms the d_in x d_out gradient.
//
// The T x T Grams are cut into 128-position blocks and only block pairs
// (t, s) with t <= s are needed: off-diagonal pairs count twice, the Grams
// being symmetric.  For every block pair of a work item the tensor core
// accumulates the A-Gram (K = d_in) and the D-Gram (K = d_out) into two TMEM
// accumulators, and the epilogue multiplies them elementwise and reduces.
// Operands are K-major rows of A_i / D_i read through 3-D tensor maps
// [B][T][d], so positions t >= T of an example read as zeros.
//
// Two kernels, chosen by the number of blocks nb = ceil(T / 128):
//
//   k_ghost_tc_pair (nb even; CTA pairs, tcgen05 cta_group::2).  A work item
//   is a pair of 256-position super-blocks (ts <= ss) of one example: CTA r
//   of the pair stages t-block 2 ts + r as its A rows and s-block 2 ss + r as
//   its half of the B rows, and the pair MMA (M = N = 256) gives CTA r the
//   block pairs (2 ts + r, 2 ss) and (2 ts + r, 2 ss + 1) in its TMEM.  Each
//   SM stages one tile per 128 x 256 product (half a tile per block pair)
//   where a single CTA stages one and a half; a diagonal item (ts == ss)
//   stages one tile per CTA and uses it as both operands.  Its one lower
//   block pair (2 ts + 1, 2 ts) is computed and not read.  For T = 512 that
//   is 8 tiles staged per example, layer and K step instead of 12: the
//   single-CTA kernel is bound by operand delivery from L2 to the SMs.
//
//   k_ghost_tc (nb odd, including T <= 128).  A work item is a strip: one
//   128-row t-block against up to two consecutive s-blocks (N = 256 MMAs).
//   Strips that start on the diagonal load each 128-row tile once and use it
//   for both operands.
//
// One launch serves up to kGhostMaxLayers layers of a step (they share B and
// T), so the few items of each layer balance across all SMs.
//
// Warp roles (384 threads, one CTA per SM):
//   warp 0 TMA producer, warp 1 TMEM allocator + MMA issuer (the leader CTA
//   of a pair), warps 2-3 idle, warps 4-11 epilogue (warp w reads TMEM lanes
//   32*(w%4)..+31, column half (w-4)/4 of each 256-column accumulator).
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
constexpr int TILE_BYTES = GT * FK * 2;  // 16 KB: one 128-position tile
constexpr int NUM_EPI_WARPS = 8;
constexpr int FIRST_EPI_WARP = 4;
constexpr int GHOST_THREADS = 128 + 32 * NUM_EPI_WARPS;
constexpr uint32_t TMEM_COLS = 512;      // A-Gram 256 + D-Gram 256
// K-major, 128-byte swizzle: rows 128 B apart, 8-row groups 1024 B apart.
constexpr uint32_t LBO = 16, SBO = 1024;

// single-CTA strips.  A stage holds SLOTS boxes of 128 rows x 64 features.
// A strip stages `nt` tiles per K step (its t-tile unless diagonal, then its
// one or two s-tiles) and fits nbox = SLOTS / nt boxes of each per stage (a
// K step of nbox * 64 features), laid out box by box: the slots of box b are
// [t-tile, s-tile 0, s-tile 1] (t-tile absent on the diagonal), so the two
// s-tiles of a 256-row B operand sit next to each other.
constexpr int STAGES = 3;
constexpr int SLOTS = 4;
constexpr int STAGE_BYTES = SLOTS * TILE_BYTES;
constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024;
constexpr uint32_t IDESC_N256 = idesc_bf16_f32(GT, 2 * GT, 0, 0);
constexpr uint32_t IDESC_N128 = idesc_bf16_f32(GT, GT, 0, 0);

// CTA pairs.  A stage holds 2 P_BOXES boxes of 128 rows x 64 features per
// CTA: for an off-diagonal item P_BOXES boxes of this CTA's s-tile and of its
// t-tile (a K step of P_BOXES * 64 features), for a diagonal item, whose
// t-tile is its s-tile, 2 P_BOXES boxes of the s-tile (a K step twice as
// long, so the same stages cover twice the load latency).  Every stage of
// either kind carries 4 P_BOXES boxes for the pair.
constexpr int P_BOXES = 2;
constexpr int P_STAGES = 3;
constexpr int P_S_OFF = 0;                          // s-tile boxes (B rows of this CTA)
constexpr int P_T_OFF = P_BOXES * TILE_BYTES;       // t-tile boxes (off-diagonal items)
constexpr int P_STAGE_BYTES = 2 * P_BOXES * TILE_BYTES;
constexpr uint32_t P_STAGE_TX = 4 * P_BOXES * TILE_BYTES;  // both CTAs' boxes of a stage
constexpr int P_SMEM_BYTES = P_STAGES * P_STAGE_BYTES + 1024;
constexpr uint32_t IDESC_PAIR = idesc_bf16_f32(2 * GT, 2 * GT, 0, 0);

struct GhostBatch {
  CUtensorMap mapA[kGhostMaxLayers];
  CUtensorMap mapD[kGhostMaxLayers];
  int d_in[kGhostMaxLayers];
  int d_out[kGhostMaxLayers];
  int row0[kGhostMaxLayers];   // partial-sum row of example 0 of the layer
  int L, B, T, nb;             // layers in this launch, examples, positions, blocks
  int n_full, n_half;          // single-CTA strips per example
  int nsb, per_ex;             // pairs: super-blocks, items per example
  float* part;
  int* err;
  int NP;
};

// Bounded wait used only at teardown (ignores the abort flag).
__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity, int* err) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer_ns() - t0 > kWaitLimitNs) {
      atomicOr(err, kErrTimeout);
      return;
    }
  }
}

// ---------------------------------------------------------------------------
// single-CTA strips
// ---------------------------------------------------------------------------
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
__device__ __forceinline__ Strip decode(int64_t item, const GhostBatch& g) {
  Strip s;
  const int per_ex = g.n_full + g.n_half;
  const int64_t per_layer = static_cast<int64_t>(g.B) * per_ex;
  s.layer = static_cast<int>(item / per_layer);
  const int64_t r = item - s.layer * per_layer;
  s.ex = static_cast<int>(r / per_ex);
  const int k = static_cast<int>(r - static_cast<int64_t>(s.ex) * per_ex);
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
  const int64_t n_items = static_cast<int64_t>(g.L) * g.B * (g.n_full + g.n_half);
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
      for (int64_t item = blockIdx.x; item < n_items; item += gridDim.x) {
        const Strip st = decode(item, g);
        const bool diag = st.tb == st.sb;
        const CUtensorMap* mA = &g.mapA[st.layer];
        const CUtensorMap* mD = &g.mapD[st.layer];
        const int nt = (diag ? 0 : 1) + st.ns;  // tiles per box
        const int nbox = SLOTS / nt;
        const int fks = nbox * FK;
        const int ka = (g.d_in[st.layer] + fks - 1) / fks;
        const int kd = (g.d_out[st.layer] + fks - 1) / fks;
        const uint32_t bytes = static_cast<uint32_t>(nbox * nt) * TILE_BYTES;
        for (int k = 0; k < ka + kd; ++k) {
          const CUtensorMap* map = k < ka ? mA : mD;
          const int f0 = (k < ka ? k : k - ka) * fks;
          if (!mbar_wait(&empty_bar[stage], phase ^ 1, abrt, g.err)) goto producer_done;
          uint8_t* sp = smem + stage * STAGE_BYTES;
          mbar_arrive_expect_tx(&full_bar[stage], bytes);
          for (int b = 0; b < nbox; ++b) {
            uint8_t* bp = sp + b * nt * TILE_BYTES;
            const int f = f0 + b * FK;
            if (!diag) {
              tma_load_3d(map, &full_bar[stage], bp, f, st.tb * GT, st.ex);
              bp += TILE_BYTES;
            }
            tma_load_3d(map, &full_bar[stage], bp, f, st.sb * GT, st.ex);
            if (st.ns == 2)
              tma_load_3d(map, &full_bar[stage], bp + TILE_BYTES, f, (st.sb + 1) * GT, st.ex);
          }
          ++uses[stage];
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
    producer_done:
      for (int s = 0; s < STAGES; ++s)
        if (uses[s] != 0) drain_wait(&full_bar[s], (uses[s] - 1) & 1, g.err);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      for (int64_t item = blockIdx.x; item < n_items; item += gridDim.x, ++it) {
        const Strip st = decode(item, g);
        const bool diag = st.tb == st.sb;
        const uint32_t idesc = st.ns == 2 ? IDESC_N256 : IDESC_N128;
        const int nt = (diag ? 0 : 1) + st.ns;
        const int nbox = SLOTS / nt;
        const int fks = nbox * FK;
        const int ka = (g.d_in[st.layer] + fks - 1) / fks;
        const int kd = (g.d_out[st.layer] + fks - 1) / fks;
        if (!mbar_wait(&tempty_bar, (it & 1) ^ 1, abrt, g.err)) goto mma_done;
        tc_fence_after();
        for (int k = 0; k < ka + kd; ++k) {
          const bool is_a = k < ka;
          const int kl = is_a ? k : k - ka;
          const uint32_t d_tmem = tmem_base + (is_a ? 0 : 2 * GT);
          if (!mbar_wait(&full_bar[stage], phase, abrt, g.err)) goto mma_done;
          tc_fence_after();
          const uint32_t sp = smem_u32(smem + stage * STAGE_BYTES);
          for (int b = 0; b < nbox; ++b) {
            const uint32_t sa = sp + b * nt * TILE_BYTES;
            const uint32_t sb = diag ? sa : sa + TILE_BYTES;
#pragma unroll
            for (int kk = 0; kk < FK / 16; ++kk) {
              const uint64_t ad = smem_desc_sw128(sa + kk * 32, LBO, SBO);
              const uint64_t bd = smem_desc_sw128(sb + kk * 32, LBO, SBO);
              mma_bf16(d_tmem, ad, bd, idesc, (kl | b | kk) != 0);
            }
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
    for (int64_t item = blockIdx.x; item < n_items; item += gridDim.x, ++it) {
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
    if (lane == 0) drain_wait(&done_bar, 0, g.err);
    __syncwarp();
    tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

// ---------------------------------------------------------------------------
// CTA pairs
// ---------------------------------------------------------------------------
struct PairItem {
  int layer, ex, ts, ss, slot;
};

// Work list: layer-major, then example, then the example's super-block pairs
// (ts, ss), ts <= ss, row by row, so the items of one example run at about
// the same time and read its rows from DRAM about once.
__device__ __forceinline__ PairItem pair_decode(int64_t item, const GhostBatch& g) {
  PairItem s;
  const int64_t per_layer = static_cast<int64_t>(g.B) * g.per_ex;
  s.layer = static_cast<int>(item / per_layer);
  const int64_t r = item - s.layer * per_layer;
  s.ex = static_cast<int>(r / g.per_ex);
  int k = static_cast<int>(r - static_cast<int64_t>(s.ex) * g.per_ex);
  s.slot = k;
  int ts = 0;
  while (k >= g.nsb - ts) {
    k -= g.nsb - ts;
    ++ts;
  }
  s.ts = ts;
  s.ss = ts + k;
  return s;
}

__global__ void __launch_bounds__(GHOST_THREADS, 1)
    k_ghost_tc_pair(const __grid_constant__ GhostBatch g) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  __shared__ uint64_t full_bar[P_STAGES], empty_bar[P_STAGES], tfull_bar, tempty_bar, done_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int64_t unit = blockIdx.x >> 1, n_units = gridDim.x >> 1;
  const int64_t n_items = static_cast<int64_t>(g.L) * g.B * g.per_ex;
  volatile int* abrt = &abort_flag;

  if (threadIdx.x == 0) {
    for (int s = 0; s < P_STAGES; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    mbar_init(&tfull_bar, 1);
    // the epilogue warps of both CTAs free the accumulators on the leader's barrier
    mbar_init(&tempty_bar, 2 * NUM_EPI_WARPS);
    mbar_init(&done_bar, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    for (int l = 0; l < g.L; ++l) {
      tma_prefetch_desc(&g.mapA[l]);
      tma_prefetch_desc(&g.mapD[l]);
    }
  }
  if (warp == 1) tmem_alloc_pair(&tmem_slot, TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // the peer's barriers exist before any remote arrive or load
  tc_fence_after();
  const uint32_t tmem_base = tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer (both CTAs) ----------------
      // Both CTAs' loads complete on the leader's full barrier; each CTA
      // waits for the MMA's release of a stage on its own empty barrier.
      int stage = 0;
      uint32_t phase = 0;
      uint32_t uses[P_STAGES] = {};
      for (int64_t item = unit; item < n_items; item += n_units) {
        const PairItem st = pair_decode(item, g);
        const bool diag = st.ts == st.ss;
        const CUtensorMap* mA = &g.mapA[st.layer];
        const CUtensorMap* mD = &g.mapD[st.layer];
        const int nbox = diag ? 2 * P_BOXES : P_BOXES;  // s-tile boxes per stage
        const int fks = nbox * FK;                      // features per K step
        const int ka = (g.d_in[st.layer] + fks - 1) / fks;
        const int kd = (g.d_out[st.layer] + fks - 1) / fks;
        const int trow = (2 * st.ts + static_cast<int>(rank)) * GT;
        const int srow = (2 * st.ss + static_cast<int>(rank)) * GT;
        for (int k = 0; k < ka + kd; ++k) {
          const CUtensorMap* map = k < ka ? mA : mD;
          const int f0 = (k < ka ? k : k - ka) * fks;
          if (!mbar_wait(&empty_bar[stage], phase ^ 1, abrt, g.err)) goto producer_done;
          uint8_t* sp = smem + stage * P_STAGE_BYTES;
          const uint32_t fb = mapa_shared(smem_u32(&full_bar[stage]), 0);
          if (leader) mbar_arrive_expect_tx(&full_bar[stage], P_STAGE_TX);
          for (int b = 0; b < nbox; ++b)
            tma_load_3d_pair(map, fb, sp + P_S_OFF + b * TILE_BYTES, f0 + b * FK, srow, st.ex);
          if (!diag) {
#pragma unroll
            for (int b = 0; b < P_BOXES; ++b)
              tma_load_3d_pair(map, fb, sp + P_T_OFF + b * TILE_BYTES, f0 + b * FK, trow, st.ex);
          }
          ++uses[stage];
          if (++stage == P_STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
    producer_done:
      // No TMA write may still be landing in shared memory when the CTA
      // exits: the leader sees completion on its full barrier, the peer
      // waits for the MMA's release of each stage it loaded.
      for (int s = 0; s < P_STAGES; ++s) {
        if (uses[s] == 0) continue;
        if (leader)
          drain_wait(&full_bar[s], (uses[s] - 1) & 1, g.err);
        else
          drain_wait(&empty_bar[s], (uses[s] - 1) & 1, g.err);
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && leader) {
      // ---------------- MMA issuer (leader CTA) ----------------
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      for (int64_t item = unit; item < n_items; item += n_units, ++it) {
        const PairItem st = pair_decode(item, g);
        const bool diag = st.ts == st.ss;
        const int nbox = diag ? 2 * P_BOXES : P_BOXES;
        const int fks = nbox * FK;
        const int ka = (g.d_in[st.layer] + fks - 1) / fks;
        const int kd = (g.d_out[st.layer] + fks - 1) / fks;
        if (!mbar_wait(&tempty_bar, (it & 1) ^ 1, abrt, g.err)) goto mma_done;
        tc_fence_after();
        for (int k = 0; k < ka + kd; ++k) {
          const bool is_a = k < ka;
          const int kl = is_a ? k : k - ka;
          const uint32_t d_tmem = tmem_base + (is_a ? 0 : 2 * GT);
          if (!mbar_wait(&full_bar[stage], phase, abrt, g.err)) goto mma_done;
          tc_fence_after();
          const uint32_t sp = smem_u32(smem + stage * P_STAGE_BYTES);
          for (int b = 0; b < nbox; ++b) {
            const uint32_t sb = sp + P_S_OFF + b * TILE_BYTES;
            const uint32_t sa = diag ? sb : sp + P_T_OFF + b * TILE_BYTES;
#pragma unroll
            for (int kk = 0; kk < FK / 16; ++kk) {
              const uint64_t ad = smem_desc_sw128(sa + kk * 32, LBO, SBO);
              const uint64_t bd = smem_desc_sw128(sb + kk * 32, LBO, SBO);
              mma_bf16_pair(d_tmem, ad, bd, IDESC_PAIR, (kl | b | kk) != 0);
            }
          }
          mma_commit_pair(&empty_bar[stage]);
          if (++stage == P_STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        mma_commit_pair(&tfull_bar);
      }
    mma_done:
      // all issued MMAs complete before TMEM is released (both CTAs wait)
      mma_commit_pair(&done_bar);
    }
  } else if (warp >= FIRST_EPI_WARP) {
    // ---------------- epilogue: weighted sum of GA * GD ----------------
    // CTA r holds rows of t-block 2 ts + r; column half h is s-block 2 ss + h.
    const int ew = warp - FIRST_EPI_WARP;
    const int quad = warp & 3;
    const int half = ew >> 2;
    const uint32_t t_lane = static_cast<uint32_t>(quad * 32) << 16;
    const uint32_t tempty_leader = mapa_shared(smem_u32(&tempty_bar), 0);
    int it = 0;
    for (int64_t item = unit; item < n_items; item += n_units, ++it) {
      const PairItem st = pair_decode(item, g);
      if (!mbar_wait(&tfull_bar, it & 1, abrt, g.err)) break;
      tc_fence_after();
      // off-diagonal items: every block pair counts twice.  A diagonal item
      // holds blocks (2ts, 2ts) and (2ts+1, 2ts+1) (once each), (2ts, 2ts+1)
      // (twice) and its mirror (2ts+1, 2ts), which is not read.
      const int r = static_cast<int>(rank);
      const float wgt = st.ts != st.ss ? 2.f : (r == half ? 1.f : (r < half ? 2.f : 0.f));
      float acc = 0.f;
      if (wgt != 0.f) {
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
      if (lane == 0) mbar_arrive_cluster(tempty_leader);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
      if (lane == 0)
        g.part[static_cast<int64_t>(g.row0[st.layer] + st.ex) * g.NP +
               (st.slot * 2 + r) * NUM_EPI_WARPS + ew] = wgt * acc;
    }
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    // the leader's last commit tells both CTAs that no MMA still writes TMEM
    if (lane == 0) drain_wait(&done_bar, 0, g.err);
    __syncwarp();
    tmem_dealloc_pair(tmem_base, TMEM_COLS);
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
bool make_map_3d(CUtensorMap* m, const void* base, int B, int T, int d) {
  const uint64_t dims[3] = {static_cast<uint64_t>(d), static_cast<uint64_t>(T),
                            static_cast<uint64_t>(B)};
  const uint64_t strides[2] = {static_cast<uint64_t>(d) * 2, static_cast<uint64_t>(T) * d * 2};
  const uint32_t box[3] = {FK, GT, 1};
  return make_tma_bf16(m, base, 3, dims, strides, box);
}

int64_t blocks_of(int64_t T) { return (T + GT - 1) / GT; }
int64_t full_strips(int64_t nb) { return (nb / 2) * ((nb + 1) / 2); }  // sum of floor((nb-t)/2)
int64_t half_strips(int64_t nb) { return (nb + 1) / 2; }
// CTA pairs serve even block counts: the super-blocks then hold no block
// past the last one, so no pair multiplies a tile of zeros.
bool use_pair(int64_t nb) { return nb % 2 == 0; }
int64_t pair_items(int64_t nb) { return (nb / 2) * (nb / 2 + 1) / 2; }

}  // namespace

bool tc_ghost_supported(int T, int64_t d_in, int64_t d_out) {
  return T >= 1 && T <= kTcGhostMaxT && d_in % 8 == 0 && d_out % 8 == 0 &&
         d_in <= kTcMaxAccum && d_out <= kTcMaxAccum && tma_encode_available();
}

int64_t tc_ghost_parts(int T) {
  const int64_t nb = blocks_of(T);
  if (use_pair(nb)) return pair_items(nb) * 2 * NUM_EPI_WARPS;
  return (full_strips(nb) + half_strips(nb)) * NUM_EPI_WARPS;
}

namespace {
cudaError_t setup_pair_kernel() {
  return setup_once_per_device(reinterpret_cast<const void*>(&k_ghost_tc_pair), [] {
    return cudaFuncSetAttribute(k_ghost_tc_pair, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                P_SMEM_BYTES);
  });
}
cudaError_t setup_strip_kernel() {
  return setup_once_per_device(reinterpret_cast<const void*>(&k_ghost_tc), [] {
    return cudaFuncSetAttribute(k_ghost_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                SMEM_BYTES);
  });
}
cudaLaunchConfig_t pair_config(cudaLaunchAttribute* attr, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(GHOST_THREADS);
  cfg.dynamicSmemBytes = P_SMEM_BYTES;
  cfg.stream = s;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cfg;
}
// CTA pairs of k_ghost_tc_pair resident at once on the current device.
int max_resident_pairs() {
  return cached_per_device(reinterpret_cast<const void*>(&k_ghost_tc_pair), [] {
    const int sms = device_sm_count();
    cudaLaunchAttribute attr[1];
    cudaLaunchConfig_t q = pair_config(attr, nullptr);
    q.gridDim = dim3(sms);
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, k_ghost_tc_pair, &q) != cudaSuccess || n < 1) {
      cudaGetLastError();
      n = sms / 2;
    }
    return n < sms / 2 ? n : sms / 2;
  });
}
}  // namespace

cudaError_t tc_ghost_prepare() {
  cudaError_t e = setup_strip_kernel();
  if (e == cudaSuccess) e = setup_pair_kernel();
  if (e == cudaSuccess && max_resident_pairs() < 1) e = cudaErrorInvalidConfiguration;
  return e;
}

cudaError_t tc_launch_ghost_batch(int L, const void* const* A, const void* const* D,
                                  const int* d_in, const int* d_out, const int* row0, int B,
                                  int T, float* part, int NP, int* err, cudaStream_t s) {
  if (L < 1 || L > kGhostMaxLayers || T < 1 || T > kTcGhostMaxT || B < 1)
    return cudaErrorInvalidValue;
  if (tc_ghost_parts(T) > NP) return cudaErrorInvalidValue;
  GhostBatch g{};
  for (int l = 0; l < L; ++l) {
    if (!make_map_3d(&g.mapA[l], A[l], B, T, d_in[l]) ||
        !make_map_3d(&g.mapD[l], D[l], B, T, d_out[l]))
      return cudaErrorInvalidValue;
    g.d_in[l] = d_in[l];
    g.d_out[l] = d_out[l];
    g.row0[l] = row0[l];
  }
  g.L = L;
  g.B = B;
  g.T = T;
  g.nb = static_cast<int>(blocks_of(T));
  g.n_full = static_cast<int>(full_strips(g.nb));
  g.n_half = static_cast<int>(half_strips(g.nb));
  g.nsb = g.nb / 2;
  g.per_ex = static_cast<int>(pair_items(g.nb));
  g.part = part;
  g.err = err;
  g.NP = NP;
  const int sms = device_sm_count();
  if (use_pair(g.nb)) {
    cudaError_t e = setup_pair_kernel();
    if (e != cudaSuccess) return e;
    cudaLaunchAttribute attr[1];
    cudaLaunchConfig_t cfg = pair_config(attr, s);
    // persistent grid: as many pairs as can be resident at once
    const int max_pairs = max_resident_pairs();
    const int64_t items = static_cast<int64_t>(L) * B * g.per_ex;
    const int64_t pairs = items < max_pairs ? items : max_pairs;
    cfg.gridDim = dim3(static_cast<unsigned>(2 * pairs));
    note_launch();
    return cudaLaunchKernelEx(&cfg, k_ghost_tc_pair, g);
  }
  cudaError_t e = setup_strip_kernel();
  if (e != cudaSuccess) return e;
  const int64_t items = static_cast<int64_t>(L) * B * (g.n_full + g.n_half);
  const int grid = static_cast<int>(items < sms ? items : sms);
  note_launch();
  k_ghost_tc<<<grid, GHOST_THREADS, SMEM_BYTES, s>>>(g);
  return cudaGetLastError();
}

cudaError_t tc_launch_ghost(const void* A, const void* D, int B, int T, int d_in, int d_out,
                            float* part, int NP, int row0, int* err, cudaStream_t s) {
  return tc_launch_ghost_batch(1, &A, &D, &d_in, &d_out, &row0, B, T, part, NP, err, s);
}

}  // namespace dpk
