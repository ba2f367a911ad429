// tcgen05 clipped-sum GEMM  S = A^T diag(c (x) 1_T) D  with the fused noise
// epilogue (Algorithm 2: sum of clipped per-example gradients, then
// out = out_scale * (S + sigma C z)), and the materialised per-example norm
// that shares its main loop (n_i = ||A_i^T D_i||_F^2 tile by tile).
//
// Operands: A is [B*T, d_in] and D is [B*T, d_out], both row-major, so as
// GEMM operands (M = d_in, N = d_out, K = B*T) both are MN-major; TMA loads
// 64-column x 64-row boxes with 128-byte swizzle straight into the canonical
// MN-major layout the tensor core reads (LBO = 8 KB between 64-element MN
// chunks, SBO = 1 KB between 8-row K groups).
//
// The clip factor varies along K (one value per example).  Instead of
// rescaling operand tiles in shared memory, the kernel folds it exactly:
// T is a multiple of the 64-row K block, so each example's contribution
// P_i = A_i^T D_i of the tile is accumulated in its own TMEM buffer (two
// buffers, 2 x 256 columns), and the epilogue warps add c_i * P_i into an
// fp32 register accumulator while the tensor core already works on the
// next example.  No extra rounding, no operand rewrite.
//
// Two variants of the same kernel:
//   single CTA (PAIR = false): tile 128 x 256, 4 stages of 48 KB;
//   CTA pair (PAIR = true, cluster of 2, tcgen05 cta_group::2): tile
//     256 x 256; each CTA stages its 128 rows of A and its 128 columns of D
//     (6 stages of 32 KB, taken two at a time when an example has an even
//     number of K blocks, then as 128-row boxes), the leader CTA issues the
//     pair MMA and its commits arrive on the barriers of both CTAs; each
//     CTA's TMEM holds its 128 rows.  Half the shared-memory bytes per MMA,
//     so the same stage memory covers 1.5x more load latency.
//
// Warp roles (3 warpgroups = 384 threads, one CTA per SM, persistent):
//   warpgroup 0: warp 0 TMA producer (one lane), warp 1 TMEM allocator +
//                MMA issuer (one lane; leader CTA only in a pair), warps 2-3
//                idle; drops to 48 regs.
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

constexpr int BM = 128, BN = 256, BK = 64;
constexpr int CHUNK = 64 * BK * 2;  // 8 KB: one 64-column chunk of 64 rows
constexpr int NUM_EPI_WARPS = 8;
constexpr int FIRST_EPI_WARP = 4;
constexpr int GEMM_THREADS = 128 + 32 * NUM_EPI_WARPS;
constexpr int REGS_CTRL = 48, REGS_EPI = 224;
constexpr uint32_t LBO = CHUNK, SBO = 1024;

// NB: tile width in output columns (N of the MMA), 256, or 128 for layers
// with d_out <= 128 (no MMA work on columns past the layer).
template <bool PAIR, int NB>
struct Cfg {
  static constexpr int B_COLS = PAIR ? NB / 2 : NB;         // D columns staged per CTA
  static constexpr int A_STAGE = BM * BK * 2;               // 16 KB
  static constexpr int B_STAGE = B_COLS * BK * 2;           // 8 / 16 / 32 KB
  static constexpr int STAGE_BYTES = A_STAGE + B_STAGE;     // 24 / 32 / 48 KB
  // 192 KB of stages whatever the tile: the operand bytes in flight set the
  // rate at which L2 delivers them (a stage's round trip is about the same
  // for every tile), so the narrow tiles get more stages: 8, 6 or 4
  static constexpr int STAGES = (192 * 1024) / STAGE_BYTES;
  static_assert(STAGES % 2 == 0 && STAGES * STAGE_BYTES == 192 * 1024, "stage split");
  static constexpr int TILE_M = PAIR ? 2 * BM : BM;
  // pipeline stages, then one 4 KB store-staging block per epilogue warp
  static constexpr int STAGING = STAGES * STAGE_BYTES;
  static constexpr int SMEM_BYTES = STAGING + NUM_EPI_WARPS * 4096 + 1024;
  static constexpr uint32_t IDESC = idesc_bf16_f32(TILE_M, NB, /*a_mn=*/1, /*b_mn=*/1);
  static constexpr uint32_t TMEM_COLS = 2 * NB;             // two accumulator buffers
  static constexpr int HALF = NB / 2;                       // columns per epilogue thread
};

// One launch serves up to kGemmMaxLayers layers of a step (same B and T):
// their tiles form one persistent work list, so the last round of tiles is
// shared by all layers instead of idling most of the GPU once per layer.
struct GemmArgs {
  CUtensorMap mapA[kGemmMaxLayers];
  CUtensorMap mapD[kGemmMaxLayers];
  CUtensorMap mapO[kGemmMaxLayers];  // fp32 outputs, 32 x 32 boxes ([split][d_in][d_out] when split)
  CUtensorMap mapT;                   // tail pieces' partial tiles [piece][TILE_M][NB] (fp32)
  // a strided convolution's parity maps 1-3 (map 0 is mapA; conv_taps)
  CUtensorMap mapS[kGemmMaxLayers][3];
  float* out[kGemmMaxLayers];
  uint64_t p_base[kGemmMaxLayers];  // global parameter index of element (0, 0)
  int d_in[kGemmMaxLayers], d_out[kGemmMaxLayers];
  int n_m[kGemmMaxLayers], n_n[kGemmMaxLayers];
  int split[kGemmMaxLayers];  // example ranges per tile (1: the whole batch)
  int conv[kGemmMaxLayers];   // 1: mapA is the NHWC input of a convolution (patch rows on the fly)
  ConvGeom cg[kGemmMaxLayers];
  int tile_start[kGemmMaxLayers + 1];  // first work item of each layer (whole tiles)
  // Tail split: a layer's tiles from tail_from on (the tiles that would
  // leave most units idle in the launch's last round) run as pieces, each
  // over about B / tail_split examples, after every whole tile of the
  // launch.  Pieces of layer l are items tile_start[L] + piece_start[l] ..;
  // piece q of the layer covers its tail tile q % n and example range
  // q / n (n tail tiles).  A clipped-sum piece stores its partial tile into
  // mapT at its piece index for the tail reduce; a norm piece writes its
  // examples' partials like a whole tile.
  int tail_from[kGemmMaxLayers], tail_split[kGemmMaxLayers];
  int piece_start[kGemmMaxLayers + 1];
  int n_items;
  int L;
  const float* c;  // clip factors [B]; nullptr: all ones (pre-scaled operand)
  float* part;     // materialised-norm partials (L == 1)
  int* err;
  int B, T;
  int NP, row0;
  int pad3d;   // 1: maps are [B][T][d] and each example's K range is padded to 64 rows
  int d_rows;  // > 0: pre-scaled mode, D row of K row k is k % d_rows (A holds [hi; lo])
  const uint64_t* key;  // device {seed, step}
  float out_scale, sigmaC;
  int add_noise, accumulate;
};

// One work item: a tile of layer l over the examples [e0, e1) of range s.
// Items are range-major within a layer, so the items in flight at once are
// different tiles of the same examples and share their operand rows in L2.
struct GemmItem {
  int l, lt, s, e0, e1;
  int z;  // tail piece index, -1 for a tile of its own
};

__device__ __forceinline__ GemmItem gemm_item(const GemmArgs& g, int item) {
  GemmItem w;
  int l = 0;
  if (item >= g.tile_start[g.L]) {
    // a tail piece (tail tiles are unsplit layers' last tiles)
    const int p = item - g.tile_start[g.L];
    while (p >= g.piece_start[l + 1]) ++l;
    const int q = p - g.piece_start[l];
    const int n = g.n_m[l] * g.n_n[l] - g.tail_from[l];
    const int r = q / n;
    w.l = l;
    w.s = 0;
    w.lt = g.tail_from[l] + (q - r * n);
    w.e0 = static_cast<int>(static_cast<int64_t>(g.B) * r / g.tail_split[l]);
    w.e1 = static_cast<int>(static_cast<int64_t>(g.B) * (r + 1) / g.tail_split[l]);
    w.z = p;
    return w;
  }
  while (item >= g.tile_start[l + 1]) ++l;
  const int li = item - g.tile_start[l];
  const int S = g.split[l];
  const int tiles = S > 1 ? g.n_m[l] * g.n_n[l] : g.tail_from[l];  // whole tiles per range
  w.l = l;
  w.s = li / tiles;
  w.lt = li - w.s * tiles;
  w.e0 = static_cast<int>(static_cast<int64_t>(g.B) * w.s / S);
  w.e1 = static_cast<int>(static_cast<int64_t>(g.B) * (w.s + 1) / S);
  w.z = -1;
  return w;
}

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

// A convolution's two A chunks of a tile: 64 channels of one kernel tap
// each, fixed for the whole work item.  cc: first channel (C_in for a chunk
// past K: a box wholly out of range, read as zeros).  The input pixel of
// output position (ho, wo) under tap offset (dy, dx) (padding included) is
// (s ho + dy, s wo + dx) for stride s.  With dy = s qy + ry (0 <= ry < s) that
// is pixel (ho + qy, wo + qx) of the parity map (ry, rx), the input's pixels
// whose row and column are ry and rx modulo s: map = ry s + rx (0 for a unit
// stride, whose one map is the input), dy, dx hold qy, qx.
struct ConvTaps {
  int cc[2], dx[2], dy[2], map[2];
};

__device__ __forceinline__ ConvTaps conv_taps(const ConvGeom& v, int m0) {
  ConvTaps t;
#pragma unroll
  for (int q = 0; q < 2; ++q) {
    const int mm = m0 + 64 * q;
    int tap = mm / v.C_in, cc = mm - tap * v.C_in;
    if (tap >= v.kh * v.kw) {
      tap = 0;
      cc = v.C_in;
    }
    const int ki = tap / v.kw;
    const int dx = (tap - ki * v.kw) - v.pad_w, dy = ki - v.pad_h;
    const int rx = ((dx % v.stride_w) + v.stride_w) % v.stride_w;
    const int ry = ((dy % v.stride_h) + v.stride_h) % v.stride_h;
    t.cc[q] = cc;
    t.dx[q] = (dx - rx) / v.stride_w;
    t.dy[q] = (dy - ry) / v.stride_h;
    t.map[q] = ry * v.stride_w + rx;
  }
  return t;
}

// TMA loads of one K block of a stage: A rows m0.. (two 64-column chunks)
// and the D columns this CTA stages, for K block kb of example ex.  The
// leader (a single CTA: itself) announces tx_bytes, the bytes the whole stage
// brings to its full barrier, with the stage's first block (0 for the rest).  For a convolution
// an A chunk is 64 channels of one kernel tap at 64 output positions
// starting at output row ho0, column wo0: one 4-D box [1 image][rows]
// [columns][64 channels] of the NHWC input at the tap's offset, whose
// out-of-range pixels (the zero padding) read as zeros.  The producer thread
// issues every stage, so nothing here divides.
// A CTA pair's stage of two K blocks reads its rows of the 2-D maps as
// 128-row boxes: one TMA copy per 64-column chunk and stage instead of one
// per chunk and K block (an in-place convolution's patch rows stay one box
// per tap and K block, placed in the same layout).  The producer's rate is set by the
// copies it issues more than by their bytes (same bytes, the launch 4%
// shorter on the LLM layers).  Such a stage holds each chunk's 128 rows
// together, the A chunks and then the D chunks 16 KB apart (the MMA's
// leading-dimension offset), and K block j of the stage starts 64 j rows in.
// Two K blocks per stage means an even number per example (T % 128 == 0);
// the pre-scaled operand (d_rows > 0) keeps 64-row boxes.
__host__ __device__ __forceinline__ bool tall_boxes(int T, int d_rows) {
  return T % (2 * BK) == 0 && d_rows == 0;
}
// An in-place convolution whose K block is whole output rows (W_out divides
// 64) reads a stage of two K blocks as one patch box of 128 positions per
// tap: 128 / W_out output rows.
__host__ __device__ __forceinline__ bool conv_tall_box(const ConvGeom& v, int T) {
  return tall_boxes(T, 0) && v.W_out <= BK;
}

template <bool PAIR, int NB, bool CONV>
__device__ __forceinline__ void issue_stage_loads(const GemmArgs& g, int layer, uint64_t* full,
                                                  bool leader, uint32_t tx_bytes, uint8_t* sa,
                                                  uint8_t* sb, int m0, int n0, int ex, int kb,
                                                  const ConvTaps& ct, int ho0, int wo0) {
  using C = Cfg<PAIR, NB>;
  const CUtensorMap* mapA = &g.mapA[layer];
  const CUtensorMap* mapD = &g.mapD[layer];
  const int arow = ex * g.T + kb * BK;                       // row of [B*T, d]
  const int drow = g.d_rows > 0 ? arow % g.d_rows : arow;    // pre-scaled: hi and lo share D
  const int trow = kb * BK;                                  // 3-D maps: position in example
  if constexpr (PAIR) {
    // both CTAs' loads complete on the leader's full barrier
    const uint32_t fb = mapa_shared(smem_u32(full), 0);
    if (leader && tx_bytes) mbar_arrive_expect_tx(full, tx_bytes);
    if (CONV && g.conv[layer]) {
      // patch rows: one box per tap and K block, or, when the stage holds two
      // K blocks of whole output rows, one box of both (conv_tall_box); D
      // rows as 128-row boxes when the stage holds two K blocks (j: this
      // block's place in it)
      const bool tall = tall_boxes(g.T, 0);
      const int j = tall ? (kb & 1) : 0;
      uint8_t* s0 = sa - j * C::STAGE_BYTES;
      const CUtensorMap* map0 = ct.map[0] ? &g.mapS[layer][ct.map[0] - 1] : mapA;
      const CUtensorMap* map1 = ct.map[1] ? &g.mapS[layer][ct.map[1] - 1] : mapA;
      if (!conv_tall_box(g.cg[layer], g.T)) {
        tma_load_4d_pair(map0, fb, tall ? s0 + j * CHUNK : sa, ct.cc[0], wo0 + ct.dx[0],
                         ho0 + ct.dy[0], ex);
        tma_load_4d_pair(map1, fb, tall ? s0 + (2 + j) * CHUNK : sa + CHUNK, ct.cc[1],
                         wo0 + ct.dx[1], ho0 + ct.dy[1], ex);
      } else if (j == 0) {
        tma_load_4d_pair(map0, fb, s0, ct.cc[0], wo0 + ct.dx[0], ho0 + ct.dy[0], ex);
        tma_load_4d_pair(map1, fb, s0 + 2 * CHUNK, ct.cc[1], wo0 + ct.dx[1], ho0 + ct.dy[1], ex);
      }
      if (!tall) {
#pragma unroll
        for (int q = 0; q < C::B_COLS / 64; ++q)
          tma_load_2d_pair(mapD, fb, sb + q * CHUNK, n0 + 64 * q, drow);
      } else if (j == 0) {
#pragma unroll
        for (int q = 0; q < C::B_COLS / 64; ++q)
          tma_load_2d_pair(mapD, fb, s0 + 2 * C::A_STAGE + q * 2 * CHUNK, n0 + 64 * q, drow);
      }
    } else if (g.pad3d) {
      tma_load_3d_pair(mapA, fb, sa, m0, trow, ex);
      tma_load_3d_pair(mapA, fb, sa + CHUNK, m0 + 64, trow, ex);
#pragma unroll
      for (int q = 0; q < C::B_COLS / 64; ++q)
        tma_load_3d_pair(mapD, fb, sb + q * CHUNK, n0 + 64 * q, trow, ex);
    } else if (tall_boxes(g.T, g.d_rows)) {
      if ((kb & 1) == 0) {  // the stage's first K block loads both
        tma_load_2d_pair(mapA, fb, sa, m0, arow);
        tma_load_2d_pair(mapA, fb, sa + 2 * CHUNK, m0 + 64, arow);
#pragma unroll
        for (int q = 0; q < C::B_COLS / 64; ++q)
          tma_load_2d_pair(mapD, fb, sa + 2 * C::A_STAGE + q * 2 * CHUNK, n0 + 64 * q, drow);
      }
    } else {
      tma_load_2d_pair(mapA, fb, sa, m0, arow);
      tma_load_2d_pair(mapA, fb, sa + CHUNK, m0 + 64, arow);
#pragma unroll
      for (int q = 0; q < C::B_COLS / 64; ++q)
        tma_load_2d_pair(mapD, fb, sb + q * CHUNK, n0 + 64 * q, drow);
    }
  } else {
    if (tx_bytes) mbar_arrive_expect_tx(full, tx_bytes);
    if (CONV && g.conv[layer]) {
      const CUtensorMap* map0 = ct.map[0] ? &g.mapS[layer][ct.map[0] - 1] : mapA;
      const CUtensorMap* map1 = ct.map[1] ? &g.mapS[layer][ct.map[1] - 1] : mapA;
      tma_load_4d(map0, full, sa, ct.cc[0], wo0 + ct.dx[0], ho0 + ct.dy[0], ex);
      tma_load_4d(map1, full, sa + CHUNK, ct.cc[1], wo0 + ct.dx[1], ho0 + ct.dy[1], ex);
#pragma unroll
      for (int q = 0; q < C::B_COLS / 64; ++q)
        tma_load_2d(mapD, full, sb + q * CHUNK, n0 + 64 * q, drow);
    } else if (g.pad3d) {
      tma_load_3d(mapA, full, sa, m0, trow, ex);
      tma_load_3d(mapA, full, sa + CHUNK, m0 + 64, trow, ex);
#pragma unroll
      for (int q = 0; q < C::B_COLS / 64; ++q)
        tma_load_3d(mapD, full, sb + q * CHUNK, n0 + 64 * q, trow, ex);
    } else {
      tma_load_2d(mapA, full, sa, m0, arow);
      tma_load_2d(mapA, full, sa + CHUNK, m0 + 64, arow);
#pragma unroll
      for (int q = 0; q < C::B_COLS / 64; ++q)
        tma_load_2d(mapD, full, sb + q * CHUNK, n0 + 64 * q, drow);
    }
  }
}

// S[4t .. 4t+3] += s * z for the warp-uniform quad slot q in [T0, T0 + N):
// a binary tree of uniform branches down to static register indices, so the
// accumulator stays in registers and each quad costs a few branches.
template <int T0, int N, int SZ>
__device__ __forceinline__ void add_noise_slot(float (&S)[SZ], int q, float4 z, float s) {
  if constexpr (N == 1) {
    S[4 * T0 + 0] = fmaf(s, z.x, S[4 * T0 + 0]);
    S[4 * T0 + 1] = fmaf(s, z.y, S[4 * T0 + 1]);
    S[4 * T0 + 2] = fmaf(s, z.z, S[4 * T0 + 2]);
    S[4 * T0 + 3] = fmaf(s, z.w, S[4 * T0 + 3]);
  } else {
    if (q < T0 + N / 2)
      add_noise_slot<T0, N / 2, SZ>(S, q, z, s);
    else
      add_noise_slot<T0 + N / 2, N / 2, SZ>(S, q, z, s);
  }
}

// Tile t of a layer -> (m tile, n tile).  Grouped raster: groups of
// kRasterM consecutive m tiles, n runs over the whole layer inside a group
// with m fastest, so the tiles in flight at one time share an A panel of
// kRasterM tiles that stays in L2 while the D panels stream past it.
constexpr int kRasterM = 8;
// most tail tiles one launch may split (the units of a GPU of 152 SMs)
constexpr int kTailMaxTiles = 152;
__host__ __device__ __forceinline__ void tile_mn(int t, int n_m, int n_n, int& mt, int& nt) {
  const int per_group = kRasterM * n_n;
  const int grp = t / per_group;
  const int r = t - grp * per_group;
  const int gm = (n_m - grp * kRasterM) < kRasterM ? (n_m - grp * kRasterM) : kRasterM;
  mt = grp * kRasterM + r % gm;
  nt = r / gm;
}

// CONV: some layer of the launch is a convolution read in place (the
// producer forms its patch rows from 4-D boxes); the dense instantiations
// carry none of that per-stage work.
template <bool NORM, bool PAIR, int NB, bool CONV>
__global__ void __launch_bounds__(GEMM_THREADS, 1)
    k_gemm_tc(const __grid_constant__ GemmArgs g) {
  using C = Cfg<PAIR, NB>;
  constexpr int STAGES = C::STAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  __shared__ uint64_t full_bar[STAGES], empty_bar[STAGES], tfull_bar[2], tempty_bar[2], done_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_flag;
  __shared__ ConvTaps s_taps;  // the producer's current convolution taps

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = PAIR ? cluster_ctarank() : 0;
  const bool leader = rank == 0;
  const int unit = PAIR ? static_cast<int>(blockIdx.x >> 1) : static_cast<int>(blockIdx.x);
  const int n_units = PAIR ? static_cast<int>(gridDim.x >> 1) : static_cast<int>(gridDim.x);
  const int kpe = (g.T + BK - 1) / BK;  // K-blocks per example
  // CTA pairs take two K blocks per stage when an example has an even number
  // of them (a stage never straddles two examples' folds): half the barrier
  // round trips per MMA, measured faster; the stage memory is the same.
  const int bps = (PAIR && (kpe % 2) == 0) ? 2 : 1;
  const int nst = bps == 2 ? STAGES / 2 : STAGES;
  const int n_tiles = g.n_items;
  volatile int* abrt = &abort_flag;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull_bar[b], 1);
      mbar_init(&tempty_bar[b], PAIR ? 2 * NUM_EPI_WARPS : NUM_EPI_WARPS);
    }
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
  if (warp == 1) {
    if constexpr (PAIR)
      tmem_alloc_pair(&tmem_slot, C::TMEM_COLS);
    else
      tmem_alloc(&tmem_slot, C::TMEM_COLS);
  }
  tc_fence_before();
  __syncthreads();
  if constexpr (PAIR) cluster_sync();  // the peer's barriers exist before any remote arrive
  tc_fence_after();
  const uint32_t tmem_base = tmem_slot;

  if (warp < FIRST_EPI_WARP) {
    // the 256-wide tile's epilogue holds 128 accumulators per thread and
    // takes registers from the control warps; the 128-wide one fits the
    // uniform allocation
    if constexpr (NB == 256) asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(REGS_CTRL));
    if (warp == 0 && lane == 0) {
      // ---------------- TMA producer (both CTAs of a pair) ----------------
      int stage = 0;
      uint32_t phase = 0;
      uint32_t uses[STAGES] = {};
      for (int tile = unit; tile < n_tiles; tile += n_units) {
        const GemmItem w = gemm_item(g, tile);
        const int l = w.l;
        int mt, nt;
        tile_mn(w.lt, g.n_m[l], g.n_n[l], mt, nt);
        const int m0 = mt * C::TILE_M + static_cast<int>(rank) * BM;
        const int n0 = nt * NB + (PAIR ? static_cast<int>(rank) * (NB / 2) : 0);
        // convolution: the tile's taps (kept in shared memory: this warp runs
        // on few registers), and how a K block advances the output position
        // (whole rows when W_out divides 64, else 64 columns)
        int rows_per_kb = 0, wout = 1;
        if (CONV && g.conv[l]) {
          s_taps = conv_taps(g.cg[l], m0);
          wout = g.cg[l].W_out;
          rows_per_kb = wout <= BK ? BK / wout : 0;
        }
        for (int ex = w.e0; ex < w.e1; ++ex) {
          int ho0 = 0, wo0 = 0;
          for (int kb = 0; kb < kpe; kb += bps) {
            if (!mbar_wait(&empty_bar[stage], phase ^ 1, abrt, g.err)) goto producer_done;
            for (int j = 0; j < bps; ++j) {
              uint8_t* sa = smem + (stage * bps + j) * C::STAGE_BYTES;
              uint8_t* sb = sa + C::A_STAGE;
              issue_stage_loads<PAIR, NB, CONV>(g, l, &full_bar[stage], leader,
                                                j == 0 ? static_cast<uint32_t>(
                                                             bps * (PAIR ? 2 : 1) * C::STAGE_BYTES)
                                                       : 0u,
                                                sa, sb, m0, n0, ex,
                                                kb + j, s_taps, ho0, wo0);
              if constexpr (CONV) {
                if (rows_per_kb) {
                  ho0 += rows_per_kb;
                } else if (wout > 1 && (wo0 += BK) == wout) {
                  wo0 = 0;
                  ++ho0;
                }
              }
            }
            ++uses[stage];
            if (++stage == nst) {
              stage = 0;
              phase ^= 1;
            }
          }
        }
      }
    producer_done:
      // No TMA write may still be landing in shared memory when the CTA exits.
      // Completion of a stage is recorded on the leader's full barrier; a
      // peer waits instead for the leader's release of each stage it loaded.
      for (int s = 0; s < STAGES; ++s) {
        if (uses[s] == 0) continue;
        if (leader)
          drain_wait(&full_bar[s], (uses[s] - 1) & 1, g.err);
        else
          drain_wait(&empty_bar[s], (uses[s] - 1) & 1, g.err);
      }
    } else if (warp == 1 && lane == 0 && leader) {
      // ---------------- MMA issuer ----------------
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      for (int tile = unit; tile < n_tiles; tile += n_units) {
        const GemmItem w = gemm_item(g, tile);
        for (int ex = w.e0; ex < w.e1; ++ex, ++it) {
          const int buf = it & 1;
          const uint32_t tph = (it >> 1) & 1;
          if (!mbar_wait(&tempty_bar[buf], tph ^ 1, abrt, g.err)) goto mma_done;
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + buf * NB;
          const bool tall = PAIR && tall_boxes(g.T, g.d_rows);
          const uint32_t lbo = tall ? 2 * CHUNK : LBO;
          for (int kb = 0; kb < kpe; kb += bps) {
            if (!mbar_wait(&full_bar[stage], phase, abrt, g.err)) goto mma_done;
            tc_fence_after();
            for (int j = 0; j < bps; ++j) {
              const uint32_t s0 = smem_u32(smem + stage * bps * C::STAGE_BYTES);
              const uint32_t sa =
                  tall ? s0 + j * BK * 128 : smem_u32(smem + (stage * bps + j) * C::STAGE_BYTES);
              const uint32_t sb = tall ? s0 + 2 * C::A_STAGE + j * BK * 128 : sa + C::A_STAGE;
#pragma unroll
              for (int kk = 0; kk < BK / 16; ++kk) {
                const uint64_t ad = smem_desc_sw128(sa + kk * 16 * 128, lbo, SBO);
                const uint64_t bd = smem_desc_sw128(sb + kk * 16 * 128, lbo, SBO);
                if constexpr (PAIR)
                  mma_bf16_pair(d_tmem, ad, bd, C::IDESC, ((kb + j) | kk) != 0);
                else
                  mma_bf16(d_tmem, ad, bd, C::IDESC, ((kb + j) | kk) != 0);
              }
            }
            if constexpr (PAIR)
              mma_commit_pair(&empty_bar[stage]);
            else
              mma_commit(&empty_bar[stage]);
            if (++stage == nst) {
              stage = 0;
              phase ^= 1;
            }
          }
          if constexpr (PAIR)
            mma_commit_pair(&tfull_bar[buf]);
          else
            mma_commit(&tfull_bar[buf]);
        }
      }
    mma_done:
      // all issued MMAs must complete before TMEM is released (both CTAs wait)
      if constexpr (PAIR)
        mma_commit_pair(&done_bar);
      else
        mma_commit(&done_bar);
    }
  } else {
    if constexpr (NB == 256) asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(REGS_EPI));
    // ---------------- fold / epilogue warps ----------------
    const int ew = warp - FIRST_EPI_WARP;
    const int quad = warp & 3;         // TMEM lane quadrant this warp may access
    const int half = ew >> 2;          // column half of the tile
    const int row = quad * 32 + lane;  // tile row held by this thread
    const uint32_t t_lane = static_cast<uint32_t>(quad * 32) << 16;
    int it = 0;
    // The tile's noise (QPT groups of 4 per thread) is generated in slices
    // of qpe groups while the tensor core works on each example and added
    // into the register accumulator (sum and noise commute), so the tile end
    // only scales and stores.
    constexpr int QPT = C::HALF / 4;
    const int qpe = (QPT + g.B - 1) / g.B;
    const uint64_t seed = g.add_noise ? g.key[0] : 0, step = g.add_noise ? g.key[1] : 0;
    for (int tile = unit; tile < n_tiles; tile += n_units) {
      const GemmItem w = gemm_item(g, tile);
      const int l = w.l, lt = w.lt;
      const int d_in = g.d_in[l], d_out = g.d_out[l];
      // a split tile or a tail piece stores its partial sum unscaled and
      // without noise; the reduce pass adds the ranges in order, then the noise
      const bool part_out = g.split[l] > 1 || w.z >= 0;
      int mt, nt;
      tile_mn(lt, g.n_m[l], g.n_n[l], mt, nt);
      const int m0 = mt * C::TILE_M + static_cast<int>(rank) * BM;
      const int n0 = nt * NB;
      const int j = m0 + row;
      const int k0 = n0 + half * C::HALF;
      const uint64_t prow = g.p_base[l] + static_cast<uint64_t>(j) * d_out;
      float S[C::HALF];
      if constexpr (!NORM) {
#pragma unroll
        for (int i = 0; i < C::HALF; ++i) S[i] = 0.f;
      }
      for (int ex = w.e0; ex < w.e1; ++ex, ++it) {
        if constexpr (!NORM) {
          if (g.add_noise && !part_out && j < d_in) {
            const int q_lo = ex * qpe;
            const int q_hi = q_lo + qpe < QPT ? q_lo + qpe : QPT;
#pragma unroll 1
            for (int q = q_lo; q < q_hi; ++q) {
              // d_out is a multiple of 8 on this path, so the four parameters
              // prow+k .. +3 sit in one output row; they form one Philox quad
              // when p_base is a multiple of 4, else they straddle two (a
              // layer after one whose size is not a multiple of 4)
              if (k0 + 4 * q >= d_out) break;
              const float4 z = gauss4_at<Root::kSqrt>(seed, step, prow + k0 + 4 * q);
              add_noise_slot<0, QPT, C::HALF>(S, q, z, g.sigmaC);
            }
          }
        }
        const int buf = it & 1;
        const uint32_t tph = (it >> 1) & 1;
        if (!mbar_wait(&tfull_bar[buf], tph, abrt, g.err)) goto epi_done;
        tc_fence_after();
        const uint32_t tcol = t_lane + buf * NB + half * C::HALF;
        float sq = 0.f;
        const float ci = NORM ? 0.f : (g.c ? g.c[ex] : 1.f);
#pragma unroll
        for (int ch = 0; ch < C::HALF / 64; ++ch) {
          uint32_t v[64];
          tmem_ld64(tmem_base + tcol + ch * 64, v);
#pragma unroll
          for (int i = 0; i < 64; ++i) {
            const float x = __uint_as_float(v[i]);
            if constexpr (NORM)
              sq = fmaf(x, x, sq);
            else
              S[ch * 64 + i] = fmaf(ci, x, S[ch * 64 + i]);
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if constexpr (PAIR)
            mbar_arrive_cluster(mapa_shared(smem_u32(&tempty_bar[buf]), 0));
          else
            mbar_arrive(&tempty_bar[buf]);
        }
        if constexpr (NORM) {
          // one partial per epilogue warp; the clip kernel sums them in order
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
          if (lane == 0)
            g.part[static_cast<int64_t>(g.row0 + ex) * g.NP +
                   (lt * (PAIR ? 2 : 1) + static_cast<int>(rank)) * NUM_EPI_WARPS + ew] = sq;
        }
      }
      if constexpr (!NORM) {
        // Store through shared memory: 4 rounds of a 32 x 32 block per warp
        // (rows of this warp's lane quadrant, 32 columns), written with the
        // 128-byte swizzle the output tensor map uses, then sent by one TMA
        // store (or reduce-add) that clips at the tensor bounds.
        uint8_t* stg = smem + C::STAGING + ew * 4096;
        const int y = m0 + quad * 32;
#pragma unroll
        for (int c4 = 0; c4 < C::HALF / 32; ++c4) {
          if (lane == 0) bulk_wait_read_all();  // previous block has been read
          __syncwarp();
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const float sc = part_out ? 1.f : g.out_scale;
            float4 v;
            v.x = sc * S[32 * c4 + 4 * k + 0];
            v.y = sc * S[32 * c4 + 4 * k + 1];
            v.z = sc * S[32 * c4 + 4 * k + 2];
            v.w = sc * S[32 * c4 + 4 * k + 3];
            *reinterpret_cast<float4*>(stg + lane * 128 + ((k ^ (lane & 7)) << 4)) = v;
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            if (w.z >= 0)
              tma_store_3d(&g.mapT, stg, k0 - n0 + 32 * c4, y - mt * C::TILE_M, w.z);
            else if (part_out)
              tma_store_3d(&g.mapO[l], stg, k0 + 32 * c4, y, w.s);
            else if (g.accumulate)
              tma_reduce_add_2d(&g.mapO[l], stg, k0 + 32 * c4, y);
            else
              tma_store_2d(&g.mapO[l], stg, k0 + 32 * c4, y);
            bulk_commit_group();
          }
        }
      }
    }
  epi_done:
    if constexpr (!NORM) {
      if (lane == 0) bulk_wait_all();  // every output write performed before exit
    }
  }

  tc_fence_before();
  __syncthreads();
  if constexpr (PAIR) cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    // the leader's last commit tells both CTAs that no MMA still writes TMEM
    if (lane == 0) drain_wait(&done_bar, 0, g.err);
    __syncwarp();
    if constexpr (PAIR)
      tmem_dealloc_pair(tmem_base, C::TMEM_COLS);
    else
      tmem_dealloc(tmem_base, C::TMEM_COLS);
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

// 3D bf16 map over [B][T][cols], box {64 cols, box_rows positions, 1 example}:
// positions t >= T of an example read as zeros.
bool make_map_3d(CUtensorMap* m, const void* base, uint64_t cols, uint64_t T, uint64_t B,
                 uint32_t box_rows) {
  const uint64_t dims[3] = {cols, T, B};
  const uint64_t strides[2] = {cols * 2, T * cols * 2};
  const uint32_t box[3] = {64, box_rows, 1};
  return make_tma_bf16(m, base, 3, dims, strides, box);
}

// CTA pairs for every layer wider than one 128-row tile.
bool use_pair(int64_t d_in) { return d_in > BM; }
// Tile width: 128 columns for layers with d_out <= 128, else 256.
int gemm_nb(int64_t d_out) { return d_out <= 128 ? 128 : BN; }

template <bool NORM, bool PAIR, int NB, bool CONV>
cudaError_t launch_gemm(GemmArgs& g, cudaStream_t s, float* tail = nullptr,
                        int64_t tail_cap = 0) {
  using C = Cfg<PAIR, NB>;
  cudaError_t e = setup_once_per_device(
      reinterpret_cast<const void*>(&k_gemm_tc<NORM, PAIR, NB, CONV>), []() -> cudaError_t {
        cudaError_t r = cudaFuncSetAttribute(k_gemm_tc<NORM, PAIR, NB, CONV>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             C::SMEM_BYTES);
        if (r != cudaSuccess) return r;
        if constexpr (NB == 256) {
          // setmaxnreg moves registers within what the block was launched with:
          // the split must fit the compiled count, else the raise never returns
          cudaFuncAttributes fa{};
          r = cudaFuncGetAttributes(&fa, k_gemm_tc<NORM, PAIR, NB, CONV>);
          if (r != cudaSuccess) return r;
          if (fa.numRegs * GEMM_THREADS < 4 * 32 * REGS_CTRL + NUM_EPI_WARPS * 32 * REGS_EPI ||
              fa.numRegs > REGS_EPI)
            return cudaErrorInvalidConfiguration;
        }
        return cudaSuccess;
      });
  if (e != cudaSuccess) return e;
  const int sms = device_sm_count();
  // whole tiles and tail pieces of every layer (a tail needs tail_split >= 2
  // on an unsplit layer; the norm kernel plans its own below)
  auto count_items = [&]() -> bool {
    g.tile_start[0] = 0;
    g.piece_start[0] = 0;
    for (int l = 0; l < g.L; ++l) {
      g.n_m[l] = (g.d_in[l] + C::TILE_M - 1) / C::TILE_M;
      g.n_n[l] = (g.d_out[l] + NB - 1) / NB;
      if (g.split[l] < 1) g.split[l] = 1;
      const int tl = g.n_m[l] * g.n_n[l];
      int whole = tl * g.split[l], pieces = 0;
      if (g.tail_split[l] >= 2) {
        if (g.split[l] != 1 || g.tail_from[l] < 0 || g.tail_from[l] >= tl ||
            g.tail_split[l] > g.B || g.d_rows > 0)
          return false;
        whole = g.tail_from[l];
        pieces = (tl - g.tail_from[l]) * g.tail_split[l];
      } else {
        g.tail_from[l] = tl;
        g.tail_split[l] = 1;
      }
      g.tile_start[l + 1] = g.tile_start[l] + whole;
      g.piece_start[l + 1] = g.piece_start[l] + pieces;
    }
    g.n_items = g.tile_start[g.L] + g.piece_start[g.L];
    return true;
  };
  if (!count_items()) return cudaErrorInvalidValue;
  if constexpr (NORM) {
    // a norm launch (one layer) splits its own last round: a piece's
    // examples keep their partial slots, so the result does not change
    auto plan_norm_tail = [&](int units) {
      const int tiles = g.tile_start[1];
      const int r = tiles % units;
      if (g.L != 1 || g.split[0] != 1 || tiles <= units || r == 0 || g.d_rows > 0) return;
      int S = units / r;
      if (S > g.B) S = g.B;
      if (S < 2) return;
      g.tail_from[0] = tiles - r;
      g.tail_split[0] = S;
      count_items();
    };
    plan_norm_tail(PAIR ? sms / 2 : sms);
  } else if (g.piece_start[g.L] > 0) {
    const int64_t bytes = static_cast<int64_t>(g.piece_start[g.L]) * C::TILE_M * NB * 4;
    if (!tail || (reinterpret_cast<uintptr_t>(tail) & 15) != 0 || bytes > tail_cap ||
        !make_tma_f32_split(&g.mapT, tail, g.piece_start[g.L], C::TILE_M, NB))
      return cudaErrorInvalidValue;
  }
  const int tiles = g.n_items;
  if constexpr (PAIR) {
    // persistent grid: as many pairs as can be resident at once
    cudaLaunchConfig_t cfg = {};
    cfg.blockDim = dim3(GEMM_THREADS);
    cfg.dynamicSmemBytes = C::SMEM_BYTES;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const int max_pairs =
        cached_per_device(reinterpret_cast<const void*>(&k_gemm_tc<NORM, PAIR, NB, CONV>), [&] {
          cudaLaunchConfig_t q = cfg;
          q.gridDim = dim3(sms);
          int n = 0;
          if (cudaOccupancyMaxActiveClusters(&n, k_gemm_tc<NORM, PAIR, NB, CONV>, &q) !=
                  cudaSuccess ||
              n < 1) {
            cudaGetLastError();
            n = sms / 2;
          }
          return n < sms / 2 ? n : sms / 2;
        });
    const int pairs = tiles < max_pairs ? tiles : max_pairs;
    cfg.gridDim = dim3(2 * pairs);
    note_launch();
    return cudaLaunchKernelEx(&cfg, k_gemm_tc<NORM, PAIR, NB, CONV>, g);
  } else {
    const int grid = tiles < sms ? tiles : sms;
    note_launch();
    k_gemm_tc<NORM, PAIR, NB, CONV><<<grid, GEMM_THREADS, C::SMEM_BYTES, s>>>(g);
    return cudaGetLastError();
  }
}

// Maps over the caller's [B][T][d] arrays of layer slot l: 2-D [B*T, d] when
// T is a multiple of the K block, else 3-D with each example's positions
// padded to it.
bool make_input_maps(const void* A, const void* D, GemmArgs& g, int l,
                     const ConvGeom* conv = nullptr) {
  g.pad3d = (g.T % BK) != 0;
  g.conv[l] = 0;
  if (conv) {
    // the NHWC input [B][H][W][C_in]; a box is 64 output positions of one
    // tap: whole output rows when W_out divides 64, else a run of 64 in a row
    if (!tc_conv_implicit_ok(*conv, g.T)) return false;
    const ConvGeom& v = *conv;
    g.conv[l] = 1;
    g.cg[l] = v;
    const uint64_t c = static_cast<uint64_t>(v.C_in);
    const uint32_t rows = v.W_out <= BK ? static_cast<uint32_t>(
                                              (conv_tall_box(v, g.T) ? 2 * BK : BK) / v.W_out)
                                        : 1u;
    const uint32_t cols = v.W_out <= BK ? static_cast<uint32_t>(v.W_out) : static_cast<uint32_t>(BK);
    const uint32_t box[4] = {64, cols, rows, 1};
    // one map per parity (ry, rx) of the stride s: the pixels (s i + ry,
    // s j + rx), i.e. the input from pixel (ry, rx) on with s times its
    // row and pixel strides (s = 1: the input itself)
    const int s = v.stride_h;
    for (int ry = 0; ry < s; ++ry)
      for (int rx = 0; rx < s; ++rx) {
        const uint64_t dims[4] = {c, static_cast<uint64_t>((v.W - rx + s - 1) / s),
                                  static_cast<uint64_t>((v.H - ry + s - 1) / s),
                                  static_cast<uint64_t>(g.B)};
        const uint64_t strides[3] = {c * 2 * s, c * v.W * 2 * s, c * v.W * v.H * 2};
        const void* base =
            static_cast<const __nv_bfloat16*>(A) + (static_cast<uint64_t>(ry) * v.W + rx) * c;
        const int k = ry * s + rx;
        if (!make_tma_bf16(k == 0 ? &g.mapA[l] : &g.mapS[l][k - 1], base, 4, dims, strides, box))
          return false;
      }
    const uint64_t rows_all = static_cast<uint64_t>(g.B) * g.T;
    return make_map_2d(&g.mapD[l], D, g.d_out[l], rows_all, tall_boxes(g.T, 0) ? 2 * BK : BK);
  }
  if (g.pad3d)
    return make_map_3d(&g.mapA[l], A, g.d_in[l], g.T, g.B, BK) &&
           make_map_3d(&g.mapD[l], D, g.d_out[l], g.T, g.B, BK);
  const uint64_t rows = static_cast<uint64_t>(g.B) * g.T;
  const uint32_t br = (use_pair(g.d_in[l]) && tall_boxes(g.T, 0)) ? 2 * BK : BK;  // tall_boxes
  return make_map_2d(&g.mapA[l], A, g.d_in[l], rows, br) &&
         make_map_2d(&g.mapD[l], D, g.d_out[l], rows, br);
}

template <bool NORM>
cudaError_t launch_any(GemmArgs& g, cudaStream_t s, float* tail = nullptr, int64_t tail_cap = 0) {
  // every layer of a launch shares the tile shape (use_pair, gemm_nb); a
  // convolution read in place always has pairs (tc_conv_implicit_ok)
  bool conv = false;
  for (int l = 0; l < g.L; ++l) conv = conv || g.conv[l];
  const bool pair = use_pair(g.d_in[0]);
  if (conv && !pair) return cudaErrorInvalidValue;
  if (gemm_nb(g.d_out[0]) == 128) {
    if (conv) return launch_gemm<NORM, true, 128, true>(g, s, tail, tail_cap);
    return pair ? launch_gemm<NORM, true, 128, false>(g, s, tail, tail_cap)
                : launch_gemm<NORM, false, 128, false>(g, s, tail, tail_cap);
  }
  if (conv) return launch_gemm<NORM, true, BN, true>(g, s, tail, tail_cap);
  return pair ? launch_gemm<NORM, true, BN, false>(g, s, tail, tail_cap)
              : launch_gemm<NORM, false, BN, false>(g, s, tail, tail_cap);
}

void set_epilogue(GemmArgs& g, const Epilogue& ep) {
  g.key = ep.key;
  g.out_scale = ep.out_scale;
  g.sigmaC = ep.sigmaC;
  g.add_noise = ep.add_noise;
  g.accumulate = ep.accumulate;
}

// Pre-scaled operand for short examples: rows [0, R) of A2 hold
// hi = RN_bf16(c_i a) and rows [R, 2R) hold lo = RN_bf16(c_i a - hi) for the
// B*T input rows (zeros in the padding rows), so hi + lo carries c_i a to
// about 2^-16 relative and S = A2^T [D; D] needs no per-example fold.
// IDX: the type of the vector index (32-bit when the 2 R d_in / 8 vectors
// fit, so that the row and column come from a 32-bit division).
template <typename IDX>
__global__ void k_prescale_hilo(const __nv_bfloat16* __restrict__ A, const float* __restrict__ c,
                                int T, int64_t BT, int64_t R, int d_in,
                                __nv_bfloat16* __restrict__ A2) {
  const IDX vpr = static_cast<IDX>(d_in / 8);  // 16-byte vectors per row
  const IDX nvec = static_cast<IDX>(2 * R) * vpr;
  for (IDX v = static_cast<IDX>(blockIdx.x) * blockDim.x + threadIdx.x; v < nvec;
       v += static_cast<IDX>(gridDim.x) * blockDim.x) {
    const int64_t row = static_cast<int64_t>(v / vpr);
    const int col = static_cast<int>(v % vpr) * 8;
    const bool lo = row >= R;
    const int64_t k = lo ? row - R : row;
    uint4 outv = make_uint4(0u, 0u, 0u, 0u);
    if (k < BT) {
      // k < B T <= 2^31 - 1
      const float ci = c[static_cast<uint32_t>(k) / static_cast<uint32_t>(T)];
      const uint4 in = *reinterpret_cast<const uint4*>(A + k * d_in + col);
      const __nv_bfloat16* x = reinterpret_cast<const __nv_bfloat16*>(&in);
      __nv_bfloat16 y[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const float p = ci * __bfloat162float(x[u]);
        const __nv_bfloat16 h = __float2bfloat16_rn(p);
        y[u] = lo ? __float2bfloat16_rn(p - __bfloat162float(h)) : h;
      }
      outv = *reinterpret_cast<const uint4*>(y);
    }
    *reinterpret_cast<uint4*>(A2 + row * d_in + col) = outv;
  }
}

int64_t prescale_rows(int B, int T) { return ((static_cast<int64_t>(B) * T + BK - 1) / BK) * BK; }

// out = out_scale (sum over ranges s of part[s] + sigma C z) for the split
// layers of a launch, one thread per 4 consecutive parameters, the ranges
// added in order.  On the tensor-core path d_in * d_out is a multiple of 64,
// so every group of 4 is whole and 16-byte aligned; its noise is one Philox
// quad, or two when p_base is not a multiple of 4.
struct SplitReduceLayer {
  const float* part;
  float* out;
  int64_t count;    // d_in * d_out
  uint64_t p_base;  // global parameter index of element 0
  int64_t q0;       // first thread of this layer in the launch
  int split;
};
struct SplitReduceBatch {
  SplitReduceLayer l[kGemmMaxLayers];
  int L;
  const uint64_t* key;
  float out_scale, sigmaC;
  int add_noise, accumulate;
};

__global__ void __launch_bounds__(256) k_split_reduce(const __grid_constant__ SplitReduceBatch g) {
  const int64_t q = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  int l = 0;
  while (l + 1 < g.L && q >= g.l[l + 1].q0) ++l;
  const SplitReduceLayer& P = g.l[l];
  const int64_t e = (q - P.q0) * 4;
  if (q < P.q0 || e >= P.count) return;
  float4 s = __ldcs(reinterpret_cast<const float4*>(P.part + e));
  for (int k = 1; k < P.split; ++k) {
    const float4 v = __ldcs(reinterpret_cast<const float4*>(P.part + k * P.count + e));
    s.x += v.x;
    s.y += v.y;
    s.z += v.z;
    s.w += v.w;
  }
  float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
  if (g.add_noise) z = gauss4_at(g.key[0], g.key[1], P.p_base + e);
  float4 v;
  v.x = g.out_scale * fmaf(g.sigmaC, z.x, s.x);
  v.y = g.out_scale * fmaf(g.sigmaC, z.y, s.y);
  v.z = g.out_scale * fmaf(g.sigmaC, z.z, s.z);
  v.w = g.out_scale * fmaf(g.sigmaC, z.w, s.w);
  float4* o = reinterpret_cast<float4*>(P.out + e);
  if (g.accumulate) {
    const float4 a = *o;
    v.x += a.x;
    v.y += a.y;
    v.z += a.z;
    v.w += a.w;
  }
  *o = v;
}

// The tail pieces of one clipped-sum launch: for each tail tile its partial
// tiles added in example order, then the noise, the output scale and the
// store (or add) into the layer's output, as for a split layer.
struct TailReduceArgs {
  const float* tail;  // [pieces][tile_m][nb]
  float* out[kGemmMaxLayers];
  uint64_t p_base[kGemmMaxLayers];
  int d_in[kGemmMaxLayers], d_out[kGemmMaxLayers];
  // per tail tile: its layer and origin, and its pieces first, first +
  // stride, ... (count of them, in example order)
  int layer[kTailMaxTiles], row0[kTailMaxTiles], col0[kTailMaxTiles];
  int first[kTailMaxTiles], stride[kTailMaxTiles], count[kTailMaxTiles];
  int n, tile_m, nb;
  const uint64_t* key;
  float out_scale, sigmaC;
  int add_noise, accumulate;
};

__global__ void __launch_bounds__(256) k_tail_reduce(const __grid_constant__ TailReduceArgs g) {
  const int per_row = g.nb / 4;
  const int per_tile = g.tile_m * per_row;
  const int64_t q = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (q >= static_cast<int64_t>(g.n) * per_tile) return;
  const int t = static_cast<int>(q / per_tile);
  const int r = static_cast<int>(q - static_cast<int64_t>(t) * per_tile);
  const int row = r / per_row, col = (r - row * per_row) * 4;
  const int l = g.layer[t];
  const int j = g.row0[t] + row, k = g.col0[t] + col;
  if (j >= g.d_in[l] || k >= g.d_out[l]) return;  // d_out is a multiple of 8
  const int64_t tile_elems = static_cast<int64_t>(g.tile_m) * g.nb;
  const float* src =
      g.tail + g.first[t] * tile_elems + static_cast<int64_t>(row) * g.nb + col;
  const int64_t step = g.stride[t] * tile_elems;
  float4 s = __ldcs(reinterpret_cast<const float4*>(src));
  for (int p = 1; p < g.count[t]; ++p) {
    const float4 v = __ldcs(reinterpret_cast<const float4*>(src + p * step));
    s.x += v.x;
    s.y += v.y;
    s.z += v.z;
    s.w += v.w;
  }
  const uint64_t e = static_cast<uint64_t>(j) * g.d_out[l] + k;
  float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
  if (g.add_noise) z = gauss4_at<Root::kSqrt>(g.key[0], g.key[1], g.p_base[l] + e);
  float4 v;
  v.x = g.out_scale * fmaf(g.sigmaC, z.x, s.x);
  v.y = g.out_scale * fmaf(g.sigmaC, z.y, s.y);
  v.z = g.out_scale * fmaf(g.sigmaC, z.z, s.z);
  v.w = g.out_scale * fmaf(g.sigmaC, z.w, s.w);
  float4* o = reinterpret_cast<float4*>(g.out[l] + e);
  if (g.accumulate) {
    const float4 a = *o;
    v.x += a.x;
    v.y += a.y;
    v.z += a.z;
    v.w += a.w;
  }
  *o = v;
}

}  // namespace

// Example ranges per tile of a layer's clipped sum or materialised norm.  A
// layer with fewer tiles than the GPU has units splits its batch into S
// ranges, S chosen to fill whole rounds of the units (the largest fraction
// tiles*S / (rounds * units), the smallest S on a tie), each range keeping
// at least 8 K-blocks of work.  S depends only on the layer's own shape (and
// the device's SM count), so a layer rounds the same in a batched launch and
// in a launch of its own.
int64_t tc_gemm_tiles(int64_t d_in, int64_t d_out) {
  const int64_t tile_m = use_pair(d_in) ? 2 * BM : BM;
  const int64_t nb = gemm_nb(d_out);
  return ((d_in + tile_m - 1) / tile_m) * ((d_out + nb - 1) / nb);
}

// Example ranges per tile.  A launch whose tiles (this layer's and the
// other_tiles of the layers sharing it) already give every unit a tile runs
// unsplit: a split writes and re-reads S partial tiles, which costs more
// than the partly empty last round it saves.  Otherwise S fills whole
// rounds: the count with the largest items / (rounds x units), the smallest
// on a tie, at least 8 K-blocks per range, at most 256.
int tc_gemm_split(int B, int T, int64_t d_in, int64_t d_out, int64_t other_tiles) {
  const bool pair = use_pair(d_in);
  const int64_t tiles = tc_gemm_tiles(d_in, d_out);
  const int64_t units = pair ? device_sm_count() / 2 : device_sm_count();
  if (tiles + other_tiles >= units || B < 2) return 1;
  const int64_t kpe = (T + BK - 1) / BK;
  int64_t smax = static_cast<int64_t>(B) * kpe / 8;
  if (smax > B) smax = B;
  if (smax > kGemmMaxSplit) smax = kGemmMaxSplit;
  int64_t best = 1;
  double best_eff = 0.0;
  for (int64_t S = 1; S <= smax; ++S) {
    const int64_t items = tiles * S + other_tiles;
    const int64_t rounds = (items + units - 1) / units;
    const double eff = static_cast<double>(items) / static_cast<double>(rounds * units);
    if (eff > best_eff + 1e-9) {
      best_eff = eff;
      best = S;
    }
  }
  return static_cast<int>(best);
}

// Patch rows on the fly: 64-channel chunks never straddle a tap (C_in a
// multiple of 64), K blocks are whole boxes of output positions (T a
// multiple of 64, W_out dividing 64 or 64 dividing W_out), stride 1 or 2 in
// both directions (a stride-2 tap reads one of four parity maps).
bool tc_conv_implicit_ok(const ConvGeom& g, int T) {
  if (g.C_in % 64 != 0 || T % BK != 0 || T != g.H_out * g.W_out) return false;
  if (!use_pair(static_cast<int64_t>(g.kh) * g.kw * g.C_in)) return false;
  // unit stride, or stride 2 in both directions (four parity maps)
  if (g.stride_h != g.stride_w || g.stride_h < 1 || g.stride_h > 2) return false;
  if (g.H < g.stride_h || g.W < g.stride_w) return false;
  if (g.W_out <= BK) return BK % g.W_out == 0;
  return g.W_out % BK == 0;
}

// Direct path: T a multiple of 64, or T >= 32 (3-D padding wastes at most half).
// (an example's product accumulates over its T positions in TMEM: T <= kTcMaxAccum)
bool tc_gemm_supported(int T, int64_t d_in, int64_t d_out) {
  return (T % BK == 0 || T >= 32) && T <= kTcMaxAccum && d_in % 8 == 0 && d_out % 8 == 0 &&
         tma_encode_available();
}

// (the whole batch, 2 B T rows of hi + lo, accumulates in one TMEM tile)
bool tc_prescaled_supported(int B, int T, int64_t d_in, int64_t d_out) {
  return T <= kPrescaleMaxT && 2 * prescale_rows(B, T) <= kTcMaxAccum && d_in % 8 == 0 &&
         d_out % 8 == 0 && tma_encode_available();
}

int64_t tc_prescaled_scratch_bytes(int B, int T, int64_t d_in) {
  return 2 * prescale_rows(B, T) * d_in * 2;
}

cudaError_t tc_launch_clipsum_prescaled(const void* A, const void* D, const float* c, int B,
                                        int T, int d_in, int d_out, float* out,
                                        const Epilogue& ep, int* err, void* scratch,
                                        cudaStream_t s) {
  const int64_t BT = static_cast<int64_t>(B) * T;
  const int64_t R = prescale_rows(B, T);
  auto* A2 = static_cast<__nv_bfloat16*>(scratch);
  const int64_t nvec = 2 * R * (d_in / 8);
  int64_t blocks = (nvec + 255) / 256;
  const int64_t cap = static_cast<int64_t>(device_sm_count()) * 8;
  note_launch();
  if (blocks > cap) blocks = cap;
  // 32-bit indices while v + the grid's stride stays below 2^32
  if (nvec + blocks * 256 < (int64_t(1) << 32))
    k_prescale_hilo<uint32_t><<<static_cast<int>(blocks), 256, 0, s>>>(
        static_cast<const __nv_bfloat16*>(A), c, T, BT, R, d_in, A2);
  else
    k_prescale_hilo<uint64_t><<<static_cast<int>(blocks), 256, 0, s>>>(
        static_cast<const __nv_bfloat16*>(A), c, T, BT, R, d_in, A2);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  GemmArgs g{};
  g.L = 1;
  g.c = nullptr;  // clip factors already applied
  g.out[0] = out;
  g.p_base[0] = ep.p_base;
  g.err = err;
  g.B = 1;
  g.T = static_cast<int>(2 * R);
  g.d_in[0] = d_in;
  g.d_out[0] = d_out;
  g.d_rows = static_cast<int>(R);
  set_epilogue(g, ep);
  if (!make_map_2d(&g.mapA[0], A2, d_in, 2 * R, BK) || !make_map_2d(&g.mapD[0], D, d_out, BT, BK) ||
      !make_tma_f32_out(&g.mapO[0], out, d_in, d_out))
    return cudaErrorInvalidValue;
  g.pad3d = 0;
  return launch_any<false>(g, s);
}

int64_t tc_mat_parts(int64_t d_in, int64_t d_out) {
  const int64_t tile_m = use_pair(d_in) ? 2 * BM : BM;
  const int64_t ctas_per_tile = use_pair(d_in) ? 2 : 1;
  const int64_t nb = gemm_nb(d_out);
  return ((d_in + tile_m - 1) / tile_m) * ((d_out + nb - 1) / nb) * ctas_per_tile *
         NUM_EPI_WARPS;
}

cudaError_t tc_launch_mat_norm(const void* A, const void* D, int B, int T, int d_in, int d_out,
                               float* part, int NP, int row0, int* err, cudaStream_t s,
                               const ConvGeom* conv) {
  GemmArgs g{};
  g.L = 1;
  g.part = part;
  g.err = err;
  g.B = B;
  g.T = T;
  g.d_in[0] = d_in;
  g.d_out[0] = d_out;
  g.split[0] = tc_gemm_split(B, T, d_in, d_out);
  g.NP = NP;
  g.row0 = row0;
  if (!make_input_maps(A, D, g, 0, conv)) return cudaErrorInvalidValue;
  return launch_any<true>(g, s);
}

cudaError_t tc_launch_clipsum_batch(int L, const void* const* A, const void* const* D,
                                    float* const* out, float* const* part, const int* d_in,
                                    const int* d_out, const uint64_t* p_base, const int* split,
                                    const float* c, int B, int T, const Epilogue& ep, int* err,
                                    cudaStream_t s, const ConvGeom* const* conv,
                                    const int* tail_from, const int* tail_split, float* tail,
                                    int64_t tail_bytes) {
  if (L < 1 || L > kGemmMaxLayers) return cudaErrorInvalidValue;
  const bool pair = use_pair(d_in[0]);
  const int nb = gemm_nb(d_out[0]);
  const int tile_m = pair ? 2 * BM : BM;
  // the planned tails' pieces must fit the scratch: else one launch per layer
  // (a layer's pieces always fit; the bits do not depend on the grouping)
  if (tail_split && L > 1) {
    int64_t pieces = 0;
    for (int l = 0; l < L; ++l)
      if (tail_split[l] >= 2)
        pieces += (tc_gemm_tiles(d_in[l], d_out[l]) - tail_from[l]) * tail_split[l];
    if (pieces * tile_m * nb * 4 > tail_bytes) {
      for (int l = 0; l < L; ++l) {
        cudaError_t e = tc_launch_clipsum_batch(
            1, A + l, D + l, out + l, part ? part + l : nullptr, d_in + l, d_out + l, p_base + l,
            split ? split + l : nullptr, c, B, T, ep, err, s, conv ? conv + l : nullptr,
            tail_from + l, tail_split + l, tail, tail_bytes);
        if (e != cudaSuccess) return e;
      }
      return cudaSuccess;
    }
  }
  GemmArgs g{};
  g.L = L;
  g.c = c;
  g.err = err;
  g.B = B;
  g.T = T;
  set_epilogue(g, ep);
  SplitReduceBatch r{};
  int64_t threads = 0;
  for (int l = 0; l < L; ++l) {
    // the caller groups layers by tile shape
    if (use_pair(d_in[l]) != pair || gemm_nb(d_out[l]) != nb) return cudaErrorInvalidValue;
    g.d_in[l] = d_in[l];
    g.d_out[l] = d_out[l];
    g.out[l] = out[l];
    g.p_base[l] = p_base[l];
    g.split[l] = split ? split[l] : tc_gemm_split(B, T, d_in[l], d_out[l]);
    if (g.split[l] < 1 || g.split[l] > kGemmMaxSplit) return cudaErrorInvalidValue;
    if (tail_split && tail_split[l] >= 2) {
      g.tail_from[l] = tail_from[l];
      g.tail_split[l] = tail_split[l];
    }
    if (!make_input_maps(A[l], D[l], g, l, conv ? conv[l] : nullptr)) return cudaErrorInvalidValue;
    if (g.split[l] > 1) {
      if (!part || !part[l] || (reinterpret_cast<uintptr_t>(part[l]) & 15) != 0 ||
          !make_tma_f32_split(&g.mapO[l], part[l], g.split[l], d_in[l], d_out[l]))
        return cudaErrorInvalidValue;
      SplitReduceLayer& R = r.l[r.L++];
      R.part = part[l];
      R.out = out[l];
      R.count = static_cast<int64_t>(d_in[l]) * d_out[l];
      R.p_base = p_base[l];
      R.q0 = threads;
      R.split = g.split[l];
      threads += R.count / 4;
    } else if (!make_tma_f32_out(&g.mapO[l], out[l], d_in[l], d_out[l])) {
      return cudaErrorInvalidValue;
    }
  }
  cudaError_t e = launch_any<false>(g, s, tail, tail_bytes);
  if (e != cudaSuccess) return e;
  if (g.piece_start[L] > 0) {
    TailReduceArgs t{};
    t.tail = tail;
    t.tile_m = tile_m;
    t.nb = nb;
    for (int l = 0; l < L; ++l) {
      t.out[l] = out[l];
      t.p_base[l] = p_base[l];
      t.d_in[l] = d_in[l];
      t.d_out[l] = d_out[l];
      const int tl = g.n_m[l] * g.n_n[l];
      const int n = tl - g.tail_from[l];
      for (int q = 0; q < n && g.tail_split[l] >= 2; ++q) {
        if (t.n == kTailMaxTiles) return cudaErrorInvalidValue;
        int mt, nt;
        tile_mn(g.tail_from[l] + q, g.n_m[l], g.n_n[l], mt, nt);
        t.layer[t.n] = l;
        t.row0[t.n] = mt * tile_m;
        t.col0[t.n] = nt * nb;
        t.first[t.n] = g.piece_start[l] + q;
        t.stride[t.n] = n;
        t.count[t.n] = g.tail_split[l];
        ++t.n;
      }
    }
    t.key = ep.key;
    t.out_scale = ep.out_scale;
    t.sigmaC = ep.sigmaC;
    t.add_noise = ep.add_noise;
    t.accumulate = ep.accumulate;
    const int64_t nthreads = static_cast<int64_t>(t.n) * tile_m * nb / 4;
    note_launch();
    k_tail_reduce<<<static_cast<int>((nthreads + 255) / 256), 256, 0, s>>>(t);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  if (r.L == 0) return cudaSuccess;
  r.key = ep.key;
  r.out_scale = ep.out_scale;
  r.sigmaC = ep.sigmaC;
  r.add_noise = ep.add_noise;
  r.accumulate = ep.accumulate;
  note_launch();
  k_split_reduce<<<static_cast<int>((threads + 255) / 256), 256, 0, s>>>(r);
  return cudaGetLastError();
}

cudaError_t tc_launch_clipsum(const void* A, const void* D, const float* c, int B, int T,
                              int d_in, int d_out, int split, float* out, float* part,
                              const Epilogue& ep, int* err, cudaStream_t s, const ConvGeom* conv,
                              int tail_from, int tail_split, float* tail, int64_t tail_bytes) {
  return tc_launch_clipsum_batch(1, &A, &D, &out, &part, &d_in, &d_out, &ep.p_base, &split, c, B,
                                 T, ep, err, s, &conv, &tail_from, &tail_split, tail, tail_bytes);
}

// Tail of a launch group of clipped sums (the layers that share one batched
// launch, in order, unsplit): with tiles > units and r = tiles mod units,
// the last r tiles become r * S pieces, S = min(units / r, B) >= 2, so the
// last round fills the units.  Returns, per layer, the first tail tile
// (tiles: none) and S (1: none).
void tc_plan_tail(int L, const int64_t* d_in, const int64_t* d_out, int B, int* tail_from,
                  int* tail_split) {
  int64_t tiles = 0;
  for (int l = 0; l < L; ++l) {
    tail_from[l] = static_cast<int>(tc_gemm_tiles(d_in[l], d_out[l]));
    tail_split[l] = 1;
    tiles += tail_from[l];
  }
  if (L < 1) return;
  const int64_t units = use_pair(d_in[0]) ? device_sm_count() / 2 : device_sm_count();
  const int64_t r = tiles % units;
  if (tiles <= units || r == 0 || r > kTailMaxTiles) return;
  int64_t S = units / r;
  if (S > B) S = B;
  if (S < 2) return;
  int64_t left = r;
  for (int l = L - 1; l >= 0 && left > 0; --l) {
    const int64_t n = left < tail_from[l] ? left : tail_from[l];
    tail_from[l] -= static_cast<int>(n);
    tail_split[l] = static_cast<int>(S);
    left -= n;
  }
}

// Scratch for the tail pieces of one clipped-sum launch: at most one partial
// tile per unit of the GPU (256 x 256 per CTA pair, 128 x 256 per CTA).
int64_t tc_tail_scratch_bytes() {
  return static_cast<int64_t>(device_sm_count()) * BM * BN * 4;
}

bool tc_clipsum_same_launch(int64_t d_in_a, int64_t d_out_a, int64_t d_in_b, int64_t d_out_b) {
  return use_pair(d_in_a) == use_pair(d_in_b) && gemm_nb(d_out_a) == gemm_nb(d_out_b);
}

}  // namespace dpk
