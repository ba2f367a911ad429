// Launchers shared between the C-ABI layer (dp_step.cu) and the kernel files.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

#include <functional>

namespace dpk {

enum InType { IN_F32 = 0, IN_BF16 = 1 };

// Longest reduction one tensor-core fp32 accumulator takes over its K
// dimension (features of a Gram, positions of an example's product): the
// accumulation drifts low by about 1.6 * 2^-24 per K = 16 step (measured on
// GB300: -3.1e-4 for a 65536-feature Gram norm, -6.2e-3 for 2^20), so 2^16
// keeps each factor of a norm below 4e-4.  Longer reductions run on CUDA
// cores, whose round-to-nearest fp32 sums do not drift.
constexpr int64_t kTcMaxAccum = 1 << 16;

// How the output tile of a clipped-sum kernel is written.
struct Epilogue {
  const uint64_t* key;  // device words {seed, step}: read by the kernel, so a
                        // captured CUDA graph picks up each step's key
  uint64_t p_base;     // global index of element (0, 0) of this layer
  float out_scale;     // applied to (S + sigmaC * z)
  float sigmaC;        // sigma * C
  int add_noise;       // 0: out_scale * S
  int accumulate;      // 1: out += value
};

// ---- per-example squared norms: partial sums into part[(row) * NP + p] ----
// row = layer * B + example; every kernel writes exactly nparts(...) entries.
// The counts are int64: a long example has ~T^2 / 8192 Gram tiles, more
// than an int holds for T of a few million; callers bound them before launch.
int64_t rank1_parts();
int64_t ghost_simt_parts(int T);
int64_t mat_simt_parts(int64_t d_in, int64_t d_out);

cudaError_t launch_norm_rank1(InType t, const void* A, const void* D, int B, int d_in, int d_out,
                              float* part, int NP, int row0, cudaStream_t s);
cudaError_t launch_norm_ghost_simt(InType t, const void* A, const void* D, int B, int T, int d_in,
                                   int d_out, float* part, int NP, int row0, cudaStream_t s);
cudaError_t launch_norm_mat_simt(InType t, const void* A, const void* D, int B, int T, int d_in,
                                 int d_out, float* part, int NP, int row0, cudaStream_t s);

// ---- cross-layer sum and clip factors ----
// mode kClipFull: s_i = sum of this context's layer norms, then c_i.
// mode kClipLocal: that sum into user_s only (a rank's share of s_i when the
//   layers are split over ranks); no clip factor.
// mode kClipGiven: s_i = s_given[i] (summed over every rank), then c_i.
constexpr int kClipFull = 0, kClipLocal = 1, kClipGiven = 2;
cudaError_t launch_clip(const float* part, int L, int B, int NP, const int* d_nparts, float C,
                        float* layer_sq, float* s_out, float* c_out, float* user_s, float* user_c,
                        int* flag, cudaStream_t s, int mode = kClipFull,
                        const float* s_given = nullptr);

// ---- clipped sum + noise (CUDA-core FFMA path) ----
cudaError_t launch_gemm_simt(InType t, const void* A, const void* D, const float* c, int B, int T,
                             int d_in, int d_out, float* out, const Epilogue& ep, cudaStream_t s);

// ---- standalone noise add: out_l[e] += scale * z_{p_base_l + e}, e < n_l ----
// One launch serves up to kNoiseMaxLayers layers; each block takes a
// contiguous chunk of kNoiseChunk Philox quads of one layer.
constexpr int kNoiseMaxLayers = 32;
constexpr int kNoiseChunk = 4096;
struct NoiseAddBatch {
  float* out[kNoiseMaxLayers];
  int64_t n[kNoiseMaxLayers];
  uint64_t p_base[kNoiseMaxLayers];
  int64_t block0[kNoiseMaxLayers + 1];  // first block of each layer (set by the launcher)
  const uint64_t* key;
  float scale;
  int L;
};
cudaError_t launch_noise_add(NoiseAddBatch& b, cudaStream_t s);

// ---- thin layers: per-example gradients stored by the norm pass ----
constexpr int kThinMax = 32;           // widest narrow side of a thin layer
constexpr int kPerGradMaxLayers = 32;  // layers per launch
struct PerGradLayer {
  const void* X;   // wide operand [B][T][n]
  const void* Y;   // narrow operand [B][T][r]
  float* G;        // per-example gradients [B][d_in][d_out]
  int n, r;        // wide and narrow widths
  int wide_is_in;  // 1: X = A (n = d_in), 0: X = D (n = d_out)
  int bulk;        // rows of X staged by bulk copies (n * elemsize % 16 == 0)
  int chunks;      // blocks per example (set by the launcher)
  int row0;        // partial-sum row of example 0
  int item0;       // first block of this layer (set by the launcher)
};
struct PerGradBatch {
  PerGradLayer l[kPerGradMaxLayers];
  float* part;
  int* err;  // sticky error word (bounded waits that gave up)
  int L, B, T, NP;
};
struct PerGradSumLayer {
  const float* G;   // [B][count]
  float* out;       // [count]
  int64_t count;    // d_in * d_out
  uint64_t p_base;  // global parameter index of element 0
  int64_t nq;       // quads (set by the launcher)
  int64_t item0;    // first block (set by the launcher)
  int vec;          // float4 path (set by the launcher)
  int split;        // threads per quad over the examples (set by the launcher)
};
struct PerGradSumBatch {
  PerGradSumLayer l[kPerGradMaxLayers];
  const float* c;
  const uint64_t* key;
  float out_scale, sigmaC;
  int add_noise, accumulate;
  int L, B;
};
int pergrad_bucket(int r);                       // 1, 2, 4, ..., 32, or 0 if too wide
int64_t pergrad_parts(InType t, int64_t d_in, int64_t d_out, int T);  // partials per example
cudaError_t launch_pergrad_norm(InType t, PerGradBatch& g, cudaStream_t s);
cudaError_t launch_pergrad_sum(PerGradSumBatch& g, cudaStream_t s);

// ---- noisy gradient + AdamW after the seed release ----
struct AdamWArgs {
  float lr, beta1, beta2, eps, weight_decay;
  float bc1, bc2;  // 1 / (1 - beta1^t), 1 / (1 - beta2^t)
};
cudaError_t launch_noise_adamw(float* grad, float* theta, float* m, float* v, int64_t n,
                               uint64_t p_base, const uint64_t* key, float noise_scale,
                               int add_noise, int write_grad, const AdamWArgs& h, cudaStream_t s);

// ---- audit gather ----
cudaError_t launch_audit(const int* idx, int n, int L, int B, const float* layer_sq,
                         const float* s_vec, const float* c_vec, const int* flag, float* rec,
                         int* flag_out, cudaStream_t s);

// ---- start of a step: device copy of the two mapped pinned key words, and
// the sticky flag cleared ----
cudaError_t launch_load_key(const uint64_t* host_key_dev, uint64_t* key, int* flag,
                            cudaStream_t s);
cudaError_t launch_set_key(uint64_t seed, uint64_t step, uint64_t* key, int* flag,
                           cudaStream_t s);

// ---- patch rows of a 2-D convolution over NHWC activations (k_conv.cu) ----
struct ConvGeom {
  int H, W, C_in, kh, kw, stride_h, stride_w, pad_h, pad_w;
  int H_out, W_out;
};
cudaError_t launch_conv_unfold(InType t, const void* x, void* a, const ConvGeom& g, int B,
                               cudaStream_t s);

// ---- per-device kernel set-up ----
// Kernel attributes (the dynamic shared-memory limit) and occupancy figures
// belong to one device.  setup_once_per_device runs setup() the first time it
// is asked for `key` (a kernel's address) on the current device, under a
// process-wide lock, and returns its status; a failed set-up runs again on
// the next call.  cached_per_device does the same for an integer (e.g. the
// CTA pairs that fit on the device at once), computed by fn() once per
// (key, device).
cudaError_t setup_once_per_device(const void* key, const std::function<cudaError_t()>& setup);
int cached_per_device(const void* key, const std::function<int()>& fn);

// ---- launch count: every launcher calls note_launch() once per kernel it
// issues (process-wide, thread-safe), read back by dp_kernel_launches() ----
void note_launch();
int64_t launch_count();

// ---- error message of the calling thread, read back by dp_last_error() ----
void set_last_error(const char* msg);

// ---- generator exports for tests ----
cudaError_t launch_debug_philox(uint64_t seed, uint64_t step, uint64_t q0, int64_t nq,
                                uint32_t* out, cudaStream_t s);
// one-warp kernel whose bounded mbarrier wait gives up after limit_ns and
// sets the timeout bit (2) of *err
cudaError_t launch_debug_wait(uint64_t limit_ns, int* err, cudaStream_t s);
cudaError_t launch_debug_gauss(uint64_t seed, uint64_t step, uint64_t p0, int64_t n, float* out,
                               cudaStream_t s);

}  // namespace dpk
