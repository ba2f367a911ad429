// Tensor-core (tcgen05 / TMEM / TMA) kernels of the DP-SGD step, bf16 inputs.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "internal.h"

namespace dpk {

// Gram-form per-example norms on tensor cores; one launch can serve up to
// kGhostMaxLayers layers of a step.
// T up to kTcGhostMaxT (a Gram of T^2 / 2 products per example; longer
// examples take the materialised form).  tc_ghost_parts(T) partial sums per
// example: CTA-pair items when ceil(T / 128) is even, single-CTA strips when
// it is odd.
constexpr int kGhostMaxLayers = 8;
constexpr int kTcGhostMaxT = 1 << 16;
bool tc_ghost_supported(int T, int64_t d_in, int64_t d_out);
int64_t tc_ghost_parts(int T);
// The once-per-device set-up of both Gram kernels (shared-memory limits, the
// resident-pair count), so that later launches make no set-up calls.
cudaError_t tc_ghost_prepare();
cudaError_t tc_launch_ghost(const void* A, const void* D, int B, int T, int d_in, int d_out,
                            float* part, int NP, int row0, int* err, cudaStream_t s);
cudaError_t tc_launch_ghost_batch(int L, const void* const* A, const void* const* D,
                                  const int* d_in, const int* d_out, const int* row0, int B,
                                  int T, float* part, int NP, int* err, cudaStream_t s);

// Clipped sum S = A^T diag(c) D with the noise epilogue, and the materialised
// per-example norm that shares its main loop.  One clipped-sum launch can
// serve up to kGemmMaxLayers layers whose tiles have the same shape
// (tc_clipsum_same_launch).
// A layer with few tiles splits its examples into tc_gemm_split ranges: the
// clipped sum then writes one partial per range into the caller's scratch
// (split * d_in * d_out fp32, 16-byte aligned) and a reduce pass adds them in
// order with the noise; the materialised norm needs no scratch.
// The split is fixed per layer when the step is planned (dp_step_init), from
// the layer's shape and the tiles of the other layers that share its launch,
// so a layer's sum rounds the same in a batched and a per-layer call.
constexpr int kGemmMaxLayers = 8;
constexpr int kGemmMaxSplit = 256;
int64_t tc_gemm_tiles(int64_t d_in, int64_t d_out);
int tc_gemm_split(int B, int T, int64_t d_in, int64_t d_out, int64_t other_tiles = 0);
bool tc_clipsum_same_launch(int64_t d_in_a, int64_t d_out_a, int64_t d_in_b, int64_t d_out_b);
// conv (per layer, NULL for a dense layer): A is then the NHWC input and the
// kernels read its patch rows directly (tc_conv_implicit_ok must hold).
// split: example ranges of each layer (as planned; NULL: tc_gemm_split alone).
// tail_from / tail_split (per layer, as planned by tc_plan_tail; NULL: no
// tail): the layer's tiles from tail_from on run as tail_split pieces of the
// batch each, into `tail` (tail_bytes, 16-byte aligned;
// tc_tail_scratch_bytes is always enough), added up by a reduce launch.
cudaError_t tc_launch_clipsum_batch(int L, const void* const* A, const void* const* D,
                                    float* const* out, float* const* part, const int* d_in,
                                    const int* d_out, const uint64_t* p_base, const int* split,
                                    const float* c, int B, int T, const Epilogue& ep, int* err,
                                    cudaStream_t s, const ConvGeom* const* conv = nullptr,
                                    const int* tail_from = nullptr,
                                    const int* tail_split = nullptr, float* tail = nullptr,
                                    int64_t tail_bytes = 0);
int64_t tc_tail_scratch_bytes();
void tc_plan_tail(int L, const int64_t* d_in, const int64_t* d_out, int B, int* tail_from,
                  int* tail_split);
bool tc_conv_implicit_ok(const ConvGeom& g, int T);
bool tc_gemm_supported(int T, int64_t d_in, int64_t d_out);
int64_t tc_mat_parts(int64_t d_in, int64_t d_out);
cudaError_t tc_launch_mat_norm(const void* A, const void* D, int B, int T, int d_in, int d_out,
                               float* part, int NP, int row0, int* err, cudaStream_t s,
                               const ConvGeom* conv = nullptr);
cudaError_t tc_launch_clipsum(const void* A, const void* D, const float* c, int B, int T,
                              int d_in, int d_out, int split, float* out, float* part,
                              const Epilogue& ep, int* err, cudaStream_t s,
                              const ConvGeom* conv = nullptr, int tail_from = 0,
                              int tail_split = 1, float* tail = nullptr, int64_t tail_bytes = 0);

// Clipped sum for short examples (T < 32): c_i folded into a bf16 hi+lo
// split of A in scratch (tc_prescaled_scratch_bytes), then one plain GEMM.
// Pre-scaled operand (c_i a as a bf16 hi + lo pair, one plain GEMM with no
// per-example fold) for T < 32, where the direct kernel's 3-D padding would
// waste more than half of every K block.  At T = 64 and 128 the direct
// kernel with its per-example fold is faster (same box, 4096 x 4096 layer at
// T = 64: 0.41 against 0.54 ms at B = 128; the 768-3072 wide block layers at
// T = 128: 0.115 against 0.295 ms).
constexpr int kPrescaleMaxT = 31;
bool tc_prescaled_supported(int B, int T, int64_t d_in, int64_t d_out);
int64_t tc_prescaled_scratch_bytes(int B, int T, int64_t d_in);
cudaError_t tc_launch_clipsum_prescaled(const void* A, const void* D, const float* c, int B,
                                        int T, int d_in, int d_out, float* out,
                                        const Epilogue& ep, int* err, void* scratch,
                                        cudaStream_t s);

// Host helpers shared by the tensor-core launchers (tc_host.cu).
bool tma_encode_available();
// bf16 tensor map, 128-byte swizzle, zero fill out of bounds; dims[0] innermost,
// strides_bytes[r] is the byte stride of dimension r+1; estrides (NULL: all 1)
// the traversal strides.
bool make_tma_bf16(CUtensorMap* m, const void* base, int rank, const uint64_t* dims,
                   const uint64_t* strides_bytes, const uint32_t* box,
                   const uint32_t* estrides = nullptr);
// fp32 output map over [rows][cols], box 32 x 32 (128-byte rows), 128-byte swizzle.
bool make_tma_f32_out(CUtensorMap* m, void* base, uint64_t rows, uint64_t cols);
// fp32 map over [split][rows][cols] partial sums, box 32 x 32 x 1, 128-byte swizzle.
bool make_tma_f32_split(CUtensorMap* m, void* base, int split, uint64_t rows, uint64_t cols);
int device_sm_count();

}  // namespace dpk
