/*
 * dp_step.h -- C ABI of the GB300 (sm_103a) DP-SGD gradient-step library.
 *
 * The library runs, on one GPU, the work the untrusted accelerator does in the
 * paper's verifiable DP-SGD protocol (Algorithm 2): per-example gradients of
 * dense layers, their L2 norms across all layers, per-example clipping, the
 * clipped sum, and the seeded Gaussian noise that the trusted side can
 * regenerate (Sec. 2.2 "DP-SGD"; Algorithms 2 and 3; Sec. 7.2 "Communication-
 * efficient split execution").  It also emits per-example audit records for
 * the partial recomputation a CPU-side checker performs (Sec. 7).
 *
 * Notation.  A step has B examples of T positions each and L dense layers;
 * layer l has weight shape d_in x d_out.  For example i the caller supplies
 *   A_{i,l} in R^{T x d_in}   activations entering layer l,
 *   D_{i,l} in R^{T x d_out}  gradients of the loss w.r.t. layer l's outputs,
 * so that the per-example weight gradient is G_{i,l} = A_{i,l}^T D_{i,l}
 * (laid out [d_in, d_out]).
 *
 * Memory layout of every A / D argument: one dense row-major array
 * [B][T][d] (example-major, then position, then feature), element type from
 * dp_config.dtype, base address 16-byte aligned, rows d * elemsize bytes
 * apart.  bf16 layers whose d_in and d_out are multiples of 8 can run on
 * tensor cores; other widths run on CUDA cores.
 * Outputs are fp32 row-major [d_in][d_out], 16-byte aligned.
 *
 * Ownership.  The caller owns every A, D and output buffer and the CUDA
 * stream; buffers are device pointers unless a parameter says "host".  The
 * context owns its scratch (per-layer norm partials, norms, clip factors,
 * audit staging, an error flag, the per-example gradients of thin layers)
 * and frees it in dp_step_destroy.
 *
 * Asynchrony.  Every call except dp_audit_emit only enqueues work on the
 * context's stream and returns; dp_audit_emit synchronises that stream.
 *
 * Errors.  Argument, shape, dtype and call-order errors are detected on the
 * host before anything is launched, and the call returns without side
 * effects.  Device-detected conditions (a non-finite squared norm) set a
 * sticky flag in the context that the next synchronising call
 * (dp_audit_emit) reports as DP_ERR_NONFINITE.  dp_last_error() returns a
 * message for the last failing call on the calling thread.
 *
 * Call order within one step:
 *   dp_step_init  ->  dp_layer_norms (every layer, any order)
 *                 ->  dp_clip_factors
 *                 ->  dp_clipped_sum_noise (any layers, any order, any number)
 *                 ->  dp_audit_emit (optional, any number of times)
 * Anything else returns DP_ERR_ORDER, except dp_clipped_sum_noise with
 * DP_NOISE_ONLY, which needs only an initialised context.
 */
#ifndef DP_STEP_H
#define DP_STEP_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct dp_ctx dp_ctx; /* opaque, owned by the library */

typedef enum {
    DP_OK = 0,
    DP_ERR_ARG = 1,         /* null pointer, misaligned buffer, bad scalar, index out of range */
    DP_ERR_SHAPE = 2,       /* shape disagrees with the context / limits exceeded */
    DP_ERR_DTYPE = 3,       /* unknown element type */
    DP_ERR_ORDER = 4,       /* call made out of the order documented above */
    DP_ERR_NONFINITE = 5,   /* a per-example squared norm was NaN or infinite */
    DP_ERR_CUDA = 6,        /* a CUDA runtime / driver call failed */
    DP_ERR_TIMEOUT = 7,     /* a bounded device wait gave up */
    DP_ERR_OOM = 8,         /* device or pinned host allocation failed */
    DP_ERR_UNSUPPORTED = 9  /* the device is not an sm_103 GPU or a path is not built */
} dp_status;

typedef enum { DP_F32 = 0, DP_BF16 = 1 } dp_dtype;

/* How the per-example squared norm ||A_i^T D_i||_F^2 of a layer is formed.
 * RANK1: T must be 1, n_i = ||a_i||^2 ||d_i||^2.
 * GHOST: n_i = sum_{t,s} (a_t . a_s)(d_t . d_s), from the two T x T Gram matrices.
 * MATERIALISED: the d_in x d_out gradient is formed tile by tile on chip,
 *   squared and summed; it is never written to memory.
 * AUTO: RANK1 when T == 1, else whichever of GHOST / MATERIALISED has the
 *   smaller arithmetic cost (T <= 2 d_in d_out / (d_in + d_out) picks GHOST),
 *   except that
 *   - a bf16 layer wider than 65536 on either side takes MATERIALISED on
 *     tensor cores instead of GHOST on CUDA cores (see dp_layer_path);
 *   - a bf16 layer with T <= 128 whose Gram form has few work items (B times
 *     the Gram layers of that T below half the SMs) takes MATERIALISED when
 *     that is faster than one Gram item, whose (d_in + d_out) / 64 feature
 *     steps run one after another on one SM (0.42 us each, measured),
 *     against 2 B T d_in d_out flops at 0.9 PFLOP/s (measured). */
typedef enum {
    DP_NORM_AUTO = 0,
    DP_NORM_RANK1 = 1,
    DP_NORM_GHOST = 2,
    DP_NORM_MATERIALISED = 3
} dp_norm_mode;

/* ---- 2-D convolutions (the CIFAR-10 WideResNet of App. B) ---------------
 * A convolution without bias over NHWC activations (a cross-correlation):
 *   y[h][w][o] = sum_{ki, kj, c} xp[h*stride_h + ki][w*stride_w + kj][c] * W[ki][kj][c][o]
 * where xp is the input with pad_h rows and pad_w columns of zeros on each
 * side.  Its per-example weight gradient sum_{h,w} patch(h,w)^T dy[h][w] is
 * the dense A_i^T D_i of a layer {d_in = K, d_out = C_out, T} with
 *   T = H_out * W_out, H_out = (H + 2 pad_h - kh) / stride_h + 1 (W_out alike),
 *   K = kh * kw * C_in,
 *   A_i[h*W_out + w][(ki*kw + kj)*C_in + c] = xp_i[h*stride_h + ki][w*stride_w + kj][c]
 *     (the patch rows dp_conv2d_unfold writes),
 *   D_i = dy_i [H_out][W_out][C_out] read as [T][C_out],
 * so the layer's output is laid out [kh][kw][C_in][C_out] (HWIO), row-major.
 * A convolution enters a step in either of two ways:
 *   - as a DP_LAYER_CONV2D layer (dp_layer.kind) with its geometry in
 *     dp_config.convs: its A argument is then the NHWC input x [B][H][W][C_in]
 *     itself, and the library forms the patch rows, on the fly inside the
 *     tensor-core kernels where the shape allows (bf16, C_in a multiple of
 *     64, T a multiple of 64, W_out dividing 64 or 64 dividing W_out), else
 *     in context scratch when the layer's norms are computed;
 *   - as a dense layer whose A is the caller's dp_conv2d_unfold output.    */
typedef struct {
    int32_t H, W;                /* input height and width, >= 1 */
    int32_t C_in;                /* input channels, >= 1 */
    int32_t kh, kw;              /* kernel height and width, >= 1 */
    int32_t stride_h, stride_w;  /* >= 1 */
    int32_t pad_h, pad_w;        /* zero rows / columns on each side, >= 0 */
} dp_conv2d;

/* One dense layer of the step: weight d_in x d_out, and the positions per
 * example its A and D carry.  T = 0 takes dp_config.T; a layer applied to one
 * position only (a classification head on the first token) gives T = 1, and
 * a bias row is a layer with d_in = 1 whose A holds ones.  All layers share B
 * and the clip factors: s_i sums every layer of the step. */
#define DP_LAYER_DENSE  0
#define DP_LAYER_CONV2D 1

typedef struct {
    int64_t d_in;
    int64_t d_out;
    int32_t T;          /* positions per example of this layer, 0 = dp_config.T */
    int32_t kind;       /* DP_LAYER_DENSE, or DP_LAYER_CONV2D: a convolution whose
                           geometry is dp_config.convs[l], with d_in = kh*kw*C_in
                           and T = H_out*W_out (or 0, which takes H_out*W_out) */
} dp_layer;

/* Parameters of Algorithm 2 for one step: batch B (also the aggregation
 * denominator when out_scale = 1/B), clip norm C, noise multiplier sigma and
 * the released per-step noise seed (seed, step). */
typedef struct {
    int32_t B;                 /* examples per step, >= 1 */
    int32_t T;                 /* positions per example of layers with T = 0, >= 1 */
    int32_t n_layers;          /* L, 1 .. 1024 */
    const dp_layer* layers;    /* host array of L layer shapes; copied by dp_step_init */
    dp_dtype dtype;            /* element type of every A and D */
    float clip_C;              /* C > 0 */
    float sigma;               /* noise multiplier, >= 0 */
    float out_scale;           /* 1 (sum) or 1/B (Algorithm 2 average); any finite value */
    uint64_t seed;             /* Philox key; the trusted side's s_noise,t */
    uint64_t step;             /* step index t; upper Philox counter words */
    dp_norm_mode norm_mode;    /* applies to every layer (AUTO picks per layer) */
    int32_t audit_capacity;    /* max records per dp_audit_emit call, 0 .. B */
    const dp_conv2d* convs;    /* host array of L geometries, read for DP_LAYER_CONV2D
                                  layers only (NULL when there are none); copied */
    uint64_t param_base;       /* global parameter index of layer 0's element (0, 0):
                                  0 for a whole model; when the layers are split over
                                  ranks, the parameters of the layers before this
                                  context's (the noise keys are global indices) */
} dp_config;

/* Flags of dp_clipped_sum_noise. */
#define DP_NO_NOISE   0x1u /* write out_scale * S only: the noiseless commitment of Algorithm 2 */
#define DP_NOISE_ONLY 0x2u /* out += out_scale * sigma * C * z; A and D are ignored (may be NULL) */
#define DP_ACCUMULATE 0x4u /* add into out instead of overwriting it (micro-batch accumulation) */
#define DP_WRITE_GRAD 0x8u /* dp_noise_adamw: also write the noisy gradient back into d_grad */

/* AdamW hyperparameters of one OptStep (App. A one-step map). */
typedef struct {
    float lr;            /* learning rate eta_t, finite */
    float beta1, beta2;  /* in [0, 1) */
    float eps;           /* >= 0, added outside the square root */
    float weight_decay;  /* decoupled weight decay lambda */
    int64_t t;           /* step count for the bias corrections, >= 1 */
} dp_adamw;

/* Create (*ctx == NULL) or re-key (*ctx != NULL) a step context.
 * Create: validates cfg, allocates scratch on the current device and binds
 *   cuda_stream (a cudaStream_t; NULL = the legacy default stream).
 * Re-key: cfg must have the same B, T, dtype and layer shapes as the context
 *   (else DP_ERR_SHAPE and the context is unchanged); clip_C, sigma,
 *   out_scale, seed, step, norm_mode, audit_capacity and the stream are
 *   replaced and the per-step call-order state is reset.  Used once per
 *   training step, and again to supply the seed the trusted side releases
 *   after the commitment (Algorithm 3, Derive/release) before a
 *   DP_NOISE_ONLY call.
 * Limits: B * T <= 2^31 - 1; every d_in, d_out in 1 .. 2^20; the device must
 *   be compute capability 10.3.  A DP_LAYER_CONV2D layer needs a valid
 *   geometry (as dp_conv2d_dims) with d_in = kh*kw*C_in and T = H_out*W_out.
 * Errors: DP_ERR_ARG, DP_ERR_SHAPE, DP_ERR_DTYPE, DP_ERR_UNSUPPORTED,
 *   DP_ERR_OOM, DP_ERR_CUDA. On failure of a create, *ctx stays NULL. */
dp_status dp_step_init(dp_ctx** ctx, const dp_config* cfg, void* cuda_stream);

/* Per-example squared gradient norms of one layer (Sec. 2.2 clipping
 * equation: ||g_t(x_i)||_2^2 restricted to layer l):
 *   n_{l,i} = ||A_{i,l}^T D_{i,l}||_F^2,  i = 0 .. B-1,
 * kept in the context.  A: [B][T][d_in], D: [B][T][d_out] device arrays; for a
 * DP_LAYER_CONV2D layer A is the NHWC input [B][H][W][C_in] and D the output
 * gradient [B][H_out][W_out][C_out].
 * Errors: DP_ERR_ARG (null / misaligned), DP_ERR_ORDER (after
 * dp_clip_factors of this step), DP_ERR_CUDA. */
dp_status dp_layer_norms(dp_ctx* ctx, int32_t layer, const void* A, const void* D);

/* The same per-example squared norms for n listed layers at once (one call
 * per step for the whole trainable set of Algorithm 2): layers[r] is a layer
 * index (each at most once), A[r] and D[r] its device arrays (host arrays of
 * n pointers).  Equivalent to dp_layer_norms on each; Gram-form tensor-core
 * layers share kernel launches, so the work of several layers balances
 * across the SMs.  Errors: as dp_layer_norms; nothing is launched if any
 * argument is invalid. */
dp_status dp_layer_norms_batch(dp_ctx* ctx, int32_t n, const int32_t* layers,
                               const void* const* A, const void* const* D);

/* Layers split over ranks (each rank's context holds a contiguous range of
 * the model's layers, dp_config.param_base placing them in the global
 * parameter vector).  Sec. 2.2's ||g_i|| runs over every trainable
 * parameter, so the squared norms of all ranks' layers are summed before
 * clipping:
 *   dp_partial_sqnorms: d_sqnorm_local[i] = sum over this context's layers
 *     of n_{l,i} (device fp32 [B]); needs every layer's norms, forms no clip
 *     factor and leaves the call-order state unchanged;
 *   dp_clip_factors_from: as dp_clip_factors, but with s_i =
 *     d_sqnorm_total[i] (device fp32 [B], e.g. the sum over ranks of their
 *     dp_partial_sqnorms) in place of this context's own sum.  Audit records
 *     then hold this total and this context's layer norms.
 * Errors: as dp_clip_factors (DP_ERR_ARG for a NULL array). */
dp_status dp_partial_sqnorms(dp_ctx* ctx, float* d_sqnorm_local);
dp_status dp_clip_factors_from(dp_ctx* ctx, const float* d_sqnorm_total, float* d_sqnorm_out,
                               float* d_clip_out);

/* Sum the per-layer norms and form the clip factors (Sec. 2.2; Algorithm 2):
 *   s_i = sum_l n_{l,i},   c_i = 1 if s_i <= C^2 else C / sqrt(s_i).
 * d_sqnorm_out [B] and d_clip_out [B] are optional device fp32 arrays that
 * receive s and c (NULL to skip).  A non-finite s_i sets the sticky flag and
 * gives c_i = NaN.
 * Errors: DP_ERR_ORDER (a layer's norms are missing), DP_ERR_ARG, DP_ERR_CUDA. */
dp_status dp_clip_factors(dp_ctx* ctx, float* d_sqnorm_out, float* d_clip_out);

/* Clipped sum and noise of one layer (Algorithm 2; Sec. 2.2 aggregation):
 *   S_l = sum_i c_i A_{i,l}^T D_{i,l} = A_l^T diag(c (x) 1_T) D_l   [d_in x d_out]
 *   out = out_scale * (S_l + sigma * C * z_l)       (flags = 0)
 *   z_p = Gaussian number of global parameter index p = off_l + j*d_out + k,
 *         off_l = sum_{l' < l} d_in^{l'} d_out^{l'};
 *   Philox4x32-10 with key = (lo32 seed, hi32 seed) and counter =
 *   (lo32 q, hi32 q, lo32 step, hi32 step), q = p >> 2, gives words x0..x3;
 *   u0 = RN_fp32((x_{2m}+1) / 2^32), u1 = RN_fp32(x_{2m+1} / 2^32);
 *   slots 2m, 2m+1 of the quad are sqrt(-2 ln u0) * (cos, sin)(2 pi u1).
 * flags: DP_NO_NOISE, DP_NOISE_ONLY, DP_ACCUMULATE (see above).
 * d_out: device fp32 [d_in][d_out], 16-byte aligned, owned by the caller.
 * Thin layers.  When one side of a layer is at most 32 wide (LoRA factors,
 *   small heads, bias rows) and either T = 1 or 8 d_in d_out < T (d_in +
 *   d_out) elemsize (and the norm mode is AUTO or MATERIALISED),
 *   dp_layer_norms stores the layer's per-example gradients G_{i,l} in the
 *   context (B d_in d_out floats), and this call sums those in example order
 *   instead of reading A and D again.  Its A and D must be the arrays given
 *   to dp_layer_norms in this step; they are checked but not read.
 * Errors: DP_ERR_ARG, DP_ERR_ORDER (clip factors not formed yet, unless
 *   DP_NOISE_ONLY), DP_ERR_CUDA. */
dp_status dp_clipped_sum_noise(dp_ctx* ctx, int32_t layer, const void* A, const void* D,
                               float* d_out, uint32_t flags);

/* Released noise on a range of the global parameter vector (Algorithm 2:
 * the noise added after the commitment), independent of layers:
 *   d_out[e] += out_scale * sigma * C * z_{p_first + e},  0 <= e < n,
 * with z as in dp_clipped_sum_noise.  It lets ranks that hold disjoint
 * slices of the summed commitment (after a reduce-scatter) each add the
 * noise of their own slice.  d_out: device fp32 [n], 16-byte aligned (the
 * kernel reads and writes whole quads when p_first is a multiple of 4).
 * Needs only an initialised context (the key of dp_step_init /
 * dp_set_noise_key).  n = 0 launches nothing.
 * Errors: DP_ERR_ARG (NULL or misaligned d_out, n < 0), DP_ERR_CUDA. */
dp_status dp_noise_add_range(dp_ctx* ctx, uint64_t p_first, int64_t n, float* d_out);

/* Clipped sum and noise of n listed layers (host arrays of n entries:
 * layer indices, each at most once, and their A, D and d_out pointers; A
 * and D may be NULL with DP_NOISE_ONLY).  Equivalent to dp_clipped_sum_noise
 * on each; tensor-core layers share kernel launches, so the last round of
 * output tiles of one layer overlaps the next layer's, and with
 * DP_NOISE_ONLY every listed layer's noise is added in one launch (per 32
 * layers).  Errors: as
 * dp_clipped_sum_noise; nothing is launched if any argument is invalid. */
dp_status dp_clipped_sum_noise_batch(dp_ctx* ctx, int32_t n, const int32_t* layers,
                                     const void* const* A, const void* const* D,
                                     float* const* d_out, uint32_t flags);

/* The GPU's update after the seed release (Algorithm 2; OptStep = AdamW as
 * in App. A), one layer, in one pass over its parameters:
 *   g~    = d_grad + out_scale * sigma * C * z          (z as above, same keys)
 *   m     = b1 m + (1 - b1) g~,   v = b2 v + (1 - b2) g~^2
 *   theta = theta - lr (m / (1 - b1^t) / (sqrt(v / (1 - b2^t)) + eps)
 *                       + weight_decay * theta)
 * d_grad holds the committed average on entry (dp_clipped_sum_noise with
 * DP_NO_NOISE); d_theta, d_m, d_v are updated in place.  All are device fp32
 * [d_in][d_out], 16-byte aligned.  flags: DP_NO_NOISE (g~ = d_grad),
 * DP_WRITE_GRAD (store g~ into d_grad).  Needs only an initialised context
 * (the key set by dp_step_init / dp_set_noise_key).
 * Errors: DP_ERR_ARG (NULL / misaligned pointers, bad hyperparameters or
 * flags), DP_ERR_CUDA. */
dp_status dp_noise_adamw(dp_ctx* ctx, int32_t layer, float* d_grad, float* d_theta, float* d_m,
                         float* d_v, const dp_adamw* hp, uint32_t flags);

/* Audit emit: for the n example indices in h_idx (host array, each in
 * 0 .. B-1, n <= audit_capacity) copy records into h_records (host memory,
 * n * dp_audit_record_bytes(L) bytes) with layout per record:
 *   int32_t example; float total_sqnorm (s_i); float clip_factor (c_i);
 *   float layer_sqnorm[L] (n_{1..L,i})
 * -- what a checker needs to recompute the audited examples (Sec. 7, partial
 * recomputation; Algorithm 1 consumes the recomputed aggregate).
 * Synchronises the context's stream.  The gather kernel reads the indices
 * and writes the records through mapped pinned staging, so the call uses no
 * copy engine and never waits behind bulk copies queued on other streams.
 * Returns DP_ERR_NONFINITE if the sticky flag was set during this step
 * (records are still written).
 * Errors: DP_ERR_ARG, DP_ERR_ORDER (before dp_clip_factors), DP_ERR_NONFINITE,
 *   DP_ERR_TIMEOUT (a tensor-core kernel gave up on a bounded wait),
 *   DP_ERR_CUDA. */
dp_status dp_audit_emit(dp_ctx* ctx, const int32_t* h_idx, int32_t n, void* h_records);

/* Bytes of one audit record for L layers: 12 + 4 L. */
int64_t dp_audit_record_bytes(int32_t n_layers);

/* Norm mode chosen for a layer (resolves DP_NORM_AUTO). */
dp_status dp_layer_norm_mode(const dp_ctx* ctx, int32_t layer, dp_norm_mode* mode_out);

/* Replace the noise key (seed, step) of CUDA graph replays without enqueuing
 * any work.  A step captured from dp_step_init on loads the key from mapped
 * pinned host memory when the graph runs (the capture's key until this call
 * replaces it), so calling this between replays keys each replay (Algorithm
 * 3's released seed s_noise,t).  The caller must not call it while a
 * previous replay that copies the key may still be pending (dp_audit_emit,
 * or any synchronisation of the stream, ensures that).  Eager steps are not
 * affected: dp_step_init fixes their key when it enqueues them.
 * Host-only; the call-order state is unchanged.  Errors: DP_ERR_ARG. */
dp_status dp_set_noise_key(dp_ctx* ctx, uint64_t seed, uint64_t step);

/* Which kernels serve a layer: *norm_tc = 1 if its per-example norms run on
 * the tcgen05 tensor cores (0: CUDA cores), *sum_tc = 1 if its clipped sum
 * does.  For bf16 layers the Gram norm does when d_in, d_out <= 65536; the
 * clipped sum and the materialised norm do when T is a multiple of 64 or
 * T >= 32 (each example padded to 64 positions) and T <= 65536, and for
 * T < 32 the clipped sum runs on a pre-scaled copy of A (c_i folded into a
 * bf16 hi + lo pair held in context scratch, no per-example fold) when
 * 2 B T <= 65536 (rounded up to 64).  The bounds are accuracy bounds: a tensor-core fp32
 * accumulator drifts low by about 1.6 * 2^-24 per 16-long step of its
 * reduction, so longer reductions run on CUDA cores.  fp32 layers never use
 * tensor cores.  Thin layers whose
 * per-example gradients are stored by the norm pass (see
 * dp_clipped_sum_noise) report *norm_tc = 2 and *sum_tc = 0: both passes run
 * on CUDA cores. */
dp_status dp_layer_path(const dp_ctx* ctx, int32_t layer, int32_t* norm_tc, int32_t* sum_tc);

/* Release the context and all of its scratch; NULL is a no-op.  Waits for
 * the context's pending work first. */
void dp_step_destroy(dp_ctx* ctx);

/* Per-example squared norms of one layer without allocating any memory.
 * The paper has no counterpart: this exists for callers that cannot call
 * cudaMalloc at the point of use (inside a CUDA stream capture in global
 * capture mode, a process whose device-memory budget is fixed at start-up,
 * or a caller that must avoid the device synchronisation allocation can
 * cause) and so cannot create a step context.
 *   d_sqnorm_out[i] = ||A_i^T D_i||_F^2, i < B, by the Gram form (the same
 *   kernels as dp_layer_norms with DP_NORM_GHOST).
 * A: [B][T][d_in], D: [B][T][d_out] device arrays of dtype, 16-byte aligned;
 * d_sqnorm_out: device fp32 [B]; cuda_stream: cudaStream_t (NULL = default).
 * Asynchronous.  Scratch is a library-owned static device array of 2^20 fp32
 * partial sums (4 MiB, held by every GPU that loads the library until exit).
 * B times the partial sums per example must not exceed 2^20, else
 * DP_ERR_SHAPE.  Per example that is, with m = ceil(ceil(T / 128) / 2):
 *   tensor cores (bf16, d_in and d_out <= 65536, T <= 65536):
 *     8 m (m + 1) when ceil(T / 128) is even, 8 m^2 when it is odd;
 *   CUDA cores (fp32, or a side or T above 65536):
 *     n (n + 1) / 2 with n = ceil(T / 64).
 * The first call on a device looks up the array's address and does the
 * kernels' per-device set-up; it should come before any stream capture.
 * Calls share the array: calls that overlap on the GPU race and must be
 * ordered by the caller.  If a tensor-core pipeline wait gives up, the
 * outputs are NaN.
 * Errors: DP_ERR_ARG, DP_ERR_DTYPE, DP_ERR_SHAPE, DP_ERR_CUDA. */
dp_status dp_layer_sqnorms_noalloc(const void* A, const void* D, int32_t B, int32_t T,
                                   int64_t d_in, int64_t d_out, dp_dtype dtype,
                                   float* d_sqnorm_out, void* cuda_stream);

/* Message of the last failing call on this thread ("" if none). */
const char* dp_last_error(void);

/* Name of a status code. */
const char* dp_status_string(dp_status s);



/* T = H_out * W_out and K = kh * kw * C_in of a convolution (host only).
 * Errors: DP_ERR_ARG (NULL argument), DP_ERR_SHAPE (a size < 1 or pad < 0,
 * a kernel larger than the padded input, T above 2^31 - 1, K above 2^20). */
dp_status dp_conv2d_dims(const dp_conv2d* conv, int32_t* T_out, int64_t* K_out);

/* Patch rows of B examples: x [B][H][W][C_in] -> a_out [B][T][K], both of
 * element type dtype, device arrays owned by the caller, 16-byte aligned and
 * not overlapping.  Values are copied and padding positions written as zero,
 * so the result is exact.  Asynchronous on stream (a cudaStream_t; NULL = the
 * legacy default stream); no context is needed.
 * Errors: DP_ERR_ARG (NULL, misaligned or overlapping arrays, B < 1),
 * DP_ERR_SHAPE (as dp_conv2d_dims, or B * T above 2^31 - 1), DP_ERR_DTYPE,
 * DP_ERR_CUDA. */
dp_status dp_conv2d_unfold(const dp_conv2d* conv, int32_t B, dp_dtype dtype, const void* x,
                           void* a_out, void* stream);

/* Number of CUDA kernels this library has issued in this process, counted on
 * the host as each launch is made, by every call above and the test exports
 * below (dp_layer_sqnorms_noalloc is not counted).  A launch made while the
 * stream is being captured into a CUDA graph counts once, at capture; graph
 * replays do not call the library and are not counted.  Thread-safe.
 * Errors: DP_ERR_ARG if count_out is NULL.                                 */
dp_status dp_kernel_launches(int64_t* count_out);

/* ---- test exports (not part of the step API) ---------------------------
 * They expose the generator the noise uses so tests can compare it with the
 * oracle: raw Philox4x32-10 blocks and the Gaussian numbers z_p.
 * d_out is a device array; stream is a cudaStream_t (NULL = default).    */

/* Make one bounded device wait run out, to exercise the failure path of the
 * tensor-core pipelines (their waits give up after 2 s, record
 * DP_ERR_TIMEOUT in the context's sticky error word and return, so the
 * context stays usable; Algorithm 1's checker then rejects the step).  A
 * one-warp kernel on the context's stream waits, with the same bounded-wait
 * helper, on an mbarrier that nothing arrives on, gives up after limit_ns
 * nanoseconds (1 .. 10^9) and sets the context's timeout bit; it issues no
 * TMA copy and no MMA.  Synchronises the stream.  Returns DP_ERR_TIMEOUT when
 * the wait gave up (dp_audit_emit of the same step then reports it too; the
 * next dp_step_init clears it).  Errors: DP_ERR_ARG (NULL context, limit out
 * of range), DP_ERR_CUDA. */
dp_status dp_debug_bounded_wait(dp_ctx* ctx, int64_t limit_ns);

/* d_out[4 r + w] = word w of the block for quad first_quad + r, r < n_quads. */
dp_status dp_debug_philox(uint64_t seed, uint64_t step, uint64_t first_quad, int64_t n_quads,
                          uint32_t* d_out, void* stream);

/* d_out[r] = z_{first_index + r} (unit variance, as defined above), r < n. */
dp_status dp_debug_gaussian(uint64_t seed, uint64_t step, uint64_t first_index, int64_t n,
                            float* d_out, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* DP_STEP_H */
