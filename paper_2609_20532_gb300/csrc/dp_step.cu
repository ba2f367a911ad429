// C-ABI layer of the DP-SGD step library: argument checking, the per-step
// call-order state machine, scratch ownership and kernel dispatch.  See
// include/dp_step.h for the contract of every entry point.
#include <cuda_runtime.h>

#include <cmath>
#include <map>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "../../include/dp_step.h"
#include "conv_thin.h"
#include "internal.h"
#include "tc.h"

namespace {

thread_local std::string g_err;

dp_status fail(dp_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  std::vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_err = buf;
  return st;
}

#define DP_CUDA(call)                                                                      \
  do {                                                                                     \
    cudaError_t e_ = (call);                                                               \
    if (e_ != cudaSuccess)                                                                 \
      return fail(DP_ERR_CUDA, "%s failed: %s", #call, cudaGetErrorString(e_));            \
  } while (0)

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

constexpr int64_t kMaxDim = 1 << 20;  // largest d_in, d_out (and convolution K)

dp_status conv_geom(const dp_conv2d* v, dpk::ConvGeom* g) {
  if (!v) return fail(DP_ERR_ARG, "conv is NULL");
  if (v->H < 1 || v->W < 1 || v->C_in < 1 || v->kh < 1 || v->kw < 1 || v->stride_h < 1 ||
      v->stride_w < 1 || v->pad_h < 0 || v->pad_w < 0)
    return fail(DP_ERR_SHAPE, "convolution sizes must be >= 1 and pads >= 0");
  const int64_t hp = static_cast<int64_t>(v->H) + 2 * static_cast<int64_t>(v->pad_h);
  const int64_t wp = static_cast<int64_t>(v->W) + 2 * static_cast<int64_t>(v->pad_w);
  if (v->kh > hp || v->kw > wp) return fail(DP_ERR_SHAPE, "kernel larger than the padded input");
  const int64_t ho = (hp - v->kh) / v->stride_h + 1, wo = (wp - v->kw) / v->stride_w + 1;
  const int64_t K = static_cast<int64_t>(v->kh) * v->kw * v->C_in;
  if (ho * wo > 0x7fffffffLL) return fail(DP_ERR_SHAPE, "H_out * W_out above 2^31 - 1");
  if (K > kMaxDim) return fail(DP_ERR_SHAPE, "kh * kw * C_in above 2^20");
  *g = dpk::ConvGeom{v->H, v->W, v->C_in, v->kh, v->kw, v->stride_h, v->stride_w,
                     v->pad_h, v->pad_w, static_cast<int>(ho), static_cast<int>(wo)};
  return DP_OK;
}

}  // namespace

namespace dpk {
void set_last_error(const char* msg) { g_err = msg; }
}  // namespace dpk

// Per-layer execution plan, fixed at init from the shapes and the norm mode.
struct LayerPlan {
  int64_t d_in, d_out;
  int T;               // positions per example of this layer
  uint64_t p_base;     // global parameter index of element (0, 0)
  dp_norm_mode mode;   // resolved norm mode
  int norm_tc;         // 1: tensor-core norm kernel
  int nparts;          // partial sums per example
  int gemm_tc;         // 0: CUDA-core clipped sum, 1: tcgen05, 2: tcgen05 on a pre-scaled operand
  int pergrad;         // 1: thin layer, per-example gradients stored by the norm pass
  int64_t g_off;       // offset (floats) of its [B][d_in][d_out] gradients in d_grads
  int split;           // tensor-core clipped sum: example ranges per tile (tc_gemm_split)
  int64_t s_off;       // offset (floats) of its [split][d_in][d_out] partials in d_split
  // tensor-core clipped sum: its tiles from tail_from on run as tail_split
  // pieces of the batch (the last round of its launch group, tc_plan_tail);
  // fixed at planning so any grouping of the calls gives the same bits
  int tail_from, tail_split;
  // tensor-core clipped sum (direct or pre-scaled) of a short batch
  // (B T <= kNoiseAfterMaxK): the noise is added by the noise-add kernel
  // after the GEMM instead of inside its epilogue, where generating it would
  // take longer than the products
  int noise_after;
  // convolutions (kind DP_LAYER_CONV2D; A is the NHWC input)
  int kind;            // dp_layer.kind as given
  int conv;            // 1: a convolution whose patch rows differ from its input
  dpk::ConvGeom cg;    // its geometry
  int implicit;        // 1: the tensor-core kernels read its patch rows from A directly
  int unfold;          // 1: its patch rows are formed in d_unf when its norms are computed
  int64_t u_off;       // byte offset of those patch rows in d_unf
  // a thin convolution whose input per example fits in shared memory: its
  // per-example gradients come straight from the NHWC input
  // (launch_conv_thin_norm), no patch rows, one norm partial per example
  int fused;
};

struct dp_ctx {
  int B = 0, T = 0, L = 0;
  dp_dtype dtype = DP_F32;
  float C = 1.f, sigma = 0.f, out_scale = 1.f;
  uint64_t seed = 0, step = 0;
  dp_norm_mode norm_mode = DP_NORM_AUTO;
  int audit_capacity = 0;
  cudaStream_t stream = nullptr;
  int device = 0;
  std::vector<LayerPlan> plan;
  int NP = 1;  // partial-sum stride
  // scratch
  float* d_part = nullptr;      // [L][B][NP]
  int* d_nparts = nullptr;      // [L]
  float* d_layer_sq = nullptr;  // [L][B]
  float* d_s = nullptr;         // [B]
  float* d_c = nullptr;         // [B]
  int* d_flag = nullptr;        // sticky error bits
  // audit staging in mapped pinned memory: the gather kernel reads the
  // indices and writes the records and the flag word over the host link
  // itself, so an audit never queues behind bulk copies on the copy engines
  int* h_idx = nullptr;         // mapped [cap]
  float* h_rec = nullptr;       // mapped [cap][3 + L]
  int* h_flag = nullptr;        // mapped
  int* h_idx_dev = nullptr;     // device views of the three
  float* h_rec_dev = nullptr;
  int* h_flag_dev = nullptr;
  uint64_t* d_key = nullptr;    // {seed, step} read by the noise kernels
  uint64_t* h_key = nullptr;    // mapped pinned source of d_key (host address)
  uint64_t* h_key_dev = nullptr;  // the same words, device address
  void* d_prescaled = nullptr;  // pre-scaled operand of short-example layers
  int64_t prescaled_bytes = 0;
  float* d_grads = nullptr;     // per-example gradients of thin layers
  int64_t grads_floats = 0;
  float* d_split = nullptr;     // partial sums of tensor-core layers whose batch is split
  int64_t split_floats = 0;
  float* d_tail = nullptr;      // partial tiles of a clipped-sum launch's tail pieces
  int64_t tail_bytes = 0;
  uint8_t* d_unf = nullptr;     // patch rows of convolutions formed in scratch
  int64_t unf_bytes = 0;
  size_t part_bytes = 0;
  // per-step state
  std::vector<char> norm_done;
  bool clip_done = false;
};

namespace {

// Partial sums one example of one layer may need.  The partial buffer holds
// L * B * NP floats; a forced Gram form on very long examples (about T^2 /
// 8192 partials) or a materialised norm of an enormous layer would exceed it.
constexpr int64_t kMaxPartsPerExample = int64_t(1) << 24;
// The tensor-core clipped sum generates its noise in the epilogue while the
// tensor core works on the examples: about 0.2 G Gaussians per second per
// launch, hidden behind the products when a tile runs over a few thousand
// rows of K = B T.  With K <= 1024 the products are the shorter part, so the
// GEMM writes the noiseless sum and the noise-add kernel (about 0.6 G
// Gaussians per second) adds the noise after it (4096 x 4096 layer: 0.080 ->
// 0.055 ms at B = 8, T = 1; 0.086 -> 0.073 ms at B = 8, T = 64; at K = 2048,
// B = 32, T = 64, the noise inside the GEMM is faster, 0.125 against 0.130).
constexpr int64_t kNoiseAfterMaxK = 1024;

dp_status check_config(const dp_config* cfg) {
  if (!cfg) return fail(DP_ERR_ARG, "cfg is NULL");
  if (cfg->B < 1 || cfg->T < 1) return fail(DP_ERR_SHAPE, "B and T must be >= 1");
  if (static_cast<int64_t>(cfg->B) * cfg->T > 0x7fffffffLL)
    return fail(DP_ERR_SHAPE, "B*T exceeds 2^31-1");
  if (cfg->n_layers < 1 || cfg->n_layers > 1024)
    return fail(DP_ERR_SHAPE, "n_layers must be in 1..1024");
  if (!cfg->layers) return fail(DP_ERR_ARG, "layers is NULL");
  if (cfg->dtype != DP_F32 && cfg->dtype != DP_BF16) return fail(DP_ERR_DTYPE, "unknown dtype");
  for (int l = 0; l < cfg->n_layers; ++l) {
    const dp_layer& ly = cfg->layers[l];
    if (ly.d_in < 1 || ly.d_out < 1 || ly.d_in > kMaxDim || ly.d_out > kMaxDim)
      return fail(DP_ERR_SHAPE, "layer %d: d_in, d_out must be in 1..2^20", l);
    if (ly.T < 0) return fail(DP_ERR_ARG, "layer %d: T must be >= 0 (0 = config T)", l);
    if (ly.kind != DP_LAYER_DENSE && ly.kind != DP_LAYER_CONV2D)
      return fail(DP_ERR_ARG, "layer %d: unknown kind %d", l, ly.kind);
    int T = ly.T > 0 ? ly.T : cfg->T;
    if (ly.kind == DP_LAYER_CONV2D) {
      if (!cfg->convs) return fail(DP_ERR_ARG, "layer %d is a convolution but convs is NULL", l);
      dpk::ConvGeom g{};
      dp_status st = conv_geom(&cfg->convs[l], &g);
      if (st != DP_OK) return st;
      if (ly.d_in != static_cast<int64_t>(g.kh) * g.kw * g.C_in)
        return fail(DP_ERR_SHAPE, "layer %d: d_in must be kh*kw*C_in", l);
      if (ly.T != 0 && ly.T != g.H_out * g.W_out)
        return fail(DP_ERR_SHAPE, "layer %d: T must be H_out*W_out (or 0)", l);
      T = g.H_out * g.W_out;
    }
    if (static_cast<int64_t>(cfg->B) * T > 0x7fffffffLL)
      return fail(DP_ERR_SHAPE, "layer %d: B*T exceeds 2^31-1", l);
    if (cfg->norm_mode == DP_NORM_RANK1 && T != 1)
      return fail(DP_ERR_SHAPE, "DP_NORM_RANK1 needs T == 1 for every layer");
    // a forced Gram form beyond the tensor cores' T bound runs on CUDA cores
    // with ceil(T/64) (ceil(T/64) + 1) / 2 partial sums per example
    if (cfg->norm_mode == DP_NORM_GHOST && T > dpk::kTcGhostMaxT &&
        dpk::ghost_simt_parts(T) > kMaxPartsPerExample)
      return fail(DP_ERR_SHAPE,
                  "layer %d: the Gram form at T = %d needs more than %lld partial sums per "
                  "example; use DP_NORM_MATERIALISED for examples this long",
                  l, T, static_cast<long long>(kMaxPartsPerExample));
  }
  if (!(cfg->clip_C > 0.f) || !std::isfinite(cfg->clip_C))
    return fail(DP_ERR_ARG, "clip_C must be finite and > 0");
  if (!(cfg->sigma >= 0.f) || !std::isfinite(cfg->sigma))
    return fail(DP_ERR_ARG, "sigma must be finite and >= 0");
  if (!std::isfinite(cfg->out_scale)) return fail(DP_ERR_ARG, "out_scale must be finite");
  if (cfg->norm_mode < DP_NORM_AUTO || cfg->norm_mode > DP_NORM_MATERIALISED)
    return fail(DP_ERR_ARG, "unknown norm_mode");
  if (cfg->audit_capacity < 0 || cfg->audit_capacity > cfg->B)
    return fail(DP_ERR_ARG, "audit_capacity must be in 0..B");
  return DP_OK;
}

dp_norm_mode resolve_mode(dp_norm_mode m, int T, int64_t d_in, int64_t d_out) {
  if (m != DP_NORM_AUTO) return m;
  if (T == 1) return DP_NORM_RANK1;
  // Multiply-adds per example: Gram form about T^2 (d_in + d_out) / 2 with
  // the symmetric half, materialised form T d_in d_out.
  const double ghost = 0.5 * double(T) * T * double(d_in + d_out);
  const double mat = double(T) * double(d_in) * double(d_out);
  return ghost <= mat ? DP_NORM_GHOST : DP_NORM_MATERIALISED;
}

// Latency term of the norm-form choice.  When the Gram form has few work
// items (B times the Gram layers that share T: fewer than half the SMs), its
// time is one item's, whose K steps run one after another on one SM: about
// 0.25 us per 64 features on the GB300 (measured: 4096 x 4096 at T = 64,
// 128 x 64 features in 32 us), while the materialised form spreads over the
// whole GPU at about 0.64 PFLOP/s for examples of one 64-position K block
// (measured at T = 64: 17.2 GFLOP in 27 us).  Both forms then reduce their
// partial sums in the clip kernel at about the same cost.  Only examples of
// one 128-position block (T <= 128) are concerned: longer ones give the Gram
// form CTA-pair items that fill the GPU and it wins by its arithmetic.
constexpr double kGramStepSeconds = 0.25e-6;
constexpr double kMatShortRate = 0.64e15;

bool gram_latency_prefers_materialised(int B, int T, int64_t d_in, int64_t d_out,
                                       int64_t gram_items, int sms) {
  if (T > 128 || gram_items * 2 >= sms) return false;
  const double steps = static_cast<double>((d_in + 63) / 64 + (d_out + 63) / 64);
  const double t_gram = steps * kGramStepSeconds;
  const double t_mat = 2.0 * B * T * static_cast<double>(d_in) * static_cast<double>(d_out) /
                       kMatShortRate;
  return t_mat < t_gram;
}

// A thin layer (narrow side <= kThinMax) stores its per-example gradients
// when writing and reading them back moves fewer bytes than reading A and D
// a second time, 8 d_in d_out < T (d_in + d_out) elem, which also makes the
// materialised norm the cheaper one (T > 4 r); and always at T = 1, where
// such a layer (a bias row, a head with few outputs) is too small for bytes
// to matter and its clipped sum would otherwise be a latency-bound K = B
// loop of its own.  A forced Gram or rank-1 mode keeps the other paths.
int layer_T(const dp_config* cfg, int l) {
  if (cfg->layers[l].kind == DP_LAYER_CONV2D) {  // geometry checked by check_config
    dpk::ConvGeom g{};
    conv_geom(&cfg->convs[l], &g);
    return g.H_out * g.W_out;
  }
  return cfg->layers[l].T > 0 ? cfg->layers[l].T : cfg->T;
}

bool use_pergrad(const dp_config* cfg, int T, int64_t d_in, int64_t d_out) {
  if (cfg->norm_mode == DP_NORM_GHOST || cfg->norm_mode == DP_NORM_RANK1) return false;
  const int64_t r = d_in < d_out ? d_in : d_out;
  if (r > dpk::kThinMax) return false;
  if (T == 1) return true;
  const double elem = cfg->dtype == DP_BF16 ? 2.0 : 4.0;
  return 8.0 * double(d_in) * double(d_out) < double(T) * double(d_in + d_out) * elem;
}

dp_status build_plan(dp_ctx* c, const dp_config* cfg) {
  c->plan.resize(cfg->n_layers);
  uint64_t off = cfg->param_base;
  int64_t grads = 0, splits = 0, unf = 0;
  int64_t NP = 1;
  const bool bf16_cfg = cfg->dtype == DP_BF16;
  // Gram-form tensor-core layers per T (they share norm launches), for the
  // latency term of the AUTO choice
  std::map<int, int64_t> gram_layers;
  if (cfg->norm_mode == DP_NORM_AUTO && bf16_cfg) {
    for (int l = 0; l < cfg->n_layers; ++l) {
      const int T = layer_T(cfg, l);
      const int64_t di = cfg->layers[l].d_in, dd = cfg->layers[l].d_out;
      if (use_pergrad(cfg, T, di, dd)) continue;
      if (resolve_mode(DP_NORM_AUTO, T, di, dd) == DP_NORM_GHOST &&
          dpk::tc_ghost_supported(T, di, dd))
        ++gram_layers[T];
    }
  }
  const int sms = gram_layers.empty() ? 0 : dpk::device_sm_count();
  // Tiles of the tensor-core clipped-sum launch each layer shares when every
  // layer is summed in one batched call in layer order (consecutive layers of
  // one tile shape and T, up to kGemmMaxLayers per launch): a layer's example
  // split is chosen for that launch, then fixed.
  std::vector<int64_t> group_tiles(cfg->n_layers, 0);
  std::vector<std::vector<int>> groups;
  {
    std::vector<int> cur;
    auto close = [&]() {
      int64_t t = 0;
      for (int l : cur) t += dpk::tc_gemm_tiles(cfg->layers[l].d_in, cfg->layers[l].d_out);
      for (int l : cur) group_tiles[l] = t;
      if (!cur.empty()) groups.push_back(cur);
      cur.clear();
    };
    for (int l = 0; l < cfg->n_layers; ++l) {
      const int T = layer_T(cfg, l);
      const int64_t di = cfg->layers[l].d_in, dd = cfg->layers[l].d_out;
      if (!bf16_cfg || use_pergrad(cfg, T, di, dd) || !dpk::tc_gemm_supported(T, di, dd))
        continue;
      if (!cur.empty()) {
        const int f = cur[0];
        if (!dpk::tc_clipsum_same_launch(cfg->layers[f].d_in, cfg->layers[f].d_out, di, dd) ||
            layer_T(cfg, f) != T)
          close();
      }
      cur.push_back(l);
      if (static_cast<int>(cur.size()) == dpk::kGemmMaxLayers) close();
    }
    close();
  }
  for (int l = 0; l < cfg->n_layers; ++l) {
    LayerPlan& p = c->plan[l];
    p.d_in = cfg->layers[l].d_in;
    p.d_out = cfg->layers[l].d_out;
    p.T = layer_T(cfg, l);
    const int T = p.T;
    p.p_base = off;
    off += static_cast<uint64_t>(p.d_in) * p.d_out;
    p.pergrad = use_pergrad(cfg, T, p.d_in, p.d_out) ? 1 : 0;
    p.fused = 0;
    p.g_off = 0;
    p.split = 1;
    p.s_off = 0;
    p.tail_from = 0;
    p.tail_split = 1;
    p.noise_after = 0;
    p.kind = cfg->layers[l].kind;
    p.conv = p.kind == DP_LAYER_CONV2D ? 1 : 0;
    p.cg = dpk::ConvGeom{};
    p.implicit = 0;
    p.unfold = 0;
    p.u_off = 0;
    if (p.conv) {
      conv_geom(&cfg->convs[l], &p.cg);
      // a 1x1, stride-1, unpadded convolution's input already is its patch rows
      const bool identity = p.cg.kh == 1 && p.cg.kw == 1 && p.cg.stride_h == 1 &&
                            p.cg.stride_w == 1 && p.cg.pad_h == 0 && p.cg.pad_w == 0;
      if (identity) p.conv = 0;
    }
    auto need_unfold = [&]() {
      p.unfold = 1;
      p.u_off = unf;
      const int64_t bytes = static_cast<int64_t>(cfg->B) * T * p.d_in *
                            (cfg->dtype == DP_BF16 ? 2 : 4);
      unf += (bytes + 255) / 256 * 256;
    };
    if (p.pergrad) {
      p.mode = DP_NORM_MATERIALISED;
      p.norm_tc = 0;
      p.gemm_tc = 0;
      p.nparts = static_cast<int>(dpk::pergrad_parts(
          cfg->dtype == DP_BF16 ? dpk::IN_BF16 : dpk::IN_F32, p.d_in, p.d_out, T));
      p.g_off = grads;
      grads += static_cast<int64_t>(cfg->B) * p.d_in * p.d_out;
      if (p.conv && dpk::conv_thin_norm_ok(p.cg, p.d_out)) {
        p.fused = 1;
        p.nparts = 1;
      } else if (p.conv) {
        need_unfold();
      }
      if (p.nparts > NP) NP = p.nparts;
      continue;
    }
    p.mode = resolve_mode(cfg->norm_mode, T, p.d_in, p.d_out);
    const bool bf16 = cfg->dtype == DP_BF16;
    // the cost model picked the Gram form for examples so long that its
    // partial sums would not fit: the materialised form needs T-independent
    // partials
    if (cfg->norm_mode == DP_NORM_AUTO && p.mode == DP_NORM_GHOST &&
        !(bf16 && dpk::tc_ghost_supported(T, p.d_in, p.d_out)) &&
        dpk::ghost_simt_parts(T) > kMaxPartsPerExample)
      p.mode = DP_NORM_MATERIALISED;
    // the cost model picked the Gram form, but a side wider than the tensor
    // cores' accumulation bound keeps it off them: the materialised form on
    // tensor cores (reductions of length T) beats the Gram form on CUDA cores
    if (cfg->norm_mode == DP_NORM_AUTO && p.mode == DP_NORM_GHOST && bf16 &&
        !dpk::tc_ghost_supported(T, p.d_in, p.d_out) && dpk::tc_gemm_supported(T, p.d_in, p.d_out))
      p.mode = DP_NORM_MATERIALISED;
    // few Gram items on short examples: the latency of one item decides
    if (cfg->norm_mode == DP_NORM_AUTO && p.mode == DP_NORM_GHOST && bf16 &&
        dpk::tc_ghost_supported(T, p.d_in, p.d_out) &&
        dpk::tc_gemm_supported(T, p.d_in, p.d_out) &&
        gram_latency_prefers_materialised(cfg->B, T, p.d_in, p.d_out,
                                          static_cast<int64_t>(cfg->B) * gram_layers[T], sms))
      p.mode = DP_NORM_MATERIALISED;
    p.norm_tc = 0;
    int64_t parts = 1;
    if (p.mode == DP_NORM_RANK1) {
      parts = dpk::rank1_parts();
    } else if (p.mode == DP_NORM_GHOST) {
      p.norm_tc = bf16 && dpk::tc_ghost_supported(T, p.d_in, p.d_out);
      parts = p.norm_tc ? dpk::tc_ghost_parts(T) : dpk::ghost_simt_parts(T);
    } else {
      p.norm_tc = bf16 && dpk::tc_gemm_supported(T, p.d_in, p.d_out);
      parts = p.norm_tc ? dpk::tc_mat_parts(p.d_in, p.d_out)
                        : dpk::mat_simt_parts(p.d_in, p.d_out);
    }
    if (parts < 1 || parts > kMaxPartsPerExample)
      return fail(DP_ERR_SHAPE,
                  "layer %d: its norm form needs %lld partial sums per example (limit %lld)%s", l,
                  static_cast<long long>(parts), static_cast<long long>(kMaxPartsPerExample),
                  p.mode == DP_NORM_GHOST ? "; use DP_NORM_MATERIALISED for examples this long"
                                          : "");
    p.nparts = static_cast<int>(parts);
    p.gemm_tc = 0;
    if (bf16 && dpk::tc_gemm_supported(T, p.d_in, p.d_out)) {
      p.gemm_tc = 1;
      p.noise_after = static_cast<int64_t>(cfg->B) * T <= kNoiseAfterMaxK ? 1 : 0;
      p.split = dpk::tc_gemm_split(cfg->B, T, p.d_in, p.d_out,
                                   group_tiles[l] - dpk::tc_gemm_tiles(p.d_in, p.d_out));
      if (p.split > 1) {
        p.s_off = splits;
        splits += static_cast<int64_t>(p.split) * p.d_in * p.d_out;
      }
      // a convolution read in place: the materialised norm (the Gram kernel
      // has no implicit loads) unless the caller forced the Gram form
      if (p.conv && cfg->norm_mode != DP_NORM_GHOST && dpk::tc_conv_implicit_ok(p.cg, T)) {
        p.implicit = 1;
        p.mode = DP_NORM_MATERIALISED;
        p.norm_tc = 1;
        p.nparts = static_cast<int>(dpk::tc_mat_parts(p.d_in, p.d_out));
      }
    } else if (bf16 && dpk::tc_prescaled_supported(cfg->B, T, p.d_in, p.d_out)) {
      p.gemm_tc = 2;
      p.noise_after = static_cast<int64_t>(cfg->B) * T <= kNoiseAfterMaxK ? 1 : 0;
      const int64_t need = dpk::tc_prescaled_scratch_bytes(cfg->B, T, p.d_in);
      if (need > c->prescaled_bytes) c->prescaled_bytes = need;
    }
    if (p.conv && !p.implicit) need_unfold();
    if (p.nparts > NP) NP = p.nparts;
  }
  // the last round of each launch group of tensor-core clipped sums
  for (const std::vector<int>& grp : groups) {
    bool ok = grp.size() <= static_cast<size_t>(dpk::kGemmMaxLayers);
    for (int l : grp) ok = ok && c->plan[l].gemm_tc == 1 && c->plan[l].split == 1;
    if (!ok) continue;
    int64_t di[dpk::kGemmMaxLayers], dd[dpk::kGemmMaxLayers];
    int tf[dpk::kGemmMaxLayers], ts[dpk::kGemmMaxLayers];
    for (size_t q = 0; q < grp.size(); ++q) {
      di[q] = c->plan[grp[q]].d_in;
      dd[q] = c->plan[grp[q]].d_out;
    }
    dpk::tc_plan_tail(static_cast<int>(grp.size()), di, dd, cfg->B, tf, ts);
    for (size_t q = 0; q < grp.size(); ++q) {
      c->plan[grp[q]].tail_from = tf[q];
      c->plan[grp[q]].tail_split = ts[q];
    }
  }
  // the partial buffer [L][B][NP] and the row index layer * B + example
  if (static_cast<double>(cfg->n_layers) * cfg->B > 0x7fffffff ||
      static_cast<double>(cfg->n_layers) * cfg->B * NP * 4.0 > 0x1p50)
    return fail(DP_ERR_SHAPE, "L * B * partial sums per example too large for the norm scratch");
  c->NP = static_cast<int>(NP);
  c->grads_floats = grads;
  c->split_floats = splits;
  c->tail_bytes = 0;
  for (const LayerPlan& p : c->plan)
    if (p.gemm_tc == 1) c->tail_bytes = dpk::tc_tail_scratch_bytes();
  c->unf_bytes = unf;
  return DP_OK;
}

void free_scratch(dp_ctx* c) {
  cudaFree(c->d_part);
  cudaFree(c->d_nparts);
  cudaFree(c->d_layer_sq);
  cudaFree(c->d_s);
  cudaFree(c->d_c);
  cudaFree(c->d_flag);
  cudaFreeHost(c->h_idx);
  cudaFreeHost(c->h_rec);
  cudaFreeHost(c->h_flag);
  cudaFree(c->d_prescaled);
  cudaFree(c->d_grads);
  cudaFree(c->d_split);
  cudaFree(c->d_tail);
  cudaFree(c->d_unf);
  c->d_prescaled = nullptr;
  c->d_grads = nullptr;
  c->d_split = nullptr;
  c->d_tail = nullptr;
  c->d_unf = nullptr;
  cudaFree(c->d_key);
  cudaFreeHost(c->h_key);
  c->d_key = nullptr;
  c->h_key = nullptr;
  c->h_key_dev = nullptr;
  c->d_part = nullptr;
  c->d_nparts = nullptr;
  c->d_layer_sq = c->d_s = c->d_c = nullptr;
  c->d_flag = nullptr;
  c->h_idx = nullptr;
  c->h_rec = nullptr;
  c->h_flag = nullptr;
}

dp_status alloc_scratch(dp_ctx* c) {
  const int L = c->L, B = c->B;
  const int cap = c->B;  // audit staging sized for the whole batch
  c->part_bytes = sizeof(float) * static_cast<size_t>(L) * B * c->NP;
#define DP_ALLOC(ptr, bytes)                                                           \
  do {                                                                                 \
    if (cudaMalloc(reinterpret_cast<void**>(&(ptr)), (bytes)) != cudaSuccess) {        \
      cudaGetLastError();                                                              \
      free_scratch(c);                                                                 \
      return fail(DP_ERR_OOM, "cudaMalloc of %zu bytes failed", size_t(bytes));        \
    }                                                                                  \
  } while (0)
  DP_ALLOC(c->d_part, c->part_bytes);
  DP_ALLOC(c->d_nparts, sizeof(int) * L);
  DP_ALLOC(c->d_layer_sq, sizeof(float) * L * B);
  DP_ALLOC(c->d_s, sizeof(float) * B);
  DP_ALLOC(c->d_c, sizeof(float) * B);
  DP_ALLOC(c->d_flag, sizeof(int));
  if (c->prescaled_bytes > 0) DP_ALLOC(c->d_prescaled, static_cast<size_t>(c->prescaled_bytes));
  if (c->grads_floats > 0) DP_ALLOC(c->d_grads, sizeof(float) * static_cast<size_t>(c->grads_floats));
  if (c->split_floats > 0) DP_ALLOC(c->d_split, sizeof(float) * static_cast<size_t>(c->split_floats));
  if (c->tail_bytes > 0) DP_ALLOC(c->d_tail, static_cast<size_t>(c->tail_bytes));
  if (c->unf_bytes > 0) DP_ALLOC(c->d_unf, static_cast<size_t>(c->unf_bytes));
  DP_ALLOC(c->d_key, 2 * sizeof(uint64_t));
#undef DP_ALLOC
  if (cudaHostAlloc(reinterpret_cast<void**>(&c->h_idx), sizeof(int) * (cap > 0 ? cap : 1),
                    cudaHostAllocMapped) != cudaSuccess ||
      cudaHostAlloc(reinterpret_cast<void**>(&c->h_rec),
                    sizeof(float) * (cap > 0 ? cap : 1) * (3 + L), cudaHostAllocMapped) !=
          cudaSuccess ||
      cudaHostAlloc(reinterpret_cast<void**>(&c->h_flag), sizeof(int), cudaHostAllocMapped) !=
          cudaSuccess ||
      cudaHostGetDevicePointer(reinterpret_cast<void**>(&c->h_idx_dev), c->h_idx, 0) !=
          cudaSuccess ||
      cudaHostGetDevicePointer(reinterpret_cast<void**>(&c->h_rec_dev), c->h_rec, 0) !=
          cudaSuccess ||
      cudaHostGetDevicePointer(reinterpret_cast<void**>(&c->h_flag_dev), c->h_flag, 0) !=
          cudaSuccess ||
      cudaHostAlloc(reinterpret_cast<void**>(&c->h_key), 2 * sizeof(uint64_t),
                    cudaHostAllocMapped) != cudaSuccess ||
      cudaHostGetDevicePointer(reinterpret_cast<void**>(&c->h_key_dev), c->h_key, 0) !=
          cudaSuccess) {
    cudaGetLastError();
    free_scratch(c);
    return fail(DP_ERR_OOM, "pinned host allocation failed");
  }
  return DP_OK;
}

dp_status upload_plan(dp_ctx* c) {
  // Pageable-source copy: returns once the source has been staged, so the
  // vector may go out of scope without a stream synchronisation.
  std::vector<int> np(c->L);
  for (int l = 0; l < c->L; ++l) np[l] = c->plan[l].nparts;
  DP_CUDA(cudaMemcpyAsync(c->d_nparts, np.data(), sizeof(int) * c->L, cudaMemcpyHostToDevice,
                          c->stream));
  return DP_OK;
}

bool same_parts(const std::vector<LayerPlan>& a, const std::vector<LayerPlan>& b) {
  if (a.size() != b.size()) return false;
  for (size_t l = 0; l < a.size(); ++l)
    if (a[l].nparts != b[l].nparts) return false;
  return true;
}

// Load the key words into device memory on the context's stream and clear
// the sticky flag, with a one-thread kernel (a step issues no copy or memset
// of its own, so nothing of it queues behind bulk host copies on the copy
// engines).  Eager: the key is a kernel argument.  Under stream capture the
// kernel reads the mapped pinned words when it runs instead, so a replay of
// the captured step uses the key current at replay time (the capture's key
// until dp_set_noise_key replaces it); an eager step leaves those words alone.
dp_status upload_key(dp_ctx* c) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  DP_CUDA(cudaStreamIsCapturing(c->stream, &cs));
  if (cs == cudaStreamCaptureStatusActive) {
    c->h_key[0] = c->seed;
    c->h_key[1] = c->step;
    DP_CUDA(dpk::launch_load_key(c->h_key_dev, c->d_key, c->d_flag, c->stream));
  } else {
    DP_CUDA(dpk::launch_set_key(c->seed, c->step, c->d_key, c->d_flag, c->stream));
  }
  return DP_OK;
}

void reset_step(dp_ctx* c) {
  c->norm_done.assign(c->L, 0);
  c->clip_done = false;
}

void set_scalars(dp_ctx* c, const dp_config* cfg, void* stream) {
  c->C = cfg->clip_C;
  c->sigma = cfg->sigma;
  c->out_scale = cfg->out_scale;
  c->seed = cfg->seed;
  c->step = cfg->step;
  c->norm_mode = cfg->norm_mode;
  c->audit_capacity = cfg->audit_capacity;
  c->stream = static_cast<cudaStream_t>(stream);
}

dp_status check_device() {
  int dev = 0;
  DP_CUDA(cudaGetDevice(&dev));
  int major = 0, minor = 0;
  DP_CUDA(cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev));
  DP_CUDA(cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev));
  if (major != 10 || minor != 3)
    return fail(DP_ERR_UNSUPPORTED, "device %d is sm_%d%d; this library is built for sm_103a",
                dev, major, minor);
  return DP_OK;
}

dp_status check_norm_args(dp_ctx* c, int32_t layer, const void* A, const void* D) {
  if (layer < 0 || layer >= c->L) return fail(DP_ERR_ARG, "layer %d out of range", layer);
  if (!A || !D) return fail(DP_ERR_ARG, "A or D is NULL");
  if (!aligned16(A) || !aligned16(D)) return fail(DP_ERR_ARG, "A and D must be 16-byte aligned");
  if (c->clip_done) return fail(DP_ERR_ORDER, "dp_layer_norms after dp_clip_factors");
  return DP_OK;
}

// The A the dense kernels read for a layer: a convolution's patch rows in
// context scratch when they are formed there, else the caller's array.
const void* dense_A(const dp_ctx* c, int32_t layer, const void* A) {
  const LayerPlan& p = c->plan[layer];
  return p.unfold ? static_cast<const void*>(c->d_unf + p.u_off) : A;
}

cudaError_t unfold_layer(dp_ctx* c, int32_t layer, const void* X) {
  const LayerPlan& p = c->plan[layer];
  return dpk::launch_conv_unfold(c->dtype == DP_BF16 ? dpk::IN_BF16 : dpk::IN_F32, X,
                                 c->d_unf + p.u_off, p.cg, c->B, c->stream);
}

void fill_pergrad(const dp_ctx* c, int32_t layer, const void* A, const void* D,
                  dpk::PerGradLayer& P) {
  const LayerPlan& p = c->plan[layer];
  P.wide_is_in = p.d_in >= p.d_out ? 1 : 0;
  P.X = P.wide_is_in ? A : D;
  P.Y = P.wide_is_in ? D : A;
  P.n = static_cast<int>(P.wide_is_in ? p.d_in : p.d_out);
  P.r = static_cast<int>(P.wide_is_in ? p.d_out : p.d_in);
  P.G = c->d_grads + p.g_off;
  P.row0 = layer * c->B;
}

void fill_pergrad_sum(const dp_ctx* c, int32_t layer, float* d_out, dpk::PerGradSumLayer& P) {
  const LayerPlan& p = c->plan[layer];
  P.G = c->d_grads + p.g_off;
  P.out = d_out;
  P.count = p.d_in * p.d_out;
  P.p_base = p.p_base;
}

dpk::PerGradSumBatch pergrad_sum_batch(const dp_ctx* c, uint32_t flags) {
  dpk::PerGradSumBatch g{};
  g.c = c->d_c;
  g.key = c->d_key;
  g.out_scale = c->out_scale;
  g.sigmaC = c->sigma * c->C;
  g.add_noise = (flags & DP_NO_NOISE) ? 0 : 1;
  g.accumulate = (flags & DP_ACCUMULATE) ? 1 : 0;
  g.B = c->B;
  return g;
}

cudaError_t launch_layer_norms(dp_ctx* c, int32_t layer, const void* A, const void* D) {
  const LayerPlan& p = c->plan[layer];
  const dpk::InType it = c->dtype == DP_BF16 ? dpk::IN_BF16 : dpk::IN_F32;
  if (p.fused)
    return dpk::launch_conv_thin_norm(it, A, D, p.cg, static_cast<int>(p.d_out), c->B,
                                      c->d_grads + p.g_off, c->d_part, c->NP, layer * c->B,
                                      c->stream);
  if (p.pergrad) {
    dpk::PerGradBatch g{};
    fill_pergrad(c, layer, A, D, g.l[0]);
    g.L = 1;
    g.part = c->d_part;
    g.err = c->d_flag;
    g.B = c->B;
    g.T = p.T;
    g.NP = c->NP;
    return dpk::launch_pergrad_norm(it, g, c->stream);
  }
  const int din = static_cast<int>(p.d_in), dout = static_cast<int>(p.d_out);
  const int row0 = layer * c->B;
  if (p.mode == DP_NORM_RANK1)
    return dpk::launch_norm_rank1(it, A, D, c->B, din, dout, c->d_part, c->NP, row0, c->stream);
  if (p.mode == DP_NORM_GHOST)
    return p.norm_tc ? dpk::tc_launch_ghost(A, D, c->B, p.T, din, dout, c->d_part, c->NP, row0,
                                            c->d_flag, c->stream)
                     : dpk::launch_norm_ghost_simt(it, A, D, c->B, p.T, din, dout, c->d_part,
                                                   c->NP, row0, c->stream);
  return p.norm_tc ? dpk::tc_launch_mat_norm(A, D, c->B, p.T, din, dout, c->d_part, c->NP, row0,
                                             c->d_flag, c->stream, p.implicit ? &p.cg : nullptr)
                   : dpk::launch_norm_mat_simt(it, A, D, c->B, p.T, din, dout, c->d_part, c->NP,
                                               row0, c->stream);
}

dp_status check_sum_args(dp_ctx* c, int32_t layer, const void* A, const void* D,
                         const float* d_out, uint32_t flags) {
  if (layer < 0 || layer >= c->L) return fail(DP_ERR_ARG, "layer %d out of range", layer);
  if (flags & ~(DP_NO_NOISE | DP_NOISE_ONLY | DP_ACCUMULATE))
    return fail(DP_ERR_ARG, "unknown flag bits 0x%x", flags);
  if ((flags & DP_NO_NOISE) && (flags & DP_NOISE_ONLY))
    return fail(DP_ERR_ARG, "DP_NO_NOISE and DP_NOISE_ONLY are exclusive");
  if (!d_out) return fail(DP_ERR_ARG, "d_out is NULL");
  if (!aligned16(d_out)) return fail(DP_ERR_ARG, "d_out must be 16-byte aligned");
  if (flags & DP_NOISE_ONLY) return DP_OK;
  if (!A || !D) return fail(DP_ERR_ARG, "A or D is NULL");
  if (!aligned16(A) || !aligned16(D)) return fail(DP_ERR_ARG, "A and D must be 16-byte aligned");
  if (!c->clip_done) return fail(DP_ERR_ORDER, "dp_clipped_sum_noise before dp_clip_factors");
  return DP_OK;
}

dpk::Epilogue make_epilogue(const dp_ctx* c, uint32_t flags, uint64_t p_base) {
  dpk::Epilogue ep{};
  ep.key = c->d_key;
  ep.p_base = p_base;
  ep.out_scale = c->out_scale;
  ep.sigmaC = c->sigma * c->C;
  ep.add_noise = (flags & DP_NO_NOISE) ? 0 : 1;
  ep.accumulate = (flags & DP_ACCUMULATE) ? 1 : 0;
  return ep;
}

// out_l += out_scale sigma C z over every parameter of layers[0 .. n), in
// launches of up to kNoiseMaxLayers layers (the DP_NOISE_ONLY arithmetic).
cudaError_t launch_noise_layers(dp_ctx* c, int n, const int32_t* layers, float* const* d_out) {
  dpk::NoiseAddBatch nb{};
  nb.key = c->d_key;
  nb.scale = c->out_scale * (c->sigma * c->C);
  for (int r = 0; r < n; ++r) {
    const LayerPlan& p = c->plan[layers[r]];
    nb.out[nb.L] = d_out[r];
    nb.n[nb.L] = p.d_in * p.d_out;
    nb.p_base[nb.L] = p.p_base;
    if (++nb.L == dpk::kNoiseMaxLayers || r == n - 1) {
      cudaError_t e = dpk::launch_noise_add(nb, c->stream);
      if (e != cudaSuccess) return e;
      nb.L = 0;
    }
  }
  return cudaSuccess;
}

cudaError_t launch_clipped_sum(dp_ctx* c, int32_t layer, const void* A, const void* D,
                               float* d_out, uint32_t flags) {
  const LayerPlan& p = c->plan[layer];
  const dpk::Epilogue ep = make_epilogue(c, flags, p.p_base);
  if (flags & DP_NOISE_ONLY) return launch_noise_layers(c, 1, &layer, &d_out);
  if (p.pergrad) {
    dpk::PerGradSumBatch g = pergrad_sum_batch(c, flags);
    fill_pergrad_sum(c, layer, d_out, g.l[0]);
    g.L = 1;
    return dpk::launch_pergrad_sum(g, c->stream);
  }
  A = dense_A(c, layer, A);
  const int din = static_cast<int>(p.d_in), dout = static_cast<int>(p.d_out);
  if (p.gemm_tc == 1) {
    const bool after = p.noise_after && ep.add_noise;
    dpk::Epilogue eg = ep;
    if (after) eg.add_noise = 0;
    cudaError_t e = dpk::tc_launch_clipsum(
        A, D, c->d_c, c->B, p.T, din, dout, p.split, d_out,
        p.split > 1 ? c->d_split + p.s_off : nullptr, eg, c->d_flag, c->stream,
        p.implicit ? &p.cg : nullptr, p.tail_from, p.tail_split, c->d_tail, c->tail_bytes);
    if (e != cudaSuccess || !after) return e;
    return launch_noise_layers(c, 1, &layer, &d_out);
  }
  if (p.gemm_tc == 2) {
    const bool after = p.noise_after && ep.add_noise;
    dpk::Epilogue eg = ep;
    if (after) eg.add_noise = 0;
    cudaError_t e = dpk::tc_launch_clipsum_prescaled(A, D, c->d_c, c->B, p.T, din, dout, d_out,
                                                     eg, c->d_flag, c->d_prescaled, c->stream);
    if (e != cudaSuccess || !after) return e;
    return launch_noise_layers(c, 1, &layer, &d_out);
  }
  return dpk::launch_gemm_simt(c->dtype == DP_BF16 ? dpk::IN_BF16 : dpk::IN_F32, A, D, c->d_c,
                               c->B, p.T, din, dout, d_out, ep, c->stream);
}

}  // namespace

extern "C" {

dp_status dp_step_init(dp_ctx** ctx, const dp_config* cfg, void* cuda_stream) {
  if (!ctx) return fail(DP_ERR_ARG, "ctx is NULL");
  dp_status st = check_config(cfg);
  if (st != DP_OK) return st;
  if (*ctx) {
    dp_ctx* c = *ctx;
    bool same = c->B == cfg->B && c->T == cfg->T && c->L == cfg->n_layers &&
                c->dtype == cfg->dtype;
    for (int l = 0; same && l < c->L; ++l) {
      same = c->plan[l].d_in == cfg->layers[l].d_in && c->plan[l].d_out == cfg->layers[l].d_out &&
             c->plan[l].T == layer_T(cfg, l) && c->plan[l].kind == cfg->layers[l].kind;
      if (same && cfg->layers[l].kind == DP_LAYER_CONV2D) {
        dpk::ConvGeom g{};
        conv_geom(&cfg->convs[l], &g);
        same = std::memcmp(&g, &c->plan[l].cg, sizeof g) == 0 || !c->plan[l].conv;
      }
    }
    if (!same) return fail(DP_ERR_SHAPE, "re-key with different shapes; destroy and re-create");
    // The norm mode may change; the partial buffer must still be large enough.
    std::vector<LayerPlan> old = c->plan;
    const int oldNP = c->NP;
    const int64_t old_pre = c->prescaled_bytes;
    const int64_t old_grads = c->grads_floats;
    const int64_t old_splits = c->split_floats;
    const int64_t old_unf = c->unf_bytes;
    st = build_plan(c, cfg);
    if (st != DP_OK) {
      c->plan = old;
      c->NP = oldNP;
      c->prescaled_bytes = old_pre;
      c->grads_floats = old_grads;
      c->split_floats = old_splits;
      c->unf_bytes = old_unf;
      return st;
    }
    c->prescaled_bytes = old_pre;  // shapes are unchanged, so is the pre-scale need
    if (c->NP > oldNP || c->grads_floats > old_grads || c->split_floats > old_splits ||
        c->unf_bytes > old_unf) {
      c->plan = old;
      c->NP = oldNP;
      c->grads_floats = old_grads;
      c->split_floats = old_splits;
      c->unf_bytes = old_unf;
      return fail(DP_ERR_SHAPE, "norm_mode change needs more scratch; destroy and re-create");
    }
    c->NP = oldNP;  // keep the allocated stride
    c->grads_floats = old_grads;
    c->split_floats = old_splits;
    c->unf_bytes = old_unf;
    set_scalars(c, cfg, cuda_stream);
    if (!same_parts(old, c->plan)) {
      st = upload_plan(c);
      if (st != DP_OK) return st;
    }
    // the key kernel also clears the sticky flag: it reports this step only
    st = upload_key(c);
    if (st != DP_OK) return st;
    reset_step(c);
    return DP_OK;
  }
  st = check_device();
  if (st != DP_OK) return st;
  dp_ctx* c = new dp_ctx();
  c->B = cfg->B;
  c->T = cfg->T;
  c->L = cfg->n_layers;
  c->dtype = cfg->dtype;
  cudaGetDevice(&c->device);
  set_scalars(c, cfg, cuda_stream);
  st = build_plan(c, cfg);
  if (st != DP_OK) {
    delete c;
    return st;
  }
  st = alloc_scratch(c);
  if (st != DP_OK) {
    delete c;
    return st;
  }
  st = upload_plan(c);
  if (st == DP_OK) st = upload_key(c);
  if (st != DP_OK) {
    free_scratch(c);
    delete c;
    return st;
  }
  reset_step(c);
  *ctx = c;
  return DP_OK;
}

dp_status dp_layer_norms(dp_ctx* c, int32_t layer, const void* A, const void* D) {
  if (!c) return fail(DP_ERR_ARG, "ctx is NULL");
  dp_status st = check_norm_args(c, layer, A, D);
  if (st != DP_OK) return st;
  cudaError_t e = c->plan[layer].unfold ? unfold_layer(c, layer, A) : cudaSuccess;
  if (e == cudaSuccess) e = launch_layer_norms(c, layer, dense_A(c, layer, A), D);
  if (e != cudaSuccess) return fail(DP_ERR_CUDA, "norm kernel launch: %s", cudaGetErrorString(e));
  c->norm_done[layer] = 1;
  return DP_OK;
}

dp_status dp_layer_norms_batch(dp_ctx* c, int32_t n, const int32_t* layers, const void* const* A,
                               const void* const* D) {
  if (!c) return fail(DP_ERR_ARG, "ctx is NULL");
  if (n < 1 || n > c->L) return fail(DP_ERR_ARG, "n=%d outside 1..L", n);
  if (!layers || !A || !D) return fail(DP_ERR_ARG, "NULL array argument");
  std::vector<char> seen(c->L, 0);
  for (int r = 0; r < n; ++r) {
    dp_status st = check_norm_args(c, layers[r], A[r], D[r]);
    if (st != DP_OK) return st;
    if (seen[layers[r]]) return fail(DP_ERR_ARG, "layer %d listed twice", layers[r]);
    seen[layers[r]] = 1;
  }
  // convolutions whose patch rows are formed in scratch: form them first;
  // from here on A is what the dense kernels read
  std::vector<const void*> Ad(n);
  for (int r = 0; r < n; ++r) {
    if (c->plan[layers[r]].unfold) {
      cudaError_t e = unfold_layer(c, layers[r], A[r]);
      if (e != cudaSuccess) return fail(DP_ERR_CUDA, "unfold kernel: %s", cudaGetErrorString(e));
    }
    Ad[r] = dense_A(c, layers[r], A[r]);
  }
  // Gram-form tensor-core layers share launches (up to kGhostMaxLayers each);
  // every other layer gets its own kernel.
  std::vector<int> grp;
  auto flush = [&]() -> cudaError_t {
    if (grp.empty()) return cudaSuccess;
    const void* a[dpk::kGhostMaxLayers];
    const void* d[dpk::kGhostMaxLayers];
    int din[dpk::kGhostMaxLayers], dout[dpk::kGhostMaxLayers], row0[dpk::kGhostMaxLayers];
    for (size_t q = 0; q < grp.size(); ++q) {
      const int r = grp[q], l = layers[r];
      a[q] = Ad[r];
      d[q] = D[r];
      din[q] = static_cast<int>(c->plan[l].d_in);
      dout[q] = static_cast<int>(c->plan[l].d_out);
      row0[q] = l * c->B;
    }
    cudaError_t e = dpk::tc_launch_ghost_batch(static_cast<int>(grp.size()), a, d, din, dout, row0,
                                               c->B, c->plan[layers[grp[0]]].T, c->d_part, c->NP,
                                               c->d_flag, c->stream);
    grp.clear();
    return e;
  };
  // Thin layers share launches too, one list per (narrow-width bucket, T).
  const dpk::InType it = c->dtype == DP_BF16 ? dpk::IN_BF16 : dpk::IN_F32;
  std::map<std::pair<int, int>, std::vector<int>> thin;
  auto flush_thin = [&](std::vector<int>& v) -> cudaError_t {
    if (v.empty()) return cudaSuccess;
    dpk::PerGradBatch g{};
    for (size_t q = 0; q < v.size(); ++q) fill_pergrad(c, layers[v[q]], Ad[v[q]], D[v[q]], g.l[q]);
    g.L = static_cast<int>(v.size());
    g.part = c->d_part;
    g.err = c->d_flag;
    g.B = c->B;
    g.T = c->plan[layers[v[0]]].T;
    g.NP = c->NP;
    v.clear();
    return dpk::launch_pergrad_norm(it, g, c->stream);
  };
  for (int r = 0; r < n; ++r) {
    const LayerPlan& p = c->plan[layers[r]];
    cudaError_t e = cudaSuccess;
    if (p.fused) {
      e = launch_layer_norms(c, layers[r], Ad[r], D[r]);
    } else if (p.pergrad) {
      const int nar = static_cast<int>(p.d_in < p.d_out ? p.d_in : p.d_out);
      std::vector<int>& v = thin[std::make_pair(dpk::pergrad_bucket(nar), p.T)];
      v.push_back(r);
      if (static_cast<int>(v.size()) == dpk::kPerGradMaxLayers) e = flush_thin(v);
    } else if (p.mode == DP_NORM_GHOST && p.norm_tc) {
      if (!grp.empty() && c->plan[layers[grp[0]]].T != p.T) e = flush();
      grp.push_back(r);
      if (static_cast<int>(grp.size()) == dpk::kGhostMaxLayers) e = flush();
    } else {
      e = launch_layer_norms(c, layers[r], Ad[r], D[r]);
    }
    if (e != cudaSuccess)
      return fail(DP_ERR_CUDA, "norm kernel launch: %s", cudaGetErrorString(e));
  }
  cudaError_t e = flush();
  for (auto it2 = thin.begin(); it2 != thin.end() && e == cudaSuccess; ++it2)
    e = flush_thin(it2->second);
  if (e != cudaSuccess) return fail(DP_ERR_CUDA, "norm kernel launch: %s", cudaGetErrorString(e));
  for (int r = 0; r < n; ++r) c->norm_done[layers[r]] = 1;
  return DP_OK;
}

dp_status dp_clip_factors(dp_ctx* c, float* d_sqnorm_out, float* d_clip_out) {
  if (!c) return fail(DP_ERR_ARG, "ctx is NULL");
  for (int l = 0; l < c->L; ++l)
    if (!c->norm_done[l]) return fail(DP_ERR_ORDER, "norms of layer %d not computed", l);
  if (c->clip_done) return fail(DP_ERR_ORDER, "dp_clip_factors already called this step");
  cudaError_t e = dpk::launch_clip(c->d_part, c->L, c->B, c->NP, c->d_nparts, c->C,
                                   c->d_layer_sq, c->d_s, c->d_c, d_sqnorm_out, d_clip_out,
                                   c->d_flag, c->stream);
  if (e != cudaSuccess) return fail(DP_ERR_CUDA, "clip kernel launch: %s", cudaGetErrorString(e));
  c->clip_done = true;
  return DP_OK;
}

dp_status dp_partial_sqnorms(dp_ctx* c, float* d_sqnorm_local) {
  if (!c) return fail(DP_ERR_ARG, "ctx is NULL");
  if (!d_sqnorm_local) return fail(DP_ERR_ARG, "d_sqnorm_local is NULL");
  for (int l = 0; l < c->L; ++l)
    if (!c->norm_done[l]) return fail(DP_ERR_ORDER, "norms of layer %d not computed", l);
  if (c->clip_done) return fail(DP_ERR_ORDER, "dp_partial_sqnorms after dp_clip_factors");
  cudaError_t e = dpk::launch_clip(c->d_part, c->L, c->B, c->NP, c->d_nparts, c->C,
                                   c->d_layer_sq, c->d_s, c->d_c, d_sqnorm_local, nullptr,
                                   c->d_flag, c->stream, dpk::kClipLocal, nullptr);
  if (e != cudaSuccess) return fail(DP_ERR_CUDA, "clip kernel launch: %s", cudaGetErrorString(e));
  return DP_OK;
}

dp_status dp_clip_factors_from(dp_ctx* c, const float* d_sqnorm_total, float* d_sqnorm_out,
                               float* d_clip_out) {
  if (!c) return fail(DP_ERR_ARG, "ctx is NULL");
  if (!d_sqnorm_total) return fail(DP_ERR_ARG, "d_sqnorm_total is NULL");
  for (int l = 0; l < c->L; ++l)
    if (!c->norm_done[l]) return fail(DP_ERR_ORDER, "norms of layer %d not computed", l);
  if (c->clip_done) return fail(DP_ERR_ORDER, "dp_clip_factors already called this step");
  cudaError_t e = dpk::launch_clip(c->d_part, c->L, c->B, c->NP, c->d_nparts, c->C,
                                   c->d_layer_sq, c->d_s, c->d_c, d_sqnorm_out, d_clip_out,
                                   c->d_flag, c->stream, dpk::kClipGiven, d_sqnorm_total);
  if (e != cudaSuccess) return fail(DP_ERR_CUDA, "clip kernel launch: %s", cudaGetErrorString(e));
  c->clip_done = true;
  return DP_OK;
}

dp_status dp_noise_add_range(dp_ctx* c, uint64_t p_first, int64_t n, float* d_out) {
  if (!c) return fail(DP_ERR_ARG, "ctx is NULL");
  if (n < 0) return fail(DP_ERR_ARG, "n < 0");
  if (n == 0) return DP_OK;
  if (!d_out) return fail(DP_ERR_ARG, "d_out is NULL");
  if (!aligned16(d_out)) return fail(DP_ERR_ARG, "d_out must be 16-byte aligned");
  dpk::NoiseAddBatch nb{};
  nb.key = c->d_key;
  nb.scale = c->out_scale * (c->sigma * c->C);
  nb.out[0] = d_out;
  nb.n[0] = n;
  nb.p_base[0] = p_first;
  nb.L = 1;
  cudaError_t e = dpk::launch_noise_add(nb, c->stream);
  if (e != cudaSuccess) return fail(DP_ERR_CUDA, "noise kernel: %s", cudaGetErrorString(e));
  return DP_OK;
}

dp_status dp_clipped_sum_noise(dp_ctx* c, int32_t layer, const void* A, const void* D,
                               float* d_out, uint32_t flags) {
  if (!c) return fail(DP_ERR_ARG, "ctx is NULL");
  dp_status st = check_sum_args(c, layer, A, D, d_out, flags);
  if (st != DP_OK) return st;
  cudaError_t e = launch_clipped_sum(c, layer, A, D, d_out, flags);
  if (e != cudaSuccess) return fail(DP_ERR_CUDA, "clipped-sum kernel: %s", cudaGetErrorString(e));
  return DP_OK;
}

dp_status dp_clipped_sum_noise_batch(dp_ctx* c, int32_t n, const int32_t* layers,
                                     const void* const* A, const void* const* D,
                                     float* const* d_out, uint32_t flags) {
  if (!c) return fail(DP_ERR_ARG, "ctx is NULL");
  if (n < 1 || n > c->L) return fail(DP_ERR_ARG, "n=%d outside 1..L", n);
  if (!layers || !d_out || (!(flags & DP_NOISE_ONLY) && (!A || !D)))
    return fail(DP_ERR_ARG, "NULL array argument");
  std::vector<char> seen(c->L, 0);
  for (int r = 0; r < n; ++r) {
    const int32_t l = layers[r];
    dp_status st = check_sum_args(c, l, (flags & DP_NOISE_ONLY) ? nullptr : A[r],
                                  (flags & DP_NOISE_ONLY) ? nullptr : D[r], d_out[r], flags);
    if (st != DP_OK) return st;
    if (seen[l]) return fail(DP_ERR_ARG, "layer %d listed twice", l);
    seen[l] = 1;
  }
  // Direct tensor-core layers with the same tile shape share launches (up to
  // kGemmMaxLayers each); every other layer gets its own kernel.
  std::vector<int> grp;
  dpk::Epilogue ep = make_epilogue(c, flags, 0);
  // noise only: every listed layer in one launch (up to kNoiseMaxLayers each)
  if (flags & DP_NOISE_ONLY) {
    cudaError_t e = launch_noise_layers(c, n, layers, d_out);
    if (e != cudaSuccess) return fail(DP_ERR_CUDA, "noise kernel: %s", cudaGetErrorString(e));
    return DP_OK;
  }
  // thin layers: one summing launch over their stored per-example gradients
  std::vector<int> thin;
  auto flush_thin = [&]() -> cudaError_t {
    if (thin.empty()) return cudaSuccess;
    dpk::PerGradSumBatch g = pergrad_sum_batch(c, flags);
    for (size_t q = 0; q < thin.size(); ++q)
      fill_pergrad_sum(c, layers[thin[q]], d_out[thin[q]], g.l[q]);
    g.L = static_cast<int>(thin.size());
    thin.clear();
    return dpk::launch_pergrad_sum(g, c->stream);
  };
  auto flush = [&]() -> cudaError_t {
    if (grp.empty()) return cudaSuccess;
    const void* a[dpk::kGemmMaxLayers];
    const void* d[dpk::kGemmMaxLayers];
    float* o[dpk::kGemmMaxLayers];
    float* part[dpk::kGemmMaxLayers];
    const dpk::ConvGeom* cg[dpk::kGemmMaxLayers];
    int din[dpk::kGemmMaxLayers], dout[dpk::kGemmMaxLayers];
    uint64_t pb[dpk::kGemmMaxLayers];
    int sp[dpk::kGemmMaxLayers], tf[dpk::kGemmMaxLayers], ts[dpk::kGemmMaxLayers];
    for (size_t q = 0; q < grp.size(); ++q) {
      const int r = grp[q];
      const LayerPlan& p = c->plan[layers[r]];
      sp[q] = p.split;
      a[q] = dense_A(c, layers[r], A[r]);
      d[q] = D[r];
      o[q] = d_out[r];
      part[q] = p.split > 1 ? c->d_split + p.s_off : nullptr;
      cg[q] = p.implicit ? &p.cg : nullptr;
      din[q] = static_cast<int>(p.d_in);
      dout[q] = static_cast<int>(p.d_out);
      pb[q] = p.p_base;
      tf[q] = p.tail_from;
      ts[q] = p.tail_split;
    }
    // the group shares B and T, hence noise_after
    const bool after = c->plan[layers[grp[0]]].noise_after && ep.add_noise;
    dpk::Epilogue eg = ep;
    if (after) eg.add_noise = 0;
    cudaError_t e = dpk::tc_launch_clipsum_batch(static_cast<int>(grp.size()), a, d, o, part, din,
                                                 dout, pb, sp, c->d_c, c->B,
                                                 c->plan[layers[grp[0]]].T, eg, c->d_flag,
                                                 c->stream, cg, tf, ts, c->d_tail,
                                                 c->tail_bytes);
    if (e == cudaSuccess && after) {
      int32_t ls[dpk::kGemmMaxLayers];
      for (size_t q = 0; q < grp.size(); ++q) ls[q] = layers[grp[q]];
      e = launch_noise_layers(c, static_cast<int>(grp.size()), ls, o);
    }
    grp.clear();
    return e;
  };
  for (int r = 0; r < n; ++r) {
    const int32_t l = layers[r];
    const LayerPlan& p = c->plan[l];
    cudaError_t e = cudaSuccess;
    if (!(flags & DP_NOISE_ONLY) && p.gemm_tc == 1) {
      const LayerPlan& p0 = c->plan[layers[grp.empty() ? r : grp[0]]];
      if (!grp.empty() && (!dpk::tc_clipsum_same_launch(p0.d_in, p0.d_out, p.d_in, p.d_out) ||
                           c->plan[layers[grp[0]]].T != p.T))
        e = flush();
      grp.push_back(r);
      if (e == cudaSuccess && static_cast<int>(grp.size()) == dpk::kGemmMaxLayers) e = flush();
    } else if (!(flags & DP_NOISE_ONLY) && p.pergrad) {
      thin.push_back(r);
      if (static_cast<int>(thin.size()) == dpk::kPerGradMaxLayers) e = flush_thin();
    } else {
      e = launch_clipped_sum(c, l, (flags & DP_NOISE_ONLY) ? nullptr : A[r],
                             (flags & DP_NOISE_ONLY) ? nullptr : D[r], d_out[r], flags);
    }
    if (e != cudaSuccess) return fail(DP_ERR_CUDA, "clipped-sum kernel: %s", cudaGetErrorString(e));
  }
  cudaError_t e = flush();
  if (e == cudaSuccess) e = flush_thin();
  if (e != cudaSuccess) return fail(DP_ERR_CUDA, "clipped-sum kernel: %s", cudaGetErrorString(e));
  return DP_OK;
}

dp_status dp_noise_adamw(dp_ctx* c, int32_t layer, float* d_grad, float* d_theta, float* d_m,
                         float* d_v, const dp_adamw* hp, uint32_t flags) {
  if (!c) return fail(DP_ERR_ARG, "ctx is NULL");
  if (layer < 0 || layer >= c->L) return fail(DP_ERR_ARG, "layer %d out of range", layer);
  if (flags & ~(DP_NO_NOISE | DP_WRITE_GRAD)) return fail(DP_ERR_ARG, "unknown flag bits 0x%x", flags);
  if (!d_grad || !d_theta || !d_m || !d_v || !hp) return fail(DP_ERR_ARG, "NULL argument");
  if (!aligned16(d_grad) || !aligned16(d_theta) || !aligned16(d_m) || !aligned16(d_v))
    return fail(DP_ERR_ARG, "gradient and optimizer arrays must be 16-byte aligned");
  if (!(hp->beta1 >= 0.f && hp->beta1 < 1.f) || !(hp->beta2 >= 0.f && hp->beta2 < 1.f) ||
      !(hp->eps >= 0.f) || !std::isfinite(hp->eps) || !std::isfinite(hp->lr) ||
      !std::isfinite(hp->weight_decay) || hp->t < 1)
    return fail(DP_ERR_ARG, "AdamW hyperparameters out of range");
  const LayerPlan& p = c->plan[layer];
  dpk::AdamWArgs h{};
  h.lr = hp->lr;
  h.beta1 = hp->beta1;
  h.beta2 = hp->beta2;
  h.eps = hp->eps;
  h.weight_decay = hp->weight_decay;
  h.bc1 = static_cast<float>(1.0 / (1.0 - std::pow(static_cast<double>(hp->beta1),
                                                  static_cast<double>(hp->t))));
  h.bc2 = static_cast<float>(1.0 / (1.0 - std::pow(static_cast<double>(hp->beta2),
                                                  static_cast<double>(hp->t))));
  DP_CUDA(dpk::launch_noise_adamw(d_grad, d_theta, d_m, d_v, p.d_in * p.d_out, p.p_base,
                                  c->d_key, c->out_scale * (c->sigma * c->C),
                                  (flags & DP_NO_NOISE) ? 0 : 1, (flags & DP_WRITE_GRAD) ? 1 : 0,
                                  h, c->stream));
  return DP_OK;
}

dp_status dp_audit_emit(dp_ctx* c, const int32_t* h_idx, int32_t n, void* h_records) {
  if (!c) return fail(DP_ERR_ARG, "ctx is NULL");
  if (n < 0 || n > c->audit_capacity)
    return fail(DP_ERR_ARG, "n=%d outside 0..audit_capacity=%d", n, c->audit_capacity);
  if (n > 0 && (!h_idx || !h_records)) return fail(DP_ERR_ARG, "h_idx or h_records is NULL");
  if (!c->clip_done) return fail(DP_ERR_ORDER, "dp_audit_emit before dp_clip_factors");
  for (int r = 0; r < n; ++r)
    if (h_idx[r] < 0 || h_idx[r] >= c->B)
      return fail(DP_ERR_ARG, "audit index %d out of range 0..%d", h_idx[r], c->B - 1);
  // The staging buffers are free here: every call synchronises before it
  // returns, so no earlier gather can still be using them.
  const size_t rec_words = static_cast<size_t>(3 + c->L);
  if (n > 0) std::memcpy(c->h_idx, h_idx, sizeof(int) * n);
  DP_CUDA(dpk::launch_audit(c->h_idx_dev, n, c->L, c->B, c->d_layer_sq, c->d_s, c->d_c,
                            c->d_flag, c->h_rec_dev, c->h_flag_dev, c->stream));
  DP_CUDA(cudaStreamSynchronize(c->stream));
  if (n > 0) std::memcpy(h_records, c->h_rec, sizeof(float) * rec_words * n);
  if (*c->h_flag & 2)
    return fail(DP_ERR_TIMEOUT, "a tensor-core kernel gave up waiting on a pipeline barrier");
  if (*c->h_flag & 1) return fail(DP_ERR_NONFINITE, "a per-example squared norm was not finite");
  return DP_OK;
}

int64_t dp_audit_record_bytes(int32_t n_layers) { return 12 + 4 * static_cast<int64_t>(n_layers); }

dp_status dp_layer_norm_mode(const dp_ctx* c, int32_t layer, dp_norm_mode* mode_out) {
  if (!c || !mode_out) return fail(DP_ERR_ARG, "NULL argument");
  if (layer < 0 || layer >= c->L) return fail(DP_ERR_ARG, "layer %d out of range", layer);
  *mode_out = c->plan[layer].mode;
  return DP_OK;
}

dp_status dp_set_noise_key(dp_ctx* c, uint64_t seed, uint64_t step) {
  if (!c) return fail(DP_ERR_ARG, "ctx is NULL");
  c->seed = seed;
  c->step = step;
  c->h_key[0] = seed;
  c->h_key[1] = step;
  return DP_OK;
}

dp_status dp_layer_path(const dp_ctx* c, int32_t layer, int32_t* norm_tc, int32_t* sum_tc) {
  if (!c || !norm_tc || !sum_tc) return fail(DP_ERR_ARG, "NULL argument");
  if (layer < 0 || layer >= c->L) return fail(DP_ERR_ARG, "layer %d out of range", layer);
  *norm_tc = c->plan[layer].pergrad ? 2 : c->plan[layer].norm_tc;
  *sum_tc = c->plan[layer].gemm_tc != 0;
  return DP_OK;
}

void dp_step_destroy(dp_ctx* c) {
  if (!c) return;
  cudaStreamSynchronize(c->stream);
  free_scratch(c);
  delete c;
}

const char* dp_last_error(void) { return g_err.c_str(); }

const char* dp_status_string(dp_status s) {
  switch (s) {
    case DP_OK: return "DP_OK";
    case DP_ERR_ARG: return "DP_ERR_ARG";
    case DP_ERR_SHAPE: return "DP_ERR_SHAPE";
    case DP_ERR_DTYPE: return "DP_ERR_DTYPE";
    case DP_ERR_ORDER: return "DP_ERR_ORDER";
    case DP_ERR_NONFINITE: return "DP_ERR_NONFINITE";
    case DP_ERR_CUDA: return "DP_ERR_CUDA";
    case DP_ERR_TIMEOUT: return "DP_ERR_TIMEOUT";
    case DP_ERR_OOM: return "DP_ERR_OOM";
    case DP_ERR_UNSUPPORTED: return "DP_ERR_UNSUPPORTED";
  }
  return "DP_ERR_UNKNOWN";
}


dp_status dp_conv2d_dims(const dp_conv2d* conv, int32_t* T_out, int64_t* K_out) {
  if (!T_out || !K_out) return fail(DP_ERR_ARG, "NULL output");
  dpk::ConvGeom g{};
  dp_status st = conv_geom(conv, &g);
  if (st != DP_OK) return st;
  *T_out = g.H_out * g.W_out;
  *K_out = static_cast<int64_t>(g.kh) * g.kw * g.C_in;
  return DP_OK;
}

dp_status dp_conv2d_unfold(const dp_conv2d* conv, int32_t B, dp_dtype dtype, const void* x,
                           void* a_out, void* stream) {
  dpk::ConvGeom g{};
  dp_status st = conv_geom(conv, &g);
  if (st != DP_OK) return st;
  if (B < 1) return fail(DP_ERR_ARG, "B must be >= 1");
  if (dtype != DP_F32 && dtype != DP_BF16) return fail(DP_ERR_DTYPE, "unknown dtype %d", dtype);
  if (!x || !a_out) return fail(DP_ERR_ARG, "x or a_out is NULL");
  if (!aligned16(x) || !aligned16(a_out)) return fail(DP_ERR_ARG, "x and a_out must be 16-byte aligned");
  if (static_cast<int64_t>(B) * g.H_out * g.W_out > 0x7fffffffLL)
    return fail(DP_ERR_SHAPE, "B * H_out * W_out above 2^31 - 1");
  const int64_t elem = dtype == DP_F32 ? 4 : 2;
  const int64_t xb = static_cast<int64_t>(B) * g.H * g.W * g.C_in * elem;
  const int64_t ab = static_cast<int64_t>(B) * g.H_out * g.W_out * g.kh * g.kw * g.C_in * elem;
  const char* xp = static_cast<const char*>(x);
  const char* ap = static_cast<const char*>(a_out);
  if (xp < ap + ab && ap < xp + xb) return fail(DP_ERR_ARG, "x and a_out overlap");
  DP_CUDA(dpk::launch_conv_unfold(dtype == DP_F32 ? dpk::IN_F32 : dpk::IN_BF16, x, a_out, g, B,
                                  static_cast<cudaStream_t>(stream)));
  return DP_OK;
}

dp_status dp_kernel_launches(int64_t* count_out) {
  if (!count_out) return fail(DP_ERR_ARG, "count_out is NULL");
  *count_out = dpk::launch_count();
  return DP_OK;
}

dp_status dp_debug_bounded_wait(dp_ctx* c, int64_t limit_ns) {
  if (!c) return fail(DP_ERR_ARG, "ctx is NULL");
  if (limit_ns < 1 || limit_ns > 1000000000)
    return fail(DP_ERR_ARG, "limit_ns must be in 1 .. 10^9");
  DP_CUDA(dpk::launch_debug_wait(static_cast<uint64_t>(limit_ns), c->d_flag, c->stream));
  DP_CUDA(cudaStreamSynchronize(c->stream));
  int flag = 0;
  DP_CUDA(cudaMemcpy(&flag, c->d_flag, sizeof(int), cudaMemcpyDeviceToHost));
  if (flag & 2) return fail(DP_ERR_TIMEOUT, "the bounded wait gave up after %lld ns",
                            static_cast<long long>(limit_ns));
  return DP_OK;
}

dp_status dp_debug_philox(uint64_t seed, uint64_t step, uint64_t first_quad, int64_t n_quads,
                          uint32_t* d_out, void* stream) {
  if (n_quads < 0) return fail(DP_ERR_ARG, "n_quads < 0");
  if (n_quads > 0 && !d_out) return fail(DP_ERR_ARG, "d_out is NULL");
  DP_CUDA(dpk::launch_debug_philox(seed, step, first_quad, n_quads, d_out,
                                   static_cast<cudaStream_t>(stream)));
  return DP_OK;
}

dp_status dp_debug_gaussian(uint64_t seed, uint64_t step, uint64_t first_index, int64_t n,
                            float* d_out, void* stream) {
  if (n < 0) return fail(DP_ERR_ARG, "n < 0");
  if (n > 0 && !d_out) return fail(DP_ERR_ARG, "d_out is NULL");
  DP_CUDA(dpk::launch_debug_gauss(seed, step, first_index, n, d_out,
                                  static_cast<cudaStream_t>(stream)));
  return DP_OK;
}

}  // extern "C"
