// Host helpers for the tensor-core launchers: the driver's tensor-map
// encoder (looked up once through the runtime, no libcuda link) and the SM
// count used to size persistent grids.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <atomic>
#include <map>
#include <mutex>
#include <utility>

#include "tc.h"

namespace dpk {

namespace {
std::atomic<int64_t> g_launches{0};
}  // namespace

void note_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }
int64_t launch_count() { return g_launches.load(std::memory_order_relaxed); }

namespace {
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    cudaDriverEntryPointQueryResult q;
    void* p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}
}  // namespace

bool tma_encode_available() { return encode_fn() != nullptr; }

bool make_tma_bf16(CUtensorMap* m, const void* base, int rank, const uint64_t* dims,
                   const uint64_t* strides_bytes, const uint32_t* box, const uint32_t* estrides) {
  auto fn = encode_fn();
  if (!fn || rank < 1 || rank > 5) return false;
  cuuint64_t d[5], st[4];
  cuuint32_t b[5], es[5];
  for (int r = 0; r < rank; ++r) {
    d[r] = dims[r];
    b[r] = box[r];
    es[r] = estrides ? estrides[r] : 1;
    if (r + 1 < rank) st[r] = strides_bytes[r];
  }
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(base), d, st, b, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

bool make_tma_f32_out(CUtensorMap* m, void* base, uint64_t rows, uint64_t cols) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t d[2] = {cols, rows};
  cuuint64_t st[1] = {cols * 4};
  cuuint32_t b[2] = {32, 32};
  cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, base, d, st, b, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool make_tma_f32_split(CUtensorMap* m, void* base, int split, uint64_t rows, uint64_t cols) {
  auto fn = encode_fn();
  if (!fn || split < 1) return false;
  cuuint64_t d[3] = {cols, rows, static_cast<cuuint64_t>(split)};
  cuuint64_t st[2] = {cols * 4, rows * cols * 4};
  cuuint32_t b[3] = {32, 32, 1};
  cuuint32_t es[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, base, d, st, b, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

namespace {
std::mutex g_setup_mu;
std::map<std::pair<const void*, int>, int> g_setup_done;   // (key, device) -> 1
std::map<std::pair<const void*, int>, int> g_cached;       // (key, device) -> value
}  // namespace

cudaError_t setup_once_per_device(const void* key, const std::function<cudaError_t()>& setup) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lk(g_setup_mu);
  const auto k = std::make_pair(key, dev);
  if (g_setup_done.count(k)) return cudaSuccess;
  e = setup();
  if (e == cudaSuccess) g_setup_done[k] = 1;
  return e;
}

int cached_per_device(const void* key, const std::function<int()>& fn) {
  int dev = 0;
  cudaGetDevice(&dev);
  std::lock_guard<std::mutex> lk(g_setup_mu);
  const auto k = std::make_pair(key, dev);
  auto it = g_cached.find(k);
  if (it != g_cached.end()) return it->second;
  const int v = fn();
  g_cached[k] = v;
  return v;
}

int device_sm_count() {
  int dev = 0, n = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  return n > 0 ? n : 1;
}

}  // namespace dpk
