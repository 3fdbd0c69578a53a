// Host-side TMA descriptor encoding (driver entry point looked up through the runtime, so the
// library does not link libcuda directly).
#include <mutex>

#include <cudaTypedefs.h>

#include "ptx.cuh"
#include "selkv_internal.cuh"

namespace selkv {
namespace {

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

}  // namespace

// Encodings are cached by (base, rows, d, box rows): the same buffers come back call after call
// (a decode step per layer), and a map depends on nothing else.
namespace {
struct MapEntry {
  const void* base;
  uint64_t rows;
  int d, box;
  CUtensorMap map;
};
constexpr int kMapCache = 128;
std::mutex g_map_mu;
MapEntry g_maps[kMapCache];
int g_map_used = 0, g_map_next = 0;
}  // namespace

bool encode_rows_bf16(CUtensorMap* map, const void* base, uint64_t rows, int d, int box_rows) {
  {
    std::lock_guard<std::mutex> lock(g_map_mu);
    for (int i = 0; i < g_map_used; ++i) {
      const MapEntry& e = g_maps[i];
      if (e.base == base && e.rows == rows && e.d == d && e.box == box_rows) {
        *map = e.map;
        return true;
      }
    }
  }
  auto fn = encode_fn();
  if (fn == nullptr) return false;
  cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)d * 2};
  cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  if (fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return false;
  std::lock_guard<std::mutex> lock(g_map_mu);
  MapEntry& e = g_maps[g_map_next];
  e.base = base;
  e.rows = rows;
  e.d = d;
  e.box = box_rows;
  e.map = *map;
  g_map_next = (g_map_next + 1) % kMapCache;
  if (g_map_used < kMapCache) ++g_map_used;
  return true;
}

}  // namespace selkv
