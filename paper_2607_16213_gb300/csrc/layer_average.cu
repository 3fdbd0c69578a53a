// Compensation averaged across layers (the overview of Sec. 3 offers it next to the per-layer
// bias of Sec. 3.6).  Each layer's bias holds alpha * ln(1 + x) for a per-slot x >= 0 (x = R - 1
// with the ratio bias, x = M with the count bias), so x = expm1(bias / alpha).  Per (sequence,
// selection unit, position) the x of every layer that kept the position are summed, a layer that
// evicted it adding 0 (R = 1, M = 0); every layer's slot holding the position then gets
// alpha * ln(1 + sum / L).
//
// Kernels, in stream order: one scatter per layer (each (unit, position) occurs at most once in
// a layer, so no two threads of a launch touch the same sum, and the layers add in order:
// reproducible), then one write over all layers.
#include "selkv_internal.cuh"

namespace selkv {
namespace {

__device__ __forceinline__ int clamp_len(const LayerAvgArgs& a, int b) {
  const int m = a.lengths[b];
  return m < 0 ? 0 : (m > a.m_cap ? a.m_cap : m);
}

__global__ __launch_bounds__(256) void avg_scatter_kernel(LayerAvgArgs a, const int32_t* kept, const float* bias) {
  const int U = a.per_head ? a.Hkv : 1;
  const int u = blockIdx.y % U, b = blockIdx.y / U;
  const int slot = blockIdx.x * blockDim.x + threadIdx.x;
  if (slot >= clamp_len(a, b)) return;
  const size_t bu = (size_t)b * U + u;
  const int p = kept[bu * a.m_cap + slot];
  if (p < 0 || p >= a.n_cap) {
    raise_flag(a.flags, SELKV_DEVERR_COUNT);
    return;
  }
  const float x = bias[((size_t)b * a.Hkv + (a.per_head ? u : 0)) * a.m_cap + slot];
  a.acc[bu * a.n_cap + p] += expm1f(x / a.alpha);
}

__global__ __launch_bounds__(256) void avg_write_kernel(LayerAvgArgs a, LayerPtrs P) {
  const int U = a.per_head ? a.Hkv : 1;
  const int u = blockIdx.y % U, b = blockIdx.y / U, l = blockIdx.z;
  const int slot = blockIdx.x * blockDim.x + threadIdx.x;
  if (slot >= clamp_len(a, b)) return;
  const size_t bu = (size_t)b * U + u;
  const int p = P.kept[l][bu * a.m_cap + slot];
  if (p < 0 || p >= a.n_cap) return;  // flagged by the scatter
  const float v = a.alpha * log1pf(a.acc[bu * a.n_cap + p] / (float)a.L);
  float* out = P.bias[l];
  if (a.per_head) {
    out[((size_t)b * a.Hkv + u) * a.m_cap + slot] = v;
  } else {
    for (int kv = 0; kv < a.Hkv; ++kv) out[((size_t)b * a.Hkv + kv) * a.m_cap + slot] = v;
  }
}

}  // namespace

cudaError_t launch_layer_average(const LayerAvgArgs& a, const LayerPtrs& P, cudaStream_t s) {
  const int U = a.per_head ? a.Hkv : 1;
  cudaError_t e = cudaMemsetAsync(a.acc, 0, (size_t)a.B * U * a.n_cap * sizeof(float), s);
  if (e != cudaSuccess) return e;
  const dim3 grid((a.m_cap + 255) / 256, a.B * U);
  for (int l = 0; l < a.L; ++l) avg_scatter_kernel<<<grid, 256, 0, s>>>(a, P.kept[l], P.bias[l]);
  avg_write_kernel<<<dim3(grid.x, grid.y, a.L), 256, 0, s>>>(a, P);
  return cudaGetLastError();
}

}  // namespace selkv
