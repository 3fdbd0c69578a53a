// Per-call set-up (sequence table, output lengths) and the value norms ||v_j|| of Eq. 1.
#include <algorithm>

#include "selkv_internal.cuh"

namespace selkv {
namespace {

// Sequence table, output lengths and the selection's initial radix states.
__global__ void setup_kernel(SeqTable tab, CompressArgs a, SelectWs w) {
  for (int b = threadIdx.x; b < a.B; b += blockDim.x) {
    a.seq_n[b] = tab.n[b];
    a.seq_m[b] = tab.m[b];
    a.lengths[b] = tab.m[b];
  }
  const int units = a.B * a.Hkv;
  for (int i = threadIdx.x; i < units + a.B; i += blockDim.x) {
    const int b = i >= units ? i - units : i / a.Hkv;
    select_init_state(a, w, i, tab.n[b], tab.m[b]);
  }
}

// Sequence table alone (the scoring entry point).
__global__ void seq_setup_kernel(SeqTable tab, int32_t* seq_n, int32_t* seq_m, int B) {
  for (int b = threadIdx.x; b < B; b += blockDim.x) {
    seq_n[b] = tab.n[b];
    seq_m[b] = tab.m[b];
  }
}

// ||v_j|| per row: D / 8 lanes per row (at most 16), each loading 8 elements at a time.
template <typename T, int D>
__global__ void vnorm_kernel(CompressArgs a) {
  constexpr int EPL = 8;                      // elements per load8
  constexpr int LPR = D / EPL < 16 ? D / EPL : 16;  // lanes per row
  constexpr int RPW = 32 / LPR;               // rows per warp step
  const int lane = threadIdx.x & 31, sub = lane / LPR, sl = lane % LPR;
  const size_t total = (size_t)a.B * a.Hkv * a.n_cap;
  const size_t nwarps = (size_t)gridDim.x * (blockDim.x / 32);
  for (size_t row0 = (blockIdx.x * (size_t)blockDim.x + threadIdx.x) / 32 * RPW; row0 < total; row0 += nwarps * RPW) {
    const size_t row = row0 + sub;
    float s = 0.f;
    bool ok = false;
    if (row < total) {
      const int j = (int)(row % a.n_cap);
      const int b = (int)(row / a.n_cap) / a.Hkv;
      ok = j < a.seq_n[b];
      if (ok) {
        const T* p = static_cast<const T*>(a.V) + row * D;
#pragma unroll
        for (int d = sl * EPL; d < D; d += LPR * EPL) {
          float x[8];
          load8(p + d, x);
#pragma unroll
          for (int e = 0; e < 8; ++e) s = fmaf(x[e], x[e], s);
        }
      }
    }
#pragma unroll
    for (int o = LPR / 2; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (ok && sl == 0) a.vnorm[row] = sqrtf(s);
  }
}

template <typename T, int D>
void launch_norms(const CompressArgs& a, cudaStream_t s) {
  const size_t rows = (size_t)a.B * a.Hkv * a.n_cap;
  const int blocks = (int)std::min<size_t>((rows + 15) / 16, 152 * 8);
  vnorm_kernel<T, D><<<blocks, 256, 0, s>>>(a);
}

}  // namespace

cudaError_t launch_setup(const CompressArgs& a, const SeqTable& tab, const SelectWs& w, cudaStream_t s) {
  setup_kernel<<<1, 256, 0, s>>>(tab, a, w);
  return cudaGetLastError();
}

cudaError_t launch_seq_setup(const CompressArgs& a, const SeqTable& tab, cudaStream_t s) {
  seq_setup_kernel<<<1, 256, 0, s>>>(tab, a.seq_n, a.seq_m, a.B);
  return cudaGetLastError();
}

cudaError_t launch_vnorm(const CompressArgs& a, cudaStream_t s) {
  if (a.dtype == SELKV_BF16) {
    if (a.D == 128) launch_norms<__nv_bfloat16, 128>(a, s); else launch_norms<__nv_bfloat16, 64>(a, s);
  } else {
    if (a.D == 128) launch_norms<float, 128>(a, s); else launch_norms<float, 64>(a, s);
  }
  return cudaGetLastError();
}

}  // namespace selkv
