// Observation-window scoring on CUDA cores (fp32 arithmetic for both storage dtypes).
//
// Per (sequence b, KV head kv) the G query heads' W window rows are stacked into R = G * W
// rows.  Row r = g * W + i is query head kv * G + g at position p = n_b - W + i and sees the
// keys j <= p (the causal re-pass of Sec. 3.1).  The cumulative attention of Eq. 5,
// averaged over the group,
//     a_j = (1/G) sum_r 2^(s'_rj - M_r) / Z_r,     s'_rj = log2(e) q_r . k_j / sqrt(d),
// needs each row's normaliser before any column can be summed, so the scores are computed
// twice: pass 1 gathers per-row (max, sum) over column chunks, a small kernel folds the
// chunks, and pass 2 recomputes the same tiles and sums columns.  Both passes use the same
// tile code, so pass 2 sees bit-identical scores.
#include "selkv_internal.cuh"

namespace selkv {

cudaError_t launch_rowstat_reduce(const CompressArgs& a, cudaStream_t s);

namespace {

constexpr int kTile = 64;   // rows and columns per tile
constexpr int kDc = 32;     // head-dimension slice staged in shared memory

// acc[i][j] = q_{r0 + 4ty + i} . k_{c0 + 4tx + j} for a 64 x 64 tile.
template <typename T, int D>
__device__ __forceinline__ void score_tile(const CompressArgs& a, int b, int kv, int n, int r0,
                                           int c0, float (&Qs)[kDc][kTile + 4],
                                           float (&Ks)[kDc][kTile + 4], float (&acc)[4][4]) {
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
  const int lrow = tid >> 2, ldd = (tid & 3) * 8;
  for (int dc = 0; dc < D; dc += kDc) {
    float x[8];
    const int r = r0 + lrow;
    if (r < a.R) {
      const int h = kv * a.G + r / a.W, i = r % a.W;
      load8(static_cast<const T*>(a.Q) + (((size_t)b * a.Hq + h) * a.W + i) * D + dc + ldd, x);
    } else {
#pragma unroll
      for (int k = 0; k < 8; ++k) x[k] = 0.f;
    }
#pragma unroll
    for (int k = 0; k < 8; ++k) Qs[ldd + k][lrow] = x[k];
    const int col = c0 + lrow;
    if (col < n) {
      load8(static_cast<const T*>(a.K) + (((size_t)b * a.Hkv + kv) * a.n_cap + col) * D + dc + ldd, x);
    } else {
#pragma unroll
      for (int k = 0; k < 8; ++k) x[k] = 0.f;
    }
#pragma unroll
    for (int k = 0; k < 8; ++k) Ks[ldd + k][lrow] = x[k];
    __syncthreads();
#pragma unroll 8
    for (int dd = 0; dd < kDc; ++dd) {
      const float4 q4 = *reinterpret_cast<const float4*>(&Qs[dd][ty * 4]);
      const float4 k4 = *reinterpret_cast<const float4*>(&Ks[dd][tx * 4]);
      const float qv[4] = {q4.x, q4.y, q4.z, q4.w};
      const float kvv[4] = {k4.x, k4.y, k4.z, k4.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(qv[i], kvv[j], acc[i][j]);
    }
    __syncthreads();
  }
}

__device__ __forceinline__ float reduce16_max(float v) {
#pragma unroll
  for (int o = 8; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float reduce16_sum(float v) {
#pragma unroll
  for (int o = 8; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Pass 1: grid (column chunk, row tile, b * Hkv); per row the (max, sum) of 2^(s' - max)
// over the chunk's visible columns.
template <typename T, int D>
__global__ __launch_bounds__(256) void rowstats_kernel(CompressArgs a) {
  __shared__ __align__(16) float Qs[kDc][kTile + 4];
  __shared__ __align__(16) float Ks[kDc][kTile + 4];
  const int chunk = blockIdx.x, r0 = blockIdx.y * kTile, bk = blockIdx.z;
  const int b = bk / a.Hkv, kv = bk % a.Hkv;
  const int n = a.seq_n[b];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float m_run[4], l_run[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) { m_run[i] = -INFINITY; l_run[i] = 0.f; }
  const int c_begin = chunk * kRowChunk;
  const int c_end = min(n, c_begin + kRowChunk);
  for (int c0 = c_begin; c0 < c_end; c0 += kTile) {
    float acc[4][4];
    score_tile<T, D>(a, b, kv, n, r0, c0, Qs, Ks, acc);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int r = r0 + ty * 4 + i;
      const int p = n - a.W + (r % a.W);
      float sv[4], tmax = -INFINITY;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int col = c0 + tx * 4 + j;
        const bool ok = r < a.R && col < n && col <= p;
        sv[j] = ok ? acc[i][j] * a.scale_log2 : -INFINITY;
        tmax = fmaxf(tmax, sv[j]);
      }
      tmax = reduce16_max(tmax);
      const float m_new = fmaxf(m_run[i], tmax);
      float ssum = 0.f;
      if (m_new != -INFINITY) {
#pragma unroll
        for (int j = 0; j < 4; ++j) ssum += exp2f(sv[j] - m_new);
      }
      ssum = reduce16_sum(ssum);
      if (m_new != -INFINITY) {
        l_run[i] = l_run[i] * exp2f(m_run[i] - m_new) + ssum;
        m_run[i] = m_new;
      }
    }
  }
  if (tx == 0) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int r = r0 + ty * 4 + i;
      if (r < a.R) a.rowpart[((size_t)bk * a.nchunks + chunk) * a.R + r] = make_float2(m_run[i], l_run[i]);
    }
  }
}

// Fold the column chunks: (M, 1 / (G * Z)) per row.
__global__ void rowstat_reduce_kernel(CompressArgs a) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= a.B * a.Hkv * a.R) return;
  const int r = idx % a.R, bk = idx / a.R;
  const int nch = a.nchunks;  // chunks without visible columns hold (-inf, 0)
  const float2* part = a.rowpart + (size_t)bk * a.nchunks * a.R + r;
  float M = -INFINITY;
  for (int c = 0; c < nch; ++c) M = fmaxf(M, part[(size_t)c * a.R].x);
  float Z = 0.f;
  for (int c = 0; c < nch; ++c) {
    const float2 p = part[(size_t)c * a.R];
    if (p.x != -INFINITY) Z += p.y * exp2f(p.x - M);
  }
  a.rowstat[idx] = make_float2(M, 1.f / ((float)a.G * Z));
}

// Pass 2: grid (column tile, b * Hkv); a_j = sum_r 2^(s'_rj - M_r) / (G Z_r).
template <typename T, int D>
__global__ __launch_bounds__(256) void colsum_kernel(CompressArgs a) {
  __shared__ __align__(16) float Qs[kDc][kTile + 4];
  __shared__ __align__(16) float Ks[kDc][kTile + 4];
  __shared__ float red[16][kTile];
  const int c0 = blockIdx.x * kTile, bk = blockIdx.y;
  const int b = bk / a.Hkv, kv = bk % a.Hkv;
  const int n = a.seq_n[b];
  if (c0 >= n) return;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float colacc[4] = {0.f, 0.f, 0.f, 0.f};
  for (int r0 = 0; r0 < a.R; r0 += kTile) {
    float acc[4][4];
    score_tile<T, D>(a, b, kv, n, r0, c0, Qs, Ks, acc);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int r = r0 + ty * 4 + i;
      if (r >= a.R) continue;
      const float2 st = a.rowstat[(size_t)bk * a.R + r];
      const int p = n - a.W + (r % a.W);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int col = c0 + tx * 4 + j;
        if (col < n && col <= p) colacc[j] += exp2f(acc[i][j] * a.scale_log2 - st.x) * st.y;
      }
    }
  }
#pragma unroll
  for (int j = 0; j < 4; ++j) red[ty][tx * 4 + j] = colacc[j];
  __syncthreads();
  if (threadIdx.x < kTile) {
    float s = 0.f;
#pragma unroll
    for (int t = 0; t < 16; ++t) s += red[t][threadIdx.x];
    const int col = c0 + threadIdx.x;
    if (col < n) a.attn[(size_t)bk * a.n_cap + col] = s;
  }
}

template <typename T, int D>
cudaError_t launch_score_t(const CompressArgs& a, cudaStream_t s, int passes) {
  const int row_tiles = (a.R + kTile - 1) / kTile;
  if (passes & kScoreRowstats) {
    rowstats_kernel<T, D><<<dim3(a.nchunks, row_tiles, a.B * a.Hkv), 256, 0, s>>>(a);
    launch_rowstat_reduce(a, s);
  }
  if (passes & kScoreColsums)
    colsum_kernel<T, D><<<dim3((a.n_cap + kTile - 1) / kTile, a.B * a.Hkv), 256, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_rowstat_reduce(const CompressArgs& a, cudaStream_t s) {
  const int nrows = a.B * a.Hkv * a.R;
  rowstat_reduce_kernel<<<(nrows + 255) / 256, 256, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_score_simt(const CompressArgs& a, cudaStream_t s, int passes) {
  if (a.dtype == SELKV_BF16)
    return a.D == 128 ? launch_score_t<__nv_bfloat16, 128>(a, s, passes) : launch_score_t<__nv_bfloat16, 64>(a, s, passes);
  return a.D == 128 ? launch_score_t<float, 128>(a, s, passes) : launch_score_t<float, 64>(a, s, passes);
}

}  // namespace selkv
