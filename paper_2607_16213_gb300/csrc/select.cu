// Contribution score, pooling and the shared-set selection of SelKV.
//
//   c_j   = a_j * ||v_j||                                   (Eq. 1, averaged over the group)
//   c^_j  = (1/K) sum_{|t| <= K/2, 0 <= j+t < n_b - m_r} c_{j+t}   (Sec. 3.2 smoothing)
//   T_kv  = top-m_s of c^ over the candidates [0, n_b - m_r)       (Eq. 2, per KV head)
//   U     = union of T_kv; if |U| > m_s keep the top-m_s of U by the score summed over KV heads
//           (the same order as the mean of Sec. 3.3); then add the recent window.
// Every top-k orders by value descending, then position ascending.  Selections are exact
// radix selects on the fp32 bit patterns (all scores are >= 0, so the unsigned order of the
// bits is the numeric order), followed by an index-ordered scan for the entries equal to the
// threshold.
#include <algorithm>
#include <climits>

#include "selkv_internal.cuh"

namespace selkv {
namespace {

__global__ void setup_kernel(SeqTable tab, int B, int32_t* seq_n, int32_t* seq_m, int32_t* lengths) {
  for (int b = threadIdx.x; b < B; b += blockDim.x) {
    seq_n[b] = tab.n[b];
    seq_m[b] = tab.m[b];
    lengths[b] = tab.m[b];
  }
}

// ||v_j|| per row; one warp per row.
template <typename T, int D>
__global__ void vnorm_kernel(CompressArgs a) {
  const int lane = threadIdx.x & 31;
  const size_t total = (size_t)a.B * a.Hkv * a.n_cap;
  const size_t nwarps = (size_t)gridDim.x * (blockDim.x / 32);
  for (size_t row = (blockIdx.x * (size_t)blockDim.x + threadIdx.x) / 32; row < total; row += nwarps) {
    const int j = (int)(row % a.n_cap);
    const int b = (int)(row / a.n_cap) / a.Hkv;
    if (j >= a.seq_n[b]) continue;
    const T* p = static_cast<const T*>(a.V) + row * D;
    float s = 0.f;
#pragma unroll
    for (int d = lane * 2; d < D; d += 64) {
      float x[2];
      load2(p + d, x);
      s = fmaf(x[0], x[0], s);
      s = fmaf(x[1], x[1], s);
    }
    s = warp_sum(s);
    if (lane == 0) a.vnorm[row] = sqrtf(s);
  }
}

// Pooled contribution score over the candidates; 0 past them.
__global__ void pool_kernel(CompressArgs a) {
  const size_t idx = blockIdx.x * (size_t)blockDim.x + threadIdx.x;
  if (idx >= (size_t)a.B * a.Hkv * a.n_cap) return;
  const int j = (int)(idx % a.n_cap);
  const size_t bk = idx / a.n_cap;
  const int b = (int)bk / a.Hkv;
  const int n = a.seq_n[b];
  if (j >= n) return;
  const int ncand = n - a.recent;
  if (j >= ncand) {
    a.score[idx] = 0.f;
    return;
  }
  const int half = a.pool_kernel / 2;
  const float* at = a.attn + bk * a.n_cap;
  const float* vn = a.vnorm + bk * a.n_cap;
  float s = 0.f;
  for (int t = -half; t <= half; ++t) {
    const int jj = j + t;
    if (jj >= 0 && jj < ncand) s += at[jj] * vn[jj];
  }
  a.score[idx] = s / (float)a.pool_kernel;
}

// Block-wide (1024 threads) exact top-k threshold over key[0..N) restricted to member[j] != 0
// (member may be NULL = everyone).  Returns T (the k-th best key's bits) and jcut (the
// position of the last entry taken among those equal to T, in position order): j is
// selected iff bits(key_j) > T or (bits(key_j) == T and j <= jcut).  Requires
// 1 <= k <= number of members.  All threads return the same values.
__device__ void block_select_top(const float* __restrict__ key, const uint8_t* __restrict__ member,
                                 int N, int k, uint32_t& T_out, int& jcut_out) {
  __shared__ uint32_t hist[256];
  __shared__ uint32_t s_prefix, s_krem, s_total;
  __shared__ int s_jcut;
  __shared__ uint32_t wcnt[32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint32_t prefix = 0, pmask = 0, krem = (uint32_t)k;
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    for (int i = tid; i < 256; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    for (int j = tid; j < N; j += blockDim.x) {
      if (member != nullptr && !member[j]) continue;
      const uint32_t u = __float_as_uint(key[j]);
      if ((u & pmask) == prefix) atomicAdd(&hist[(u >> shift) & 255u], 1u);
    }
    __syncthreads();
    if (warp == 0) {
      uint32_t c[8], tot = 0;
#pragma unroll
      for (int t = 0; t < 8; ++t) {
        c[t] = hist[255 - 8 * lane - t];
        tot += c[t];
      }
      uint32_t incl = tot;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t v = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += v;
      }
      const unsigned bal = __ballot_sync(0xffffffffu, incl >= krem);
      const int L = __ffs(bal) - 1;
      if (lane == L) {
        uint32_t cum = incl - tot;
        int dg = 255 - 8 * lane - 7;
#pragma unroll
        for (int t = 0; t < 8; ++t) {
          if (cum + c[t] >= krem) {
            dg = 255 - 8 * lane - t;
            break;
          }
          cum += c[t];
        }
        s_prefix = prefix | ((uint32_t)dg << shift);
        s_krem = krem - cum;
      }
    }
    __syncthreads();
    prefix = s_prefix;
    krem = s_krem;
    pmask |= 255u << shift;
    __syncthreads();
  }
  // krem entries equal to `prefix` are taken, lowest positions first.
  if (tid == 0) s_jcut = INT_MAX;
  uint32_t base = 0;
  for (int j0 = 0; j0 < N; j0 += blockDim.x) {
    const int j = j0 + tid;
    const bool f = j < N && (member == nullptr || member[j]) && __float_as_uint(key[j]) == prefix;
    const unsigned bal = __ballot_sync(0xffffffffu, f);
    if (lane == 0) wcnt[warp] = __popc(bal);
    __syncthreads();
    if (warp == 0) {
      const uint32_t v = wcnt[lane];
      uint32_t incl = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t w = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += w;
      }
      wcnt[lane] = incl - v;
      if (lane == 31) s_total = incl;
    }
    __syncthreads();
    const uint32_t rank = base + wcnt[warp] + __popc(bal & ((1u << lane) - 1u)) + 1u;
    if (f && rank == krem) s_jcut = j;
    base += s_total;
    __syncthreads();
    if (base >= krem) break;
  }
  __syncthreads();
  T_out = prefix;
  jcut_out = s_jcut;
}

// Per (b, kv): threshold of the KV head's own top-m_s (Eq. 2).
__global__ __launch_bounds__(1024) void topk_kernel(CompressArgs a) {
  const int bk = blockIdx.x, b = bk / a.Hkv;
  const int n = a.seq_n[b];
  const int ncand = n - a.recent;
  const int k = a.seq_m[b] - a.recent;
  const float* sc = a.score + (size_t)bk * a.n_cap;
  uint32_t T = 0xffffffffu;
  int jcut = -1;
  if (k > 0) block_select_top(sc, nullptr, ncand, k, T, jcut);
  if (threadIdx.x == 0) a.thr[bk] = make_uint2(T, (uint32_t)jcut);
  if (a.dbg_topk != nullptr) {
    for (int j = threadIdx.x; j < n; j += blockDim.x) {
      const uint32_t u = __float_as_uint(sc[j]);
      a.dbg_topk[(size_t)bk * a.n_cap + j] = (j < ncand && k > 0 && (u > T || (u == T && j <= jcut))) ? 1 : 0;
    }
  }
}

// Block-wide exclusive scan of a 0/1 flag (1024 threads).  Returns the rank of this thread's
// flag among the set flags and the block total.
__device__ __forceinline__ uint32_t block_rank(bool f, uint32_t& total, uint32_t* wcnt) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const unsigned bal = __ballot_sync(0xffffffffu, f);
  if (lane == 0) wcnt[warp] = __popc(bal);
  __syncthreads();
  if (warp == 0) {
    const uint32_t v = wcnt[lane];
    uint32_t incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t w = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += w;
    }
    wcnt[lane] = incl - v;
    if (lane == 31) wcnt[32] = incl;
  }
  __syncthreads();
  const uint32_t r = wcnt[warp] + __popc(bal & ((1u << lane) - 1u));
  total = wcnt[32];
  __syncthreads();
  return r;
}

// Per sequence: union over KV heads, trim by the summed score, recent window, compaction.
__global__ __launch_bounds__(1024) void trim_compact_kernel(CompressArgs a, float* tkey, uint8_t* uflag) {
  __shared__ uint32_t wcnt[33];
  __shared__ uint32_t s_ucount;
  const int b = blockIdx.x;
  const int n = a.seq_n[b];
  const int ncand = n - a.recent;
  const int k = a.seq_m[b] - a.recent;
  float* tk = tkey + (size_t)b * a.n_cap;
  uint8_t* uf = uflag + (size_t)b * a.n_cap;
  if (threadIdx.x == 0) s_ucount = 0;
  __syncthreads();
  uint32_t local = 0;
  for (int j = threadIdx.x; j < ncand; j += blockDim.x) {
    bool in = false;
    float sum = 0.f;
    for (int kv = 0; kv < a.Hkv; ++kv) {
      const size_t bk = (size_t)b * a.Hkv + kv;
      const float s = a.score[bk * a.n_cap + j];
      const uint32_t u = __float_as_uint(s);
      const uint2 t = a.thr[bk];
      in |= (u > t.x) || (u == t.x && j <= (int)t.y);
      sum += s;
    }
    uf[j] = in ? 1 : 0;
    tk[j] = sum;
    local += in ? 1u : 0u;
  }
  atomicAdd(&s_ucount, local);
  __syncthreads();
  const bool trim = (int)s_ucount > k;
  uint32_t T2 = 0;
  int jcut2 = INT_MAX;
  if (trim && k > 0) block_select_top(tk, uf, ncand, k, T2, jcut2);
  uint32_t base = 0;
  for (int j0 = 0; j0 < n; j0 += blockDim.x) {
    const int j = j0 + threadIdx.x;
    bool kept = false;
    if (j < ncand) {
      kept = uf[j] != 0;
      if (trim && kept) {
        if (k <= 0) {
          kept = false;
        } else {
          const uint32_t u = __float_as_uint(tk[j]);
          kept = u > T2 || (u == T2 && j <= jcut2);
        }
      }
    } else if (j < n) {
      kept = true;
    }
    uint32_t total;
    const uint32_t r = block_rank(kept, total, wcnt);
    if (j < n) {
      a.kflag[(size_t)b * a.n_cap + j] = kept ? 1 : 0;
      a.slot_of[(size_t)b * a.n_cap + j] = kept ? (int)(base + r) : -1;
      if (kept && a.dbg_kept_idx != nullptr && (int)(base + r) < a.m_cap)
        a.dbg_kept_idx[(size_t)b * a.m_cap + base + r] = j;
    }
    base += total;
  }
  if (threadIdx.x == 0 && (int)base != a.seq_m[b]) raise_flag(a.flags, SELKV_DEVERR_COUNT);
}

template <typename T, int D>
void launch_norms(const CompressArgs& a, cudaStream_t s) {
  const size_t rows = (size_t)a.B * a.Hkv * a.n_cap;
  const int blocks = (int)std::min<size_t>((rows + 7) / 8, 152 * 16);
  vnorm_kernel<T, D><<<blocks, 256, 0, s>>>(a);
}

}  // namespace

cudaError_t launch_setup(const CompressArgs& a, const SeqTable& tab, cudaStream_t s) {
  setup_kernel<<<1, 256, 0, s>>>(tab, a.B, a.seq_n, a.seq_m, a.lengths);
  return cudaGetLastError();
}

cudaError_t launch_norm_pool(const CompressArgs& a, cudaStream_t s) {
  if (a.dtype == SELKV_BF16) {
    if (a.D == 128) launch_norms<__nv_bfloat16, 128>(a, s); else launch_norms<__nv_bfloat16, 64>(a, s);
  } else {
    if (a.D == 128) launch_norms<float, 128>(a, s); else launch_norms<float, 64>(a, s);
  }
  const size_t total = (size_t)a.B * a.Hkv * a.n_cap;
  pool_kernel<<<(unsigned)((total + 255) / 256), 256, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_select(const CompressArgs& a, float* tkey, uint8_t* uflag, cudaStream_t s) {
  topk_kernel<<<a.B * a.Hkv, 1024, 0, s>>>(a);
  trim_compact_kernel<<<a.B, 1024, 0, s>>>(a, tkey, uflag);
  return cudaGetLastError();
}

}  // namespace selkv
