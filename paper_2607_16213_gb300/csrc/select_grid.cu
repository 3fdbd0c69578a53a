// Pooling and the shared-set selection of SelKV, spread over the whole GPU.
//
//   c^_j  = (1/K) sum_{|t| <= K/2, 0 <= j+t < n_b - m_r} a_{j+t} ||v_{j+t}||   (Eq. 1, Sec. 3.2)
//   T_kv  = top-m_s of c^ over the candidates [0, n_b - m_r)                    (Eq. 2)
//   U     = union over KV heads; if |U| > m_s, keep the top-m_s of U by the score summed
//           over KV heads (the order of the mean of Sec. 3.3); then the recent window.
// Every top-k orders by value descending, then position ascending, and is an exact radix
// select on the fp32 bit patterns (scores are >= 0, so unsigned order = numeric order), done
// in three digit passes (11, 11, 10 bits).  Each pass is one grid-wide histogram: CTAs count
// digits in shared memory and add them to a per-unit global histogram; the last CTA of a unit
// to arrive (one atomic add, no waiting) picks the digit and narrows the unit's prefix.  After
// the last pass `count_eq` entries equal the threshold T; when more of them exist than are
// still needed, the CTA that picked the last digit finds the position of the last one taken.
// A unit selects j iff bits(key_j) > T or (bits(key_j) == T and j <= jcut).
#include <climits>

#include "selkv_internal.cuh"

namespace selkv {
namespace {

#ifndef SELKV_SEL_MINB
#define SELKV_SEL_MINB 4  // CTAs per SM the pooling and union kernels are compiled for (full occupancy)
#endif
constexpr int kBlock = 512;                 // threads per CTA
constexpr int kPerThread = 2;               // positions per thread
constexpr int kSpan = kBlock * kPerThread;  // positions per CTA
constexpr int kBins = 2048;
__device__ __constant__ int kShift[3] = {21, 10, 0};
__device__ __constant__ uint32_t kMask[3] = {0u, 0xFFE00000u, 0xFFFFFC00u};
__device__ __constant__ uint32_t kDigitMask[3] = {2047u, 2047u, 1023u};

__device__ __forceinline__ bool selected(uint32_t u, int j, const RadixState& s) {
  return u > s.prefix || (u == s.prefix && j <= s.jcut);
}

// Add this CTA's shared histogram to the unit's global one, then arrive; the last CTA of the
// unit (of `nblocks`) reads the unit's histogram back into `sh` (one round of loads), picks
// the digit of `pass` and narrows the unit's state.  The pick uses the whole CTA: thread t
// sums `per` consecutive bins counted from the top digit down, a CTA-wide scan of those sums
// finds the thread whose bins reach the krem-th entry, and that thread walks its bins.
__device__ void flush_and_select(uint32_t* sh, uint32_t* ghist, RadixState* st, int pass, int nblocks,
                                 bool* s_last) {
  __shared__ uint32_t s_wsum[32];
  const int bins = pass == 2 ? 1024 : kBins;
  __syncthreads();
  for (int i = threadIdx.x; i < bins; i += blockDim.x)
    if (sh[i] != 0u) atomicAdd(&ghist[i], sh[i]);
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) *s_last = atomicAdd(&st->arrive, 1u) == (uint32_t)nblocks - 1u;
  __syncthreads();
  if (!*s_last) return;
  __threadfence();
  for (int i = threadIdx.x; i < bins; i += blockDim.x) sh[i] = __ldcg(&ghist[i]);
  __syncthreads();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nwarps = blockDim.x >> 5;
  const int per = bins >= (int)blockDim.x ? bins / (int)blockDim.x : 1;
  const int owners = bins / per;             // threads that own bins (the rest own none)
  const int hi = bins - 1 - tid * per;       // this thread's bins: hi, hi-1, ..., hi-per+1
  uint32_t tot = 0;
  if (tid < owners)
    for (int t = 0; t < per; ++t) tot += sh[hi - t];
  uint32_t incl = tot;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t v = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += v;
  }
  if (lane == 31) s_wsum[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    const uint32_t v = lane < nwarps ? s_wsum[lane] : 0u;
    uint32_t w = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t x = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += x;
    }
    if (lane < nwarps) s_wsum[lane] = w - v;  // entries in the bins of the warps before
  }
  __syncthreads();
  incl += s_wsum[warp];
  const uint32_t krem = st->krem;
  const uint32_t excl = incl - tot;
  // the owner of the krem-th entry; if fewer entries remain than krem, the owner of bin 0;
  // with krem = 0, the owner of the top bin
  const bool mine = tid < owners && ((excl < krem && incl >= krem) || (tid == owners - 1 && incl < krem) ||
                                     (krem == 0u && tid == 0));
  if (mine) {
    uint32_t cum = excl;
    int dg = hi - per + 1;
    uint32_t cnt = 0;
    for (int t = 0; t < per; ++t) {
      const uint32_t c = sh[hi - t];
      if (cum + c >= krem) {
        dg = hi - t;
        cnt = c;
        break;
      }
      cum += c;
    }
    st->prefix |= (uint32_t)dg << kShift[pass];
    st->krem = krem - cum;
    if (pass == 2) st->count_eq = cnt;
    st->arrive = 0u;
  }
}

// Pooling of Eq. 1's score over the candidates, fused with digit pass 0 of each KV head's
// top-m_s.  Grid (position blocks, B * Hkv).
__global__ __launch_bounds__(kBlock, SELKV_SEL_MINB) void pool_hist0_kernel(CompressArgs a, SelectWs w) {
  __shared__ uint32_t sh[kBins];
  __shared__ bool s_last;
  const int u = blockIdx.y, b = u / a.Hkv;
  const int n = a.seq_n[b], ncand = n - a.recent;
  RadixState* st = &w.topk[u];
  const bool active = st->active != 0u;
  for (int i = threadIdx.x; i < kBins; i += kBlock) sh[i] = 0u;
  __syncthreads();
  const int half = a.pool_kernel / 2;
  const float* at = a.attn + (size_t)u * a.n_cap;
  const float* vn = a.vnorm + (size_t)u * a.n_cap;
  float* sc = a.score + (size_t)u * a.n_cap;
  const int j0 = blockIdx.x * kSpan;
#pragma unroll 1
  for (int e = 0; e < kPerThread; ++e) {
    const int j = j0 + e * kBlock + threadIdx.x;
    if (j >= n) continue;
    float s = 0.f;
    if (j < ncand) {
      for (int t = -half; t <= half; ++t) {
        const int jj = j + t;
        if (jj >= 0 && jj < ncand) s += at[jj] * vn[jj];
      }
      s = s / (float)a.pool_kernel;
      if (active) atomicAdd(&sh[__float_as_uint(s) >> 21], 1u);
    }
    sc[j] = s;
  }
  if (active) flush_and_select(sh, w.topk_hist + (size_t)u * 3 * kBins, st, 0, gridDim.x, &s_last);
}

// After the last pass: when more entries equal the threshold than are still needed, find the
// position of the last one taken (lowest positions first).  Run by the CTA that picked the
// last digit of unit u, right after picking it.
__device__ __noinline__ void resolve_tie(const CompressArgs& a, RadixState* st, const float* key, const uint8_t* member, int u,
                            int per_seq) {
  __shared__ uint32_t wcnt[32];
  __shared__ uint32_t s_total;
  __shared__ int s_jcut;
  const int b = u / per_seq;
  __syncthreads();
  const uint32_t T = __ldcg(&st->prefix), krem = __ldcg(&st->krem);
  if (__ldcg(&st->count_eq) == krem) {
    if (threadIdx.x == 0) st->jcut = INT_MAX;
    return;
  }
  const int ncand = a.seq_n[b] - a.recent;
  const float* k = key + (size_t)u * a.n_cap;
  const uint8_t* mb = member != nullptr ? member + (size_t)u * a.n_cap : nullptr;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  if (threadIdx.x == 0) s_jcut = INT_MAX;
  uint32_t base = 0;
  for (int j0 = 0; j0 < ncand; j0 += blockDim.x) {
    const int j = j0 + threadIdx.x;
    const bool f = j < ncand && (mb == nullptr || mb[j]) && __float_as_uint(k[j]) == T;
    const unsigned bal = __ballot_sync(0xffffffffu, f);
    if (lane == 0) wcnt[warp] = __popc(bal);
    __syncthreads();
    if (warp == 0) {
      const uint32_t v = lane < nwarps ? wcnt[lane] : 0u;
      uint32_t incl = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t t = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += t;
      }
      if (lane < nwarps) wcnt[lane] = incl - v;
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
  if (threadIdx.x == 0) st->jcut = s_jcut;
}

// Digit pass `pass` (1 or 2) of a set of units.  Unit u's keys are key[u * stride + j] for
// j < len(u); member (optional) filters them.  Grid (position blocks, units).
__global__ __launch_bounds__(kBlock) void hist_kernel(CompressArgs a, RadixState* states, uint32_t* hist,
                                                      const float* key, const uint8_t* member, int per_seq,
                                                      int pass) {
  __shared__ uint32_t sh[kBins];
  __shared__ bool s_last;
  const int u = blockIdx.y, b = u / per_seq;
  RadixState* st = &states[u];
  if (st->active == 0u) return;
  const int ncand = a.seq_n[b] - a.recent;
  const int bins = pass == 2 ? 1024 : kBins;
  for (int i = threadIdx.x; i < bins; i += kBlock) sh[i] = 0u;
  __syncthreads();
  const uint32_t prefix = st->prefix, mask = kMask[pass], dmask = kDigitMask[pass];
  const int shift = kShift[pass];
  const float* k = key + (size_t)u * a.n_cap;
  const uint8_t* mb = member != nullptr ? member + (size_t)u * a.n_cap : nullptr;
  const int j0 = blockIdx.x * kSpan;
#pragma unroll
  for (int e = 0; e < kPerThread; ++e) {
    const int j = j0 + e * kBlock + threadIdx.x;
    if (j >= ncand || (mb != nullptr && !mb[j])) continue;
    const uint32_t x = __float_as_uint(k[j]);
    if ((x & mask) == prefix) atomicAdd(&sh[(x >> shift) & dmask], 1u);
  }
  flush_and_select(sh, hist + ((size_t)u * 3 + pass) * kBins, st, pass, gridDim.x, &s_last);
  if (pass == 2 && s_last) {
    __threadfence();
    resolve_tie(a, st, key, member, u, per_seq);
  }
}

// Union over KV heads, the trim key (score summed over KV heads), |U|, and digit pass 0 of
// the trim.  Grid (position blocks, B).
__global__ __launch_bounds__(kBlock, SELKV_SEL_MINB) void union_kernel(CompressArgs a, SelectWs w) {
  __shared__ uint32_t sh[kBins];
  __shared__ uint32_t s_cnt;
  __shared__ bool s_last;
  __shared__ uint32_t s_prefix[32];
  __shared__ int s_jcut[32];
  const int b = blockIdx.y;
  const int n = a.seq_n[b], ncand = n - a.recent;
  for (int i = threadIdx.x; i < kBins; i += kBlock) sh[i] = 0u;
  if (threadIdx.x == 0) s_cnt = 0u;
  if (threadIdx.x < a.Hkv) {
    const RadixState t = w.topk[(size_t)b * a.Hkv + threadIdx.x];
    s_prefix[threadIdx.x] = t.prefix;
    s_jcut[threadIdx.x] = t.jcut;
  }
  __syncthreads();
  const int j0 = blockIdx.x * kSpan;
  uint32_t cnt = 0;
#pragma unroll 1
  for (int e = 0; e < kPerThread; ++e) {
    const int j = j0 + e * kBlock + threadIdx.x;
    if (j >= n) continue;
    bool in = false;
    float sum = 0.f;
    for (int kv = 0; kv < a.Hkv; ++kv) {
      const size_t u = (size_t)b * a.Hkv + kv;
      const float s = a.score[u * a.n_cap + j];
      const uint32_t x = __float_as_uint(s);
      const bool mem = j < ncand && (x > s_prefix[kv] || (x == s_prefix[kv] && j <= s_jcut[kv]));
      if (a.dbg_topk != nullptr) a.dbg_topk[u * a.n_cap + j] = mem ? 1 : 0;
      in |= mem;
      sum += s;
    }
    if (j < ncand) {
      w.uflag[(size_t)b * a.n_cap + j] = in ? 1 : 0;
      w.tkey[(size_t)b * a.n_cap + j] = sum;
      if (in) {
        ++cnt;
        atomicAdd(&sh[__float_as_uint(sum) >> 21], 1u);
      }
    }
  }
  atomicAdd(&s_cnt, cnt);
  __syncthreads();
  RadixState* st = &w.trim[b];
  if (threadIdx.x == 0 && s_cnt) atomicAdd(&st->ucount, s_cnt);
  flush_and_select(sh, w.trim_hist + (size_t)b * 3 * kBins, st, 0, gridDim.x, &s_last);
  __syncthreads();
  // the last CTA decides whether the union needs trimming (flush_and_select left its digit)
  if (s_last && threadIdx.x == 0) {
    __threadfence();
    const uint32_t k = (uint32_t)(a.seq_m[b] - a.recent);
    if (__ldcg(&st->ucount) <= k) {  // no trim: every member of the union is kept
      st->active = 0u;
      st->prefix = 0u;
      st->jcut = INT_MAX;
    }
  }
}

// Kept flags and per-block counts.  Shared mode: the trimmed union, then the recent window;
// grid (blocks, B).  Per-head mode: the KV head's own top-m_s (whose choice it also reports),
// then the recent window; grid (blocks, B * Hkv).
__global__ __launch_bounds__(kBlock) void compact_count_kernel(CompressArgs a, SelectWs w) {
  __shared__ uint32_t s_cnt;
  const int u = blockIdx.y, b = a.per_head ? u / a.Hkv : u;
  const int n = a.seq_n[b], ncand = n - a.recent;
  const RadixState st = a.per_head ? w.topk[u] : w.trim[b];
  if (threadIdx.x == 0) s_cnt = 0u;
  __syncthreads();
  const int j0 = blockIdx.x * kSpan;
  uint32_t cnt = 0;
#pragma unroll
  for (int e = 0; e < kPerThread; ++e) {
    const int j = j0 + e * kBlock + threadIdx.x;
    if (j >= n) continue;
    bool kept = true;
    if (j < ncand) {
      if (a.per_head) {
        kept = selected(__float_as_uint(a.score[(size_t)u * a.n_cap + j]), j, st);
        if (a.dbg_topk != nullptr) a.dbg_topk[(size_t)u * a.n_cap + j] = kept ? 1 : 0;
      } else {
        kept = w.uflag[(size_t)b * a.n_cap + j] != 0 &&
               selected(__float_as_uint(w.tkey[(size_t)b * a.n_cap + j]), j, st);
      }
    } else if (a.per_head && a.dbg_topk != nullptr) {
      a.dbg_topk[(size_t)u * a.n_cap + j] = 0;
    }
    a.kflag[(size_t)u * a.n_cap + j] = kept ? 1 : 0;
    cnt += kept ? 1u : 0u;
  }
  atomicAdd(&s_cnt, cnt);
  __syncthreads();
  if (threadIdx.x == 0) w.blkcnt[(size_t)u * gridDim.x + blockIdx.x] = s_cnt;
}

// Slots in position order: block offset (sum of earlier blocks) + rank within the block.
__global__ __launch_bounds__(kBlock) void compact_write_kernel(CompressArgs a, SelectWs w) {
  __shared__ uint32_t wcnt[kBlock / 32 + 1];
  __shared__ uint32_t s_off;
  const int u = blockIdx.y, blk = blockIdx.x, b = a.per_head ? u / a.Hkv : u;
  const int n = a.seq_n[b];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (warp == 0) {
    uint32_t s = 0;
    for (int i = lane; i < blk; i += 32) s += w.blkcnt[(size_t)u * gridDim.x + i];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (lane == 0) s_off = s;
  }
  __syncthreads();
  uint32_t base = s_off;
  const int j0 = blk * kSpan;
  for (int e = 0; e < kPerThread; ++e) {
    const int j = j0 + e * kBlock + threadIdx.x;
    const bool kept = j < n && a.kflag[(size_t)u * a.n_cap + j] != 0;
    const unsigned bal = __ballot_sync(0xffffffffu, kept);
    if (lane == 0) wcnt[warp] = __popc(bal);
    __syncthreads();
    if (warp == 0) {
      const uint32_t v = lane < kBlock / 32 ? wcnt[lane] : 0u;
      uint32_t incl = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t t = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += t;
      }
      if (lane < kBlock / 32) wcnt[lane] = incl - v;
      if (lane == kBlock / 32 - 1) wcnt[kBlock / 32] = incl;
    }
    __syncthreads();
    const uint32_t slot = base + wcnt[warp] + __popc(bal & ((1u << lane) - 1u));
    if (j < n) {
      a.slot_of[(size_t)u * a.n_cap + j] = kept ? (int)slot : -1;
      // with the full cosine routing: the evicted positions in order (slot = kept ones before j)
      if (!kept && a.routing == SELKV_ROUTE_COSINE) a.ev_pos[(size_t)u * a.n_cap + (j - (int)slot)] = j;
      if (kept && (int)slot < a.m_cap) {
        a.kept_pos[(size_t)u * a.m_cap + slot] = j;
        if (a.dbg_kept_idx != nullptr) a.dbg_kept_idx[(size_t)u * a.m_cap + slot] = j;
      }
    }
    base += wcnt[kBlock / 32];
    __syncthreads();
  }
  if (blk == (int)gridDim.x - 1 && threadIdx.x == 0 && (int)base != a.seq_m[b]) raise_flag(a.flags, SELKV_DEVERR_COUNT);
}

}  // namespace

size_t select_ws_bytes(int B, int Hkv, int n_cap) {
  const size_t units = (size_t)B * Hkv;
  const size_t blocks = (size_t)(n_cap + kSpan - 1) / kSpan;
  // seven regions, each start rounded up to 256 bytes
  return (units + B) * sizeof(RadixState) + (units + B) * 3 * kBins * 4 + units * blocks * 4 +
         (size_t)B * n_cap * 5 + 7 * 256;
}

SelectWs carve_select_ws(void* base, int B, int Hkv, int n_cap) {
  const size_t units = (size_t)B * Hkv;
  const size_t blocks = (size_t)(n_cap + kSpan - 1) / kSpan;
  char* p = static_cast<char*>(base);
  auto take = [&](size_t bytes) {
    char* r = p;
    p += (bytes + 255) & ~size_t(255);
    return r;
  };
  SelectWs w{};
  w.topk = reinterpret_cast<RadixState*>(take(units * sizeof(RadixState)));
  w.trim = reinterpret_cast<RadixState*>(take((size_t)B * sizeof(RadixState)));
  w.topk_hist = reinterpret_cast<uint32_t*>(take(units * 3 * kBins * 4));
  w.trim_hist = reinterpret_cast<uint32_t*>(take((size_t)B * 3 * kBins * 4));
  w.hist_bytes = (size_t)(reinterpret_cast<char*>(w.trim_hist) - reinterpret_cast<char*>(w.topk_hist)) +
                 (size_t)B * 3 * kBins * 4;
  w.blkcnt = reinterpret_cast<uint32_t*>(take(units * blocks * 4));  // per selection unit
  w.tkey = reinterpret_cast<float*>(take((size_t)B * n_cap * 4));
  w.uflag = reinterpret_cast<uint8_t*>(take((size_t)B * n_cap));
  return w;
}

// Pooling and the whole selection: 8 kernels (5 in the per-head mode) and one memset, all on
// `s`, no host sync (the radix states are initialised by the set-up kernel).
cudaError_t launch_select_grid(const CompressArgs& a, const SelectWs& w, cudaStream_t s) {
  const int units = a.B * a.Hkv;
  const int blocks = (a.n_cap + kSpan - 1) / kSpan;
  cudaError_t e = cudaMemsetAsync(w.topk_hist, 0, w.hist_bytes, s);
  if (e != cudaSuccess) return e;
  pool_hist0_kernel<<<dim3(blocks, units), kBlock, 0, s>>>(a, w);
  for (int pass = 1; pass < 3; ++pass)
    hist_kernel<<<dim3(blocks, units), kBlock, 0, s>>>(a, w.topk, w.topk_hist, a.score, nullptr, a.Hkv, pass);
  if (!a.per_head) {  // union over KV heads and the trim (shared mode only)
    union_kernel<<<dim3(blocks, a.B), kBlock, 0, s>>>(a, w);
    for (int pass = 1; pass < 3; ++pass)
      hist_kernel<<<dim3(blocks, a.B), kBlock, 0, s>>>(a, w.trim, w.trim_hist, w.tkey, w.uflag, 1, pass);
  }
  const int sel_units = a.per_head ? units : a.B;
  compact_count_kernel<<<dim3(blocks, sel_units), kBlock, 0, s>>>(a, w);
  compact_write_kernel<<<dim3(blocks, sel_units), kBlock, 0, s>>>(a, w);
  return cudaGetLastError();
}

}  // namespace selkv
