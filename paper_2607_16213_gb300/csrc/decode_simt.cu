// Compensated decode attention on CUDA cores for fp32 caches (bf16 caches use decode_tc.cu).
//
//   out[b][h] = sum_i softmax_i(q_h . k_i / sqrt(d) + bias_i) v_i      (Alg. 1 decode,
//                                                                     Sec. 3.6 compensation)
// Split-K flash decoding: CTA (split s, KV head kv, sequence b) streams a contiguous slice of
// the compressed rows once for all G query heads of the group, keeping a running max / sum
// per head in the base-2 domain (the bias is folded into the logit before the max).  Each CTA
// leaves (max, sum, unnormalised output) in the workspace; the last CTA of a (b, kv) to
// arrive (one atomic add, no waiting) folds the splits in split order, so the result does
// not depend on scheduling.  With k_new / v_new the new row joins the softmax with bias 0 and
// is then written at row lengths[b]; the last (b, kv) of a sequence bumps lengths[b].
#include <algorithm>

#include "decode_common.cuh"
#include "selkv_internal.cuh"

namespace selkv {
namespace {

constexpr int kWarps = 4;

template <typename T, int D, int GM>
__global__ __launch_bounds__(kWarps * 32) void decode_simt_kernel(DecodeArgs a) {
  constexpr int PER = D / 32;
  __shared__ __align__(16) float qs[GM][D];
  __shared__ float wm[kWarps][GM], wl[kWarps][GM];
  __shared__ float wo[kWarps][GM][D];
  __shared__ bool s_last;
  const int s = blockIdx.x, kv = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int G = a.G, S = a.splits;
  const size_t bk = (size_t)b * a.Hkv + kv;

  int L = a.lengths[b];
  if (L < 0 || L > a.m_cap) {
    if (tid == 0 && s == 0 && kv == 0) raise_flag(a.flags, SELKV_DEVERR_LENGTH);
    L = L < 0 ? 0 : a.m_cap;
  }
  bool app = a.k_new != nullptr;
  if (app && L + 1 > a.m_cap) {
    if (tid == 0 && s == 0 && kv == 0) raise_flag(a.flags, SELKV_DEVERR_CAPACITY);
    app = false;
  }
  const int total = L + (app ? 1 : 0);
  const int chunk = ((total + S - 1) / S + 31) / 32 * 32;
  const int lo = s * chunk, hi = min(total, lo + chunk);

  for (int i = tid; i < G * D; i += blockDim.x) {
    const int g = i / D, d = i % D;
    qs[g][d] = load1(static_cast<const T*>(a.q) + ((size_t)b * a.Hq + kv * G + g) * D + d) * a.scale_log2;
  }
  __syncthreads();

  const T* Kb = static_cast<const T*>(a.Kc) + bk * a.m_cap * D;
  const T* Vb = static_cast<const T*>(a.Vc) + bk * a.m_cap * D;
  const T* kn = app ? static_cast<const T*>(a.k_new) + bk * D : nullptr;
  const T* vnw = app ? static_cast<const T*>(a.v_new) + bk * D : nullptr;
  const float* bias = a.bias != nullptr ? a.bias + bk * a.m_cap : nullptr;

  float m[GM], l[GM], o[GM][PER], pg[GM];
#pragma unroll
  for (int g = 0; g < GM; ++g) {
    m[g] = -INFINITY;
    l[g] = 0.f;
#pragma unroll
    for (int e = 0; e < PER; ++e) o[g][e] = 0.f;
  }
  for (int t0 = lo + warp * 32; t0 < hi; t0 += kWarps * 32) {
    const int key = t0 + lane;
    const bool valid = key < hi;
    float sc[GM];
#pragma unroll
    for (int g = 0; g < GM; ++g) sc[g] = 0.f;
    if (valid) {
      const T* kr = key < L ? Kb + (size_t)key * D : kn;
#pragma unroll 4
      for (int d = 0; d < D; d += 8) {
        float x[8];
        load8(kr + d, x);
#pragma unroll
        for (int g = 0; g < GM; ++g) {
          if (g < G) {
#pragma unroll
            for (int e = 0; e < 8; ++e) sc[g] = fmaf(qs[g][d + e], x[e], sc[g]);
          }
        }
      }
    }
    const float bv = (valid && key < L && bias != nullptr) ? bias[key] * kLog2e : 0.f;
#pragma unroll
    for (int g = 0; g < GM; ++g) {
      if (g >= G) break;
      const float v = valid ? sc[g] + bv : -INFINITY;
      const float mn = fmaxf(m[g], warp_max(v));
      const float corr = exp2f(m[g] - mn);
      const float p = exp2f(v - mn);
      l[g] = l[g] * corr + warp_sum(p);
#pragma unroll
      for (int e = 0; e < PER; ++e) o[g][e] *= corr;
      m[g] = mn;
      pg[g] = p;
    }
    const int nk = min(32, hi - t0);
    for (int k = 0; k < nk; ++k) {
      const int key2 = t0 + k;
      const T* vr = key2 < L ? Vb + (size_t)key2 * D : vnw;
      float v[PER];
      if constexpr (PER == 4) load4(vr + lane * 4, v); else load2(vr + lane * 2, v);
#pragma unroll
      for (int g = 0; g < GM; ++g) {
        if (g >= G) break;
        const float pk = __shfl_sync(0xffffffffu, pg[g], k);
#pragma unroll
        for (int e = 0; e < PER; ++e) o[g][e] = fmaf(pk, v[e], o[g][e]);
      }
    }
  }
  // fold the warps
#pragma unroll
  for (int g = 0; g < GM; ++g) {
    if (g >= G) break;
    if (lane == 0) {
      wm[warp][g] = m[g];
      wl[warp][g] = l[g];
    }
#pragma unroll
    for (int e = 0; e < PER; ++e) wo[warp][g][lane * PER + e] = o[g][e];
  }
  __syncthreads();
  write_split_partial<kWarps>(a, b, kv, s, &wo[0][0][0], &wm[0][0], &wl[0][0], GM, D, false);
  if (!arrive_last(a, bk, &s_last)) return;
  combine_splits<T>(a, b, kv, &wo[0][0][0]);
  if (app) write_append_row<T>(a, bk, L, threadIdx.x, blockDim.x);
  finish_lengths(a, b, bk, L, app);
}

template <typename T, int D>
cudaError_t launch_t(const DecodeArgs& a, cudaStream_t st) {
  const dim3 grid(a.splits, a.Hkv, a.B);
  const int th = kWarps * 32;
  if (a.G <= 1) decode_simt_kernel<T, D, 1><<<grid, th, 0, st>>>(a);
  else if (a.G <= 2) decode_simt_kernel<T, D, 2><<<grid, th, 0, st>>>(a);
  else if (a.G <= 4) decode_simt_kernel<T, D, 4><<<grid, th, 0, st>>>(a);
  else if (a.G <= 8) decode_simt_kernel<T, D, 8><<<grid, th, 0, st>>>(a);
  else decode_simt_kernel<T, D, 16><<<grid, th, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace

#ifndef SELKV_DEC_CTAS_PER_SM
#define SELKV_DEC_CTAS_PER_SM 1  // decode CTAs planned per SM when splitting the rows
#endif
#ifndef SELKV_DEC_FILL_ROWS
#define SELKV_DEC_FILL_ROWS 256  // a CTA's fixed cost in the split model, in rows streamed
#endif
#ifndef SELKV_DEC_BACKFILL_WAVES
#define SELKV_DEC_BACKFILL_WAVES 3  // one split over at least this many waves of units ...
#endif
#ifndef SELKV_DEC_BACKFILL_MAX_ROWS
#define SELKV_DEC_BACKFILL_MAX_ROWS 8192  // ... of at most this many rows: fractional waves
#endif
#ifndef SELKV_DEC_MAX_SPLITS
#define SELKV_DEC_MAX_SPLITS 64  // most splits of one (sequence, KV head)
#endif

// Split count of each (sequence, KV head).  The B * Hkv * S CTAs run in waves of
// CTAS_PER_SM * num_sms; a wave lasts about as long as streaming one CTA's rows plus a fixed
// fill-and-fold cost worth kFillRows rows.  S minimises waves * (rows per CTA + kFillRows) over
// the capacity m_cap, fewest splits on ties.  With `unit_walk` (the tensor-core decode), one
// split over more units than slots with at most SELKV_DEC_UNITS_MAX_ROWS rows runs as
// persistent CTAs that pay the fixed cost once: waves * rows + kFillRows.  There too, one split
// over at least BACKFILL_WAVES waves of units of at most BACKFILL_MAX_ROWS rows counts its waves as
// units / slots: the block scheduler starts each unit as a slot frees, so ragged units pack
// (batch 64 x 8k at 50%: 151.0 -> 144.0 us per launch, 64 x 32k at 10%: 129.6 -> 120.7; with
// longer units the last ones started leave a tail: 64 x 32k at 50% 490 -> 496, 64 x 128k at
// 25% 924 -> 972, so those keep their splits).  (Serving sweep, batch 8 x 32k at 50%: 256
// rows of fixed cost pick more splits than 512 did, 85.7 -> 71.0 us per launch; batch 4 x 8k:
// 4 splits either way.)
int decode_splits(int B, int Hkv, int m_cap, int num_sms, bool unit_walk) {
  constexpr long kFillRows = SELKV_DEC_FILL_ROWS;
  const long units = (long)B * Hkv;
  const long slots = std::max(1L, (long)SELKV_DEC_CTAS_PER_SM * num_sms);
  const int smax = std::max(1, std::min(SELKV_DEC_MAX_SPLITS, (m_cap + 63) / 64));
  int best = 1;
  long best_cost = -1;
  for (int S = 1; S <= smax; ++S) {
    // costs in units of rows x slots, so that fractional waves stay integral
    const long waves = (units * S + slots - 1) / slots * slots;
    const long rows = ((long)(m_cap + S - 1) / S + 63) / 64 * 64;
    const bool walk = unit_walk && S == 1 && units > slots && m_cap <= SELKV_DEC_UNITS_MAX_ROWS;
    const bool backfill = unit_walk && S == 1 && !walk && units >= (long)SELKV_DEC_BACKFILL_WAVES * slots &&
                          m_cap <= SELKV_DEC_BACKFILL_MAX_ROWS;
    const long cost = walk ? waves * rows + kFillRows * slots
                           : (backfill ? units : waves) * (rows + kFillRows);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best = S;
    }
  }
  return best;
}

cudaError_t launch_decode(const DecodeArgs& a, cudaStream_t st) {
  if (a.dtype == SELKV_BF16) return launch_decode_tc(a, st);
  return a.D == 128 ? launch_t<float, 128>(a, st) : launch_t<float, 64>(a, st);
}

}  // namespace selkv
