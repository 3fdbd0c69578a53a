// Bucket-attention routing, soft cosine gate, gated merge, attention ratio and the
// compressed-cache write-out of SelKV (Eq. 3-6, Sec. 3.6 GQA bias).
//
// One CTA per (bucket X, sequence b) with one warp per KV head.  Under Eq. 3 (argmax over the
// kept tokens of the bucket of the cumulative attention a) every evicted token of a bucket
// routes to the same kept token tau_X, so the merge is a gather: the CTA of a non-empty bucket
// X collects, in ascending position order, the evicted tokens of X and of the empty buckets
// whose nearest non-empty ring resolves to X, accumulates
//     num = sum g_j a_j v_j,   den = sum g_j a_j,   g_j = clamp(cos(v_j, v_tau), 0, 1),
// and writes v~_tau = (a_tau v_tau + num) / (a_tau + den), R_tau = (a_tau + den) / a_tau.
// Every kept token of X is copied to its slot of K_c / V_c (keys unchanged), and
// bias = alpha * ln(mean over KV heads of R) is written once all warps have their R.
// No floating-point atomics: the summation order is fixed, so results are reproducible.
#include <climits>

#include "selkv_internal.cuh"

namespace selkv {
namespace {

template <typename T, int D, int MAXT>
__global__ __launch_bounds__(MAXT) void merge_kernel(CompressArgs a) {
  constexpr int PER = D / 32;  // elements of a row per lane
  __shared__ float Rs[32][33];
  const int X = blockIdx.x, b = blockIdx.y;
  const int kv = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n = a.seq_n[b];
  const int Bs = a.bucket;
  const int nb = (n + Bs - 1) / Bs;
  if (X >= nb) return;
  const uint8_t* kf = a.kflag + (size_t)b * a.n_cap;
  auto bucket_mask = [&](int e) -> uint32_t {
    const int p = e * Bs + lane;
    const bool k = lane < Bs && p < n && kf[p] != 0;
    return __ballot_sync(0xffffffffu, k);
  };
  const size_t bk = (size_t)b * a.Hkv + kv;
  const float* A = a.attn + bk * a.n_cap;
  const float* vn = a.vnorm + bk * a.n_cap;
  const T* Vb = static_cast<const T*>(a.V) + bk * a.n_cap * D;
  const int base = X * Bs;
  const int cntX = min(Bs, n - base);
  // this lane's position of bucket X: a and ||v||, fetched together with the kept flags
  const float A_l = lane < cntX ? A[base + lane] : -INFINITY;
  const float vn_l = lane < cntX ? vn[base + lane] : 0.f;
  const uint32_t mX = bucket_mask(X);
  if (mX == 0u) {
    // Empty bucket: under EXPAND a neighbour's CTA owns these tokens; under DROP (or with
    // nothing kept at all) they stay without target.
    if (a.empty_bucket == SELKV_EMPTY_DROP || a.seq_m[b] == 0) {
      if (lane < cntX) {
        const size_t o = bk * a.n_cap + base + lane;
        if (a.dbg_target) a.dbg_target[o] = -1;
        if (a.dbg_gate) a.dbg_gate[o] = 0.f;
        if (a.dbg_decision) a.dbg_decision[o] = 0;
      }
    }
    return;
  }
  // argmax of a over the kept tokens of a bucket (larger a, then lower position).
  auto best_of = [&](float v, int idx) -> int {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float v2 = __shfl_xor_sync(0xffffffffu, v, o);
      const int i2 = __shfl_xor_sync(0xffffffffu, idx, o);
      if (v2 > v || (v2 == v && i2 < idx)) { v = v2; idx = i2; }
    }
    return idx;
  };
  auto best_in = [&](int e, uint32_t mask) -> int {
    const bool in = (mask >> lane) & 1u;
    return best_of(in ? A[e * Bs + lane] : -INFINITY, in ? e * Bs + lane : INT_MAX);
  };
  const bool inX = (mX >> lane) & 1u;
  const int tau = best_of(inX ? A_l : -INFINITY, inX ? base + lane : INT_MAX);
  const float a_tau = __shfl_sync(0xffffffffu, A_l, tau - base);
  const float vn_tau = __shfl_sync(0xffffffffu, vn_l, tau - base);
  int lo_b = X, hi_b = X;  // buckets whose evicted tokens route to tau
  if (a.empty_bucket == SELKV_EMPTY_EXPAND) {
    int L = X - 1;
    uint32_t mL = 0u;
    while (L >= 0 && (mL = bucket_mask(L)) == 0u) --L;
    if (L < 0) {
      lo_b = 0;
    } else if (L < X - 1) {
      // empty e in (L, X): X is nearer iff X - e < e - L; at equal distance the ring holds
      // both buckets and X wins only with a strictly larger a (tau_L has the lower index).
      lo_b = (X + L) / 2 + 1;
      if (((X + L) & 1) == 0 && a_tau > A[best_in(L, mL)]) lo_b = (X + L) / 2;
    }
    int Rb = X + 1;
    uint32_t mR = 0u;
    while (Rb < nb && (mR = bucket_mask(Rb)) == 0u) ++Rb;
    if (Rb >= nb) {
      hi_b = nb - 1;
    } else if (Rb > X + 1) {
      hi_b = (X + Rb - 1) / 2;
      if (((X + Rb) & 1) == 0 && a_tau >= A[best_in(Rb, mR)]) hi_b = (X + Rb) / 2;
    }
  }
  float vt[PER];
  if constexpr (PER == 4) load4(Vb + (size_t)tau * D + lane * 4, vt); else load2(Vb + (size_t)tau * D + lane * 2, vt);

  float num[PER];
#pragma unroll
  for (int e = 0; e < PER; ++e) num[e] = 0.f;
  float den = 0.f;
  // Contributors in ascending position order, a batch at a time: their loads are independent
  // and their dot-product reductions interleave (the sums stay in position order).
  constexpr int kBatch = MAXT <= 256 ? 8 : 4;
  for (int e = lo_b; e <= hi_b; ++e) {
    const int eb = e * Bs;
    const int cnt_e = min(Bs, n - eb);
    const uint32_t valid = cnt_e >= 32 ? 0xffffffffu : ((1u << cnt_e) - 1u);
    const bool own = e == X;
    uint32_t rem = valid & ~(own ? mX : 0u);
    // a and ||v|| of bucket e, one position per lane
    const float Ae = own ? A_l : (lane < cnt_e ? A[eb + lane] : 0.f);
    const float Ne = own ? vn_l : (lane < cnt_e ? vn[eb + lane] : 0.f);
    while (rem) {
      int pos[kBatch];
      int nb_ = 0;
#pragma unroll
      for (int k = 0; k < kBatch; ++k) {
        pos[k] = -1;
        if (rem) {
          pos[k] = eb + __ffs(rem) - 1;
          rem &= rem - 1u;
          ++nb_;
        }
      }
      float vj[kBatch][PER];
      float dot[kBatch];
#pragma unroll
      for (int k = 0; k < kBatch; ++k) {
        if (pos[k] >= 0) {
          if constexpr (PER == 4) load4(Vb + (size_t)pos[k] * D + lane * 4, vj[k]);
          else load2(Vb + (size_t)pos[k] * D + lane * 2, vj[k]);
        } else {
#pragma unroll
          for (int t = 0; t < PER; ++t) vj[k][t] = 0.f;
        }
        dot[k] = 0.f;
#pragma unroll
        for (int t = 0; t < PER; ++t) dot[k] = fmaf(vj[k][t], vt[t], dot[k]);
      }
      if (a.gate_mode == SELKV_GATE_COSINE) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1)
#pragma unroll
          for (int k = 0; k < kBatch; ++k) dot[k] += __shfl_xor_sync(0xffffffffu, dot[k], o);
      }
#pragma unroll
      for (int k = 0; k < kBatch; ++k) {
        if (k >= nb_) break;
        const int src = pos[k] - eb;
        const float ak = __shfl_sync(0xffffffffu, Ae, src);
        const float nk = __shfl_sync(0xffffffffu, Ne, src);
        float g;
        if (a.gate_mode == SELKV_GATE_OPEN) {
          g = 1.f;
        } else if (a.gate_mode == SELKV_GATE_CLOSED) {
          g = 0.f;
        } else {
          const float sim = (nk == 0.f || vn_tau == 0.f) ? 0.f : dot[k] / (nk * vn_tau);
          g = fminf(fmaxf(sim, 0.f), 1.f);
        }
        const float w = g * ak;
#pragma unroll
        for (int t = 0; t < PER; ++t) num[t] = fmaf(w, vj[k][t], num[t]);
        den += w;
        if (lane == k) {
          const size_t o = bk * a.n_cap + pos[k];
          if (a.dbg_target) a.dbg_target[o] = tau;
          if (a.dbg_gate) a.dbg_gate[o] = g;
          if (a.dbg_decision) a.dbg_decision[o] = g > 0.f ? 1 : 0;
        }
      }
    }
  }
  const float tot = a_tau + den;
  float vm[PER];
#pragma unroll
  for (int t = 0; t < PER; ++t) vm[t] = tot > 0.f ? (a_tau * vt[t] + num[t]) / tot : vt[t];
  const float R_tau = a_tau > 0.f ? tot / a_tau : 1.f;

  // Kept tokens of X, four at a time (loads first, then stores).
  const T* Kb = static_cast<const T*>(a.K) + bk * a.n_cap * D;
  T* Kc = static_cast<T*>(a.Kc) + bk * a.m_cap * D;
  T* Vc = static_cast<T*>(a.Vc) + bk * a.m_cap * D;
  const int32_t* so = a.slot_of + (size_t)b * a.n_cap;
  uint32_t rem = mX;
  while (rem) {
    constexpr int kCopy = 4;
    int tk[kCopy], sl[kCopy];
#pragma unroll
    for (int k = 0; k < kCopy; ++k) {
      tk[k] = -1;
      sl[k] = -1;
      if (rem) {
        tk[k] = __ffs(rem) - 1;
        rem &= rem - 1u;
        sl[k] = so[base + tk[k]];
        if (sl[k] < 0 || sl[k] >= a.m_cap) {
          if (lane == 0) raise_flag(a.flags, SELKV_DEVERR_COUNT);
          sl[k] = -1;
        }
      }
    }
    float kx[kCopy][PER], vx[kCopy][PER];
#pragma unroll
    for (int k = 0; k < kCopy; ++k) {
      if (sl[k] < 0) continue;
      const int p = base + tk[k];
      if constexpr (PER == 4) {
        load4(Kb + (size_t)p * D + lane * 4, kx[k]);
        if (p != tau) load4(Vb + (size_t)p * D + lane * 4, vx[k]);
      } else {
        load2(Kb + (size_t)p * D + lane * 2, kx[k]);
        if (p != tau) load2(Vb + (size_t)p * D + lane * 2, vx[k]);
      }
      if (p == tau) {
#pragma unroll
        for (int e = 0; e < PER; ++e) vx[k][e] = vm[e];
      }
    }
#pragma unroll
    for (int k = 0; k < kCopy; ++k) {
      if (sl[k] < 0) continue;
      const int p = base + tk[k];
      const int slot = sl[k];
      if constexpr (PER == 4) {
        store4(Kc + (size_t)slot * D + lane * 4, kx[k]);
        store4(Vc + (size_t)slot * D + lane * 4, vx[k]);
      } else {
        store1(Kc + (size_t)slot * D + lane * 2, kx[k][0]);
        store1(Kc + (size_t)slot * D + lane * 2 + 1, kx[k][1]);
        store1(Vc + (size_t)slot * D + lane * 2, vx[k][0]);
        store1(Vc + (size_t)slot * D + lane * 2 + 1, vx[k][1]);
      }
      if (lane == 0) {
        const float Rv = (p == tau) ? R_tau : 1.f;
        Rs[kv][tk[k]] = Rv;
        const size_t o = bk * a.n_cap + p;
        if (a.dbg_target) a.dbg_target[o] = -1;
        if (a.dbg_gate) a.dbg_gate[o] = 0.f;
        if (a.dbg_decision) a.dbg_decision[o] = 2;
        if (a.dbg_ratio) a.dbg_ratio[bk * a.m_cap + slot] = Rv;
      }
    }
  }
  __syncthreads();
  // bias = alpha * ln(mean over KV heads of R) (Sec. 3.6, GQA), the same row for every head.
  if (inX) {
    const int slot = so[base + lane];
    if (slot >= 0 && slot < a.m_cap) {
      float s = 0.f;
      for (int h = 0; h < a.Hkv; ++h) s += Rs[h][lane];
      a.bias[bk * a.m_cap + slot] = a.alpha * logf(s / (float)a.Hkv);
    }
  }
}

template <typename T, int D>
void launch_merge_t(const CompressArgs& a, dim3 grid, int threads, cudaStream_t s) {
  if (threads <= 256) merge_kernel<T, D, 256><<<grid, threads, 0, s>>>(a);
  else merge_kernel<T, D, 1024><<<grid, threads, 0, s>>>(a);
}

}  // namespace

cudaError_t launch_merge(const CompressArgs& a, cudaStream_t s) {
  const int nb = (a.n_cap + a.bucket - 1) / a.bucket;
  const dim3 grid(nb, a.B);
  const int threads = 32 * a.Hkv;
  if (a.dtype == SELKV_BF16) {
    if (a.D == 128) launch_merge_t<__nv_bfloat16, 128>(a, grid, threads, s);
    else launch_merge_t<__nv_bfloat16, 64>(a, grid, threads, s);
  } else {
    if (a.D == 128) launch_merge_t<float, 128>(a, grid, threads, s);
    else launch_merge_t<float, 64>(a, grid, threads, s);
  }
  return cudaGetLastError();
}

}  // namespace selkv
