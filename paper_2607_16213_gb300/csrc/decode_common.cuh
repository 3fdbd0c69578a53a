// Split-K bookkeeping shared by the decode kernels: the per-split partial layout, the fold of
// a CTA's warp states into one partial, the last-CTA combine of the splits, the append and the
// length update.
//
// Partial layout in the workspace: one record per (b, kv) of decode_record_floats(G, S, D)
// floats, 16-byte aligned:
//   o  [G][S][D]   unnormalised output of each split (fp32)
//   ml [G][S]      (running max in base 2, running sum) of each split, padded to 16 bytes
#pragma once

#include "ptx.cuh"
#include "selkv_internal.cuh"

namespace selkv {

struct PartialView {
  float* base;
  size_t rec;  // floats per (b, kv) record
  int G, S, D;
  __device__ __forceinline__ float* record(size_t bk) const { return base + bk * rec; }
  __device__ __forceinline__ float* o(size_t bk, int g, int s) const {
    return record(bk) + ((size_t)g * S + s) * D;
  }
  __device__ __forceinline__ float2* ml(size_t bk, int g, int s) const {
    return reinterpret_cast<float2*>(record(bk) + (size_t)G * S * D) + g * S + s;
  }
};

__device__ __forceinline__ PartialView partial_view(const DecodeArgs& a) {
  return {a.partial, decode_record_floats(a.G, a.splits, a.D), a.G, a.splits, a.D};
}

// Griddepcontrol (programmatic dependent launch): a no-op for kernels launched without it.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Fold NW warp states (max wm[w*rs+g], sum wl[w*rs+g], output wo[(w*rs+g)*ld+d]) of heads
// g < G into this split's partial.  An aborted CTA leaves an empty partial.
template <int NW>
__device__ __forceinline__ void write_split_partial(const DecodeArgs& a, int b, int kv, int s,
                                                    const float* wo, const float* wm, const float* wl,
                                                    int rs, int ld, bool aborted) {
  const int G = a.G, D = a.D;
  const PartialView pv = partial_view(a);
  const size_t bk = (size_t)b * a.Hkv + kv;
  for (int i = threadIdx.x; i < G * D; i += blockDim.x) {
    const int g = i / D, d = i % D;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < NW; ++w) M = fmaxf(M, wm[w * rs + g]);
    float sl = 0.f, so = 0.f;
    if (M != -INFINITY && !aborted) {
#pragma unroll
      for (int w = 0; w < NW; ++w) {
        const float f = exp2f(wm[w * rs + g] - M);
        sl += wl[w * rs + g] * f;
        so += wo[(w * rs + g) * ld + d] * f;
      }
    } else {
      M = -INFINITY;
    }
    pv.o(bk, g, s)[d] = so;
    if (d == 0) *pv.ml(bk, g, s) = make_float2(M, sl);
  }
}

// One atomic arrival per CTA on the (b, kv) counter; true for the last of the S splits.  The
// CTA barrier orders every thread's partial stores before thread 0's acquire-release bump,
// which publishes them (release is cumulative) and, in the last CTA, acquires the other
// splits' partials before the barrier that lets its threads read them.
__device__ __forceinline__ bool arrive_last(const DecodeArgs& a, size_t bk, bool* s_flag) {
  __syncthreads();
  if (threadIdx.x == 0) *s_flag = atom_add_acq_rel_gpu(&a.cnt_head[bk], 1u) == (uint32_t)a.splits - 1u;
  __syncthreads();
  return *s_flag;
}

// Fold the S split partials of (b, kv) in split order and write out[b][kv*G + g].  Each
// thread owns an output quad: one pass takes the max over the splits, a second sums the
// splits' outputs and sums with weights 2^(max_t - max); the loads of both passes are
// independent of each other, so a pass costs about one memory round trip.
template <typename T>
__device__ __forceinline__ void combine_splits(const DecodeArgs& a, int b, int kv, float* /*scratch*/) {
  const int G = a.G, D = a.D, S = a.splits;
  const PartialView pv = partial_view(a);
  const size_t bk = (size_t)b * a.Hkv + kv;
  const size_t bh0 = bk * G;
  const int D4 = D / 4;
  for (int i = threadIdx.x; i < G * D4; i += blockDim.x) {
    const int g = i / D4, d4 = i % D4;
    const float4* op = reinterpret_cast<const float4*>(pv.o(bk, g, 0)) + d4;
    const float2* mp = pv.ml(bk, g, 0);
    float M = -INFINITY;
#pragma unroll 8
    for (int t = 0; t < S; ++t) M = fmaxf(M, __ldcg(mp + t).x);
    float L = 0.f;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    if (M != -INFINITY) {
#pragma unroll 8
      for (int t = 0; t < S; ++t) {
        const float2 ml = __ldcg(mp + t);
        const float4 v = __ldcg(op + (size_t)t * D4);
        const float w = exp2f(ml.x - M);
        L = fmaf(ml.y, w, L);
        acc.x = fmaf(v.x, w, acc.x);
        acc.y = fmaf(v.y, w, acc.y);
        acc.z = fmaf(v.z, w, acc.z);
        acc.w = fmaf(v.w, w, acc.w);
      }
    }
    const float inv = L > 0.f ? 1.f / L : 0.f;
    const float r[4] = {acc.x * inv, acc.y * inv, acc.z * inv, acc.w * inv};
    store4(static_cast<T*>(a.out) + (bh0 + g) * D + d4 * 4, r);
  }
}

// Write the appended row (k_new, v_new) at row L of K_c / V_c with bias 0.  No CTA of this
// launch reads row L (they read rows below L), so any one CTA may do it.
template <typename T>
__device__ __forceinline__ void write_append_row(const DecodeArgs& a, size_t bk, int L, int tid, int nthreads) {
  const int D = a.D;
  const uint4* kn = reinterpret_cast<const uint4*>(static_cast<const T*>(a.k_new) + bk * D);
  const uint4* vn = reinterpret_cast<const uint4*>(static_cast<const T*>(a.v_new) + bk * D);
  uint4* Kw = reinterpret_cast<uint4*>(static_cast<T*>(a.Kc) + (bk * a.m_cap + L) * D);
  uint4* Vw = reinterpret_cast<uint4*>(static_cast<T*>(a.Vc) + (bk * a.m_cap + L) * D);
  const int n16 = D * (int)sizeof(T) / 16;
  for (int i = tid; i < n16; i += nthreads) {
    Kw[i] = kn[i];
    Vw[i] = vn[i];
  }
  if (a.bias != nullptr && tid == 0) a.bias[bk * a.m_cap + L] = 0.f;
}

// Length bookkeeping of the last CTA of (b, kv), split in two so the atomic's round trip
// overlaps the combine; thread `owner` does both halves.  begin: reset the (b, kv) counter
// and count this head on the sequence's counter; every CTA of the sequence has read
// lengths[b] before its own arrival, so the last head to count may advance it.  end: that
// head writes lengths[b] = L + 1.  The count is acquire-release: it acquires the heads that
// counted before it and releases this head's own split CTAs' reads of lengths[b] (acquired
// through their arrivals) to the head that writes it.  A CTA that leaves early (a timed-out
// wait) still runs end, so the sequence's counter is reset for the next launch.
__device__ __forceinline__ uint32_t finish_lengths_begin(const DecodeArgs& a, int b, size_t bk, bool app,
                                                         int owner = 0) {
  uint32_t old = 0u;
  if ((int)threadIdx.x == owner) {
    a.cnt_head[bk] = 0u;
    if (app) old = atom_add_acq_rel_gpu(&a.cnt_seq[b], 1u);
  }
  return old;
}
__device__ __forceinline__ void finish_lengths_end(const DecodeArgs& a, int b, int L, bool app, uint32_t old,
                                                   int owner = 0) {
  if ((int)threadIdx.x == owner && app && old == (uint32_t)a.Hkv - 1u) {
    a.lengths[b] = L + 1;
    a.cnt_seq[b] = 0u;
  }
}
__device__ __forceinline__ void finish_lengths(const DecodeArgs& a, int b, size_t bk, int L, bool app) {
  finish_lengths_end(a, b, L, app, finish_lengths_begin(a, b, bk, app));
}

}  // namespace selkv
