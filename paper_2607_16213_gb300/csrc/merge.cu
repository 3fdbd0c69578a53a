// Bucket-attention routing, soft cosine gate, gated merge, attention ratio and the
// compressed-cache write-out of SelKV (Eq. 3-6, Sec. 3.6 GQA bias).  With the full cosine
// routing the route and merge kernels give way to those of route_cosine.cu, launched after
// the copy.
//
// Under Eq. 3 (argmax over the kept tokens of a bucket of the cumulative attention a) every
// evicted token of a bucket routes to the same kept token tau_X, so the merge is a gather.
// The kernels, in stream order:
//   route  warp per (bucket X, sequence b): tau_X and a(tau_X) for every KV head (-1 / -inf
//          for a bucket with no kept token);
//   copy   (only with RoPE repositioning or the cosine routing) every kept token's key and
//          value row to its slot of K_c / V_c and ratio 1 for the slot; a thread per 16
//          bytes, coalesced.  Keys are unchanged, or, with RoPE repositioning (Eq. 7),
//          turned by the shift from their position to their slot;
//   merge  one-warp CTA per (non-empty bucket X, KV head, sequence b): the evicted tokens of X and of
//          the empty buckets that the nearest-ring rule gives to X, in ascending position
//          order, 16 at a time: g_j = clamp(cos(v_j, v_tau), 0, 1) and
//              v~_tau = (a_tau v_tau + sum g_j a_j v_j) / (a_tau + sum g_j a_j),
//              R_tau  = (a_tau + sum g_j a_j) / a_tau,
//          written over tau's slot; without the copy kernel the same warp then copies X's
//          kept key rows and its other kept value rows to their slots (ratio 1);
//   bias   bias = alpha * ln(mean over KV heads of R) for every slot (the same row for every
//          KV head).
// No floating-point atomics: every sum has a fixed order, so results are reproducible.
#include <climits>

#include "ptx.cuh"
#include "selkv_internal.cuh"

namespace selkv {
namespace {

constexpr int kWarpsPerCta = 8;
constexpr int kBatch = 16;  // contributors per merge batch

// argmax over the lanes of (value, position): larger value, then lower position
__device__ __forceinline__ void argmax_lanes(float& v, int& idx) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float v2 = __shfl_xor_sync(0xffffffffu, v, o);
    const int i2 = __shfl_xor_sync(0xffffffffu, idx, o);
    if (v2 > v || (v2 == v && i2 < idx)) {
      v = v2;
      idx = i2;
    }
  }
}

__global__ __launch_bounds__(kWarpsPerCta * 32) void route_kernel(CompressArgs a) {
  const int lane = threadIdx.x & 31;
  const int X = blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5), b = blockIdx.y;
  const int n = a.seq_n[b], Bs = a.bucket;
  const int nb = (n + Bs - 1) / Bs;
  if (X >= nb) return;
  const int p = X * Bs + lane;
  const bool valid = lane < Bs && p < n;
  bool kept = valid && a.kflag[sel_unit(a, b, 0) * a.n_cap + p] != 0;
  for (int kv = 0; kv < a.Hkv; ++kv) {
    const size_t bk = (size_t)b * a.Hkv + kv;
    if (a.per_head && kv > 0) kept = valid && a.kflag[bk * a.n_cap + p] != 0;
    float v = kept ? a.attn[bk * a.n_cap + p] : -INFINITY;
    int idx = kept ? p : INT_MAX;
    argmax_lanes(v, idx);
    if (lane == 0) {
      a.tau[bk * a.nbk + X] = idx == INT_MAX ? -1 : idx;
      a.atau[bk * a.nbk + X] = v;
    }
  }
}

// RoPE repositioning tables (Eq. 7): for frequency f, w_f = theta^(-2f/d); row c < rope_hi
// holds (cos, sin) of (256 c) w_f for every f, and row rope_hi + c those of c w_f (c < 256),
// so a shift e = 256 e_hi + e_lo composes two rows (the frequencies of a row are contiguous).
// Angles are reduced modulo 2 pi in fp64 before the sine and cosine, so shifts of 10^5
// positions stay accurate to fp32 rounding.
constexpr int kRopeRowsPerThread = 8;
__global__ void rope_table_kernel(CompressArgs a) {
  const int half = a.D / 2, rows = a.rope_hi + 256;
  const int groups = (rows + kRopeRowsPerThread - 1) / kRopeRowsPerThread;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= half * groups) return;
  const int f = i % half, c0 = (i / half) * kRopeRowsPerThread;
  const double w = pow((double)a.rope_theta, -2.0 * f / a.D);
  const double two_pi = 6.283185307179586;
  for (int c = c0; c < min(rows, c0 + kRopeRowsPerThread); ++c) {
    const double e = c < a.rope_hi ? 256.0 * c : (double)(c - a.rope_hi);
    double ang = e * w;
    ang -= two_pi * rint(ang / two_pi);  // in [-pi, pi], exact to fp64 rounding
    float sn, cs;
    sincosf((float)ang, &sn, &cs);
    a.rope_tab[(size_t)c * half + f] = make_float2(cs, sn);
  }
}

// (cos, sin) of e w_f for the N consecutive frequencies f0 .. f0 + N - 1 (f0 and N even),
// from the coarse and the fine row of e.
template <int N>
__device__ __forceinline__ void rope_angles(const CompressArgs& a, int f0, int e, float2 (&cs)[N]) {
  const int half = a.D / 2;
  const float4* h = reinterpret_cast<const float4*>(a.rope_tab + (size_t)(e >> 8) * half + f0);
  const float4* l = reinterpret_cast<const float4*>(a.rope_tab + (size_t)(a.rope_hi + (e & 255)) * half + f0);
#pragma unroll
  for (int t = 0; t < N / 2; ++t) {
    const float4 hv = h[t], lv = l[t];
    cs[2 * t] = make_float2(hv.x * lv.x - hv.y * lv.y, hv.y * lv.x + hv.x * lv.y);
    cs[2 * t + 1] = make_float2(hv.z * lv.z - hv.w * lv.w, hv.w * lv.z + hv.z * lv.w);
  }
}

// Turn the pair (x, y) back by e w_f (from position j to slot j - e).
__device__ __forceinline__ void rope_back(float& x, float& y, float2 cs) {
  const float nx = x * cs.x + y * cs.y, ny = y * cs.x - x * cs.y;
  x = nx;
  y = ny;
}

template <typename T>
__device__ __forceinline__ void unpack16(const uint4& u, float* x);
template <>
__device__ __forceinline__ void unpack16<__nv_bfloat16>(const uint4& u, float* x) {
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    x[2 * i] = bf16_lo(w[i]);
    x[2 * i + 1] = bf16_hi(w[i]);
  }
}
template <>
__device__ __forceinline__ void unpack16<float>(const uint4& u, float* x) {
  x[0] = __uint_as_float(u.x);
  x[1] = __uint_as_float(u.y);
  x[2] = __uint_as_float(u.z);
  x[3] = __uint_as_float(u.w);
}
template <typename T>
__device__ __forceinline__ void unpack8(const uint2& u, float* x);
template <>
__device__ __forceinline__ void unpack8<__nv_bfloat16>(const uint2& u, float* x) {
  x[0] = bf16_lo(u.x);
  x[1] = bf16_hi(u.x);
  x[2] = bf16_lo(u.y);
  x[3] = bf16_hi(u.y);
}
template <>
__device__ __forceinline__ void unpack8<float>(const uint2& u, float* x) {
  x[0] = __uint_as_float(u.x);
  x[1] = __uint_as_float(u.y);
}
template <typename T>
__device__ __forceinline__ uint2 pack8(const float* x);
template <>
__device__ __forceinline__ uint2 pack8<__nv_bfloat16>(const float* x) {
  return make_uint2(pack_bf16(x[0], x[1]), pack_bf16(x[2], x[3]));
}
template <>
__device__ __forceinline__ uint2 pack8<float>(const float* x) {
  return make_uint2(__float_as_uint(x[0]), __float_as_uint(x[1]));
}
template <typename T>
__device__ __forceinline__ uint4 pack16(const float* x);
template <>
__device__ __forceinline__ uint4 pack16<__nv_bfloat16>(const float* x) {
  return make_uint4(pack_bf16(x[0], x[1]), pack_bf16(x[2], x[3]), pack_bf16(x[4], x[5]), pack_bf16(x[6], x[7]));
}
template <>
__device__ __forceinline__ uint4 pack16<float>(const float* x) {
  return make_uint4(__float_as_uint(x[0]), __float_as_uint(x[1]), __float_as_uint(x[2]), __float_as_uint(x[3]));
}

// One thread per 16 bytes of a kept row: the K and V rows of slot s of (b, kv).  With RoPE
// repositioning a key row is turned by the shift e = position - slot; in the HALF layout the
// thread of piece p takes the 8-byte pieces p and p + (pieces per row) of the row, so its
// elements pair with the ones d/2 further on (the pairs (f, f + d/2)).
template <typename T, int D>
__global__ __launch_bounds__(256) void copy_kernel(CompressArgs a) {
  constexpr int kPieces = D * (int)sizeof(T) / 16;  // 16-byte pieces per row
  constexpr int kEpp = 16 / (int)sizeof(T);          // elements per piece
  const int b = blockIdx.y;
  const int m = a.seq_m[b];
  const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int piece = (int)(i % kPieces);
  const size_t row = i / kPieces;  // over (kv, slot, tensor)
  const int tensor = (int)(row & 1);
  const size_t ks = row >> 1;
  const int slot = (int)(ks % a.m_cap);
  const int kv = (int)(ks / a.m_cap);
  if (kv >= a.Hkv || slot >= m) return;
  const int pos = a.kept_pos[sel_unit(a, b, kv) * a.m_cap + slot];
  const size_t bk = (size_t)b * a.Hkv + kv;
  if (pos < 0 || pos >= a.n_cap) {
    if (piece == 0 && tensor == 0) raise_flag(a.flags, SELKV_DEVERR_COUNT);
    return;
  }
  const uint4* src = reinterpret_cast<const uint4*>(static_cast<const T*>(tensor ? a.V : a.K) + (bk * a.n_cap + pos) * D);
  uint4* dst = reinterpret_cast<uint4*>(static_cast<T*>(tensor ? a.Vc : a.Kc) + (bk * a.m_cap + slot) * D);
  if (tensor == 0 && a.rope != SELKV_ROPE_OFF) {
    const int e = max(0, pos - slot);  // kept positions ascend with their slots
    if (a.rope == SELKV_ROPE_HALF) {
      // lane `piece` takes elements [h0, h0 + kEpp/2) of the first half and their partners
      // (+ d/2) in the second half: 8-byte pieces, every lane of the row busy
      constexpr int kH = kEpp / 2;
      const int h0 = piece * kH;
      const uint2* s8 = reinterpret_cast<const uint2*>(src);
      uint2* d8 = reinterpret_cast<uint2*>(dst);
      const uint2 xu = s8[piece], yu = s8[piece + kPieces];
      float x[kH], y[kH];
      unpack8<T>(xu, x);
      unpack8<T>(yu, y);
      float2 cs[kH];
      rope_angles<kH>(a, h0, e, cs);
#pragma unroll
      for (int t = 0; t < kH; ++t) rope_back(x[t], y[t], cs[t]);
      d8[piece] = pack8<T>(x);
      d8[piece + kPieces] = pack8<T>(y);
    } else {
      float x[kEpp];
      unpack16<T>(src[piece], x);
      float2 cs[kEpp / 2];
      rope_angles<kEpp / 2>(a, piece * kEpp / 2, e, cs);
#pragma unroll
      for (int t = 0; t < kEpp; t += 2) rope_back(x[t], x[t + 1], cs[t / 2]);
      dst[piece] = pack16<T>(x);
    }
  } else {
    dst[piece] = src[piece];
  }
  if (piece == 0 && tensor == 1 && a.routing == SELKV_ROUTE_COSINE) {
    const float nv = a.vnorm[bk * a.n_cap + pos];
    a.cos_invn[bk * a.cos_mpad + slot] = nv > 0.f ? 1.f / nv : 0.f;
    a.cos_tslot[bk * a.n_cap + pos] = -1;  // a kept token routes nowhere
  }
  if (piece == 0 && tensor == 0) {
    a.ratio[bk * a.m_cap + slot] = 1.f;
    a.mcount[bk * a.m_cap + slot] = 0.f;
    if (a.dbg_ratio) a.dbg_ratio[bk * a.m_cap + slot] = 1.f;
    const size_t o = bk * a.n_cap + pos;
    if (a.dbg_target) a.dbg_target[o] = -1;
    if (a.dbg_gate) a.dbg_gate[o] = 0.f;
    if (a.dbg_decision) a.dbg_decision[o] = 2;
  }
}

// Sum kBatch per-lane partials p[k] over the 32 lanes with the batch spread over the lanes:
// each butterfly level keeps half of the values and adds the partner's copy of them, so lanes
// 2k and 2k + 1 end with the full sum of value k.  The pairs added at each level are those
// of a plain xor butterfly over all 32 lanes, so every sum is bitwise that of a per-value
// all-reduce.
__device__ __forceinline__ float transpose_reduce16(const float (&p)[kBatch], int lane) {
  float q[8];
  {
    const bool up = lane & 16;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float mine = up ? p[8 + i] : p[i], other = up ? p[i] : p[8 + i];
      q[i] = mine + __shfl_xor_sync(0xffffffffu, other, 16);
    }
  }
  float r[4];
  {
    const bool up = lane & 8;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float mine = up ? q[4 + i] : q[i], other = up ? q[i] : q[4 + i];
      r[i] = mine + __shfl_xor_sync(0xffffffffu, other, 8);
    }
  }
  float s[2];
  {
    const bool up = lane & 4;
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const float mine = up ? r[2 + i] : r[i], other = up ? r[i] : r[2 + i];
      s[i] = mine + __shfl_xor_sync(0xffffffffu, other, 4);
    }
  }
  const bool up = lane & 2;
  const float mine = up ? s[1] : s[0], other = up ? s[0] : s[1];
  const float t = mine + __shfl_xor_sync(0xffffffffu, other, 2);
  return t + __shfl_xor_sync(0xffffffffu, t, 1);
}

#ifndef SELKV_MERGE_COPY
#define SELKV_MERGE_COPY 1  // bucket routing without repositioning: the merge warps copy the kept rows
#endif
template <int BYTES>
struct RawOf;
template <>
struct RawOf<4> { using type = uint32_t; };
template <>
struct RawOf<8> { using type = uint2; };
template <>
struct RawOf<16> { using type = uint4; };

// Copy of bucket X's kept rows into their slots: every key row, and every value row but the
// merge target's (written merged by the caller); ratio 1 and count 0 for the slots other
// than the target's.  Loads of up to 8 kept positions are issued before their stores.  The
// same work as copy_kernel does for every slot, done by the warp that owns the bucket.
template <typename T, int D>
__device__ __forceinline__ void copy_kept_rows(const CompressArgs& a, size_t bk, int base, bool keptX, int slotX,
                                               int tau, int lane) {
  constexpr int PER = D / 32;
  using Raw = typename RawOf<PER * (int)sizeof(T)>::type;
  const T* Kb = static_cast<const T*>(a.K) + bk * a.n_cap * D;
  const T* Vb = static_cast<const T*>(a.V) + bk * a.n_cap * D;
  T* Kc = static_cast<T*>(a.Kc) + bk * a.m_cap * D;
  T* Vc = static_cast<T*>(a.Vc) + bk * a.m_cap * D;
  if (keptX) {
    if (slotX < 0 || slotX >= a.m_cap) {
      raise_flag(a.flags, SELKV_DEVERR_COUNT);
    } else if (base + lane != tau) {
      a.ratio[bk * a.m_cap + slotX] = 1.f;
      a.mcount[bk * a.m_cap + slotX] = 0.f;
      if (a.dbg_ratio) a.dbg_ratio[bk * a.m_cap + slotX] = 1.f;
    }
    const size_t o = bk * a.n_cap + base + lane;
    if (a.dbg_target) a.dbg_target[o] = -1;
    if (a.dbg_gate) a.dbg_gate[o] = 0.f;
    if (a.dbg_decision) a.dbg_decision[o] = 2;
  }
  uint32_t km = __ballot_sync(0xffffffffu, keptX && slotX >= 0 && slotX < a.m_cap);
  while (km) {
    constexpr int kN = 4;
    int pos[kN], slot[kN];
    Raw kr[kN], vr[kN];
#pragma unroll
    for (int i = 0; i < kN; ++i) {
      const int bit = km ? __ffs(km) - 1 : -1;
      km &= km ? km - 1u : 0u;
      pos[i] = bit < 0 ? -1 : base + bit;
      slot[i] = __shfl_sync(0xffffffffu, slotX, bit < 0 ? 0 : bit);
      if (pos[i] >= 0) {
        kr[i] = *reinterpret_cast<const Raw*>(Kb + (size_t)pos[i] * D + lane * PER);
        if (pos[i] != tau) vr[i] = *reinterpret_cast<const Raw*>(Vb + (size_t)pos[i] * D + lane * PER);
      }
    }
#pragma unroll
    for (int i = 0; i < kN; ++i) {
      if (pos[i] < 0) continue;
      *reinterpret_cast<Raw*>(Kc + (size_t)slot[i] * D + lane * PER) = kr[i];
      if (pos[i] != tau) *reinterpret_cast<Raw*>(Vc + (size_t)slot[i] * D + lane * PER) = vr[i];
    }
  }
}

template <typename T, int D>
#ifndef SELKV_MERGE_MINB
#define SELKV_MERGE_MINB 32  // one-warp merge CTAs resident per SM (32: the most an SM holds)
#endif
__global__ __launch_bounds__(32, SELKV_MERGE_MINB) void merge_kernel(CompressArgs a) {
  constexpr int PER = D / 32;  // elements of a row per lane
  const int lane = threadIdx.x;
  const int X = blockIdx.x;
  const int kv = blockIdx.y % a.Hkv, b = blockIdx.y / a.Hkv;
  const int n = a.seq_n[b], Bs = a.bucket;
  const int nb = (n + Bs - 1) / Bs;
  if (X >= nb) return;
  const size_t bk = (size_t)b * a.Hkv + kv;
  const int32_t* tau_of = a.tau + bk * a.nbk;
  const float* atau_of = a.atau + bk * a.nbk;
  const int base = X * Bs;
  const bool inX = lane < min(Bs, n - base);
  // One round of independent loads: tau_X and a(tau_X), the 32 buckets on either side (for
  // the nearest non-empty ones), and the kept flags of X.
  const int tau = tau_of[X];
  const float a_tau = atau_of[X];
  const bool expand = a.empty_bucket == SELKV_EMPTY_EXPAND;
  const int eL = X - 1 - lane, eR = X + 1 + lane;
  const int tl = (expand && eL >= 0) ? tau_of[eL] : -1;
  const int tr = (expand && eR < nb) ? tau_of[eR] : -1;
  const float al = (expand && eL >= 0) ? atau_of[eL] : 0.f;
  const float ar = (expand && eR < nb) ? atau_of[eR] : 0.f;
  const size_t su = sel_unit(a, b, kv);
  const bool keptX = inX && a.kflag[su * a.n_cap + base + lane] != 0;
  const float* A = a.attn + bk * a.n_cap;
  const float* vn = a.vnorm + bk * a.n_cap;
  const float AX = inX ? A[base + lane] : 0.f;
  const float NX = inX ? vn[base + lane] : 0.f;
  const bool fuse_copy = SELKV_MERGE_COPY && a.rope == SELKV_ROPE_OFF;
  const int slotX = (fuse_copy && inX) ? a.slot_of[su * a.n_cap + base + lane] : -1;
  if (tau < 0) {  // (then X keeps no token: nothing to copy)
    // Empty bucket: under EXPAND a neighbour's warp owns these tokens; under DROP (or with
    // nothing kept at all) they stay without target.
    if (a.empty_bucket == SELKV_EMPTY_DROP || a.seq_m[b] == 0) {
      if (inX) {
        const size_t o = bk * a.n_cap + base + lane;
        if (a.dbg_target) a.dbg_target[o] = -1;
        if (a.dbg_gate) a.dbg_gate[o] = 0.f;
        if (a.dbg_decision) a.dbg_decision[o] = 0;
      }
    }
    return;
  }
  const T* Vb = static_cast<const T*>(a.V) + bk * a.n_cap * D;
  const float vn_tau = __shfl_sync(0xffffffffu, NX, tau - base);
  RowSlice<T, PER> vt;
  vt.load(Vb + (size_t)tau * D + lane * PER);

  int lo_b = X, hi_b = X;  // buckets whose evicted tokens route to tau
  if (expand) {
    // nearest non-empty buckets L < X and R > X (a further probe only past 32 empty ones)
    int L = -1, R = -1;
    float aL = 0.f, aR = 0.f;
    uint32_t m = __ballot_sync(0xffffffffu, tl >= 0);
    if (m) {
      L = X - __ffs(m);
      aL = __shfl_sync(0xffffffffu, al, __ffs(m) - 1);
    } else {
      for (int e0 = X - 33; e0 >= 0 && L < 0; e0 -= 32) {
        const int e = e0 - lane;
        const uint32_t mm = __ballot_sync(0xffffffffu, e >= 0 && tau_of[e] >= 0);
        if (mm) L = e0 - (__ffs(mm) - 1);
      }
      if (L >= 0) aL = atau_of[L];
    }
    m = __ballot_sync(0xffffffffu, tr >= 0);
    if (m) {
      R = X + __ffs(m);
      aR = __shfl_sync(0xffffffffu, ar, __ffs(m) - 1);
    } else {
      for (int e0 = X + 33; e0 < nb && R < 0; e0 += 32) {
        const int e = e0 + lane;
        const uint32_t mm = __ballot_sync(0xffffffffu, e < nb && tau_of[e] >= 0);
        if (mm) R = e0 + (__ffs(mm) - 1);
      }
      if (R >= 0) aR = atau_of[R];
    }
    // An empty e between L and X goes to the nearer one; at equal distance both are in the
    // ring and X wins only with a strictly larger a (tau_L has the lower index).  Towards R,
    // X wins ties at equal distance (tau_X has the lower index).
    if (L < 0) {
      lo_b = 0;
    } else if (L < X - 1) {
      lo_b = (X + L) / 2 + 1;
      if (((X + L) & 1) == 0 && a_tau > aL) lo_b = (X + L) / 2;
    }
    if (R < 0) {
      hi_b = nb - 1;
    } else if (R > X + 1) {
      hi_b = (X + R - 1) / 2;
      if (((X + R) & 1) == 0 && a_tau >= aR) hi_b = (X + R) / 2;
    }
  }
  // Contributors: every position of buckets lo_b..hi_b except the kept tokens of X (the other
  // buckets of the range are empty), in ascending order, up to kBatch at a time per bucket.
  const uint32_t evX = __ballot_sync(0xffffffffu, inX && !keptX);
  float num[PER];
#pragma unroll
  for (int t = 0; t < PER; ++t) num[t] = 0.f;
  float den = 0.f;
  int merged = 0;             // contributors with g > 0 (the count bias)
  const int own = lane >> 1;  // contributor owned by this lane pair within a batch
  for (int e = lo_b; e <= hi_b; ++e) {
    const int eb = e * Bs;
    const int cnt_e = min(Bs, n - eb);
    uint32_t rem = e == X ? evX : (cnt_e >= 32 ? 0xffffffffu : ((1u << cnt_e) - 1u));
    // a and ||v|| of bucket e, one position per lane
    const float Ae = e == X ? AX : (lane < cnt_e ? A[eb + lane] : 0.f);
    const float Ne = e == X ? NX : (lane < cnt_e ? vn[eb + lane] : 0.f);
    while (rem) {
      // the (up to) kBatch lowest contributors left in this bucket
      const int cut = __fns(rem, 0, kBatch + 1);  // position of the (kBatch+1)-th set bit
      const uint32_t bm = (cut < 0 || cut > 31) ? rem : (rem & ((1u << cut) - 1u));
      rem &= ~bm;
      const int cnt = __popc(bm);
      RowSlice<T, PER> vj[kBatch];
      {
        uint32_t r = bm;
#pragma unroll
        for (int k = 0; k < kBatch; ++k) {
          if (r) {
            vj[k].load(Vb + (size_t)(eb + __ffs(r) - 1) * D + lane * PER);
            r &= r - 1u;
          } else {
            vj[k].zero();
          }
        }
      }
      const int ob = own < cnt ? (int)__fns(bm, 0, own + 1) : -1;  // bit of the owned contributor
      const float ak = __shfl_sync(0xffffffffu, Ae, ob < 0 ? 0 : ob);
      const float nk = __shfl_sync(0xffffffffu, Ne, ob < 0 ? 0 : ob);
      float g;
      if (a.gate_mode == SELKV_GATE_OPEN) {
        g = 1.f;
      } else if (a.gate_mode == SELKV_GATE_CLOSED) {
        g = 0.f;
      } else {
        float part[kBatch];
#pragma unroll
        for (int k = 0; k < kBatch; ++k) {
          part[k] = 0.f;
#pragma unroll
          for (int t = 0; t < PER; ++t) part[k] = fmaf(vj[k][t], vt[t], part[k]);
        }
        const float dot = transpose_reduce16(part, lane);
        const float sim = (nk == 0.f || vn_tau == 0.f) ? 0.f : dot / (nk * vn_tau);
        g = fminf(fmaxf(sim, 0.f), 1.f);
      }
      const float w = ob >= 0 ? g * ak : 0.f;
      merged += __popc(__ballot_sync(0xffffffffu, ob >= 0 && g > 0.f) & 0x55555555u);
      if (ob >= 0 && (lane & 1) == 0) {
        const size_t o = bk * a.n_cap + eb + ob;
        if (a.dbg_target) a.dbg_target[o] = tau;
        if (a.dbg_gate) a.dbg_gate[o] = g;
        if (a.dbg_decision) a.dbg_decision[o] = g > 0.f ? 1 : 0;
      }
#pragma unroll
      for (int k = 0; k < kBatch; ++k) {
        if (k >= cnt) break;
        const float wk = __shfl_sync(0xffffffffu, w, 2 * k);
#pragma unroll
        for (int t = 0; t < PER; ++t) num[t] = fmaf(wk, vj[k][t], num[t]);
        den += wk;
      }
    }
  }
  const float tot = a_tau + den;
  float vm[PER];
#pragma unroll
  for (int t = 0; t < PER; ++t) vm[t] = tot > 0.f ? (a_tau * vt[t] + num[t]) / tot : vt[t];
  const float R_tau = a_tau > 0.f ? tot / a_tau : 1.f;
  const int slot = a.slot_of[su * a.n_cap + tau];
  if (slot < 0 || slot >= a.m_cap) {
    if (lane == 0) raise_flag(a.flags, SELKV_DEVERR_COUNT);
    return;
  }
  T* Vc = static_cast<T*>(a.Vc) + (bk * a.m_cap + slot) * D + lane * PER;
  if constexpr (PER == 4) {
    store4(Vc, vm);
  } else {
    store1(Vc, vm[0]);
    store1(Vc + 1, vm[1]);
  }
  if (lane == 0) {
    a.ratio[bk * a.m_cap + slot] = R_tau;
    a.mcount[bk * a.m_cap + slot] = (float)merged;
    if (a.dbg_ratio) a.dbg_ratio[bk * a.m_cap + slot] = R_tau;
  }
  if (fuse_copy) copy_kept_rows<T, D>(a, bk, base, keptX, slotX, tau, lane);
}

// bias[b][kv][slot] = alpha * ln(mean over KV heads of R[b][kv][slot])   (Sec. 3.6, GQA);
// per-head mode: alpha * ln R[b][kv][slot] of each head, no averaging (Sec. 3.6, MHA).  The
// count variant uses ln(1 + M) of the merge counts M instead of ln R.
__global__ __launch_bounds__(256) void bias_kernel(CompressArgs a) {
  const int b = blockIdx.y;
  const int slot = blockIdx.x * blockDim.x + threadIdx.x;
  if (slot >= a.seq_m[b]) return;
  const float* src = a.bias_count ? a.mcount : a.ratio;
  if (a.per_head) {
    for (int kv = 0; kv < a.Hkv; ++kv) {
      const size_t o = ((size_t)b * a.Hkv + kv) * a.m_cap + slot;
      a.bias[o] = a.alpha * (a.bias_count ? log1pf(src[o]) : logf(src[o]));
    }
    return;
  }
  float s = 0.f;
  for (int kv = 0; kv < a.Hkv; ++kv) s += src[((size_t)b * a.Hkv + kv) * a.m_cap + slot];
  const float mean = s / (float)a.Hkv;
  const float bias = a.alpha * (a.bias_count ? log1pf(mean) : logf(mean));
  for (int kv = 0; kv < a.Hkv; ++kv) a.bias[((size_t)b * a.Hkv + kv) * a.m_cap + slot] = bias;
}

template <typename T, int D>
void launch_merge_t(const CompressArgs& a, cudaStream_t s) {
  constexpr int kPieces = D * (int)sizeof(T) / 16;
  const size_t copy_threads = (size_t)a.Hkv * a.m_cap * 2 * kPieces;
  // with the bucket routing and no repositioning the merge warps copy the kept rows themselves
  if (!merge_copies_kept_rows(a))
    copy_kernel<T, D><<<dim3((unsigned)((copy_threads + 255) / 256), a.B), 256, 0, s>>>(a);
  if (a.routing == SELKV_ROUTE_BUCKET) merge_kernel<T, D><<<dim3(a.nbk, a.B * a.Hkv), 32, 0, s>>>(a);
}

}  // namespace

bool merge_copies_kept_rows(const CompressArgs& a) {
  return SELKV_MERGE_COPY && a.routing == SELKV_ROUTE_BUCKET && a.rope == SELKV_ROPE_OFF;
}

cudaError_t launch_merge(const CompressArgs& a, cudaStream_t s) {
  if (a.rope != SELKV_ROPE_OFF) {
    const int groups = (a.rope_hi + 256 + kRopeRowsPerThread - 1) / kRopeRowsPerThread;
    const int threads = a.D / 2 * groups;
    rope_table_kernel<<<(threads + 127) / 128, 128, 0, s>>>(a);
  }
  if (a.routing == SELKV_ROUTE_BUCKET)
    route_kernel<<<dim3((a.nbk + kWarpsPerCta - 1) / kWarpsPerCta, a.B), kWarpsPerCta * 32, 0, s>>>(a);
  if (a.dtype == SELKV_BF16) {
    if (a.D == 128) launch_merge_t<__nv_bfloat16, 128>(a, s);
    else launch_merge_t<__nv_bfloat16, 64>(a, s);
  } else {
    if (a.D == 128) launch_merge_t<float, 128>(a, s);
    else launch_merge_t<float, 64>(a, s);
  }
  if (a.routing == SELKV_ROUTE_COSINE) {
    const cudaError_t e = launch_route_cosine(a, s);
    if (e != cudaSuccess) return e;
  }
  bias_kernel<<<dim3((a.m_cap + 255) / 256, a.B), 256, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace selkv
