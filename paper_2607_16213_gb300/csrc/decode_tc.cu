// Compensated decode attention for bf16 caches: TMA-fed, tensor-core split-K flash decoding.
//
//   out[b][h] = sum_i softmax_i(q_h . k_i / sqrt(d) + bias_i) v_i     (Alg. 1 decode, Sec. 3.6)
//
// CTA (split s, KV head kv, sequence b) owns a contiguous slice of the compressed rows, cut
// at multiples of 64 rows.  A producer warp streams 128-row K and V tiles into a STAGES-deep
// ring of shared-memory buffers with 2D TMA loads (64-row boxes, 128-byte swizzle, completion
// on an mbarrier per stage; a slice's last tile may be a single box high).  Eight consumer
// warps each take 16 rows of a tile: S = Q K^T for all G query heads of the group at once
// (mma.sync m16n8k16, bf16 in, fp32 accumulate; the G heads are the M rows, so one K tile
// serves the whole group), the scale and the fp32 bias are applied to S before the running
// max, then O += P V on the tensor cores.  The rows of one warp stream form one flash-decoding
// state; the warp states and then the splits are folded in a fixed order, the splits by the
// last CTA of (b, kv) to arrive (one atomic add, no waiting), which brings every split's
// partial into the idle ring with one bulk copy.  The appended row
// (k_new, v_new) joins the last split with bias 0 and is then written at row lengths[b].
//
// Every mbarrier wait is bounded: on timeout the CTA raises SELKV_DEVERR_TIMEOUT, stops, and
// waits (bounded again) for the copies it has issued before leaving.  Launched with
// programmatic dependent launch: while the previous kernel of the stream finishes, the CTA
// sets up its barriers and loads the first tiles of its slice, planned from a length read
// without ordering, into the ring (only rows that no kernel still running can be writing:
// below that length minus one).  After griddepcontrol.wait the slice is planned again from
// the length read in order, and an early tile is kept only where the two plans agree; the
// query, the bias and the lengths used for the result are all read after the wait.
#include <algorithm>

#include "decode_common.cuh"
#include "ptx.cuh"
#include "selkv_internal.cuh"

namespace selkv {
namespace {

#ifndef SELKV_DEC_TILE
#define SELKV_DEC_TILE 128     // rows per tile (multiple of 16, at most 256)
#endif
#ifndef SELKV_DEC_STAGES
#define SELKV_DEC_STAGES 2     // tiles in flight per CTA
#endif
#ifndef SELKV_DEC_PDL
#define SELKV_DEC_PDL 1        // launch with programmatic dependent launch
#endif
#ifndef SELKV_DEC_PF_ROWS
#define SELKV_DEC_PF_ROWS 128  // rows prefetched into L2 before griddepcontrol.wait when no tile is preloaded
#endif
#ifndef SELKV_DEC_PRELOAD
#define SELKV_DEC_PRELOAD 2    // tiles of the slice loaded into the ring before griddepcontrol.wait
#endif
#ifndef SELKV_DEC_PRELOAD_WAVE
#define SELKV_DEC_PRELOAD_WAVE 1  // only CTAs of the grid's first wave load early
#endif
#ifndef SELKV_DEC_PRELOAD_MIN
#define SELKV_DEC_PRELOAD_MIN 8  // ... on slices of at least this many tiles
#endif
#ifndef SELKV_DEC_PF_QB
#define SELKV_DEC_PF_QB 2  // tiles of bias rows (and the group's queries) prefetched into L2 before the wait
#endif
#ifndef SELKV_DEC_UNITS
#define SELKV_DEC_UNITS 1  // persistent unit-walking CTAs when every (b, kv) has one split and they outnumber the SMs
#endif
#ifndef SELKV_DEC_MINBLOCKS
#define SELKV_DEC_MINBLOCKS 1  // CTAs resident per SM (register / shared-memory budget)
#endif

constexpr int kTile = SELKV_DEC_TILE;
constexpr int kConsumers = kTile / 16;  // consumer warps, 16 rows of a tile each
constexpr int kThreads = (kConsumers + 1) * 32;
constexpr int kStages = SELKV_DEC_STAGES;
constexpr int kBoxRows = 64;   // TMA box height; split boundaries fall on multiples of it
constexpr int kHalves = kTile / kBoxRows;
static_assert(kTile % kBoxRows == 0, "tile is whole boxes");

template <int D>
struct Cfg {
  static constexpr int kBoxes = D / 64;                // 128-byte-wide boxes per row
  static constexpr int kBoxBytes = kTile * 128;        // one 128-byte column of a tile
  static constexpr int kPieceBytes = kBoxRows * 128;   // one TMA box: kBoxRows rows x 128 bytes
  static constexpr int kTileBytes = kTile * D * 2;     // K (or V) tile
  static constexpr int kStageBytes = 2 * kTileBytes;
  static constexpr int kRingBytes = kStages * kStageBytes;
  // after the ring: full[kStages], empty[kStages], pre[kStages], comb, abort flag (8 bytes),
  // warp states
  static constexpr int kSmemBytes = kRingBytes + 1024 /*align*/ + (3 * kStages + 2) * 8 + 2 * kConsumers * 16 * 4;
  static constexpr int kFoldLd = D + 8;                // fold row stride (floats): conflict-free float2 stores
  static_assert(kConsumers * 16 * kFoldLd * 4 <= kRingBytes, "fold scratch fits");
};

// Combine of (b, kv) by its last CTA when S <= 32, with no shared memory and no barrier.
// Two lanes own each output float4 (lanes l and l ^ 16: the first and the second half of the
// splits); every partial they need is loaded into registers at once, next to the (max, sum)
// of split `lane` of the item's head, so the whole combine costs one L2 round trip.  The
// weights 2^(max_t - max) and the normaliser come from warp reductions and shuffles; each
// lane sums its splits in split order and the two halves are added.  The producer warp's
// lane 0 does the length bookkeeping.
constexpr int kRegSplits = 32;
template <int D>
__device__ __forceinline__ void combine_registers(const DecodeArgs& a, int b, int kv, size_t bk, int L, bool app) {
  constexpr int D4 = D / 4;
  constexpr int kHalf = kRegSplits / 2;
  static_assert(D4 % 16 == 0, "a warp's 16 items share one head");
  const int G = a.G, S = a.splits;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, nwarps = blockDim.x >> 5;
  const int owner = blockDim.x - 32;
  const PartialView pv = partial_view(a);
  const uint32_t seq_old = finish_lengths_begin(a, b, bk, app, owner);
  const int Sh = (S + 1) / 2;
  const int half = lane >> 4;
  const int t0 = half * Sh, cnt = min(S, t0 + Sh) - t0;
  const int items = G * D4, per_pass = nwarps * 16;
  for (int base = 0; base < items; base += per_pass) {
    const int wbase = base + warp * 16;  // first item of this warp (uniform)
    if (wbase >= items) break;
    const int g = wbase / D4, d4 = wbase % D4 + (lane & 15);
    const float4* op = reinterpret_cast<const float4*>(pv.o(bk, g, 0)) + d4;
    float4 v[kHalf];
#pragma unroll
    for (int j = 0; j < kHalf; ++j)
      v[j] = j < cnt ? __ldcg(op + (size_t)(t0 + j) * D4) : make_float4(0.f, 0.f, 0.f, 0.f);
    const float2 ml = lane < S ? __ldcg(pv.ml(bk, g, lane)) : make_float2(-INFINITY, 0.f);
    const float M = warp_max(ml.x);
    const float w = (lane < S && M != -INFINITY) ? exp2f(ml.x - M) : 0.f;
    const float Ls = warp_sum(ml.y * w);
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int j = 0; j < kHalf; ++j) {
      const float wj = __shfl_sync(0xffffffffu, w, (t0 + j) & 31);
      if (j < cnt) {
        acc.x = fmaf(v[j].x, wj, acc.x);
        acc.y = fmaf(v[j].y, wj, acc.y);
        acc.z = fmaf(v[j].z, wj, acc.z);
        acc.w = fmaf(v[j].w, wj, acc.w);
      }
    }
    const float ox = __shfl_xor_sync(0xffffffffu, acc.x, 16);
    const float oy = __shfl_xor_sync(0xffffffffu, acc.y, 16);
    const float oz = __shfl_xor_sync(0xffffffffu, acc.z, 16);
    const float ow = __shfl_xor_sync(0xffffffffu, acc.w, 16);
    if (half == 0) {
      const float iv = Ls > 0.f ? 1.f / Ls : 0.f;
      const float r[4] = {(acc.x + ox) * iv, (acc.y + oy) * iv, (acc.z + oz) * iv, (acc.w + ow) * iv};
      store4(static_cast<__nv_bfloat16*>(a.out) + (bk * G + g) * D + d4 * 4, r);
    }
  }
  finish_lengths_end(a, b, L, app, seq_old, owner);
}

// Combine of (b, kv) by its last CTA: one bulk copy brings the whole partial record (every
// split's output and (max, sum)) into the idle ring; a warp per head turns the maxima into
// weights 2^(max_t - max) and the normaliser; each output float4 is then summed over the
// splits by two lanes (first and second half of the splits, in split order) and the halves
// added.  The producer warp's lane 0, which issues no loads here, does the length
// bookkeeping.  A record too large for the ring falls back to combine_splits.
template <int D>
__device__ __forceinline__ void combine_record(const DecodeArgs& a, int b, int kv, size_t bk, unsigned char* smem,
                                               int smem_bytes, uint64_t* bar, int L, bool app) {
  constexpr int D4 = D / 4;
  const int G = a.G, S = a.splits;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, nwarps = blockDim.x >> 5;
  const int owner = blockDim.x - 32;
  const PartialView pv = partial_view(a);
  const uint32_t rec_bytes = (uint32_t)(pv.rec * 4);
  if ((size_t)rec_bytes + (size_t)G * (S + 1) * 4 > (size_t)smem_bytes) {
    const uint32_t old = finish_lengths_begin(a, b, bk, app, owner);
    combine_splits<__nv_bfloat16>(a, b, kv, nullptr);
    finish_lengths_end(a, b, L, app, old, owner);
    return;
  }
  // the ring was last touched through the generic proxy; the bulk copy writes it through the
  // async proxy, and reads the other splits' generic-proxy stores acquired by arrive_last
  fence_proxy_async_all();
  __syncthreads();
  if (tid == 0) {
    mbar_arrive_expect_tx(bar, rec_bytes);
    bulk_load(smem, pv.record(bk), rec_bytes, bar);
  }
  const uint32_t seq_old = finish_lengths_begin(a, b, bk, app, owner);
  const float* os = reinterpret_cast<const float*>(smem);                              // [G][S][D]
  const float2* mls = reinterpret_cast<const float2*>(smem + (size_t)G * S * D * 4);   // [G][S]
  float* wts = reinterpret_cast<float*>(smem + rec_bytes);                              // [G][S]
  float* inv = wts + G * S;                                                             // [G]
  if (!mbar_wait(bar, 0)) {
    if (tid == 0) raise_flag(a.flags, SELKV_DEVERR_TIMEOUT);
    mbar_wait(bar, 0);  // the copy must land before the CTA leaves
    finish_lengths_end(a, b, L, app, seq_old, owner);  // the sequence counter must not stay raised
    return;
  }
  for (int g = warp; g < G; g += nwarps) {
    float M = -INFINITY;
    for (int t = lane; t < S; t += 32) M = fmaxf(M, mls[g * S + t].x);
    M = warp_max(M);
    float Ls = 0.f;
    for (int t = lane; t < S; t += 32) {
      const float2 ml = mls[g * S + t];
      const float w = M == -INFINITY ? 0.f : exp2f(ml.x - M);
      wts[g * S + t] = w;
      Ls = fmaf(ml.y, w, Ls);
    }
    Ls = warp_sum(Ls);
    if (lane == 0) inv[g] = Ls > 0.f ? 1.f / Ls : 0.f;
  }
  __syncthreads();
  const int Sh = (S + 1) / 2;
  const int items = G * D4, per_pass = nwarps * 16;
  for (int base = 0; base < items; base += per_pass) {
    const int item = base + warp * 16 + (lane & 15);
    const int half = lane >> 4;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    const int g = item / D4, d4 = item % D4;
    if (item < items) {
      const int t0 = half * Sh, t1 = min(S, t0 + Sh);
      const float4* op = reinterpret_cast<const float4*>(os + (size_t)g * S * D) + d4;
      const float* wp = wts + g * S;
      for (int t = t0; t < t1; t += 8) {
        float4 v[8];
        float w[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const bool ok = t + j < t1;
          v[j] = ok ? op[(t + j) * D4] : make_float4(0.f, 0.f, 0.f, 0.f);
          w[j] = ok ? wp[t + j] : 0.f;
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          acc.x = fmaf(v[j].x, w[j], acc.x);
          acc.y = fmaf(v[j].y, w[j], acc.y);
          acc.z = fmaf(v[j].z, w[j], acc.z);
          acc.w = fmaf(v[j].w, w[j], acc.w);
        }
      }
    }
    const float ox = __shfl_xor_sync(0xffffffffu, acc.x, 16);
    const float oy = __shfl_xor_sync(0xffffffffu, acc.y, 16);
    const float oz = __shfl_xor_sync(0xffffffffu, acc.z, 16);
    const float ow = __shfl_xor_sync(0xffffffffu, acc.w, 16);
    if (item < items && half == 0) {
      const float iv = inv[g];
      const float r[4] = {(acc.x + ox) * iv, (acc.y + oy) * iv, (acc.z + oz) * iv, (acc.w + ow) * iv};
      store4(static_cast<__nv_bfloat16*>(a.out) + (bk * G + g) * D + d4 * 4, r);
    }
  }
  finish_lengths_end(a, b, L, app, seq_old, owner);
}

template <int D, bool ROWS16>
__global__ __launch_bounds__(kThreads, SELKV_DEC_MINBLOCKS) void decode_tc_kernel(const __grid_constant__ CUtensorMap tmK,
                                                                 const __grid_constant__ CUtensorMap tmV,
                                                                 DecodeArgs a) {
  using C = Cfg<D>;
  constexpr int NT = D / 8;   // n-tiles of the output (8 columns each)
  constexpr int KS = D / 16;  // k-steps of Q K^T
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::kRingBytes);
  uint64_t* empty = full + kStages;
  uint64_t* pre = empty + kStages;   // completion of the tiles loaded before griddepcontrol.wait
  uint64_t* comb = pre + kStages;    // completion of the combine's bulk copy
  volatile int* s_abort = reinterpret_cast<volatile int*>(comb + 1);
  float* wm = reinterpret_cast<float*>(comb + 2);  // [kConsumers][16] warp maxima (base 2)
  float* wl = wm + kConsumers * 16;                // [kConsumers][16] warp sums
  __shared__ bool s_last;
  __shared__ float s_inv[16];  // one split: 1 / sum per query head of the group
  __shared__ int s_pre_lo, s_pre_n;  // slice start and tile count of the early loads

  const int s = blockIdx.x, kv = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = a.G, S = a.splits;
  const size_t bk = (size_t)b * a.Hkv + kv;

  if (warp == kConsumers && lane == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], kConsumers);
      mbar_init(&pre[i], 1);
    }
    mbar_init(comb, 1);
    *s_abort = 0;
    fence_mbar_init();
    prefetch_tensormap(&tmK);
    prefetch_tensormap(&tmV);
    // Before griddepcontrol.wait, while the previous kernel of the stream finishes (its split
    // combines leave HBM idle), this CTA starts on its slice as planned from a length read
    // without ordering, which may be stale.  Rows below that length minus one are rows no
    // kernel that may still be running writes: the previous kernel is at most appending the
    // row at the length it read (a decode of this cache), and anything before it has
    // completed (the contract in selkv.h).  Whole tiles below that bound are loaded into the
    // ring; after the wait they are used only if the slice, planned again from the true
    // length, starts at the same row and covers them.  Only CTAs of the grid's first wave
    // (later waves start while HBM is busy anyway) with slices of at least
    // SELKV_DEC_PRELOAD_MIN tiles load early: on short slices the early loads are a large
    // share of the work and they compete with the previous kernel's last CTAs; such slices
    // prefetch their first rows into L2 instead.
    const int Lg = min(max(ld_relaxed_gpu(a.lengths + b), 0), a.m_cap);
    const int chk = ((Lg + S - 1) / S + kBoxRows - 1) / kBoxRows * kBoxRows;
    const int plo = min(Lg, s * chk), phi = min(Lg, plo + chk);
    int npre = 0;
#if SELKV_DEC_PRELOAD
    const int safe = min(phi, Lg - 1);
    const bool first_wave = SELKV_DEC_PRELOAD_WAVE == 0 ||
                            (int)(blockIdx.x + gridDim.x * (blockIdx.y + gridDim.y * blockIdx.z)) < kPlanSMs;
    const int max_pre = (first_wave && phi - plo >= SELKV_DEC_PRELOAD_MIN * kTile) ? min(kStages, SELKV_DEC_PRELOAD) : 0;
    for (; npre < max_pre && plo + (npre + 1) * kTile <= safe; ++npre) {
      unsigned char* base = smem + npre * C::kStageBytes;
      mbar_arrive_expect_tx(&pre[npre], C::kStageBytes);
      for (int h = 0; h < kHalves; ++h) {
        const int y = (int)(bk * a.m_cap) + plo + npre * kTile + h * kBoxRows;
#pragma unroll
        for (int bx = 0; bx < C::kBoxes; ++bx)
          tma_load_2d(base + bx * C::kBoxBytes + h * C::kPieceBytes, &tmK, bx * 64, y, &pre[npre]);
#pragma unroll
        for (int bx = 0; bx < C::kBoxes; ++bx)
          tma_load_2d(base + C::kTileBytes + bx * C::kBoxBytes + h * C::kPieceBytes, &tmV, bx * 64, y, &pre[npre]);
      }
    }
#endif
    s_pre_lo = plo;
    s_pre_n = npre;
#if SELKV_DEC_PF_ROWS > 0
    // no tile loaded early: the slice's first rows go to L2 (a prefetch; nothing computed
    // depends on it, so it may cover any row of the early plan)
    const int prow = npre > 0 ? 0 : min(phi - plo, SELKV_DEC_PF_ROWS);
    const char* kp = static_cast<const char*>(a.Kc) + (bk * a.m_cap + plo) * (size_t)(D * 2);
    const char* vp = static_cast<const char*>(a.Vc) + (bk * a.m_cap + plo) * (size_t)(D * 2);
    for (int r = 0; r < prow; r += kBoxRows) {
      const uint32_t bytes = (uint32_t)(min(kBoxRows, prow - r) * D * 2);
      bulk_prefetch_l2(kp + (size_t)r * D * 2, bytes);
      bulk_prefetch_l2(vp + (size_t)r * D * 2, bytes);
    }
#endif
#if SELKV_DEC_PF_QB > 0
    // The group's queries and the bias of the slice's first rows go to L2 as well: the first
    // tiles are then waiting on nothing but L2 hits after the wait.  The previous kernel may
    // still write these (q, the bias): a prefetch only moves lines into L2, where its writes
    // land, and the values used are loaded after the wait.
    {
      const char* qp = static_cast<const char*>(a.q) + ((size_t)b * a.Hq + (size_t)kv * G) * D * 2;
      for (int off = 0; off < G * D * 2; off += 128) prefetch_l2(qp + off);
      if (a.bias != nullptr) {
        const char* bp = reinterpret_cast<const char*>(a.bias + bk * a.m_cap + plo);
        const int nb = min(phi - plo, SELKV_DEC_PF_QB * kTile) * 4;  // bytes, inside row bk's bias
        if (nb > 0) {
          for (int off = 0; off < nb; off += 128) prefetch_l2(bp + off);
          prefetch_l2(bp + nb - 1);
        }
      }
    }
#endif
  }
  // Everything above touches only this CTA's shared memory; everything below may read what
  // the previous kernel in the stream wrote (lengths, the cache, the workspace).
  pdl_wait();
  pdl_launch_dependents();
  int L = a.lengths[b];  // in flight across the barrier below
  __syncthreads();
  if (L < 0 || L > a.m_cap) {
    if (tid == 0 && s == 0 && kv == 0) raise_flag(a.flags, SELKV_DEVERR_LENGTH);
    L = L < 0 ? 0 : a.m_cap;
  }
  bool app = a.k_new != nullptr;
  if (app && L + 1 > a.m_cap) {
    if (tid == 0 && s == 0 && kv == 0) raise_flag(a.flags, SELKV_DEVERR_CAPACITY);
    app = false;
  }
  const int chunk = ((L + S - 1) / S + kBoxRows - 1) / kBoxRows * kBoxRows;
  const int lo = min(L, s * chunk), hi = min(L, lo + chunk);
  const int ntiles = (hi - lo + kTile - 1) / kTile;
  const int row0 = (int)(bk * a.m_cap) + lo;

  float o[NT][4];
  float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};
#pragma unroll
  for (int nt = 0; nt < NT; ++nt)
#pragma unroll
    for (int e = 0; e < 4; ++e) o[nt][e] = 0.f;
  const int g0 = lane >> 2, c2 = (lane & 3) * 2;

  if (warp == kConsumers) {
    // ---------------- producer ----------------
    if (lane == 0) {
      int issued = 0;
      const int npre = s_pre_n;
      uint32_t pre_seen = 0u;  // early loads known to have landed
      for (int t = 0; t < ntiles; ++t) {
        const int st = t % kStages;
        if (!mbar_wait(&empty[st], ((t / kStages) & 1) ^ 1)) {
          *s_abort = 1;
          raise_flag(a.flags, SELKV_DEVERR_TIMEOUT);
          break;
        }
        if (*s_abort) break;
        if (t < npre) {
          // the early load into this stage lands before the stage is released or reloaded
          if (!mbar_wait(&pre[st], 0)) {
            *s_abort = 1;
            raise_flag(a.flags, SELKV_DEVERR_TIMEOUT);
            break;
          }
          pre_seen |= 1u << st;
          if (lo == s_pre_lo && lo + (t + 1) * kTile <= hi) {
            mbar_arrive(&full[st]);  // the tile is already in place
            issued = t + 1;
            continue;
          }
        }
        unsigned char* base = smem + st * C::kStageBytes;
        // a split's last tile may be cut at a box boundary: load only the boxes it covers
        const int nh = min(kHalves, (hi - lo - t * kTile + kBoxRows - 1) / kBoxRows);
        mbar_arrive_expect_tx(&full[st], 2 * nh * C::kBoxes * C::kPieceBytes);
        for (int h = 0; h < nh; ++h) {
          const int y = row0 + t * kTile + h * kBoxRows;
#pragma unroll
          for (int bx = 0; bx < C::kBoxes; ++bx)
            tma_load_2d(base + bx * C::kBoxBytes + h * C::kPieceBytes, &tmK, bx * 64, y, &full[st]);
#pragma unroll
          for (int bx = 0; bx < C::kBoxes; ++bx)
            tma_load_2d(base + C::kTileBytes + bx * C::kBoxBytes + h * C::kPieceBytes, &tmV, bx * 64, y, &full[st]);
        }
        issued = t + 1;
      }
      // every issued copy must have landed before the ring is reused or the CTA exits
      for (int t = max(0, issued - kStages); t < issued; ++t) mbar_wait(&full[t % kStages], (t / kStages) & 1);
      for (int st = 0; st < npre; ++st)
        if (!(pre_seen & (1u << st))) mbar_wait(&pre[st], 0);
    }
  } else {
    // ---------------- consumers ----------------
    const __nv_bfloat16* qg = static_cast<const __nv_bfloat16*>(a.q) + ((size_t)b * a.Hq + (size_t)kv * G) * D;
    uint32_t qa[KS][4];
#pragma unroll
    for (int ks = 0; ks < KS; ++ks) {
      const int d0 = ks * 16 + c2;
      qa[ks][0] = g0 < G ? *reinterpret_cast<const uint32_t*>(qg + (size_t)g0 * D + d0) : 0u;
      qa[ks][2] = g0 < G ? *reinterpret_cast<const uint32_t*>(qg + (size_t)g0 * D + d0 + 8) : 0u;
      qa[ks][1] = (ROWS16 && g0 + 8 < G) ? *reinterpret_cast<const uint32_t*>(qg + (size_t)(g0 + 8) * D + d0) : 0u;
      qa[ks][3] = (ROWS16 && g0 + 8 < G) ? *reinterpret_cast<const uint32_t*>(qg + (size_t)(g0 + 8) * D + d0 + 8) : 0u;
    }
    const float* brow = a.bias != nullptr ? a.bias + bk * a.m_cap : nullptr;
    const float sc = a.scale_log2;
    // bias of this lane's four keys, fetched one tile ahead so its latency hides behind a tile
    auto fetch_bias = [&](int t, float (&dst)[2][2]) {
#pragma unroll
      for (int nt = 0; nt < 2; ++nt)
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int key = lo + t * kTile + warp * 16 + nt * 8 + c2 + e;
          dst[nt][e] = (brow != nullptr && key < hi) ? __ldg(brow + key) * kLog2e : 0.f;
        }
    };
    float bnext[2][2];
    fetch_bias(0, bnext);
    for (int t = 0; t < ntiles; ++t) {
      float bv[2][2];
#pragma unroll
      for (int nt = 0; nt < 2; ++nt)
#pragma unroll
        for (int e = 0; e < 2; ++e) bv[nt][e] = bnext[nt][e];
      if (t + 1 < ntiles) fetch_bias(t + 1, bnext);
      const int st = t % kStages;
      if (!mbar_wait(&full[st], (t / kStages) & 1)) {
        *s_abort = 1;
        if (lane == 0) raise_flag(a.flags, SELKV_DEVERR_TIMEOUT);
        break;
      }
      const int key0 = lo + t * kTile + warp * 16;
      const int nvalid = hi - key0;
      if (nvalid > 0) {
        const uint32_t Kt = smem_u32(smem + st * C::kStageBytes);
        const uint32_t Vt = Kt + C::kTileBytes;
        // S = Q K^T over this warp's 16 rows (two 8-row n-tiles)
        float sacc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
        const int mi = lane >> 3, ri = lane & 7;
#pragma unroll
        for (int ks = 0; ks < KS; ++ks) {
          const int krow = (mi >> 1) * 8 + ri;      // row within the warp's 16
          const int chunk16 = ks * 2 + (mi & 1);    // 16-byte chunk along d
          uint32_t kb[4];
          ldmatrix_x4(kb, Kt + (chunk16 >> 3) * C::kBoxBytes + swz128(warp * 16 + krow, chunk16 & 7));
          mma_bf16_16816(sacc[0], qa[ks], kb[0], kb[1]);
          mma_bf16_16816(sacc[1], qa[ks], kb[2], kb[3]);
        }
        // logits (base 2), masked past `hi`
        float tmax[2] = {-INFINITY, -INFINITY};
#pragma unroll
        for (int nt = 0; nt < 2; ++nt)
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const bool ok = key0 + nt * 8 + c2 + e < hi;
#pragma unroll
            for (int r = 0; r < 2; ++r) {
              const float v = ok ? fmaf(sacc[nt][r * 2 + e], sc, bv[nt][e]) : -INFINITY;
              sacc[nt][r * 2 + e] = v;
              tmax[r] = fmaxf(tmax[r], v);
            }
          }
        float corr[2], mref[2];
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          tmax[r] = fmaxf(tmax[r], __shfl_xor_sync(0xffffffffu, tmax[r], 1));
          tmax[r] = fmaxf(tmax[r], __shfl_xor_sync(0xffffffffu, tmax[r], 2));
          const float mn = fmaxf(mrow[r], tmax[r]);
          mref[r] = mn == -INFINITY ? 0.f : mn;
          corr[r] = exp2f(mrow[r] - mref[r]);
          mrow[r] = mn;
        }
        float p[2][4];
        float psum[2] = {0.f, 0.f};
#pragma unroll
        for (int nt = 0; nt < 2; ++nt)
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            p[nt][i] = exp2f(sacc[nt][i] - mref[i >> 1]);
            psum[i >> 1] += p[nt][i];
          }
#pragma unroll
        for (int r = 0; r < 2; ++r) lrow[r] = lrow[r] * corr[r] + psum[r];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          o[nt][0] *= corr[0];
          o[nt][1] *= corr[0];
          o[nt][2] *= corr[1];
          o[nt][3] *= corr[1];
        }
        uint32_t pa[4];
        pa[0] = pack_bf16(p[0][0], p[0][1]);
        pa[1] = pack_bf16(p[0][2], p[0][3]);
        pa[2] = pack_bf16(p[1][0], p[1][1]);
        pa[3] = pack_bf16(p[1][2], p[1][3]);
        // rows past `hi` may hold anything (even NaN): zero them before P V
        const bool zeroed = nvalid < 16;
        if (zeroed) {
          unsigned char* vt = smem + st * C::kStageBytes + C::kTileBytes;
          for (int i = lane; i < (16 - nvalid) * C::kBoxes * 8; i += 32) {
            const int r = warp * 16 + nvalid + i / (C::kBoxes * 8);
            const int rem = i % (C::kBoxes * 8);
            *reinterpret_cast<uint4*>(vt + (rem >> 3) * C::kBoxBytes + r * 128 + (rem & 7) * 16) = make_uint4(0, 0, 0, 0);
          }
          __syncwarp();
        }
        // O += P V
#pragma unroll
        for (int nt = 0; nt < NT; nt += 2) {
          const int vrow = (mi & 1) * 8 + ri;       // row within the warp's 16
          const int chunk16 = nt + (mi >> 1);       // 16-byte chunk along d
          uint32_t vb[4];
          ldmatrix_x4_trans(vb, Vt + (chunk16 >> 3) * C::kBoxBytes + swz128(warp * 16 + vrow, chunk16 & 7));
          mma_bf16_16816(o[nt], pa, vb[0], vb[1]);
          mma_bf16_16816(o[nt + 1], pa, vb[2], vb[3]);
        }
        if (zeroed) fence_proxy_async_smem();
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[st]);
    }
    // the appended row joins the last split (warp 0), bias 0
    if (app && s == S - 1 && warp == 0 && !*s_abort) {
      const __nv_bfloat16* kn = static_cast<const __nv_bfloat16*>(a.k_new) + bk * D;
      const __nv_bfloat16* vn = static_cast<const __nv_bfloat16*>(a.v_new) + bk * D;
      float sv[2] = {-INFINITY, -INFINITY};
      for (int g = 0; g < G; ++g) {
        float part = 0.f;
        for (int d = lane; d < D; d += 32) part = fmaf(__bfloat162float(qg[(size_t)g * D + d]), __bfloat162float(kn[d]), part);
        part = warp_sum(part) * sc;
        if (g == g0) sv[0] = part;
        if (g == g0 + 8) sv[1] = part;
      }
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        if (g0 + r * 8 >= G) continue;
        const float mn = fmaxf(mrow[r], sv[r]);
        const float cr = exp2f(mrow[r] - mn);
        const float pn = exp2f(sv[r] - mn);
        lrow[r] = lrow[r] * cr + ((lane & 3) == 0 ? pn : 0.f);
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          const float v0 = __bfloat162float(vn[nt * 8 + c2]);
          const float v1 = __bfloat162float(vn[nt * 8 + c2 + 1]);
          o[nt][r * 2] = o[nt][r * 2] * cr + pn * v0;
          o[nt][r * 2 + 1] = o[nt][r * 2 + 1] * cr + pn * v1;
        }
        mrow[r] = mn;
      }
      write_append_row<__nv_bfloat16>(a, bk, L, lane, 32);
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 1);
      lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 2);
    }
  }
  // Fold the warp states into this split's partial.  The warps' (max, sum) live outside the
  // ring, so one barrier both drains the ring and publishes them; each warp then scales its
  // own output by 2^(m_w - max) while storing it, and the partial output is the sum over
  // the warps in warp order.  An aborted CTA leaves an empty partial.
  if (warp < kConsumers && (lane & 3) == 0) {
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int g = g0 + r * 8;
      if (g >= G) continue;
      wm[warp * 16 + g] = mrow[r];
      wl[warp * 16 + g] = lrow[r];
    }
  }
  __syncthreads();  // the ring is idle (drained) from here on: reuse it for the fold
  const bool aborted = *s_abort != 0;
  const PartialView pv = partial_view(a);
  float* wo = reinterpret_cast<float*>(smem);  // [kConsumers][16][kFoldLd], scaled outputs
  if (warp < kConsumers) {
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int g = g0 + r * 8;
      if (g >= G) continue;
      float M = -INFINITY;
#pragma unroll
      for (int w = 0; w < kConsumers; ++w) M = fmaxf(M, wm[w * 16 + g]);
      const float f = M == -INFINITY ? 0.f : exp2f(mrow[r] - M);
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
        *reinterpret_cast<float2*>(wo + (warp * 16 + g) * C::kFoldLd + nt * 8 + c2) =
            make_float2(o[nt][r * 2] * f, o[nt][r * 2 + 1] * f);
      if (warp == 0 && (lane & 3) == 0) {
        float Ls = 0.f;
        if (M != -INFINITY) {
#pragma unroll
          for (int w = 0; w < kConsumers; ++w) Ls = fmaf(wl[w * 16 + g], exp2f(wm[w * 16 + g] - M), Ls);
        }
        if (S == 1) s_inv[g] = (Ls > 0.f && !aborted) ? 1.f / Ls : 0.f;
        else *pv.ml(bk, g, s) = aborted ? make_float2(-INFINITY, 0.f) : make_float2(M, Ls);
      }
    }
  }
  __syncthreads();
  {
    constexpr int D4 = D / 4;
    for (int i = tid; i < G * D4; i += blockDim.x) {
      const int g = i / D4, d4 = i % D4;
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int w = 0; w < kConsumers; ++w) {
        const float4 v = *reinterpret_cast<const float4*>(wo + (w * 16 + g) * C::kFoldLd + d4 * 4);
        acc.x += v.x;
        acc.y += v.y;
        acc.z += v.z;
        acc.w += v.w;
      }
      if (aborted) acc = make_float4(0.f, 0.f, 0.f, 0.f);
      if (S == 1) {
        // the CTA holds the whole of (b, kv): its fold is the output
        const float iv = s_inv[g];
        const float r[4] = {acc.x * iv, acc.y * iv, acc.z * iv, acc.w * iv};
        store4(static_cast<__nv_bfloat16*>(a.out) + (bk * G + g) * D + d4 * 4, r);
      } else {
        reinterpret_cast<float4*>(pv.o(bk, g, s))[d4] = acc;
      }
    }
  }
  if (S == 1) {
    // no split to wait for: only the length bookkeeping of the sequence remains
    if (tid == 0) {
      const uint32_t old = finish_lengths_begin(a, b, bk, app, 0);
      finish_lengths_end(a, b, L, app, old, 0);
    }
    return;
  }
  if (!arrive_last(a, bk, &s_last)) return;
  if (S <= kRegSplits)
    combine_registers<D>(a, b, kv, bk, L, app);
  else
    combine_record<D>(a, b, kv, bk, smem, C::kRingBytes, comb, L, app);
}

// ---- one split per (b, kv), more units than CTAs: persistent CTAs ------------------------------
// When the split model gives every (b, kv) a single CTA and there are more of them than SMs,
// a grid of kUnitsCtas CTAs walks the units instead: CTA p takes units p, p + P, p + 2P, ...
// in turn.  The producer streams the next unit's tiles while the consumer warps fold the
// previous one (the ring runs on across units), so the start and drain of a CTA are paid once
// per CTA instead of once per unit.  Each unit is held whole by one CTA: its fold is its output.
// The group's queries (and the appended row) are staged in shared memory per unit, so the
// mma fragments are not held in registers across the tiles.
template <int D, bool ROWS16>
struct UCfg {
  using C = Cfg<D>;
  static constexpr int kRows = ROWS16 ? 16 : 8;          // group rows a warp state holds
  static constexpr int kFoldLd = D + 8;
  static constexpr int kFoldBytes = kConsumers * kRows * kFoldLd * 4;
  static constexpr int kQLd = D + 8;                     // staged query row stride (bf16)
  static constexpr int kQBytes = 16 * kQLd * 2 + 2 * D * 2;  // queries (16 rows), k_new, v_new
  // ring | fold scratch | queries | full, empty, pre [kStages] | abort | warp (max, sum), appended row
  static constexpr int kSmemBytes =
      1024 + C::kRingBytes + kFoldBytes + kQBytes + 3 * kStages * 8 + 8 + 2 * (kConsumers + 1) * 16 * 4;
  static_assert((C::kRingBytes + kFoldBytes) % 16 == 0 && kQBytes % 16 == 0, "query rows 16-byte aligned");
};

template <int D, bool ROWS16>
__global__ __launch_bounds__(kThreads, 1) void decode_units_kernel(const __grid_constant__ CUtensorMap tmK,
                                                                   const __grid_constant__ CUtensorMap tmV,
                                                                   DecodeArgs a) {
  using C = Cfg<D>;
  using U = UCfg<D, ROWS16>;
  constexpr int NT = D / 8;
  constexpr int KS = D / 16;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  float* wo = reinterpret_cast<float*>(smem + C::kRingBytes);  // [kConsumers][kRows][kFoldLd]
  __nv_bfloat16* sq = reinterpret_cast<__nv_bfloat16*>(smem + C::kRingBytes + U::kFoldBytes);  // [16][kQLd]
  __nv_bfloat16* snew = sq + 16 * U::kQLd;                                                   // [2][D]
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::kRingBytes + U::kFoldBytes + U::kQBytes);
  uint64_t* empty = full + kStages;
  uint64_t* pre = empty + kStages;
  volatile int* s_abort = reinterpret_cast<volatile int*>(pre + kStages);
  float* wm = reinterpret_cast<float*>(pre + kStages + 1);  // [kConsumers][16]
  float* wl = wm + kConsumers * 16;                         // [kConsumers][16]
  float* apm = wl + kConsumers * 16;                        // [16] appended row's logit
  float* apw = apm + 16;                                    // [16] its weight / the normaliser
  __shared__ int s_pre_n;
  __shared__ float s_inv[16];  // 1 / normaliser per query head of the unit

  const int p = blockIdx.x, P = gridDim.x;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = a.G;
  const int units = a.B * a.Hkv;
  constexpr int kBar = 1;  // named barrier of the consumer warps
  constexpr int kCons = kConsumers * 32;

  if (warp == kConsumers && lane == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], kConsumers);
      mbar_init(&pre[i], 1);
    }
    *s_abort = 0;
    fence_mbar_init();
    prefetch_tensormap(&tmK);
    prefetch_tensormap(&tmV);
    // Before griddepcontrol.wait: the first unit's first tiles below its (possibly stale)
    // length minus one, as in the split kernel; kept after the wait if the length still covers them.
    int npre = 0;
    if (p < units) {
      const int b = p / a.Hkv;
      const size_t bk = (size_t)p;
      const int Lg = min(max(ld_relaxed_gpu(a.lengths + b), 0), a.m_cap);
      const int safe = Lg - 1;
      const int max_pre = Lg >= SELKV_DEC_PRELOAD_MIN * kTile ? min(kStages, SELKV_DEC_PRELOAD) : 0;
      for (; npre < max_pre && (npre + 1) * kTile <= safe; ++npre) {
        unsigned char* base = smem + npre * C::kStageBytes;
        mbar_arrive_expect_tx(&pre[npre], C::kStageBytes);
        for (int h = 0; h < kHalves; ++h) {
          const int y = (int)(bk * a.m_cap) + npre * kTile + h * kBoxRows;
#pragma unroll
          for (int bx = 0; bx < C::kBoxes; ++bx)
            tma_load_2d(base + bx * C::kBoxBytes + h * C::kPieceBytes, &tmK, bx * 64, y, &pre[npre]);
#pragma unroll
          for (int bx = 0; bx < C::kBoxes; ++bx)
            tma_load_2d(base + C::kTileBytes + bx * C::kBoxBytes + h * C::kPieceBytes, &tmV, bx * 64, y, &pre[npre]);
        }
      }
      const char* qp = static_cast<const char*>(a.q) + ((size_t)b * a.Hq + (size_t)(p % a.Hkv) * G) * D * 2;
      for (int off = 0; off < G * D * 2; off += 128) prefetch_l2(qp + off);
    }
    s_pre_n = npre;
  }
  pdl_wait();
  pdl_launch_dependents();
  __syncthreads();
  const bool has_new = a.k_new != nullptr;

  if (warp == kConsumers) {
    // ---------------- producer ----------------
    if (lane == 0) {
      const int npre = s_pre_n;
      uint32_t pre_seen = 0u;
      int issued = 0;  // tiles handed to the consumers so far, over all of this CTA's units
      bool stop = false;
      for (int u = p; u < units && !stop; u += P) {
        const int L = min(max(a.lengths[u / a.Hkv], 0), a.m_cap);
        const int nt = (L + kTile - 1) / kTile;
        const int row0 = (int)((size_t)u * a.m_cap);
        for (int t = 0; t < nt; ++t) {
          const int tg = issued, st = tg % kStages;
          if (!mbar_wait(&empty[st], ((tg / kStages) & 1) ^ 1)) {
            *s_abort = 1;
            raise_flag(a.flags, SELKV_DEVERR_TIMEOUT);
            stop = true;
            break;
          }
          if (*s_abort) {
            stop = true;
            break;
          }
          if (tg < npre) {
            // the early load into this stage lands before the stage is released or reloaded
            if (!mbar_wait(&pre[st], 0)) {
              *s_abort = 1;
              raise_flag(a.flags, SELKV_DEVERR_TIMEOUT);
              stop = true;
              break;
            }
            pre_seen |= 1u << st;
            if (u == p && (t + 1) * kTile <= L) {
              mbar_arrive(&full[st]);  // the tile is already in place
              issued = tg + 1;
              continue;
            }
          }
          unsigned char* base = smem + st * C::kStageBytes;
          const int nh = min(kHalves, (L - t * kTile + kBoxRows - 1) / kBoxRows);
          mbar_arrive_expect_tx(&full[st], 2 * nh * C::kBoxes * C::kPieceBytes);
          for (int h = 0; h < nh; ++h) {
            const int y = row0 + t * kTile + h * kBoxRows;
#pragma unroll
            for (int bx = 0; bx < C::kBoxes; ++bx)
              tma_load_2d(base + bx * C::kBoxBytes + h * C::kPieceBytes, &tmK, bx * 64, y, &full[st]);
#pragma unroll
            for (int bx = 0; bx < C::kBoxes; ++bx)
              tma_load_2d(base + C::kTileBytes + bx * C::kBoxBytes + h * C::kPieceBytes, &tmV, bx * 64, y, &full[st]);
          }
          issued = tg + 1;
        }
      }
      for (int tg = max(0, issued - kStages); tg < issued; ++tg) mbar_wait(&full[tg % kStages], (tg / kStages) & 1);
      for (int st = 0; st < npre; ++st)
        if (!(pre_seen & (1u << st))) mbar_wait(&pre[st], 0);
    }
    return;
  }
  // ---------------- consumers ----------------
  const int g0 = lane >> 2, c2 = (lane & 3) * 2;
  const float sc = a.scale_log2;
  int tg = 0;  // tiles consumed so far, in step with the producer
  for (int u = p; u < units; u += P) {
    const int b = u / a.Hkv;
    const size_t bk = (size_t)u;
    int L = a.lengths[b];
    if (L < 0 || L > a.m_cap) {
      if (tid == 0 && u % a.Hkv == 0) raise_flag(a.flags, SELKV_DEVERR_LENGTH);
      L = L < 0 ? 0 : a.m_cap;
    }
    const bool app = has_new && L + 1 <= a.m_cap;
    const int nt = (L + kTile - 1) / kTile;
    float o[NT][4];
    float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};
#pragma unroll
    for (int n8 = 0; n8 < NT; ++n8)
#pragma unroll
      for (int e = 0; e < 4; ++e) o[n8][e] = 0.f;
    {
      const __nv_bfloat16* qg = static_cast<const __nv_bfloat16*>(a.q) + ((size_t)b * a.Hq + (size_t)(u - b * a.Hkv) * G) * D;
      for (int i = tid; i < 16 * (D / 8); i += kCons) {
        const int row = i / (D / 8), c8 = i % (D / 8);
        const uint4 v = row < G ? *reinterpret_cast<const uint4*>(qg + (size_t)row * D + c8 * 8) : make_uint4(0, 0, 0, 0);
        *reinterpret_cast<uint4*>(sq + row * U::kQLd + c8 * 8) = v;
      }
      if (app) {
        // the appended row: into shared memory for the fold, and into the cache at row L (no
        // tile of this launch reads it)
        for (int i = tid; i < 2 * (D / 8); i += kCons) {
          const bool isv = i >= D / 8;
          const int c8 = isv ? i - D / 8 : i;
          const uint4 v = *reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(isv ? a.v_new : a.k_new) +
                                                          bk * D + c8 * 8);
          *reinterpret_cast<uint4*>(snew + (isv ? D : 0) + c8 * 8) = v;
          *reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(isv ? a.Vc : a.Kc) + (bk * a.m_cap + L) * D + c8 * 8) = v;
        }
        if (tid == 0 && a.bias != nullptr) a.bias[bk * a.m_cap + L] = 0.f;
      }
    }
    named_bar_sync(kBar, kCons);
    const uint32_t qs = smem_u32(sq) + (uint32_t)(((lane & 15) * U::kQLd + (lane >> 4) * 8) * 2);
    const float* brow = a.bias != nullptr ? a.bias + bk * a.m_cap : nullptr;
    auto fetch_bias = [&](int t, float (&dst)[2][2]) {
#pragma unroll
      for (int n2 = 0; n2 < 2; ++n2)
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int key = t * kTile + warp * 16 + n2 * 8 + c2 + e;
          dst[n2][e] = (brow != nullptr && key < L) ? __ldg(brow + key) * kLog2e : 0.f;
        }
    };
    float bnext[2][2];
    if (nt > 0) fetch_bias(0, bnext);
    for (int t = 0; t < nt; ++t, ++tg) {
      float bv[2][2];
#pragma unroll
      for (int n2 = 0; n2 < 2; ++n2)
#pragma unroll
        for (int e = 0; e < 2; ++e) bv[n2][e] = bnext[n2][e];
      if (t + 1 < nt) fetch_bias(t + 1, bnext);
      const int st = tg % kStages;
      if (!__all_sync(0xffffffffu, *s_abort == 0)) break;
      if (!__all_sync(0xffffffffu, mbar_wait(&full[st], (tg / kStages) & 1))) {
        *s_abort = 1;
        if (lane == 0) raise_flag(a.flags, SELKV_DEVERR_TIMEOUT);
        break;
      }
      const int key0 = t * kTile + warp * 16;
      const int nvalid = L - key0;
      if (nvalid > 0) {
        const uint32_t Kt = smem_u32(smem + st * C::kStageBytes);
        const uint32_t Vt = Kt + C::kTileBytes;
        float sacc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
        const int mi = lane >> 3, ri = lane & 7;
#pragma unroll
        for (int ks = 0; ks < KS; ++ks) {
          const int krow = (mi >> 1) * 8 + ri;
          const int chunk16 = ks * 2 + (mi & 1);
          uint32_t kb[4], qf[4];
          ldmatrix_x4(kb, Kt + (chunk16 >> 3) * C::kBoxBytes + swz128(warp * 16 + krow, chunk16 & 7));
          ldmatrix_x4(qf, qs + ks * 32);
          mma_bf16_16816(sacc[0], qf, kb[0], kb[1]);
          mma_bf16_16816(sacc[1], qf, kb[2], kb[3]);
        }
        float tmax[2] = {-INFINITY, -INFINITY};
#pragma unroll
        for (int n2 = 0; n2 < 2; ++n2)
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const bool ok = key0 + n2 * 8 + c2 + e < L;
#pragma unroll
            for (int r = 0; r < 2; ++r) {
              const float v = ok ? fmaf(sacc[n2][r * 2 + e], sc, bv[n2][e]) : -INFINITY;
              sacc[n2][r * 2 + e] = v;
              tmax[r] = fmaxf(tmax[r], v);
            }
          }
        float corr[2], mref[2];
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          tmax[r] = fmaxf(tmax[r], __shfl_xor_sync(0xffffffffu, tmax[r], 1));
          tmax[r] = fmaxf(tmax[r], __shfl_xor_sync(0xffffffffu, tmax[r], 2));
          const float mn = fmaxf(mrow[r], tmax[r]);
          mref[r] = mn == -INFINITY ? 0.f : mn;
          corr[r] = exp2f(mrow[r] - mref[r]);
          mrow[r] = mn;
        }
        float pr[2][4];
        float psum[2] = {0.f, 0.f};
#pragma unroll
        for (int n2 = 0; n2 < 2; ++n2)
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            pr[n2][i] = exp2f(sacc[n2][i] - mref[i >> 1]);
            psum[i >> 1] += pr[n2][i];
          }
#pragma unroll
        for (int r = 0; r < 2; ++r) lrow[r] = lrow[r] * corr[r] + psum[r];
#pragma unroll
        for (int n8 = 0; n8 < NT; ++n8) {
          o[n8][0] *= corr[0];
          o[n8][1] *= corr[0];
          o[n8][2] *= corr[1];
          o[n8][3] *= corr[1];
        }
        uint32_t pa[4];
        pa[0] = pack_bf16(pr[0][0], pr[0][1]);
        pa[1] = pack_bf16(pr[0][2], pr[0][3]);
        pa[2] = pack_bf16(pr[1][0], pr[1][1]);
        pa[3] = pack_bf16(pr[1][2], pr[1][3]);
        const bool zeroed = nvalid < 16;
        if (zeroed) {
          unsigned char* vt = smem + st * C::kStageBytes + C::kTileBytes;
          for (int i = lane; i < (16 - nvalid) * C::kBoxes * 8; i += 32) {
            const int r = warp * 16 + nvalid + i / (C::kBoxes * 8);
            const int rem = i % (C::kBoxes * 8);
            *reinterpret_cast<uint4*>(vt + (rem >> 3) * C::kBoxBytes + r * 128 + (rem & 7) * 16) = make_uint4(0, 0, 0, 0);
          }
          __syncwarp();
        }
#pragma unroll
        for (int n8 = 0; n8 < NT; n8 += 2) {
          const int vrow = (mi & 1) * 8 + ri;
          const int chunk16 = n8 + (mi >> 1);
          uint32_t vb[4];
          ldmatrix_x4_trans(vb, Vt + (chunk16 >> 3) * C::kBoxBytes + swz128(warp * 16 + vrow, chunk16 & 7));
          mma_bf16_16816(o[n8], pa, vb[0], vb[1]);
          mma_bf16_16816(o[n8 + 1], pa, vb[2], vb[3]);
        }
        if (zeroed) fence_proxy_async_smem();
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[st]);
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 1);
      lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 2);
    }
    // Fold the warp states (and the appended row, bias 0) into the unit's output, among the
    // consumer warps only: the producer is already loading the next unit.
    if (app) {
      for (int g = warp; g < G; g += kConsumers) {
        float part = 0.f;
        for (int d = lane; d < D; d += 32)
          part = fmaf(__bfloat162float(sq[g * U::kQLd + d]), __bfloat162float(snew[d]), part);
        part = warp_sum(part) * sc;
        if (lane == 0) apm[g] = part;
      }
    }
    if ((lane & 3) == 0) {
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        const int g = g0 + r * 8;
        if (g >= G) continue;
        wm[warp * 16 + g] = mrow[r];
        wl[warp * 16 + g] = lrow[r];
      }
    }
    named_bar_sync(kBar, kCons);
    const bool aborted = *s_abort != 0;
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int g = g0 + r * 8;
      if (g >= G) continue;
      float M = app ? apm[g] : -INFINITY;
#pragma unroll
      for (int w = 0; w < kConsumers; ++w) M = fmaxf(M, wm[w * 16 + g]);
      const float f = M == -INFINITY ? 0.f : exp2f(mrow[r] - M);
#pragma unroll
      for (int n8 = 0; n8 < NT; ++n8)
        *reinterpret_cast<float2*>(wo + (warp * U::kRows + g) * U::kFoldLd + n8 * 8 + c2) =
            make_float2(o[n8][r * 2] * f, o[n8][r * 2 + 1] * f);
      if (warp == 0 && (lane & 3) == 0) {
        float Ls = 0.f;
        if (M != -INFINITY) {
#pragma unroll
          for (int w = 0; w < kConsumers; ++w) Ls = fmaf(wl[w * 16 + g], exp2f(wm[w * 16 + g] - M), Ls);
        }
        const float wa = app ? exp2f(apm[g] - M) : 0.f;  // M >= apm[g] > -inf when app
        Ls += wa;
        const float inv = (Ls > 0.f && !aborted) ? 1.f / Ls : 0.f;
        apw[g] = wa * inv;   // the appended row's share of the output
        s_inv[g] = inv;
      }
    }
    named_bar_sync(kBar, kCons);
    {
      constexpr int D4 = D / 4;
      for (int i = tid; i < G * D4; i += kCons) {
        const int g = i / D4, d4 = i % D4;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int w = 0; w < kConsumers; ++w) {
          const float4 v = *reinterpret_cast<const float4*>(wo + (w * U::kRows + g) * U::kFoldLd + d4 * 4);
          acc.x += v.x;
          acc.y += v.y;
          acc.z += v.z;
          acc.w += v.w;
        }
        const float inv = s_inv[g];
        float r[4] = {acc.x * inv, acc.y * inv, acc.z * inv, acc.w * inv};
        if (app) {
          const float wa = apw[g];
          const __nv_bfloat16* vn = snew + D + d4 * 4;
#pragma unroll
          for (int e = 0; e < 4; ++e) r[e] = fmaf(wa, __bfloat162float(vn[e]), r[e]);
        }
        store4(static_cast<__nv_bfloat16*>(a.out) + (bk * G + g) * D + d4 * 4, r);
      }
    }
    // The sequence's length advances once all its KV heads are done: each has read it by now.
    if (tid == 0 && has_new) {
      if (app) {
        if (atom_add_acq_rel_gpu(&a.cnt_seq[b], 1u) == (uint32_t)a.Hkv - 1u) {
          a.lengths[b] = L + 1;
          a.cnt_seq[b] = 0u;
        }
      } else if (u % a.Hkv == 0) {
        raise_flag(a.flags, SELKV_DEVERR_CAPACITY);
      }
    }
    // the next unit rewrites the staged queries, the warp states and the fold scratch only
    // after every consumer has passed this barrier
    named_bar_sync(kBar, kCons);
  }
}

template <int D, bool R16>
cudaError_t launch_tc_t(const DecodeArgs& a, cudaStream_t st) {
  CUtensorMap tk, tv;
  const uint64_t rows = (uint64_t)a.B * a.Hkv * a.m_cap;
  if (!encode_rows_bf16(&tk, a.Kc, rows, D, kBoxRows) || !encode_rows_bf16(&tv, a.Vc, rows, D, kBoxRows))
    return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(kThreads);
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = SELKV_DEC_PDL ? 1 : 0;
  if (SELKV_DEC_UNITS && a.splits == 1 && a.B * a.Hkv > kPlanSMs && a.m_cap <= SELKV_DEC_UNITS_MAX_ROWS) {
    // one split per (b, kv), more units than SMs, short units: persistent CTAs walk the units
    // (with longer units the static walk balances worse than the hardware's CTA scheduling)
    cudaError_t e = set_smem_once<decode_units_kernel<D, R16>>(UCfg<D, R16>::kSmemBytes);
    if (e != cudaSuccess) return e;
    cfg.gridDim = dim3(kPlanSMs, 1, 1);
    cfg.dynamicSmemBytes = UCfg<D, R16>::kSmemBytes;
    return cudaLaunchKernelEx(&cfg, decode_units_kernel<D, R16>, tk, tv, a);
  }
  cudaError_t e = set_smem_once<decode_tc_kernel<D, R16>>(Cfg<D>::kSmemBytes);
  if (e != cudaSuccess) return e;
  cfg.gridDim = dim3(a.splits, a.Hkv, a.B);
  cfg.dynamicSmemBytes = Cfg<D>::kSmemBytes;
  return cudaLaunchKernelEx(&cfg, decode_tc_kernel<D, R16>, tk, tv, a);
}

}  // namespace

cudaError_t launch_decode_tc(const DecodeArgs& a, cudaStream_t st) {
  if (a.D == 128) return a.G > 8 ? launch_tc_t<128, true>(a, st) : launch_tc_t<128, false>(a, st);
  return a.G > 8 ? launch_tc_t<64, true>(a, st) : launch_tc_t<64, false>(a, st);
}

}  // namespace selkv
