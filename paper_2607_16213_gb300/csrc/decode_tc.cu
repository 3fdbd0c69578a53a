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
// last CTA of (b, kv) to arrive (one atomic add, no waiting), which stages every split's
// partial in the idle ring with one round of asynchronous copies.  The appended row
// (k_new, v_new) joins the last split with bias 0 and is then written at row lengths[b].
//
// Every mbarrier wait is bounded: on timeout the CTA raises SELKV_DEVERR_TIMEOUT, stops, and
// waits (bounded again) for the copies it has issued before leaving.  Launched with
// programmatic dependent launch: the barrier set-up overlaps the previous kernel's tail, and
// nothing another kernel may have written is read before griddepcontrol.wait.
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
  static constexpr int kSmemBytes = kRingBytes + 1024 /*align*/ + 2 * kStages * 8 + 64;
  static_assert(kConsumers * 16 * D * 4 + kConsumers * 16 * 8 <= kRingBytes, "fold scratch fits");
};

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
  volatile int* s_abort = reinterpret_cast<volatile int*>(empty + kStages);
  __shared__ bool s_last;

  const int s = blockIdx.x, kv = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = a.G, S = a.splits;
  const size_t bk = (size_t)b * a.Hkv + kv;

  if (tid == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], kConsumers);
    }
    *s_abort = 0;
    fence_mbar_init();
  }
  if (warp == kConsumers && lane == 0) {
    prefetch_tensormap(&tmK);
    prefetch_tensormap(&tmV);
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
      for (int t = 0; t < ntiles; ++t) {
        const int st = t % kStages;
        if (!mbar_wait(&empty[st], ((t / kStages) & 1) ^ 1)) {
          *s_abort = 1;
          raise_flag(a.flags, SELKV_DEVERR_TIMEOUT);
          break;
        }
        if (*s_abort) break;
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
  __syncthreads();  // the ring is idle (drained) from here on: reuse it for the fold

  float* wo = reinterpret_cast<float*>(smem);                  // [kConsumers][16][D]
  float* wm = wo + kConsumers * 16 * D;                         // [kConsumers][16]
  float* wl = wm + kConsumers * 16;                             // [kConsumers][16]
  if (warp < kConsumers) {
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int g = g0 + r * 8;
      if (g >= G) continue;
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        wo[(warp * 16 + g) * D + nt * 8 + c2] = o[nt][r * 2];
        wo[(warp * 16 + g) * D + nt * 8 + c2 + 1] = o[nt][r * 2 + 1];
      }
      if ((lane & 3) == 0) {
        wm[warp * 16 + g] = mrow[r];
        wl[warp * 16 + g] = lrow[r];
      }
    }
  }
  __syncthreads();
  write_split_partial<kConsumers>(a, b, kv, s, wo, wm, wl, 16, *s_abort != 0);
  if (!arrive_last(a, bk, &s_last)) return;
  const uint32_t seq_old = finish_lengths_begin(a, b, bk, app);
  combine_splits_staged<__nv_bfloat16>(a, b, kv, smem, C::kRingBytes);
  finish_lengths_end(a, b, L, app, seq_old);
}

template <int D, bool R16>
cudaError_t launch_tc_t(const DecodeArgs& a, cudaStream_t st) {
  CUtensorMap tk, tv;
  const uint64_t rows = (uint64_t)a.B * a.Hkv * a.m_cap;
  if (!encode_rows_bf16(&tk, a.Kc, rows, D, kBoxRows) || !encode_rows_bf16(&tv, a.Vc, rows, D, kBoxRows))
    return cudaErrorInvalidValue;
  auto kern = decode_tc_kernel<D, R16>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<D>::kSmemBytes);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.splits, a.Hkv, a.B);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = Cfg<D>::kSmemBytes;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = SELKV_DEC_PDL ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, tk, tv, a);
}

}  // namespace

cudaError_t launch_decode_tc(const DecodeArgs& a, cudaStream_t st) {
  if (a.D == 128) return a.G > 8 ? launch_tc_t<128, true>(a, st) : launch_tc_t<128, false>(a, st);
  return a.G > 8 ? launch_tc_t<64, true>(a, st) : launch_tc_t<64, false>(a, st);
}

}  // namespace selkv
