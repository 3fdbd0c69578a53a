// Observation-window scoring on the 5th-generation tensor cores (bf16 caches).
//
// Per (sequence b, KV head kv) the G query heads' W window rows are stacked into R = G W rows
// (row r = g W + i is query head kv G + g at position p = n_b - W + i, which sees keys j <= p:
// the causal re-pass of Sec. 3.1).  With s'_rj = log2(e) q_r . k_j / sqrt(d):
//   pass 1: per row, over a slice of the keys: (max_j s'_rj, sum_j 2^(s'_rj - max)),
//   (fold)  M_r, Z_r over the slices (rowstat_reduce_kernel),
//   pass 2: a_j = sum_r 2^(s'_rj - M_r) / (G Z_r)   (Eq. 5's a, mean over the group).
// Both passes are one kernel: a TMA producer warp streams 128-key K tiles (and the group's Q
// once) into shared memory with 128-byte swizzling; one thread issues tcgen05.mma (bf16 in,
// fp32 accumulate) into one of two tensor-memory accumulators; eight epilogue warps read the
// accumulator with tcgen05.ld and reduce it while the next tile is multiplied.  Pass 1 puts
// the query rows in the accumulator lanes (M = 128 rows per MMA, N = 128 keys), so each
// epilogue thread owns a row; pass 2 puts the keys in the lanes (M = 128 keys, N = R rows),
// so each epilogue thread owns a column sum.
//
// Every wait is bounded; on timeout the CTA raises SELKV_DEVERR_TIMEOUT, keeps the barrier
// protocol of its epilogue warps, lets issued copies and MMAs finish (bounded) and frees its
// tensor memory before leaving.
#include <cudaTypedefs.h>

#include "ptx.cuh"
#include "selkv_internal.cuh"

namespace selkv {
namespace {

constexpr int kKeys = 128;  // keys per tile
constexpr int kEpiWarps = 8;
constexpr int kProducerWarp = 8, kMmaWarp = 9;
constexpr int kThreads = (kEpiWarps + 2) * 32;
constexpr int kStages = 4;
constexpr uint32_t kTmemCols = 512;  // two accumulators of up to 256 fp32 columns

template <int D>
struct SCfg {
  static constexpr int kBoxes = D / 64;                  // 128-byte-wide boxes per row
  static constexpr int kKTile = kKeys * D * 2;           // one K tile
  static constexpr int kQBytes = 256 * D * 2;            // the group's Q, up to 256 rows
  static constexpr int kRing = kStages * kKTile;
  static constexpr int kMisc = 256 + 256 * 8 + 2 * 128 * 4;
  static constexpr int kSmem = 1024 + kQBytes + kRing + kMisc;
};

template <int D, int PASS>
__global__ __launch_bounds__(kThreads, 1) void score_tc_kernel(const __grid_constant__ CUtensorMap tmQ,
                                                                const __grid_constant__ CUtensorMap tmK,
                                                                CompressArgs a) {
  using C = SCfg<D>;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  unsigned char* Qs = smem;                  // [kBoxes][Rq rows][128 B]
  unsigned char* Ks = smem + C::kQBytes;     // [kStages][kBoxes][kKeys rows][128 B]
  unsigned char* misc = Ks + C::kRing;
  uint64_t* full = reinterpret_cast<uint64_t*>(misc);
  uint64_t* empty = full + kStages;
  uint64_t* tfull = empty + kStages;
  uint64_t* tempty = tfull + 2;
  uint64_t* qbar = tempty + 2;
  uint64_t* done = qbar + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float2* rstat = reinterpret_cast<float2*>(misc + 256);            // pass 2: (M, 1/(G Z))
  float* colpart = reinterpret_cast<float*>(misc + 256 + 256 * 8);  // pass 2: [2][kKeys]

  const int split = blockIdx.x, kv = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n = a.seq_n[b];
  const int R = a.R;
  const int Rp = (R + 15) & ~15;              // N of the pass-2 MMA
  const int Rq = R > 128 ? 256 : 128;         // rows of Q staged (whole TMA boxes)
  const int MT = (R + 127) / 128;             // pass-1 M tiles
  const int ntiles_all = (n + kKeys - 1) / kKeys;
  const int per = (ntiles_all + a.nchunks - 1) / a.nchunks;
  const int t_begin = split * per;
  const int nt = max(0, min(ntiles_all, t_begin + per) - t_begin);
  const size_t bk = (size_t)b * a.Hkv + kv;
  const int krow0 = (int)(bk * a.n_cap) + t_begin * kKeys;
  const int qrow0 = (b * a.Hq + kv * a.G) * a.W;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], kEpiWarps);
    }
    mbar_init(qbar, 1);
    mbar_init(done, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == kMmaWarp) tmem_alloc(tmem_slot, kTmemCols);
  if (PASS == 2)
    for (int r = threadIdx.x; r < 256; r += blockDim.x)
      rstat[r] = r < R ? a.rowstat[bk * R + r] : make_float2(0.f, 0.f);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == kProducerWarp) {
    if (lane == 0 && nt > 0) {
      prefetch_tensormap(&tmQ);
      prefetch_tensormap(&tmK);
      mbar_arrive_expect_tx(qbar, C::kBoxes * Rq * 128);
      for (int bx = 0; bx < C::kBoxes; ++bx)
        for (int r0 = 0; r0 < Rq; r0 += 128) tma_load_2d(Qs + (bx * Rq + r0) * 128, &tmQ, bx * 64, qrow0 + r0, qbar);
      int issued = 0;
      for (int t = 0; t < nt; ++t) {
        const int st = t % kStages;
        if (!mbar_wait(&empty[st], ((t / kStages) & 1) ^ 1) || *abort_flag) {
          *abort_flag = 1;
          raise_flag(a.flags, SELKV_DEVERR_TIMEOUT);
          break;
        }
        mbar_arrive_expect_tx(&full[st], C::kKTile);
        for (int bx = 0; bx < C::kBoxes; ++bx)
          tma_load_2d(Ks + st * C::kKTile + bx * kKeys * 128, &tmK, bx * 64, krow0 + t * kKeys, &full[st]);
        issued = t + 1;
      }
      for (int t = max(0, issued - kStages); t < issued; ++t) mbar_wait(&full[t % kStages], (t / kStages) & 1);
      mbar_wait(qbar, 0);
    }
  } else if (warp == kMmaWarp) {
    if (lane == 0 && nt > 0) {
      bool ok = mbar_wait(qbar, 0);
      const uint32_t idesc = PASS == 1 ? umma_idesc_bf16(128, kKeys) : umma_idesc_bf16(128, Rp);
      const uint32_t qbase = smem_u32(Qs);
      int t = 0;
      for (; ok && t < nt; ++t) {
        const int st = t % kStages, buf = t & 1;
        if (!mbar_wait(&full[st], (t / kStages) & 1) || !mbar_wait(&tempty[buf], ((t >> 1) & 1) ^ 1) ||
            *abort_flag) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t kbase = smem_u32(Ks + st * C::kKTile);
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
          const uint32_t koff = (ks >> 2) * (kKeys * 128) + (ks & 3) * 32;
          const uint32_t qoff = (ks >> 2) * (Rq * 128) + (ks & 3) * 32;
          if (PASS == 1) {
            for (int mt = 0; mt < MT; ++mt)
              umma_bf16(tmem + buf * 256 + mt * 128, umma_desc_sw128(qbase + qoff + mt * 128 * 128),
                        umma_desc_sw128(kbase + koff), idesc, ks > 0);
          } else {
            umma_bf16(tmem + buf * 256, umma_desc_sw128(kbase + koff), umma_desc_sw128(qbase + qoff), idesc, ks > 0);
          }
        }
        umma_commit(&empty[st]);
        umma_commit(&tfull[buf]);
      }
      if (!ok) {
        *abort_flag = 1;
        raise_flag(a.flags, SELKV_DEVERR_TIMEOUT);
      }
      umma_commit(done);  // every MMA issued above has completed once this arrives
      mbar_wait(done, 0);
    }
  } else {
    // ---------------- epilogue: warps 0-7 ----------------
    const int wg = warp >> 2, q = warp & 3;
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    const float sc = a.scale_log2;
    // lane 0 waits, the warp follows its verdict (tcgen05.ld below needs the whole warp)
    auto warp_wait = [&](uint64_t* bar, uint32_t parity) -> bool {
      int ok = 0;
      if (lane == 0) {
        ok = !*abort_flag && mbar_wait(bar, parity);
        if (!ok && !*abort_flag) {
          *abort_flag = 1;
          raise_flag(a.flags, SELKV_DEVERR_TIMEOUT);
        }
      }
      return __shfl_sync(0xffffffffu, ok, 0) != 0;
    };
    if (PASS == 1) {
      const int r = wg * 128 + q * 32 + lane;  // query row owned by this thread
      const bool row_ok = r < R;
      const int p = n - a.W + (r % a.W);        // its last visible key
      float m_run = -INFINITY, l_run = 0.f;
      for (int t = 0; t < nt; ++t) {
        const int buf = t & 1;
        const bool ok = warp_wait(&tfull[buf], (t >> 1) & 1);
        tc_fence_after();
        if (ok && wg < MT) {
          const int key0 = (t_begin + t) * kKeys;
          const bool full_tile = key0 + kKeys - 1 <= n - a.W;  // every row sees every key
#pragma unroll 1
          for (int c = 0; c < kKeys; c += 32) {
            float v[32];
            tmem_ld32(tmem + lane_base + buf * 256 + wg * 128 + c, v);
            float cm[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
            if (full_tile && row_ok) {
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                v[i] *= sc;
                cm[i & 3] = fmaxf(cm[i & 3], v[i]);
              }
            } else {
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                v[i] = (row_ok && key0 + c + i <= p) ? v[i] * sc : -INFINITY;
                cm[i & 3] = fmaxf(cm[i & 3], v[i]);
              }
            }
            const float mn = fmaxf(m_run, fmaxf(fmaxf(cm[0], cm[1]), fmaxf(cm[2], cm[3])));
            if (mn != -INFINITY) {
              float s4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
              for (int i = 0; i < 32; ++i) s4[i & 3] += ex2_approx(v[i] - mn);
              l_run = l_run * ex2_approx(m_run - mn) + ((s4[0] + s4[1]) + (s4[2] + s4[3]));
              m_run = mn;
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty[buf]);
      }
      if (row_ok) a.rowpart[(bk * a.nchunks + split) * R + r] = make_float2(m_run, l_run);
    } else {
      const int klane = q * 32 + lane;   // key owned by this thread within the tile
      const int r_lo = wg * 128, r_hi = min(R, r_lo + 128);
      for (int t = 0; t < nt; ++t) {
        const int buf = t & 1;
        const bool ok = warp_wait(&tfull[buf], (t >> 1) & 1);
        tc_fence_after();
        const int j = (t_begin + t) * kKeys + klane;
        const int jrel = j - (n - a.W);  // > 0: only rows with (r mod W) >= jrel see key j
        float acc = 0.f;
        if (ok) {
#pragma unroll 1
          for (int c = r_lo; c < r_hi; c += 32) {
            float v[32];
            tmem_ld32(tmem + lane_base + buf * 256 + c, v);
            const int cnt = min(32, r_hi - c);
            if (jrel <= 0 && cnt == 32) {
              float a4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
              for (int i = 0; i < 32; i += 2) {
                const float4 st = *reinterpret_cast<const float4*>(&rstat[c + i]);  // rows c+i, c+i+1
                a4[i & 3] = fmaf(ex2_approx(fmaf(v[i], sc, -st.x)), st.y, a4[i & 3]);
                a4[(i + 1) & 3] = fmaf(ex2_approx(fmaf(v[i + 1], sc, -st.z)), st.w, a4[(i + 1) & 3]);
              }
              acc += (a4[0] + a4[1]) + (a4[2] + a4[3]);
            } else {
#pragma unroll
              for (int i = 0; i < 32; ++i)
                if (i < cnt && (jrel <= 0 || (c + i) % a.W >= jrel)) {
                  const float2 st = rstat[c + i];
                  acc = fmaf(ex2_approx(fmaf(v[i], sc, -st.x)), st.y, acc);
                }
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty[buf]);
        // fold the two row halves (warpgroups) of this key
        float* cp = colpart + (t & 1) * kKeys;
        if (wg == 1) cp[klane] = acc;
        named_bar_sync(1, kEpiWarps * 32);
        if (wg == 0 && j < n) a.attn[bk * a.n_cap + j] = acc + cp[klane];
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

template <int D>
cudaError_t launch_tc_t(const CompressArgs& a, cudaStream_t st) {
  CUtensorMap tq, tk;
  if (!encode_rows_bf16(&tq, a.Q, (uint64_t)a.B * a.Hq * a.W, D, 128) ||
      !encode_rows_bf16(&tk, a.K, (uint64_t)a.B * a.Hkv * a.n_cap, D, 128))
    return cudaErrorInvalidValue;
  const dim3 grid(a.nchunks, a.Hkv, a.B);
  auto k1 = score_tc_kernel<D, 1>;
  auto k2 = score_tc_kernel<D, 2>;
  cudaError_t e = cudaFuncSetAttribute(k1, cudaFuncAttributeMaxDynamicSharedMemorySize, SCfg<D>::kSmem);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(k2, cudaFuncAttributeMaxDynamicSharedMemorySize, SCfg<D>::kSmem);
  if (e != cudaSuccess) return e;
  k1<<<grid, kThreads, SCfg<D>::kSmem, st>>>(tq, tk, a);
  e = launch_rowstat_reduce(a, st);
  if (e != cudaSuccess) return e;
  k2<<<grid, kThreads, SCfg<D>::kSmem, st>>>(tq, tk, a);
  return cudaGetLastError();
}

}  // namespace

bool score_uses_tc(int dtype, int D, int R) { return dtype == SELKV_BF16 && (D == 64 || D == 128) && R >= 1 && R <= 256; }

int score_tc_splits(int B, int Hkv, int n_cap, int num_sms) {
  const int units = B * Hkv;
  const int tiles = (n_cap + kKeys - 1) / kKeys;
  int s = num_sms / units;
  if (s < 1) s = 1;
  if (s > tiles) s = tiles;
  return s < 1 ? 1 : s;
}

cudaError_t launch_score_tc(const CompressArgs& a, cudaStream_t st) {
  return a.D == 128 ? launch_tc_t<128>(a, st) : launch_tc_t<64>(a, st);
}

}  // namespace selkv
