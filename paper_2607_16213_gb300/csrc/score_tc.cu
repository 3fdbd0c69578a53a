// Observation-window scoring on the 5th-generation tensor cores (bf16 caches).
//
// Per (sequence b, KV head kv) the G query heads' W window rows are stacked into R = G W rows
// (row r = g W + i is query head kv G + g at position p = n_b - W + i, which sees keys j <= p:
// the causal re-pass of Sec. 3.1).  With s'_rj = log2(e) q_r . k_j / sqrt(d):
//   pass 1: per row, over a slice of the keys: (max_j s'_rj, sum_j 2^(s'_rj - max)),
//   (fold)  M_r, Z_r over the slices (rowstat_reduce_kernel),
//   pass 2: a_j = sum_r 2^(s'_rj - M_r) / (G Z_r) = sum_r 2^(s'_rj - M_r - log2(G Z_r))
//           (Eq. 5's a, mean over the group).
// Both passes are one kernel: a TMA producer warp streams K tiles (and the group's Q once)
// into shared memory with 128-byte swizzling; one thread issues tcgen05.mma (bf16 in, fp32
// accumulate, N = 256 so each instruction carries a full-width product) into one of two
// tensor-memory accumulators; sixteen epilogue warps (four per scheduler) read the
// accumulator with tcgen05.ld and reduce it while the next tile is multiplied.  Pass 1 puts
// 128 query rows in the accumulator lanes (M = 128) and 256 keys in its columns, so a CTA
// owns one half of the R rows; an epilogue thread owns a row and a quarter of each tile's
// keys, and the four quarter states of a row are folded at the end.  Pass 2 puts 128 keys in
// the lanes and the R rows in the columns; an epilogue thread owns a key and a quarter of the
// rows, and the four quarters' column sums of a key are added in shared memory in a fixed
// order before a_j is written.
//
// Every wait is bounded; on timeout the CTA raises SELKV_DEVERR_TIMEOUT, keeps the barrier
// protocol of its epilogue warps, lets issued copies and MMAs finish (bounded) and frees its
// tensor memory before leaving.
#include <cudaTypedefs.h>

#include "ptx.cuh"
#include "selkv_internal.cuh"

namespace selkv {
namespace {

constexpr uint32_t kTmemCols = 512;  // two accumulators of up to 256 fp32 columns
#ifndef SELKV_P1_KEYS
#define SELKV_P1_KEYS 256  // pass 1: keys per tile (the MMA's N), a multiple of 32
#endif
#ifndef SELKV_P1_CPW
#define SELKV_P1_CPW 2     // pass 1: 32-column accumulator chunks per epilogue warp and tile
#endif
// Epilogue warps: pass 1 splits a tile's keys over the warps of each TMEM lane quarter (32
// columns x SELKV_P1_CPW per warp), pass 2 splits the rows over four warps per lane quarter.
// A TMA producer warp and an MMA warp follow them.
constexpr int kP1Parts = SELKV_P1_KEYS / (32 * SELKV_P1_CPW);
static_assert(kP1Parts * 32 * SELKV_P1_CPW == SELKV_P1_KEYS && kP1Parts >= 1, "pass-1 tile split");
static_assert(4 * kP1Parts + 2 <= 32 && SELKV_P1_KEYS <= 256, "pass-1 warps per CTA");
__host__ __device__ constexpr int epi_warps(int pass) { return pass == 1 ? 4 * kP1Parts : 16; }
__host__ __device__ constexpr int cta_threads(int pass) { return (epi_warps(pass) + 2) * 32; }

#ifndef SELKV_P2_PIPE
#define SELKV_P2_PIPE 1   // pass 2: pipelined 16-column TMEM loads on full, unmasked tiles
#endif

// Pass 2, one thread's key over 64 rows of a tile (no causal mask): the sum over the rows of
// 2^(v sc - M_r - log2(G Z_r)).  The accumulator is read 16 columns at a time, each load
// issued before the arithmetic on the previous one so its latency overlaps that work; row
// pairs are packed (f32x2) and summed in four interleaved partial sums.
__device__ __forceinline__ void colsum_accum16(const float (&v)[16], uint32_t rn, uint64_t sc2,
                                               uint64_t& a01, uint64_t& a23) {
#pragma unroll
  for (int i = 0; i < 16; i += 4) {
    const float4 nm = lds_f4(rn + i * 4);  // -(M + log2(G Z)) of rows i .. i+3
    float x0, x1, x2, x3;
    unpack_f2(ffma2(pack_f2(v[i], v[i + 1]), sc2, pack_f2(nm.x, nm.y)), x0, x1);
    unpack_f2(ffma2(pack_f2(v[i + 2], v[i + 3]), sc2, pack_f2(nm.z, nm.w)), x2, x3);
    a01 = fadd2(a01, pack_f2(ex2_approx(x0), ex2_approx(x1)));
    a23 = fadd2(a23, pack_f2(ex2_approx(x2), ex2_approx(x3)));
  }
}
__device__ __forceinline__ float colsum64(uint32_t taddr, uint32_t rn, float sc) {
  const uint64_t sc2 = pack_f2(sc, sc);
  uint64_t a01 = pack_f2(0.f, 0.f), a23 = a01;
  float va[16], vb[16];
  tmem_ld16_issue(taddr, va);
  tmem_wait_ld16(va);
#pragma unroll
  for (int c = 0; c < 4; c += 2) {
    tmem_ld16_issue(taddr + (c + 1) * 16, vb);
    colsum_accum16(va, rn + c * 64, sc2, a01, a23);
    tmem_wait_ld16(vb);
    if (c + 2 < 4) tmem_ld16_issue(taddr + (c + 2) * 16, va);
    colsum_accum16(vb, rn + (c + 1) * 64, sc2, a01, a23);
    if (c + 2 < 4) tmem_wait_ld16(va);
  }
  float s0, s1, s2, s3;
  unpack_f2(a01, s0, s1);
  unpack_f2(a23, s2, s3);
  return (s0 + s1) + (s2 + s3);
}

// HALVES (pass 2): 1 when the R rows fit one accumulator of 256 columns, 2 when they take two
// (R up to 512): each key tile is then multiplied by the two 256-row halves of Q in turn, the
// halves alternating between the two accumulators, and the K ring is shortened to make room
// for the 512 staged rows.
template <int D, int PASS, int HALVES = 1>
struct SCfg {
  static constexpr int kKeys = PASS == 1 ? SELKV_P1_KEYS : 128;        // keys per tile
  static constexpr int kStages = PASS == 1 ? 2 : (HALVES == 2 ? 2 : 4);  // K tiles in flight
  static constexpr int kRows = PASS == 1 ? 128 : 256 * HALVES;          // Q rows staged per CTA
  static constexpr int kBoxes = D / 64;                  // 128-byte-wide boxes per row
  static constexpr int kKTile = kKeys * D * 2;           // one K tile
  static constexpr int kQBytes = kRows * D * 2;
  static constexpr int kRing = kStages * kKTile;
  // barriers | -(M + log2(G Z)) of up to 512 rows | pass 1: [parts][128] float2, pass 2: [2][4][128] float
  static constexpr int kMisc = 256 + 256 * 8 + (kP1Parts * 128 * 8 > 4096 ? kP1Parts * 128 * 8 : 4096);
  static constexpr int kSmem = 1024 + kQBytes + kRing + kMisc;
};

template <int D, int PASS, int HALVES>
__global__ __launch_bounds__(cta_threads(PASS), 1) void score_tc_kernel(const __grid_constant__ CUtensorMap tmQ,
                                                                        const __grid_constant__ CUtensorMap tmK,
                                                                        CompressArgs a) {
  using C = SCfg<D, PASS, HALVES>;
  constexpr int kEpiWarps = epi_warps(PASS);
  constexpr int kProducerWarp = kEpiWarps, kMmaWarp = kEpiWarps + 1;
  constexpr int kKeys = C::kKeys, kStages = C::kStages;
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
  // pass 2: per lane quarter and column-sum buffer, "the other three parts' sums are in" and
  // "part 0 has read them"
  uint64_t* cs_full = reinterpret_cast<uint64_t*>(misc + 128);  // [4][2]
  uint64_t* cs_empty = cs_full + 8;                              // [4][2]
  float* rneg = reinterpret_cast<float*>(misc + 256);               // pass 2: -(M + log2(G Z)) per row
  float* colpart = reinterpret_cast<float*>(misc + 256 + 256 * 8);  // pass 1: [parts][128] float2; pass 2: [2][4][128]

  const int kv = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n = a.seq_n[b];
  const int R = a.R;
  const int Rp = (R + 15) & ~15;              // N of the pass-2 MMAs over all halves
  const int MT = (R + 127) / 128;             // 128-row halves of the R rows
  const int h = PASS == 1 ? (int)blockIdx.x % MT : 0;           // pass 1: this CTA's rows
  const int split = PASS == 1 ? (int)blockIdx.x / MT : (int)blockIdx.x;
  const int nsplit = PASS == 1 ? (int)gridDim.x / MT : (int)gridDim.x;
  const int Rq = PASS == 1 ? 128 : (HALVES == 2 ? 512 : (R > 128 ? 256 : 128));  // Q rows staged (whole boxes)
  const int ntiles_all = (n + kKeys - 1) / kKeys;
  const int per = (ntiles_all + nsplit - 1) / nsplit;
  const int t_begin = split * per;
  const int nt = max(0, min(ntiles_all, t_begin + per) - t_begin);
  const size_t bk = (size_t)b * a.Hkv + kv;
  const int krow0 = (int)(bk * a.n_cap) + t_begin * kKeys;
  const int qrow0 = (b * a.Hq + kv * a.G) * a.W + h * 128;

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
    for (int i = 0; i < 8; ++i) {
      mbar_init(&cs_full[i], 3 * 32);
      mbar_init(&cs_empty[i], 32);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == kMmaWarp) tmem_alloc(tmem_slot, kTmemCols);
  if (PASS == 2)
    for (int r = threadIdx.x; r < 256 * HALVES; r += blockDim.x) {
      // 2^(s' - M) / (G Z) = 2^(s' - (M + log2(G Z))): the normaliser joins the exponent
      const float2 st = r < R ? a.rowstat[bk * R + r] : make_float2(0.f, 0.f);
      rneg[r] = st.y > 0.f ? -(st.x - log2f(st.y)) : -INFINITY;
    }
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
      const uint32_t qbase = smem_u32(Qs);
      int u = 0;  // accumulator use: one per (key tile, row half)
      for (int t = 0; ok && t < nt; ++t) {
        const int st = t % kStages;
        if (!mbar_wait(&full[st], (t / kStages) & 1) || *abort_flag) {
          ok = false;
          break;
        }
        const uint32_t kbase = smem_u32(Ks + st * C::kKTile);
        for (int ph = 0; ph < HALVES; ++ph, ++u) {
          const int buf = u & 1;
          if (!mbar_wait(&tempty[buf], ((u >> 1) & 1) ^ 1) || *abort_flag) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t idesc = PASS == 1 ? umma_idesc_bf16(128, kKeys) : umma_idesc_bf16(128, min(256, Rp - ph * 256));
#pragma unroll
          for (int ks = 0; ks < D / 16; ++ks) {
            const uint32_t koff = (ks >> 2) * (kKeys * 128) + (ks & 3) * 32;
            const uint32_t qoff = (ks >> 2) * (Rq * 128) + (ks & 3) * 32 + ph * 256 * 128;
            if (PASS == 1) {
              umma_bf16(tmem + buf * 256, umma_desc_sw128(qbase + qoff), umma_desc_sw128(kbase + koff), idesc, ks > 0);
            } else {
              umma_bf16(tmem + buf * 256, umma_desc_sw128(kbase + koff), umma_desc_sw128(qbase + qoff), idesc, ks > 0);
            }
          }
          umma_commit(&tfull[buf]);
        }
        if (!ok) break;
        umma_commit(&empty[st]);
      }
      if (!ok) {
        *abort_flag = 1;
        raise_flag(a.flags, SELKV_DEVERR_TIMEOUT);
      }
      umma_commit(done);  // every MMA issued above has completed once this arrives
      mbar_wait(done, 0);
    }
  } else {
    // ---------------- epilogue: warps 0-15 ----------------
    const int q = warp & 3, part = warp >> 2;  // lane quarter of TMEM, and which part of the work
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    const float sc = a.scale_log2;
    // lane 0 waits, the warp follows its outcome (tcgen05.ld below needs the whole warp)
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
      const int r = h * 128 + q * 32 + lane;    // query row owned by this thread
      const bool row_ok = r < R;
      const int p = n - a.W + (r % a.W);        // its last visible key
      float m_run = -INFINITY, l_run = 0.f;     // running max (base 2, scaled) and sum
      for (int t = 0; t < nt; ++t) {
        const int buf = t & 1;
        const bool ok = warp_wait(&tfull[buf], (t >> 1) & 1);
        tc_fence_after();
        constexpr int kCols = 32 * SELKV_P1_CPW;           // this warp's keys of the tile
        const int key0 = (t_begin + t) * kKeys + part * kCols;
        const bool full_quarter = key0 + kCols - 1 <= n - a.W;  // every row sees every key of the part
        // (pass 1 reads the accumulator 32 columns at a time, each load waited for before its
        // arithmetic: pipelined loads measured slower here, 16-column ones because the running
        // max then needs a correction every 16 keys, 32-column ones by half a microsecond)
        if (ok) {
#pragma unroll 1
          for (int c = 0; c < kCols; c += 32) {
            float v[32];
            tmem_ld32(tmem + lane_base + buf * 256 + part * kCols + c, v);
            float cm[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
            if (full_quarter && row_ok) {
#pragma unroll
              for (int i = 0; i < 32; ++i) cm[i & 3] = fmaxf(cm[i & 3], v[i]);
            } else {
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                v[i] = (row_ok && key0 + c + i <= p) ? v[i] : -INFINITY;
                cm[i & 3] = fmaxf(cm[i & 3], v[i]);
              }
            }
            // the scale is positive, so max(v) * scale is the max of the scaled logits
            const float mn = fmaxf(m_run, fmaxf(fmaxf(cm[0], cm[1]), fmaxf(cm[2], cm[3])) * sc);
            if (mn != -INFINITY) {
              // 2^(v sc - mn), pairs packed; sums in four interleaved lanes as (0,1) and (2,3)
              const uint64_t sc2 = pack_f2(sc, sc), nm2 = pack_f2(-mn, -mn);
              uint64_t s01 = pack_f2(0.f, 0.f), s23 = s01;
#pragma unroll
              for (int i = 0; i < 32; i += 4) {
                float x0, x1, x2, x3;
                unpack_f2(ffma2(pack_f2(v[i], v[i + 1]), sc2, nm2), x0, x1);
                unpack_f2(ffma2(pack_f2(v[i + 2], v[i + 3]), sc2, nm2), x2, x3);
                s01 = fadd2(s01, pack_f2(ex2_approx(x0), ex2_approx(x1)));
                s23 = fadd2(s23, pack_f2(ex2_approx(x2), ex2_approx(x3)));
              }
              float s0, s1, s2, s3;
              unpack_f2(s01, s0, s1);
              unpack_f2(s23, s2, s3);
              l_run = l_run * ex2_approx(m_run - mn) + ((s0 + s1) + (s2 + s3));
              m_run = mn;
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty[buf]);
      }
      // fold the key parts of each row in part order (parts 1.. via shared memory)
      float2* st4 = reinterpret_cast<float2*>(colpart);  // [parts][128]
      if (part > 0) st4[part * 128 + q * 32 + lane] = make_float2(m_run, l_run);
      named_bar_sync(1, kEpiWarps * 32);
      if (part == 0 && row_ok) {
        float2 o[kP1Parts];
        o[0] = make_float2(m_run, l_run);
#pragma unroll
        for (int k = 1; k < kP1Parts; ++k) o[k] = st4[k * 128 + q * 32 + lane];
        float M = o[0].x;
#pragma unroll
        for (int k = 1; k < kP1Parts; ++k) M = fmaxf(M, o[k].x);
        float L = 0.f;
        if (M != -INFINITY) {
#pragma unroll
          for (int k = 0; k < kP1Parts; ++k) L += o[k].y * ex2_approx(o[k].x - M);
        }
        a.rowpart[(bk * a.nchunks + split) * R + r] = make_float2(M, L);
      }
    } else {
      const int klane = q * 32 + lane;   // key owned by this thread within the tile
      int u = 0;                         // accumulator use, as counted by the MMA thread
      for (int t = 0; t < nt; ++t) {
        const int j = (t_begin + t) * kKeys + klane;
        const int jrel = j - (n - a.W);  // > 0: only rows with (r mod W) >= jrel see key j
        // every key of this warp is seen by every row: the whole tile is unmasked
        const bool unmasked = (t_begin + t) * kKeys + q * 32 + 31 <= n - a.W;
        float acc = 0.f;
        for (int ph = 0; ph < HALVES; ++ph, ++u) {
          const int buf = u & 1;
          const bool ok = warp_wait(&tfull[buf], (u >> 1) & 1);
          tc_fence_after();
          // this part's 64 rows of the half: accumulator columns from c0, rows from r_lo
          const int c0 = part * 64, r_lo = ph * 256 + c0, r_hi = min(R, r_lo + 64);
          const uint32_t tcol = tmem + lane_base + buf * 256 + c0;
          if (ok && SELKV_P2_PIPE && r_hi - r_lo == 64 && unmasked) {
            acc += colsum64(tcol, smem_u32(rneg + r_lo), sc);
          } else if (ok) {
#pragma unroll 1
            for (int c = r_lo; c < r_hi; c += 32) {
              float v[32];
              tmem_ld32(tcol + (c - r_lo), v);
              const int cnt = min(32, r_hi - c);
              if (jrel <= 0 && cnt == 32) {
                // sum over rows of 2^(v sc - M_r - log2(G Z_r)), pairs of rows packed; four
                // interleaved partial sums as (0,1) and (2,3)
                const uint64_t sc2 = pack_f2(sc, sc);
                uint64_t a01 = pack_f2(0.f, 0.f), a23 = a01;
#pragma unroll
                for (int i = 0; i < 32; i += 4) {
                  const float4 nm = *reinterpret_cast<const float4*>(&rneg[c + i]);  // rows c+i .. c+i+3
                  float x0, x1, x2, x3;
                  unpack_f2(ffma2(pack_f2(v[i], v[i + 1]), sc2, pack_f2(nm.x, nm.y)), x0, x1);
                  unpack_f2(ffma2(pack_f2(v[i + 2], v[i + 3]), sc2, pack_f2(nm.z, nm.w)), x2, x3);
                  a01 = fadd2(a01, pack_f2(ex2_approx(x0), ex2_approx(x1)));
                  a23 = fadd2(a23, pack_f2(ex2_approx(x2), ex2_approx(x3)));
                }
                float s0, s1, s2, s3;
                unpack_f2(a01, s0, s1);
                unpack_f2(a23, s2, s3);
                acc += (s0 + s1) + (s2 + s3);
              } else {
#pragma unroll
                for (int i = 0; i < 32; ++i)
                  if (i < cnt && (jrel <= 0 || (c + i) % a.W >= jrel))
                    acc += ex2_approx(fmaf(v[i], sc, rneg[c + i]));
              }
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&tempty[buf]);
        }
        // The four row quarters' column sums of key j meet in shared memory (two buffers,
        // alternating by tile): parts 1-3 leave theirs and go on, part 0 adds them to its own in
        // quarter order and writes a_j.  A part reuses a buffer only once part 0 has read it.
        const int cb = t & 1;
        float* cs = colpart + cb * 512;  // [4][128]
        uint64_t* cfull = &cs_full[q * 2 + cb];
        uint64_t* cempty = &cs_empty[q * 2 + cb];
        // bounded wait of every lane (each lane acquires what it then reads or overwrites)
        auto lane_wait = [&](uint64_t* bar, uint32_t parity) {
          if (*abort_flag) return;
          if (!mbar_wait(bar, parity)) {
            *abort_flag = 1;
            raise_flag(a.flags, SELKV_DEVERR_TIMEOUT);
          }
        };
        if (part > 0) {
          if (t >= 2) lane_wait(cempty, ((t >> 1) - 1) & 1);
          cs[part * 128 + klane] = acc;
          mbar_arrive(cfull);
        } else {
          lane_wait(cfull, (t >> 1) & 1);
          const float sum = ((acc + cs[128 + klane]) + cs[256 + klane]) + cs[384 + klane];
          mbar_arrive(cempty);
          if (j < n) a.attn[bk * a.n_cap + j] = sum;
        }
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

// Splits of the keys of one (sequence, KV head): enough CTAs for one per SM, each CTA
// owning `row_parts` x (a slice of `keys`-key tiles).
int splits_for(int B, int Hkv, int n_cap, int num_sms, int row_parts, int keys) {
  const int units = B * Hkv * row_parts;
  const int tiles = (n_cap + keys - 1) / keys;
  int s = num_sms / units;
  if (s > tiles) s = tiles;
  return s < 1 ? 1 : s;
}

template <int D, int HALVES>
cudaError_t launch_tc_t(const CompressArgs& a, cudaStream_t st, int passes) {
  using C1 = SCfg<D, 1>;
  using C2 = SCfg<D, 2, HALVES>;
  CUtensorMap tq, tk1, tk2;
  if (!encode_rows_bf16(&tq, a.Q, (uint64_t)a.B * a.Hq * a.W, D, 128) ||
      !encode_rows_bf16(&tk1, a.K, (uint64_t)a.B * a.Hkv * a.n_cap, D, C1::kKeys) ||
      !encode_rows_bf16(&tk2, a.K, (uint64_t)a.B * a.Hkv * a.n_cap, D, C2::kKeys))
    return cudaErrorInvalidValue;
  const int MT = (a.R + 127) / 128;
  const dim3 grid1(a.nchunks * MT, a.Hkv, a.B);
  const dim3 grid2(splits_for(a.B, a.Hkv, a.n_cap, kPlanSMs, 1, C2::kKeys), a.Hkv, a.B);
  auto k1 = score_tc_kernel<D, 1, 1>;
  auto k2 = score_tc_kernel<D, 2, HALVES>;
  cudaError_t e = set_smem_once<score_tc_kernel<D, 1, 1>>(C1::kSmem);
  if (e == cudaSuccess) e = set_smem_once<score_tc_kernel<D, 2, HALVES>>(C2::kSmem);
  if (e != cudaSuccess) return e;
  if (passes & kScoreRowstats) {
    k1<<<grid1, cta_threads(1), C1::kSmem, st>>>(tq, tk1, a);
    e = launch_rowstat_reduce(a, st);
    if (e != cudaSuccess) return e;
  }
  if (passes & kScoreColsums) k2<<<grid2, cta_threads(2), C2::kSmem, st>>>(tq, tk2, a);
  return cudaGetLastError();
}

}  // namespace

// The window rows of a KV group, R = G W, go to the tensor cores up to 512 (two 256-row halves
// in the column-sum pass); wider groups take the CUDA-core path.
bool score_uses_tc(int dtype, int D, int R) { return dtype == SELKV_BF16 && (D == 64 || D == 128) && R >= 1 && R <= 512; }

int score_tc_splits(int B, int Hkv, int n_cap, int R, int num_sms) {
  return splits_for(B, Hkv, n_cap, num_sms, (R + 127) / 128, SCfg<128, 1>::kKeys);
}

cudaError_t launch_score_tc(const CompressArgs& a, cudaStream_t st, int passes) {
  if (a.R > 256) return a.D == 128 ? launch_tc_t<128, 2>(a, st, passes) : launch_tc_t<64, 2>(a, st, passes);
  return a.D == 128 ? launch_tc_t<128, 1>(a, st, passes) : launch_tc_t<64, 1>(a, st, passes);
}

}  // namespace selkv
