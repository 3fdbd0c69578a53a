// Full cosine routing: the alternative that Sec. 3.4 sets against the bucket routing.  Every
// evicted token j of a KV head goes to the kept token i of that head with the largest
// cos(v_j, v_i) over all kept tokens (original values, ties to the lower position, a zero norm
// gives cosine 0); gate, merge (Eq. 4-6) and bias are those of the bucket routing.
//
// For a fixed j the cosine orders the kept tokens as s_ji = (v_j . v_i) / ||v_i|| does, so the
// routing is a row argmax of the product V V_kept^T scaled by column: a dense contraction of
// |S| |E| d multiply-adds per KV head, run on the tensor cores for bf16 caches.  Kernels, in
// stream order (after the copy kernel has put the kept rows into V_c and 1 / ||v_i|| into
// cos_invn):
//   argmax   a CTA per 128 evicted positions of one (sequence, KV head): their value rows are
//            gathered once into shared memory (the MMA's A), 256-slot tiles of the kept rows
//            stream in by TMA (B), tcgen05.mma accumulates 128 x 256 products in tensor memory,
//            and sixteen epilogue warps keep each row's running (max s_ji, slot) over a quarter
//            of each tile's columns; the quarters are folded in column order at the end.  The
//            row's target, gate g = clamp(s / ||v_j||, 0, 1) and decision are written there.
//            fp32 caches use a CUDA-core kernel with the same outputs.
//   rank     stable counting sort of the contributors (g > 0) by target slot, part 1: a warp per
//            (chunk of positions, block of 2048 slots) walks its chunk in ascending order and
//            gives each contributor its rank among the earlier ones of the chunk with the
//            same target, keeping per-slot counts in shared memory;
//   colscan  per slot, the counts of the chunks turned into their exclusive prefix, and the total;
//   slotscan exclusive prefix of the totals over the slots: the slot's first entry;
//   scatter  each contributor to base[slot] + prefix[chunk][slot] + rank: the contributors of a
//            slot end up grouped, in ascending position order;
//   merge    a warp per kept slot with contributors: Eq. 5 and Eq. 6 over them in that order.
// Every sum runs in a fixed order; no floating-point atomics.
#include <climits>
#include <cudaTypedefs.h>

#include "ptx.cuh"
#include "selkv_internal.cuh"

namespace selkv {
namespace {

// ---- row finish: target, gate and decision of position j --------------------------------
// (Evicted positions only; the copy kernel writes the entries of the kept ones.)
__device__ __forceinline__ void cos_finish(const CompressArgs& a, int b, int kv, int j, float best, int bcol) {
  const size_t bk = (size_t)b * a.Hkv + kv;
  const size_t o = bk * a.n_cap + j;
  const size_t su = sel_unit(a, b, kv);
  float g = 0.f;
  int tpos = -1;
  if (bcol >= 0) {
    tpos = a.kept_pos[su * a.m_cap + bcol];
    const float nj = a.vnorm[o];
    const float sim = nj > 0.f ? best / nj : 0.f;
    g = a.gate_mode == SELKV_GATE_OPEN ? 1.f : a.gate_mode == SELKV_GATE_CLOSED ? 0.f : fminf(fmaxf(sim, 0.f), 1.f);
  }
  a.cos_tslot[o] = g > 0.f ? bcol : -1;
  a.cos_g[o] = g;
  if (a.dbg_target) a.dbg_target[o] = tpos;
  if (a.dbg_gate) a.dbg_gate[o] = g;
  if (a.dbg_decision) a.dbg_decision[o] = g > 0.f ? 1 : 0;
}

// (s, c) replaces (best, bcol) if it is larger, or equal at a lower slot
__device__ __forceinline__ void argmax_take(float& best, int& bcol, float s, int c) {
  if (c >= 0 && (bcol < 0 || s > best || (s == best && c < bcol))) {
    best = s;
    bcol = c;
  }
}

// ---- argmax on the tensor cores (bf16) ----------------------------------------------------
constexpr int kEpiWarps = 16;
constexpr int kProducerWarp = 16, kMmaWarp = 17;
constexpr int kThreads = (kEpiWarps + 2) * 32;
constexpr int kCols = 256;                 // kept slots per tile: the MMA's N
constexpr int kChunkBytes = kCols * 128;   // one 64-element-wide box of a tile
constexpr int kRingChunks = 4;             // two tiles in flight at d = 128
constexpr uint32_t kTmemCols = 512;        // two 256-column accumulators

template <int D>
struct CosCfg {
  static constexpr int kBoxes = D / 64;
  static constexpr int kABytes = 128 * D * 2;
  static constexpr int kRing = kRingChunks * kChunkBytes;
  static constexpr int kMisc = 256 + 3 * 128 * 8;
  static constexpr int kSmem = 1024 + kABytes + kRing + kMisc;
  static_assert(kSmem <= 227 * 1024, "shared memory per CTA");
};

__device__ __forceinline__ uint64_t fmul2(uint64_t x, uint64_t y) {
  uint64_t d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(x), "l"(y));
  return d;
}

template <int D>
__global__ __launch_bounds__(kThreads, 1) void cos_tc_kernel(const __grid_constant__ CUtensorMap tmB, CompressArgs a) {
  using C = CosCfg<D>;
  const int kv = blockIdx.y, b = blockIdx.z;
  const int n = a.seq_n[b], m = a.seq_m[b], ne = n - m;
  const int r0 = blockIdx.x * 128;
  if (r0 >= ne) return;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  unsigned char* As = smem;                 // [kBoxes][128 rows][128 B]
  unsigned char* ring = smem + C::kABytes;  // [kRingChunks][256 rows][128 B]
  unsigned char* misc = ring + C::kRing;
  uint64_t* full = reinterpret_cast<uint64_t*>(misc);
  uint64_t* empty = full + kRingChunks;
  uint64_t* tfull = empty + kRingChunks;
  uint64_t* tempty = tfull + 2;
  uint64_t* abar = tempty + 2;
  uint64_t* done = abar + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float2* fold = reinterpret_cast<float2*>(misc + 256);  // [3][128] (best, slot) of quarters 1-3

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const size_t bk = (size_t)b * a.Hkv + kv;
  const size_t su = sel_unit(a, b, kv);
  const int nt = (m + kCols - 1) / kCols;
  const int nchunks = nt * C::kBoxes;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kRingChunks; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], kEpiWarps);
    }
    mbar_init(abar, 1);
    mbar_init(done, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == kMmaWarp) tmem_alloc(tmem_slot, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == kProducerWarp) {
    if (lane == 0 && nt > 0) {
      prefetch_tensormap(&tmB);
      const int brow0 = (int)(bk * a.m_cap);
      int issued = 0;
      for (int c = 0; c < nchunks; ++c) {
        const int st = c % kRingChunks;
        if (!mbar_wait(&empty[st], ((c / kRingChunks) & 1) ^ 1) || *abort_flag) {
          *abort_flag = 1;
          raise_flag(a.flags, SELKV_DEVERR_TIMEOUT);
          break;
        }
        mbar_arrive_expect_tx(&full[st], kChunkBytes);
        tma_load_2d(ring + st * kChunkBytes, &tmB, (c % C::kBoxes) * 64, brow0 + (c / C::kBoxes) * kCols, &full[st]);
        issued = c + 1;
      }
      for (int c = max(0, issued - kRingChunks); c < issued; ++c)
        mbar_wait(&full[c % kRingChunks], (c / kRingChunks) & 1);
    }
  } else if (warp == kMmaWarp) {
    if (lane == 0 && nt > 0) {
      bool ok = mbar_wait(abar, 0);
      const uint32_t idesc = umma_idesc_bf16(128, kCols);
      const uint32_t abase = smem_u32(As), rbase = smem_u32(ring);
      for (int t = 0; ok && t < nt; ++t) {
        const int buf = t & 1;
        if (!mbar_wait(&tempty[buf], ((t >> 1) & 1) ^ 1) || *abort_flag) {
          ok = false;
          break;
        }
        for (int bx = 0; bx < C::kBoxes; ++bx) {
          const int c = t * C::kBoxes + bx, st = c % kRingChunks;
          if (!mbar_wait(&full[st], (c / kRingChunks) & 1) || *abort_flag) {
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int ks = 0; ks < 4; ++ks)
            umma_bf16(tmem + buf * kCols, umma_desc_sw128(abase + bx * 128 * 128 + ks * 32),
                      umma_desc_sw128(rbase + st * kChunkBytes + ks * 32), idesc, (bx | ks) > 0);
          umma_commit(&empty[st]);  // the stage is free once these MMAs have read it
        }
        if (!ok) break;
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
    // ---------------- epilogue: warps 0-15 ----------------
    const int32_t* ev = a.ev_pos + su * a.n_cap;  // evicted positions, ascending
    {
      // gather the 128 evicted value rows into the swizzled A layout (rows past the evicted
      // count repeat the last one; their results are not written)
      constexpr int kRowChunks = D / 8;  // 16-byte pieces per row
      const __nv_bfloat16* Vb = static_cast<const __nv_bfloat16*>(a.V) + bk * a.n_cap * D;
      const uint32_t abase = smem_u32(As);
      for (int i = threadIdx.x; i < 128 * kRowChunks; i += kEpiWarps * 32) {
        const int r = i / kRowChunks, ch = i % kRowChunks;
        const int j = ev[min(r0 + r, ne - 1)];
        cp_async16_cg(abase + (ch >> 3) * (128 * 128) + swz128(r, ch & 7), Vb + (size_t)j * D + ch * 8);
      }
      cp_async_wait_all();
      fence_proxy_async_smem();  // visible to the tensor cores (async proxy)
      named_bar_sync(1, kEpiWarps * 32);
      if (threadIdx.x == 0) mbar_arrive(abar);
    }
    const int q = warp & 3, part = warp >> 2;  // TMEM lane quarter (rows), column quarter of a tile
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    const float* invn = a.cos_invn + bk * a.cos_mpad;
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
    float best = -INFINITY;
    int bcol = -1;
    for (int t = 0; t < nt; ++t) {
      const int buf = t & 1;
      const bool ok = warp_wait(&tfull[buf], (t >> 1) & 1);
      tc_fence_after();
      if (ok) {
#pragma unroll 1
        for (int c = 0; c < 64; c += 32) {
          float v[32];
          tmem_ld32(tmem + lane_base + buf * kCols + part * 64 + c, v);
          const int col0 = t * kCols + part * 64 + c;
          if (col0 >= m) continue;  // uniform across the warp
          // s = acc / ||v_i||, pairs packed; slots past m take -inf
          const float4* w4 = reinterpret_cast<const float4*>(invn + col0);
#pragma unroll
          for (int i = 0; i < 32; i += 4) {
            const float4 w = __ldg(w4 + i / 4);
            unpack_f2(fmul2(pack_f2(v[i], v[i + 1]), pack_f2(w.x, w.y)), v[i], v[i + 1]);
            unpack_f2(fmul2(pack_f2(v[i + 2], v[i + 3]), pack_f2(w.z, w.w)), v[i + 2], v[i + 3]);
          }
          if (col0 + 32 > m) {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = col0 + i < m ? v[i] : -INFINITY;
          }
          const float cmax = max32(v);
          if (cmax > best) {  // strictly larger: an equal value at a later slot does not win
            int first = 31;   // the lowest slot holding the maximum
#pragma unroll
            for (int i = 30; i >= 0; --i) first = v[i] == cmax ? i : first;
            best = cmax;
            bcol = col0 + first;
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[buf]);
    }
    // fold the four column quarters of each row (their columns interleave: compare slots)
    const int r = q * 32 + lane;
    if (part > 0) fold[(part - 1) * 128 + r] = make_float2(best, __int_as_float(bcol));
    named_bar_sync(1, kEpiWarps * 32);
    if (part == 0 && r0 + r < ne) {
#pragma unroll
      for (int k = 0; k < 3; ++k) {
        const float2 f = fold[k * 128 + r];
        argmax_take(best, bcol, f.x, __float_as_int(f.y));
      }
      cos_finish(a, b, kv, ev[r0 + r], best, bcol);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ---- argmax on the CUDA cores (fp32 caches) ----------------------------------------------
// A warp per evicted position j: lane l takes the slots l, l + 32, ... in ascending order, then
// the warp reduces (max, lower slot).
constexpr int kSimtRows = 8;
template <typename T, int D>
__global__ __launch_bounds__(kSimtRows * 32) void cos_simt_kernel(CompressArgs a) {
  const int kv = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int e = blockIdx.x * kSimtRows + warp;  // evicted rank
  const int n = a.seq_n[b], m = a.seq_m[b];
  __shared__ float vj[kSimtRows][D];
  if (e >= n - m) return;
  const size_t bk = (size_t)b * a.Hkv + kv;
  const int j = a.ev_pos[sel_unit(a, b, kv) * a.n_cap + e];
  const T* row = static_cast<const T*>(a.V) + (bk * a.n_cap + j) * D;
  for (int d = lane; d < D; d += 32) vj[warp][d] = load1(row + d);
  __syncwarp();
  const T* Vc = static_cast<const T*>(a.Vc) + bk * a.m_cap * D;
  const float* invn = a.cos_invn + bk * a.cos_mpad;
  float best = -INFINITY;
  int bcol = -1;
  for (int i = lane; i < m; i += 32) {
    const T* ri = Vc + (size_t)i * D;
    float acc = 0.f;
#pragma unroll 8
    for (int d = 0; d < D; ++d) acc = fmaf(vj[warp][d], load1(ri + d), acc);
    const float s = acc * invn[i];
    if (s > best || bcol < 0) {
      best = s;
      bcol = i;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float s2 = __shfl_xor_sync(0xffffffffu, best, o);
    const int c2 = __shfl_xor_sync(0xffffffffu, bcol, o);
    argmax_take(best, bcol, s2, c2);
  }
  if (lane == 0) cos_finish(a, b, kv, j, best, bcol);
}

// ---- stable counting sort of the contributors by target slot ------------------------------
constexpr int kRankSlots = 2048;

__global__ __launch_bounds__(32) void cos_rank_kernel(CompressArgs a) {
  const int c = blockIdx.x, s0 = blockIdx.y * kRankSlots;
  const int bk = blockIdx.z, b = bk / a.Hkv;
  const int n = a.seq_n[b], m = a.seq_m[b];
  if (s0 >= m) return;
  const int ns = min(kRankSlots, m - s0);
  const int lane = threadIdx.x;
  __shared__ int cnt[kRankSlots];
  for (int k = lane; k < kRankSlots; k += 32) cnt[k] = 0;
  __syncwarp();
  const int j_lo = c * a.cos_chunk, j_hi = min(n, j_lo + a.cos_chunk);
  const int32_t* ts = a.cos_tslot + (size_t)bk * a.n_cap;
  int32_t* rank = a.cos_rank + (size_t)bk * a.n_cap;
  constexpr int kRounds = 8;  // targets loaded ahead, 32 positions per round
  for (int j0 = j_lo; j0 < j_hi; j0 += kRounds * 32) {
    int tv[kRounds];
#pragma unroll
    for (int k = 0; k < kRounds; ++k) {
      const int j = j0 + k * 32 + lane;
      tv[k] = j < j_hi ? ts[j] : -1;
    }
#pragma unroll
    for (int k = 0; k < kRounds; ++k) {
      const int j = j0 + k * 32 + lane, t = tv[k];
      const bool mine = t >= s0 && t < s0 + ns;
      const uint32_t peers = __match_any_sync(0xffffffffu, mine ? t : -1);
      const int before = mine ? cnt[t - s0] : 0;
      __syncwarp();
      if (mine) {
        const int lt = __popc(peers & ((1u << lane) - 1u));
        if (lt == 0) cnt[t - s0] = before + __popc(peers);
        rank[j] = before + lt;
      }
      __syncwarp();
    }
  }
  int32_t* out = a.cos_cnt + ((size_t)bk * a.cos_chunks + c) * a.m_cap + s0;
  for (int k = lane; k < ns; k += 32) out[k] = cnt[k];
}

__global__ __launch_bounds__(256) void cos_colscan_kernel(CompressArgs a) {
  const int bk = blockIdx.y, b = bk / a.Hkv;
  const int slot = blockIdx.x * blockDim.x + threadIdx.x;
  if (slot >= a.seq_m[b]) return;
  int32_t* col = a.cos_cnt + (size_t)bk * a.cos_chunks * a.m_cap + slot;
  int x[kMaxCosChunks];
#pragma unroll
  for (int c = 0; c < kMaxCosChunks; ++c) x[c] = c < a.cos_chunks ? col[(size_t)c * a.m_cap] : 0;
  int run = 0;
#pragma unroll
  for (int c = 0; c < kMaxCosChunks; ++c) {
    if (c < a.cos_chunks) col[(size_t)c * a.m_cap] = run;
    run += x[c];
  }
  a.cos_seg[(size_t)bk * a.m_cap + slot].y = run;
}

__global__ __launch_bounds__(1024) void cos_slotscan_kernel(CompressArgs a) {
  const int bk = blockIdx.x, b = bk / a.Hkv;
  const int m = a.seq_m[b];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __shared__ int wsum[32];
  int2* seg = a.cos_seg + (size_t)bk * a.m_cap;
  int carry = 0;
  for (int s0 = 0; s0 < m; s0 += 4096) {
    const int s = s0 + 4 * threadIdx.x;  // four consecutive slots per thread
    int e[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) e[k] = s + k < m ? seg[s + k].y : 0;
    const int x = (e[0] + e[1]) + (e[2] + e[3]);
    int v = x;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, v, o);
      if (lane >= o) v += y;
    }
    if (lane == 31) wsum[warp] = v;
    __syncthreads();
    if (warp == 0) {
      int w = wsum[lane];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, w, o);
        if (lane >= o) w += y;
      }
      wsum[lane] = w;
    }
    __syncthreads();
    int run = carry + (warp > 0 ? wsum[warp - 1] : 0) + v - x;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      if (s + k < m) seg[s + k].x = run;
      run += e[k];
    }
    carry += wsum[31];
    __syncthreads();  // wsum is rewritten by the next round
  }
}

__global__ __launch_bounds__(256) void cos_scatter_kernel(CompressArgs a) {
  const int bk = blockIdx.y, b = bk / a.Hkv;
  const int n = a.seq_n[b];
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= n) return;
  const size_t o = (size_t)bk * a.n_cap + j;
  const int t = a.cos_tslot[o];
  if (t < 0) return;
  const int c = j / a.cos_chunk;
  const int dest = a.cos_seg[(size_t)bk * a.m_cap + t].x +
                   a.cos_cnt[((size_t)bk * a.cos_chunks + c) * a.m_cap + t] + a.cos_rank[o];
  if (dest < 0 || dest >= n) {
    raise_flag(a.flags, SELKV_DEVERR_COUNT);
    return;
  }
  a.cos_order[(size_t)bk * a.n_cap + dest] = j;
}

// ---- gated merge over each slot's contributors (Eq. 5, Eq. 6) ----------------------------
constexpr int kMergeWarps = 8;
constexpr int kBatch = 8;  // contributor rows in flight per lane

template <typename T, int D>
__global__ __launch_bounds__(kMergeWarps * 32) void cos_merge_kernel(CompressArgs a) {
  constexpr int PER = D / 32;
  const int bk = blockIdx.y, b = bk / a.Hkv, kv = bk % a.Hkv;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int slot = blockIdx.x * kMergeWarps + warp;
  if (slot >= a.seq_m[b]) return;
  const size_t sm = (size_t)bk * a.m_cap + slot;
  const int2 sg = a.cos_seg[sm];  // (first entry, contributors)
  const int pos = a.kept_pos[sel_unit(a, b, kv) * a.m_cap + slot];
  const int cnt = sg.y, beg = sg.x;
  if (cnt == 0) return;  // V_c keeps the kept value, R = 1 (copy kernel)
  const T* Vb = static_cast<const T*>(a.V) + (size_t)bk * a.n_cap * D;
  const float* A = a.attn + (size_t)bk * a.n_cap;
  const float* Gt = a.cos_g + (size_t)bk * a.n_cap;
  const int32_t* ord = a.cos_order + (size_t)bk * a.n_cap + beg;
  RowSlice<T, PER> vi;
  vi.load(Vb + (size_t)pos * D + lane * PER);
  const float a_i = A[pos];
  float num[PER];
#pragma unroll
  for (int t = 0; t < PER; ++t) num[t] = 0.f;
  float den = 0.f;
  for (int e0 = 0; e0 < cnt; e0 += 32) {
    const int k = min(32, cnt - e0);
    const int jj = lane < k ? ord[e0 + lane] : 0;
    const float w = lane < k ? Gt[jj] * A[jj] : 0.f;
    for (int k0 = 0; k0 < k; k0 += kBatch) {
      RowSlice<T, PER> vj[kBatch];
#pragma unroll
      for (int kk = 0; kk < kBatch; ++kk) {
        const int jx = __shfl_sync(0xffffffffu, jj, (k0 + kk) & 31);
        if (k0 + kk < k) vj[kk].load(Vb + (size_t)jx * D + lane * PER);
        else vj[kk].zero();
      }
#pragma unroll
      for (int kk = 0; kk < kBatch; ++kk) {
        const float wk = __shfl_sync(0xffffffffu, w, (k0 + kk) & 31);
        if (k0 + kk >= k) break;
#pragma unroll
        for (int t = 0; t < PER; ++t) num[t] = fmaf(wk, vj[kk][t], num[t]);
        den += wk;
      }
    }
  }
  const float tot = a_i + den;
  float vm[PER];
#pragma unroll
  for (int t = 0; t < PER; ++t) vm[t] = tot > 0.f ? (a_i * vi[t] + num[t]) / tot : vi[t];
  T* Vc = static_cast<T*>(a.Vc) + sm * D + lane * PER;
  if constexpr (PER == 4) {
    store4(Vc, vm);
  } else {
    store1(Vc, vm[0]);
    store1(Vc + 1, vm[1]);
  }
  if (lane == 0) {
    const float R = a_i > 0.f ? tot / a_i : 1.f;
    a.ratio[sm] = R;
    a.mcount[sm] = (float)cnt;
    if (a.dbg_ratio) a.dbg_ratio[sm] = R;
  }
}

template <int D>
cudaError_t launch_argmax_tc(const CompressArgs& a, cudaStream_t st) {
  using C = CosCfg<D>;
  if ((uint64_t)a.B * a.Hkv * a.m_cap >= (1ull << 31)) return cudaErrorInvalidValue;  // 32-bit TMA rows
  CUtensorMap tb;
  if (!encode_rows_bf16(&tb, a.Vc, (uint64_t)a.B * a.Hkv * a.m_cap, D, kCols)) return cudaErrorInvalidValue;
  cudaError_t e = set_smem_once<cos_tc_kernel<D>>(C::kSmem);
  if (e != cudaSuccess) return e;
  cos_tc_kernel<D><<<dim3((a.n_cap + 127) / 128, a.Hkv, a.B), kThreads, C::kSmem, st>>>(tb, a);
  return cudaGetLastError();
}

template <typename T, int D>
void launch_rest(const CompressArgs& a, cudaStream_t st) {
  const unsigned bkn = (unsigned)(a.B * a.Hkv);
  cos_rank_kernel<<<dim3(a.cos_chunks, (a.m_cap + kRankSlots - 1) / kRankSlots, bkn), 32, 0, st>>>(a);
  cos_colscan_kernel<<<dim3((a.m_cap + 255) / 256, bkn), 256, 0, st>>>(a);
  cos_slotscan_kernel<<<bkn, 1024, 0, st>>>(a);
  cos_scatter_kernel<<<dim3((a.n_cap + 255) / 256, bkn), 256, 0, st>>>(a);
  cos_merge_kernel<T, D><<<dim3((a.m_cap + kMergeWarps - 1) / kMergeWarps, bkn), kMergeWarps * 32, 0, st>>>(a);
}

}  // namespace

int cosine_kernels(int, int) { return 6; }

cudaError_t launch_route_cosine(const CompressArgs& a, cudaStream_t st) {
  if (a.m_cap < 1) return cudaSuccess;
  cudaError_t e = cudaSuccess;
  if (a.dtype == SELKV_BF16) {
    e = a.D == 128 ? launch_argmax_tc<128>(a, st) : launch_argmax_tc<64>(a, st);
    if (e != cudaSuccess) return e;
    if (a.D == 128) launch_rest<__nv_bfloat16, 128>(a, st);
    else launch_rest<__nv_bfloat16, 64>(a, st);
  } else {
    const dim3 grid((a.n_cap + kSimtRows - 1) / kSimtRows, a.Hkv, a.B);
    if (a.D == 128) {
      cos_simt_kernel<float, 128><<<grid, kSimtRows * 32, 0, st>>>(a);
      launch_rest<float, 128>(a, st);
    } else {
      cos_simt_kernel<float, 64><<<grid, kSimtRows * 32, 0, st>>>(a);
      launch_rest<float, 64>(a, st);
    }
  }
  return cudaGetLastError();
}

}  // namespace selkv
