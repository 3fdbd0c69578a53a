// Internal declarations shared by the SelKV kernels and the C-ABI host code.
#pragma once

#include <atomic>

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/selkv.h"

namespace selkv {

// Every workspace starts with this header; the rest is carved by the host planners.
struct WsHeader {
  uint32_t flags;  // SELKV_DEVERR_* bits, sticky until selkv_workspace_error
  uint32_t pad[63];
};
static_assert(sizeof(WsHeader) == 256, "header is 256 bytes");

constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ void raise_flag(uint32_t* flags, uint32_t bit) { atomicOr(flags, bit); }

// ---- element access: storage dtype -> fp32 ------------------------------------------------
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// Load 8 consecutive elements starting at p (16-byte aligned for bf16, 32-byte for fp32).
__device__ __forceinline__ void load8(const __nv_bfloat16* p, float (&x)[8]) {
  const uint4 u = *reinterpret_cast<const uint4*>(p);
  x[0] = bf16_lo(u.x); x[1] = bf16_hi(u.x);
  x[2] = bf16_lo(u.y); x[3] = bf16_hi(u.y);
  x[4] = bf16_lo(u.z); x[5] = bf16_hi(u.z);
  x[6] = bf16_lo(u.w); x[7] = bf16_hi(u.w);
}
__device__ __forceinline__ void load8(const float* p, float (&x)[8]) {
  const float4 a = reinterpret_cast<const float4*>(p)[0];
  const float4 b = reinterpret_cast<const float4*>(p)[1];
  x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w;
  x[4] = b.x; x[5] = b.y; x[6] = b.z; x[7] = b.w;
}
// Load 4 consecutive elements (8-byte aligned for bf16, 16-byte for fp32).
__device__ __forceinline__ void load4(const __nv_bfloat16* p, float (&x)[4]) {
  const uint2 u = *reinterpret_cast<const uint2*>(p);
  x[0] = bf16_lo(u.x); x[1] = bf16_hi(u.x);
  x[2] = bf16_lo(u.y); x[3] = bf16_hi(u.y);
}
__device__ __forceinline__ void load4(const float* p, float (&x)[4]) {
  const float4 a = *reinterpret_cast<const float4*>(p);
  x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w;
}
__device__ __forceinline__ void load2(const __nv_bfloat16* p, float (&x)[2]) {
  const uint32_t u = *reinterpret_cast<const uint32_t*>(p);
  x[0] = bf16_lo(u); x[1] = bf16_hi(u);
}
__device__ __forceinline__ void load2(const float* p, float (&x)[2]) {
  const float2 a = *reinterpret_cast<const float2*>(p);
  x[0] = a.x; x[1] = a.y;
}
__device__ __forceinline__ float load1(const __nv_bfloat16* p) { return __bfloat162float(*p); }
__device__ __forceinline__ float load1(const float* p) { return *p; }

__device__ __forceinline__ void store1(__nv_bfloat16* p, float v) { *p = __float2bfloat16_rn(v); }
__device__ __forceinline__ void store1(float* p, float v) { *p = v; }
__device__ __forceinline__ void store4(__nv_bfloat16* p, const float (&x)[4]) {
  __nv_bfloat162 a = __floats2bfloat162_rn(x[0], x[1]);
  __nv_bfloat162 b = __floats2bfloat162_rn(x[2], x[3]);
  uint2 u;
  u.x = *reinterpret_cast<uint32_t*>(&a);
  u.y = *reinterpret_cast<uint32_t*>(&b);
  *reinterpret_cast<uint2*>(p) = u;
}
__device__ __forceinline__ void store4(float* p, const float (&x)[4]) {
  *reinterpret_cast<float4*>(p) = make_float4(x[0], x[1], x[2], x[3]);
}

// One lane's PER consecutive elements of a row, kept in the storage type.
template <typename T, int PER>
struct RowSlice;
template <>
struct RowSlice<__nv_bfloat16, 4> {
  uint2 w;
  __device__ __forceinline__ void load(const __nv_bfloat16* p) { w = *reinterpret_cast<const uint2*>(p); }
  __device__ __forceinline__ void zero() { w = make_uint2(0u, 0u); }
  __device__ __forceinline__ float operator[](int e) const {
    const uint32_t x = e < 2 ? w.x : w.y;
    return (e & 1) ? bf16_hi(x) : bf16_lo(x);
  }
};
template <>
struct RowSlice<__nv_bfloat16, 2> {
  uint32_t w;
  __device__ __forceinline__ void load(const __nv_bfloat16* p) { w = *reinterpret_cast<const uint32_t*>(p); }
  __device__ __forceinline__ void zero() { w = 0u; }
  __device__ __forceinline__ float operator[](int e) const { return (e & 1) ? bf16_hi(w) : bf16_lo(w); }
};
template <int PER>
struct RowSlice<float, PER> {
  float x[PER];
  __device__ __forceinline__ void load(const float* p) {
    if constexpr (PER == 4) {
      const float4 v = *reinterpret_cast<const float4*>(p);
      x[0] = v.x;
      x[1] = v.y;
      x[2] = v.z;
      x[3] = v.w;
    } else {
      const float2 v = *reinterpret_cast<const float2*>(p);
      x[0] = v.x;
      x[1] = v.y;
    }
  }
  __device__ __forceinline__ void zero() {
#pragma unroll
    for (int e = 0; e < PER; ++e) x[e] = 0.f;
  }
  __device__ __forceinline__ float operator[](int e) const { return x[e]; }
};

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// ---- compress -----------------------------------------------------------------------------
struct SeqTable {
  int32_t n[SELKV_MAX_BATCH];  // prefill length n_b
  int32_t m[SELKV_MAX_BATCH];  // budget m_b = floor(rho * n_b)
};

struct CompressArgs {
  int dtype, B, Hq, Hkv, G, D, W, n_cap, m_cap;
  int R;          // observation rows per KV head: G * W
  int nchunks;    // column chunks of the row-statistics pass
  float alpha;
  int pool_kernel, bucket, recent, gate_mode, empty_bucket;
  int per_head;   // SELKV_SELECT_PER_HEAD: selection units are (b, kv), not b
  int rope;       // selkv_rope layout of the kept keys' repositioning (0: off)
  int bias_count; // SELKV_BIAS_COUNT: bias from merge counts instead of ratios
  float rope_theta;
  int rope_hi;    // coarse table entries: position shifts up to 256 * rope_hi
  float2* rope_tab;  // [rope_hi + 256][d/2] (cos, sin) of e * w_f: rows e = 256 c (c < rope_hi), then e = c
  float scale_log2;  // log2(e) / sqrt(d)
  const void* K;
  const void* V;
  const void* Q;
  void* Kc;
  void* Vc;
  float* bias;
  int32_t* lengths;
  // debug outputs (nullable)
  uint8_t* dbg_topk;
  int32_t* dbg_kept_idx;
  int32_t* dbg_target;
  float* dbg_gate;
  uint8_t* dbg_decision;
  float* dbg_ratio;
  // workspace arrays
  uint32_t* flags;
  int32_t* seq_n;
  int32_t* seq_m;
  float2* rowpart;   // [B][Hkv][nchunks][R] (max, sum) of 2^(s' - max) per column chunk
  float2* rowstat;   // [B][Hkv][R] (M, 1 / (G * Z))
  float* attn;       // [B][Hkv][n_cap]
  float* vnorm;      // [B][Hkv][n_cap]
  float* score;      // [B][Hkv][n_cap]
  uint8_t* kflag;    // [units][n_cap] 1 = kept (units: B, or B * Hkv in per-head mode)
  int32_t* slot_of;  // [units][n_cap] slot of a kept position, -1 otherwise
  int32_t* kept_pos; // [units][m_cap] position of each slot
  int nbk;           // buckets per sequence at n_cap: ceil(n_cap / bucket)
  int32_t* tau;      // [B][Hkv][nbk] merge target of each bucket (-1: no kept token)
  float* atau;       // [B][Hkv][nbk] a of that target
  float* ratio;      // [B][Hkv][m_cap] attention ratio R of each slot
  float* mcount;     // [B][Hkv][m_cap] evicted tokens merged into each slot (g > 0)
  // full cosine routing (routing == SELKV_ROUTE_COSINE)
  int routing;
  int cos_chunks;      // position chunks of the stable counting sort by target slot
  int cos_chunk;       // positions per chunk (a multiple of 32)
  int cos_mpad;        // m_cap rounded up to a whole 256-slot tile
  int32_t* ev_pos;     // [units][n_cap] evicted positions in ascending order
  int32_t* cos_tslot;  // [B][Hkv][n_cap] target slot of an evicted j merged with g > 0, else -1
  float* cos_g;        // [B][Hkv][n_cap] gate g of an evicted j
  float* cos_invn;     // [B][Hkv][cos_mpad] 1 / ||v|| of each slot's kept value (0 for a zero norm)
  int32_t* cos_rank;   // [B][Hkv][n_cap] rank of j among the earlier j of its chunk with its target
  int32_t* cos_order;  // [B][Hkv][n_cap] contributors grouped by target slot, ascending within
  int32_t* cos_cnt;    // [B][Hkv][cos_chunks][m_cap] contributors per (chunk, slot), then their prefix
  int2* cos_seg;       // [B][Hkv][m_cap] (first entry in cos_order, contributors) of each slot
};

// SM count used to plan grids and splits: fixed, so that workspace sizes and results do
// not depend on which device answers (GB300: 152 SMs).
constexpr int kPlanSMs = 152;

// Selection unit of (b, kv): the sequence in the shared mode, the KV head in the per-head mode.
__host__ __device__ __forceinline__ size_t sel_unit(const CompressArgs& a, int b, int kv) {
  return a.per_head ? (size_t)b * a.Hkv + kv : (size_t)b;
}

// Coarse RoPE table entries for caches of n_cap rows: position shifts e < n_cap split as
// e = 256 e_hi + e_lo.
__host__ __device__ constexpr int rope_coarse(int n_cap) { return n_cap / 256 + 1; }

constexpr int kRowChunk = 512;  // columns per CTA in the row-statistics pass

// Grid-wide exact radix selection (select_grid.cu).
struct RadixState {
  uint32_t prefix;    // threshold bits fixed so far (the threshold T after the last pass)
  uint32_t krem;      // entries still to take among those matching `prefix`
  uint32_t count_eq;  // after the last pass: entries equal to T
  int32_t jcut;       // last position taken among the entries equal to T
  uint32_t active;    // a selection is still being narrowed
  uint32_t arrive;    // CTAs of the current pass that have finished (self-resetting)
  uint32_t ucount;    // trim only: size of the union
  uint32_t pad;
};
struct SelectWs {
  RadixState* topk;     // [B * Hkv]
  RadixState* trim;     // [B]
  uint32_t* topk_hist;  // [B * Hkv][3][2048]
  uint32_t* trim_hist;  // [B][3][2048]
  size_t hist_bytes;    // both histogram arrays (contiguous)
  uint32_t* blkcnt;     // [B][position blocks]
  float* tkey;          // [B][n_cap] score summed over KV heads
  uint8_t* uflag;       // [B][n_cap] member of the union
};
// Initial radix state i of units + B: top-m_s per (b, kv), then the trim per b.  Called by
// the set-up kernel with seq_n and seq_m of this call.
__device__ __forceinline__ void select_init_state(const CompressArgs& a, const SelectWs& w, int i, int n_b, int m_b) {
  const int units = a.B * a.Hkv;
  const bool trim = i >= units;
  const int b = trim ? i - units : i / a.Hkv;
  (void)b;
  const int k = m_b - a.recent;
  const int ncand = n_b - a.recent;
  RadixState s{};
  s.krem = (uint32_t)max(k, 0);
  s.jcut = INT_MAX;
  if (trim) {
    s.active = k > 0 ? 1u : 0u;  // the union kernel switches it off when |U| <= m_s
  } else if (k <= 0) {
    s.prefix = 0xffffffffu;  // select nothing
    s.jcut = -1;
  } else if (k >= ncand) {
    s.prefix = 0u;  // select every candidate
  } else {
    s.active = 1u;
  }
  if (trim) w.trim[i - units] = s; else w.topk[i] = s;
}

size_t select_ws_bytes(int B, int Hkv, int n_cap);
SelectWs carve_select_ws(void* base, int B, int Hkv, int n_cap);
cudaError_t launch_select_grid(const CompressArgs& a, const SelectWs& w, cudaStream_t s);

// Scoring: tensor-core path for bf16 with G W <= 256 rows, CUDA-core path otherwise.
bool score_uses_tc(int dtype, int D, int R);
int score_tc_splits(int B, int Hkv, int n_cap, int R, int num_sms);  // pass-1 key splits
// passes: bit 0 = row statistics (pass 1 and their fold), bit 1 = column sums (pass 2)
constexpr int kScoreRowstats = 1, kScoreColsums = 2, kScoreAll = 3;
cudaError_t launch_score_tc(const CompressArgs& a, cudaStream_t s, int passes = kScoreAll);
cudaError_t launch_score_simt(const CompressArgs& a, cudaStream_t s, int passes = kScoreAll);
cudaError_t launch_seq_setup(const CompressArgs& a, const SeqTable& tab, cudaStream_t s);
cudaError_t launch_rowstat_reduce(const CompressArgs& a, cudaStream_t s);
// Compensation averaged across layers (layer_average.cu).
constexpr int kMaxLayers = 128;
struct LayerPtrs {
  const int32_t* kept[kMaxLayers];  // each layer's kept positions [B][units per b][m_cap]
  float* bias[kMaxLayers];          // each layer's bias [B][Hkv][m_cap], read and rewritten
};
struct LayerAvgArgs {
  int B, Hkv, m_cap, n_cap, per_head, L;
  float alpha;
  const int32_t* lengths;  // [B] compressed lengths
  float* acc;              // [B][units per b][n_cap] sum over layers of expm1(bias / alpha)
  uint32_t* flags;
};
cudaError_t launch_layer_average(const LayerAvgArgs& a, const LayerPtrs& P, cudaStream_t s);
// Full cosine routing after the kept rows are in place: argmax, gate, grouping and merge.
cudaError_t launch_route_cosine(const CompressArgs& a, cudaStream_t s);
int cosine_kernels(int dtype, int D);  // kernels launch_route_cosine enqueues
// Chunks of the counting sort for caches of n_cap positions, and the chunk length.
constexpr int kMaxCosChunks = 32;
__host__ __device__ constexpr int cos_chunks_for(int n_cap) {
  return n_cap <= 2048 ? 1 : (n_cap + 2047) / 2048 < kMaxCosChunks ? (n_cap + 2047) / 2048 : kMaxCosChunks;
}
__host__ __device__ constexpr int cos_chunk_len(int n_cap) {
  return ((n_cap + cos_chunks_for(n_cap) - 1) / cos_chunks_for(n_cap) + 31) / 32 * 32;
}

// ---- decode -------------------------------------------------------------------------------
struct DecodeArgs {
  int dtype, B, Hq, Hkv, G, D, m_cap, splits;
  float scale_log2;  // log2(e) / sqrt(d)
  const void* q;
  void* Kc;
  void* Vc;
  float* bias;
  int32_t* lengths;
  const void* k_new;
  const void* v_new;
  void* out;
  uint32_t* flags;
  uint32_t* cnt_head;  // [B][Hkv] arrivals per (b, kv) (self-resetting)
  uint32_t* cnt_seq;   // [B] (b, kv) completions per sequence (self-resetting)
  float* partial;      // [B][Hkv] records of decode_record_floats(G, splits, D) floats
};

// Floats of one (sequence, KV head) record of split partials: the unnormalised outputs
// o [G][S][D], then the (max in base 2, sum) pairs [G][S] padded to a 16-byte multiple, so
// every record starts 16-byte aligned and can be moved with one bulk copy.
__host__ __device__ constexpr size_t decode_record_floats(int G, int S, int D) {
  return (size_t)G * S * D + (((size_t)G * S * 2 + 3) & ~(size_t)3);
}

// cudaFuncSetAttribute(MaxDynamicSharedMemorySize) once per kernel and device (the attribute
// persists; repeating it costs host time on every launch).  Keyed by the kernel itself.
template <auto Kern>
cudaError_t set_smem_once(int bytes) {
  static std::atomic<uint64_t> done{0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = dev < 64 ? (uint64_t)1 << dev : 0;
  if (bit != 0 && (done.load(std::memory_order_acquire) & bit)) return cudaSuccess;
  e = cudaFuncSetAttribute(Kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess && bit != 0) done.fetch_or(bit, std::memory_order_acq_rel);
  return e;
}

// True when the merge kernel copies the kept rows itself (bucket routing, no repositioning),
// so the separate copy kernel is not launched.
bool merge_copies_kept_rows(const CompressArgs& a);

// SELKV_ERR_CUDA, with `e` kept for selkv_last_cuda_error on this thread.
selkv_status cuda_fail(cudaError_t e);

#ifndef SELKV_DEC_UNITS_MAX_ROWS
#define SELKV_DEC_UNITS_MAX_ROWS 2112  // persistent unit-walking decode: most rows of a unit
#endif
// Splits per (b, kv) of a decode launch; unit_walk: the tensor-core decode, which walks many
// short one-split units with persistent CTAs.
int decode_splits(int B, int Hkv, int m_cap, int num_sms, bool unit_walk);
cudaError_t launch_decode(const DecodeArgs& a, cudaStream_t s);     // dispatch by dtype
cudaError_t launch_decode_tc(const DecodeArgs& a, cudaStream_t s);  // bf16: TMA + tensor cores

}  // namespace selkv
