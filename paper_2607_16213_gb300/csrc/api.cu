// C-ABI entry points of the SelKV library: argument validation, workspace planning and
// kernel launches.  Host code only; every step of the method runs in the kernels.
#include <atomic>
#include <cmath>
#include <cstring>
#include <mutex>

#include "selkv_internal.cuh"

namespace selkv {
cudaError_t launch_setup(const CompressArgs& a, const SeqTable& tab, const SelectWs& w, cudaStream_t s);
cudaError_t launch_vnorm(const CompressArgs& a, cudaStream_t s);
cudaError_t launch_merge(const CompressArgs& a, cudaStream_t s);

namespace {

// Kernels enqueued by each call (diagnostic count, see selkv_kernel_launches).
std::atomic<uint64_t> g_launches{0};
constexpr int kDecodeKernels = 1;

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

bool shape_ok(const selkv_shape* s) {
  if (s == nullptr) return false;
  if (s->dtype != SELKV_BF16 && s->dtype != SELKV_FP32) return false;
  if (s->batch < 1 || s->batch > SELKV_MAX_BATCH) return false;
  if (s->num_kv_heads < 1 || s->num_kv_heads > 32 || s->num_q_heads < 1) return false;
  if (s->num_q_heads % s->num_kv_heads != 0) return false;
  if (s->num_q_heads / s->num_kv_heads > 16) return false;
  if (s->head_dim < 1 || s->n_cap < 0 || s->m_cap < 0 || s->obs_window < 0) return false;
  return true;
}

size_t round256(size_t x) { return (x + 255) & ~size_t(255); }

// A side stream per device: the value-norm pass (HBM-bound) runs on it next to the scoring
// passes (bound by the exponentials), forked from and joined back to the caller's stream with
// events, a pattern that also records into a CUDA graph.  Created on first use outside a
// capture; if it cannot be had, the pass runs on the caller's stream.
struct SideStream {
  cudaStream_t s = nullptr;
  cudaEvent_t fork = nullptr, join = nullptr;
  bool ready = false, failed = false;
};
constexpr int kMaxDevices = 64;
std::mutex g_side_mu;
SideStream g_side[kMaxDevices];

// Requires g_side_mu.
SideStream* side_stream(cudaStream_t caller) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  SideStream& x = g_side[dev];
  if (!x.ready && !x.failed) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(caller, &cs) != cudaSuccess || cs != cudaStreamCaptureStatusNone) return nullptr;
    x.ready = cudaStreamCreateWithFlags(&x.s, cudaStreamNonBlocking) == cudaSuccess &&
              cudaEventCreateWithFlags(&x.fork, cudaEventDisableTiming) == cudaSuccess &&
              cudaEventCreateWithFlags(&x.join, cudaEventDisableTiming) == cudaSuccess;
    x.failed = !x.ready;
  }
  return x.ready ? &x : nullptr;
}

// Key slices of the scoring's first pass (one row-statistics partial per slice and row).
int score_chunks(const selkv_shape& s, int R) {
  return score_uses_tc(s.dtype, s.head_dim, R) ? score_tc_splits(s.batch, s.num_kv_heads, s.n_cap, R, kPlanSMs)
                                               : (int)(((size_t)s.n_cap + kRowChunk - 1) / kRowChunk);
}

struct CompressPlan {
  size_t seq_n, seq_m, rowpart, rowstat, attn, vnorm, rope_tab, mcount, score, kflag, slot, kept_pos, tau, atau, ratio, select, total;
  size_t ev_pos, cos_invn, cos_rank, cos_order, cos_cnt, cos_seg;
  int nchunks, R;
};

CompressPlan plan_compress(const selkv_shape& s) {
  CompressPlan p{};
  size_t off = sizeof(WsHeader);
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += round256(bytes);
    return o;
  };
  const size_t B = s.batch, Hkv = s.num_kv_heads, n = s.n_cap;
  p.R = (s.num_q_heads / s.num_kv_heads) * s.obs_window;
  p.nchunks = score_chunks(s, p.R);
  p.seq_n = take(B * 4);
  p.seq_m = take(B * 4);
  p.rowpart = take(B * Hkv * (size_t)p.nchunks * p.R * sizeof(float2));
  p.rowstat = take(B * Hkv * (size_t)p.R * sizeof(float2));
  p.attn = take(B * Hkv * n * 4);
  p.vnorm = take(B * Hkv * n * 4);
  p.score = take(B * Hkv * n * 4);
  // kept flags, slot maps: per sequence, or per KV head in the per-head mode (sized for that)
  p.kflag = take(B * Hkv * n);
  p.slot = take(B * Hkv * n * 4);
  p.kept_pos = take(B * Hkv * (size_t)s.m_cap * 4);
  // merge targets per bucket, sized for the smallest bucket (the size is a call parameter)
  p.tau = take(B * Hkv * n * 4);
  p.atau = take(B * Hkv * n * 4);
  p.ratio = take(B * Hkv * (size_t)s.m_cap * 4);
  p.mcount = take(B * Hkv * (size_t)s.m_cap * 4);
  // RoPE repositioning tables (used only with params->rope): coarse and fine (cos, sin)
  p.rope_tab = take((size_t)(s.head_dim / 2) * (rope_coarse(s.n_cap) + 256) * 8);
  // full cosine routing (used only with params->routing == COSINE; its target slots and gates
  // live in tau / atau)
  const size_t mpad = ((size_t)s.m_cap + 255) / 256 * 256;
  p.ev_pos = take(B * Hkv * n * 4);
  p.cos_invn = take(B * Hkv * mpad * 4);
  p.cos_rank = take(B * Hkv * n * 4);
  p.cos_order = take(B * Hkv * n * 4);
  p.cos_cnt = take(B * Hkv * (size_t)cos_chunks_for(s.n_cap) * s.m_cap * 4);
  p.cos_seg = take(B * Hkv * (size_t)s.m_cap * 8);
  p.select = take(select_ws_bytes(s.batch, s.num_kv_heads, s.n_cap));
  p.total = off;
  return p;
}

struct ScorePlan {
  size_t seq_n, seq_m, rowpart, rowstat, total;
  int nchunks, R;
};

ScorePlan plan_score(const selkv_shape& s) {
  ScorePlan p{};
  size_t off = sizeof(WsHeader);
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += round256(bytes);
    return o;
  };
  const size_t B = s.batch, Hkv = s.num_kv_heads;
  p.R = (s.num_q_heads / s.num_kv_heads) * s.obs_window;
  p.nchunks = score_chunks(s, p.R);
  p.seq_n = take(B * 4);
  p.seq_m = take(B * 4);
  p.rowpart = take(B * Hkv * (size_t)p.nchunks * p.R * sizeof(float2));
  p.rowstat = take(B * Hkv * (size_t)p.R * sizeof(float2));
  p.total = off;
  return p;
}

struct DecodePlan {
  size_t cnt_head, cnt_seq, partial, total;
  int splits;
};

DecodePlan plan_decode(const selkv_shape& s) {
  DecodePlan p{};
  size_t off = sizeof(WsHeader);
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += round256(bytes);
    return o;
  };
  p.splits = decode_splits(s.batch, s.num_kv_heads, s.m_cap, kPlanSMs, s.dtype == SELKV_BF16);
  p.cnt_head = take((size_t)s.batch * s.num_kv_heads * 4);
  p.cnt_seq = take((size_t)s.batch * 4);
  p.partial = take((size_t)s.batch * s.num_kv_heads *
                   decode_record_floats(s.num_q_heads / s.num_kv_heads, p.splits, s.head_dim) * 4);
  p.total = off;
  return p;
}

template <typename T>
T* at(void* ws, size_t off) {
  return reinterpret_cast<T*>(static_cast<char*>(ws) + off);
}

}  // namespace

void note_launches(int kernels) { g_launches += (uint64_t)kernels; }

// Kernels one selkv_compress call enqueues, mirroring the launch code: set-up and value norms;
// the scoring's two passes and the fold of the row statistics between them; the selection
// (pooling with digit pass 0 and digit passes 1-2 of each KV head's top-k, then, in the
// shared mode only, the union with the trim's pass 0 and its passes 1-2; finally the
// compaction's count and write); the RoPE tables when repositioning;
// the routing and merge (bucket: route and merge, plus the kept-row copy unless the merge
// does it; cosine: the copy and the cosine kernels); the bias.
int compress_kernel_count(const CompressArgs& a) {
  int k = 2 + 3;
  k += a.per_head ? 5 : 8;
  if (a.rope != SELKV_ROPE_OFF) k += 1;
  if (a.routing == SELKV_ROUTE_COSINE)
    k += 1 + (a.m_cap > 0 ? cosine_kernels(a.dtype, a.D) : 0);
  else
    k += 2 + (merge_copies_kept_rows(a) ? 0 : 1);
  return k + 1;
}

}  // namespace selkv

namespace selkv {
namespace {
thread_local cudaError_t g_last_cuda = cudaSuccess;
}  // namespace
selkv_status cuda_fail(cudaError_t e) {
  g_last_cuda = e;
  return SELKV_ERR_CUDA;
}
}  // namespace selkv

using namespace selkv;

extern "C" {

const char* selkv_status_string(selkv_status status) {
  switch (status) {
    case SELKV_OK: return "ok";
    case SELKV_ERR_INVALID_ARG: return "invalid argument";
    case SELKV_ERR_UNSUPPORTED: return "unsupported configuration";
    case SELKV_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
    case SELKV_ERR_CUDA: return "CUDA error";
    case SELKV_ERR_DEVICE: return "device reported an error";
  }
  return "unknown status";
}

int selkv_last_cuda_error(const char** name) {
  const cudaError_t e = g_last_cuda;
  if (name != nullptr) *name = cudaGetErrorName(e);
  return (int)e;
}

uint64_t selkv_kernel_launches(void) { return g_launches.load(); }

selkv_status selkv_workspace_init(void* workspace, size_t workspace_bytes, selkv_stream_t stream) {
  if (workspace == nullptr || !aligned(workspace, 256) || workspace_bytes < sizeof(WsHeader))
    return SELKV_ERR_WORKSPACE;
  const cudaError_t e = cudaMemsetAsync(workspace, 0, workspace_bytes, reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e);
  return SELKV_OK;
}

selkv_status selkv_workspace_error(void* workspace, selkv_stream_t stream, uint32_t* flags) {
  if (workspace == nullptr || flags == nullptr) return SELKV_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  uint32_t f = 0;
  if (const cudaError_t e = cudaMemcpyAsync(&f, workspace, sizeof(f), cudaMemcpyDeviceToHost, st); e != cudaSuccess)
    return cuda_fail(e);
  if (const cudaError_t e = cudaStreamSynchronize(st); e != cudaSuccess) return cuda_fail(e);
  *flags = f;
  if (f != 0) {
    if (const cudaError_t e = cudaMemsetAsync(workspace, 0, sizeof(uint32_t), st); e != cudaSuccess) return cuda_fail(e);
    if (const cudaError_t e = cudaStreamSynchronize(st); e != cudaSuccess) return cuda_fail(e);
    return SELKV_ERR_DEVICE;
  }
  return SELKV_OK;
}

size_t selkv_compress_workspace_size(const selkv_shape* shape) {
  if (!shape_ok(shape)) return 0;
  return plan_compress(*shape).total;
}

selkv_status selkv_compress(const selkv_shape* shape, const int32_t* n_len, double rho,
                            const selkv_params* params, const void* K, const void* V,
                            const void* Q_obs, void* K_c, void* V_c, float* bias,
                            int32_t* lengths, const selkv_compress_debug* debug,
                            void* workspace, size_t workspace_bytes, selkv_stream_t stream) {
  if (!shape_ok(shape) || params == nullptr || n_len == nullptr) return SELKV_ERR_INVALID_ARG;
  const selkv_shape& s = *shape;
  if (s.head_dim != 64 && s.head_dim != 128) return SELKV_ERR_UNSUPPORTED;
  if (s.obs_window < 1 || s.n_cap < 1) return SELKV_ERR_INVALID_ARG;
  const selkv_params& p = *params;
  if (!std::isfinite(p.alpha) || p.pool_kernel < 1 || (p.pool_kernel & 1) == 0 || p.recent < 0 ||
      p.bucket < 1 || p.gate_mode < 0 || p.gate_mode > 2 || p.empty_bucket < 0 || p.empty_bucket > 1 ||
      p.select_mode < 0 || p.select_mode > 1 || p.rope < 0 || p.rope > 2 || p.bias_mode < 0 || p.bias_mode > 1 ||
      p.routing < 0 || p.routing > 1 ||
      (p.rope != 0 && !(std::isfinite(p.rope_theta) && p.rope_theta > 0.f)))
    return SELKV_ERR_INVALID_ARG;
  if (p.bucket > 32) return SELKV_ERR_UNSUPPORTED;
  if (!(rho > 0.0 && rho <= 1.0)) return SELKV_ERR_INVALID_ARG;
  const void* tensors[] = {K, V, Q_obs, K_c, V_c, bias, lengths};
  for (const void* t : tensors)
    if (t == nullptr || !aligned(t, 16)) return SELKV_ERR_INVALID_ARG;
  if (debug != nullptr) {
    const void* dbg[] = {debug->attn, debug->score, debug->topk, debug->kept_idx,
                         debug->target, debug->gate, debug->decision, debug->ratio};
    for (const void* t : dbg)
      if (t != nullptr && !aligned(t, 16)) return SELKV_ERR_INVALID_ARG;
  }
  static thread_local SeqTable tab;
  for (int b = 0; b < s.batch; ++b) {
    const int n = n_len[b];
    if (n < s.obs_window || n > s.n_cap) return SELKV_ERR_INVALID_ARG;
    const double mm = std::floor(rho * (double)n);
    const int m = (int)mm;
    if (m - p.recent < 0 || m > s.m_cap || m > n) return SELKV_ERR_INVALID_ARG;
    tab.n[b] = n;
    tab.m[b] = m;
  }
  const CompressPlan plan = plan_compress(s);
  if (workspace == nullptr || !aligned(workspace, 256)) return SELKV_ERR_WORKSPACE;
  if (workspace_bytes < plan.total) return SELKV_ERR_WORKSPACE;

  CompressArgs a{};
  a.dtype = s.dtype;
  a.B = s.batch;
  a.Hq = s.num_q_heads;
  a.Hkv = s.num_kv_heads;
  a.G = s.num_q_heads / s.num_kv_heads;
  a.D = s.head_dim;
  a.W = s.obs_window;
  a.n_cap = s.n_cap;
  a.m_cap = s.m_cap;
  a.R = plan.R;
  a.nchunks = plan.nchunks;
  a.alpha = p.alpha;
  a.pool_kernel = p.pool_kernel;
  a.bucket = p.bucket;
  a.recent = p.recent;
  a.gate_mode = p.gate_mode;
  a.empty_bucket = p.empty_bucket;
  a.per_head = p.select_mode == SELKV_SELECT_PER_HEAD ? 1 : 0;
  a.rope = p.rope;
  a.bias_count = p.bias_mode == SELKV_BIAS_COUNT ? 1 : 0;
  a.rope_theta = p.rope_theta;
  a.rope_hi = rope_coarse(s.n_cap);
  a.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)s.head_dim));
  a.K = K;
  a.V = V;
  a.Q = Q_obs;
  a.Kc = K_c;
  a.Vc = V_c;
  a.bias = bias;
  a.lengths = lengths;
  a.flags = at<uint32_t>(workspace, 0);
  a.seq_n = at<int32_t>(workspace, plan.seq_n);
  a.seq_m = at<int32_t>(workspace, plan.seq_m);
  a.rowpart = at<float2>(workspace, plan.rowpart);
  a.rowstat = at<float2>(workspace, plan.rowstat);
  a.attn = (debug && debug->attn) ? debug->attn : at<float>(workspace, plan.attn);
  a.vnorm = at<float>(workspace, plan.vnorm);
  a.score = (debug && debug->score) ? debug->score : at<float>(workspace, plan.score);
  a.kflag = at<uint8_t>(workspace, plan.kflag);
  a.slot_of = at<int32_t>(workspace, plan.slot);
  a.kept_pos = at<int32_t>(workspace, plan.kept_pos);
  a.nbk = (s.n_cap + p.bucket - 1) / p.bucket;
  a.tau = at<int32_t>(workspace, plan.tau);
  a.atau = at<float>(workspace, plan.atau);
  a.ratio = at<float>(workspace, plan.ratio);
  a.mcount = at<float>(workspace, plan.mcount);
  a.rope_tab = at<float2>(workspace, plan.rope_tab);
  a.routing = p.routing;
  a.cos_chunks = cos_chunks_for(s.n_cap);
  a.cos_chunk = cos_chunk_len(s.n_cap);
  a.cos_mpad = (s.m_cap + 255) / 256 * 256;
  a.cos_tslot = a.tau;
  a.cos_g = a.atau;
  a.ev_pos = at<int32_t>(workspace, plan.ev_pos);
  a.cos_invn = at<float>(workspace, plan.cos_invn);
  a.cos_rank = at<int32_t>(workspace, plan.cos_rank);
  a.cos_order = at<int32_t>(workspace, plan.cos_order);
  a.cos_cnt = at<int32_t>(workspace, plan.cos_cnt);
  a.cos_seg = at<int2>(workspace, plan.cos_seg);
  if (debug != nullptr) {
    a.dbg_topk = debug->topk;
    a.dbg_kept_idx = debug->kept_idx;
    a.dbg_target = debug->target;
    a.dbg_gate = debug->gate;
    a.dbg_decision = debug->decision;
    a.dbg_ratio = debug->ratio;
  }
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const SelectWs sw = carve_select_ws(at<char>(workspace, plan.select), s.batch, s.num_kv_heads, s.n_cap);
  cudaError_t e = launch_setup(a, tab, sw, st);
  {
    // value norms on the side stream (they need seq_n from the set-up; selection needs them)
    std::lock_guard<std::mutex> lock(g_side_mu);
    SideStream* side = e == cudaSuccess ? side_stream(st) : nullptr;
    if (side != nullptr) {
      e = cudaEventRecord(side->fork, st);
      if (e == cudaSuccess) e = cudaStreamWaitEvent(side->s, side->fork, 0);
      if (e == cudaSuccess) e = launch_vnorm(a, side->s);
      if (e == cudaSuccess) e = cudaEventRecord(side->join, side->s);
    }
    if (e == cudaSuccess) e = score_uses_tc(a.dtype, a.D, a.R) ? launch_score_tc(a, st) : launch_score_simt(a, st);
    if (e == cudaSuccess) e = side != nullptr ? cudaStreamWaitEvent(st, side->join, 0) : launch_vnorm(a, st);
  }
  if (e == cudaSuccess)
    e = launch_select_grid(a, sw, st);
  if (e == cudaSuccess) e = launch_merge(a, st);
  g_launches += (uint64_t)compress_kernel_count(a);
  return e == cudaSuccess ? SELKV_OK : cuda_fail(e);
}

size_t selkv_score_workspace_size(const selkv_shape* shape) {
  if (!shape_ok(shape)) return 0;
  return plan_score(*shape).total;
}

selkv_status selkv_score(const selkv_shape* shape, const int32_t* n_len, const void* K, const void* Q_obs,
                         float* attn, int32_t passes, void* workspace, size_t workspace_bytes,
                         selkv_stream_t stream) {
  if (!shape_ok(shape) || n_len == nullptr) return SELKV_ERR_INVALID_ARG;
  const selkv_shape& s = *shape;
  if (s.head_dim != 64 && s.head_dim != 128) return SELKV_ERR_UNSUPPORTED;
  if (s.obs_window < 1 || s.n_cap < 1) return SELKV_ERR_INVALID_ARG;
  if (passes != SELKV_SCORE_ROWSTATS && passes != SELKV_SCORE_COLSUMS && passes != SELKV_SCORE_ALL)
    return SELKV_ERR_INVALID_ARG;
  if (K == nullptr || Q_obs == nullptr || !aligned(K, 16) || !aligned(Q_obs, 16)) return SELKV_ERR_INVALID_ARG;
  if ((passes & SELKV_SCORE_COLSUMS) && (attn == nullptr || !aligned(attn, 16))) return SELKV_ERR_INVALID_ARG;
  static thread_local SeqTable tab;
  for (int b = 0; b < s.batch; ++b) {
    const int n = n_len[b];
    if (n < s.obs_window || n > s.n_cap) return SELKV_ERR_INVALID_ARG;
    tab.n[b] = n;
    tab.m[b] = 0;
  }
  const ScorePlan plan = plan_score(s);
  if (workspace == nullptr || !aligned(workspace, 256)) return SELKV_ERR_WORKSPACE;
  if (workspace_bytes < plan.total) return SELKV_ERR_WORKSPACE;
  CompressArgs a{};
  a.dtype = s.dtype;
  a.B = s.batch;
  a.Hq = s.num_q_heads;
  a.Hkv = s.num_kv_heads;
  a.G = s.num_q_heads / s.num_kv_heads;
  a.D = s.head_dim;
  a.W = s.obs_window;
  a.n_cap = s.n_cap;
  a.m_cap = s.m_cap;
  a.R = plan.R;
  a.nchunks = plan.nchunks;
  a.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)s.head_dim));
  a.K = K;
  a.Q = Q_obs;
  a.attn = attn;
  a.flags = at<uint32_t>(workspace, 0);
  a.seq_n = at<int32_t>(workspace, plan.seq_n);
  a.seq_m = at<int32_t>(workspace, plan.seq_m);
  a.rowpart = at<float2>(workspace, plan.rowpart);
  a.rowstat = at<float2>(workspace, plan.rowstat);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = cudaSuccess;
  int kernels = 0;
  if (passes & SELKV_SCORE_ROWSTATS) {  // the column-sum pass reuses the table of its row-statistics call
    e = launch_seq_setup(a, tab, st);
    kernels += 3;
  }
  if (passes & SELKV_SCORE_COLSUMS) kernels += 1;
  if (e == cudaSuccess)
    e = score_uses_tc(a.dtype, a.D, a.R) ? launch_score_tc(a, st, passes) : launch_score_simt(a, st, passes);
  g_launches += (uint64_t)kernels;
  return e == cudaSuccess ? SELKV_OK : cuda_fail(e);
}

size_t selkv_layer_average_workspace_size(const selkv_shape* shape) {
  if (!shape_ok(shape)) return 0;
  return sizeof(WsHeader) + round256((size_t)shape->batch * shape->num_kv_heads * shape->n_cap * sizeof(float));
}

selkv_status selkv_layer_average_bias(const selkv_shape* shape, const selkv_params* params, int32_t num_layers,
                                      const int32_t* const* kept_idx, float* const* bias,
                                      const int32_t* lengths, void* workspace, size_t workspace_bytes,
                                      selkv_stream_t stream) {
  if (!shape_ok(shape) || params == nullptr || kept_idx == nullptr || bias == nullptr || lengths == nullptr)
    return SELKV_ERR_INVALID_ARG;
  if (num_layers < 1 || num_layers > kMaxLayers) return SELKV_ERR_INVALID_ARG;
  const selkv_params& p = *params;
  if (!std::isfinite(p.alpha) || p.select_mode < 0 || p.select_mode > 1 || p.bias_mode < 0 || p.bias_mode > 1)
    return SELKV_ERR_INVALID_ARG;
  if (!aligned(lengths, 4)) return SELKV_ERR_INVALID_ARG;
  LayerPtrs P{};
  for (int l = 0; l < num_layers; ++l) {
    if (kept_idx[l] == nullptr || bias[l] == nullptr || !aligned(kept_idx[l], 16) || !aligned(bias[l], 16))
      return SELKV_ERR_INVALID_ARG;
    P.kept[l] = kept_idx[l];
    P.bias[l] = bias[l];
  }
  const selkv_shape& s = *shape;
  if (workspace == nullptr || !aligned(workspace, 256)) return SELKV_ERR_WORKSPACE;
  if (workspace_bytes < selkv_layer_average_workspace_size(shape)) return SELKV_ERR_WORKSPACE;
  if (p.alpha == 0.f || s.m_cap < 1) return SELKV_OK;  // every bias is 0 and stays 0
  LayerAvgArgs a{};
  a.B = s.batch;
  a.Hkv = s.num_kv_heads;
  a.m_cap = s.m_cap;
  a.n_cap = s.n_cap;
  a.per_head = p.select_mode == SELKV_SELECT_PER_HEAD ? 1 : 0;
  a.L = num_layers;
  a.alpha = p.alpha;
  a.lengths = lengths;
  a.flags = at<uint32_t>(workspace, 0);
  a.acc = at<float>(workspace, sizeof(WsHeader));
  const cudaError_t e = launch_layer_average(a, P, reinterpret_cast<cudaStream_t>(stream));
  g_launches += (uint64_t)num_layers + 1;
  return e == cudaSuccess ? SELKV_OK : cuda_fail(e);
}

size_t selkv_decode_workspace_size(const selkv_shape* shape) {
  if (!shape_ok(shape)) return 0;
  return plan_decode(*shape).total;
}

selkv_status selkv_decode_attn(const selkv_shape* shape, const void* q, void* K_c, void* V_c,
                               float* bias, int32_t* lengths, const void* k_new,
                               const void* v_new, void* out, void* workspace,
                               size_t workspace_bytes, selkv_stream_t stream) {
  if (!shape_ok(shape)) return SELKV_ERR_INVALID_ARG;
  const selkv_shape& s = *shape;
  if (s.head_dim != 64 && s.head_dim != 128) return SELKV_ERR_UNSUPPORTED;
  if (s.m_cap < 1) return SELKV_ERR_INVALID_ARG;
  const void* tensors[] = {q, K_c, V_c, lengths, out};
  for (const void* t : tensors)
    if (t == nullptr || !aligned(t, 16)) return SELKV_ERR_INVALID_ARG;
  if ((k_new == nullptr) != (v_new == nullptr)) return SELKV_ERR_INVALID_ARG;
  if (k_new != nullptr && (!aligned(k_new, 16) || !aligned(v_new, 16))) return SELKV_ERR_INVALID_ARG;
  if (bias != nullptr && !aligned(bias, 16)) return SELKV_ERR_INVALID_ARG;
  const DecodePlan plan = plan_decode(s);
  if (workspace == nullptr || !aligned(workspace, 256)) return SELKV_ERR_WORKSPACE;
  if (workspace_bytes < plan.total) return SELKV_ERR_WORKSPACE;
  DecodeArgs a{};
  a.dtype = s.dtype;
  a.B = s.batch;
  a.Hq = s.num_q_heads;
  a.Hkv = s.num_kv_heads;
  a.G = s.num_q_heads / s.num_kv_heads;
  a.D = s.head_dim;
  a.m_cap = s.m_cap;
  a.splits = plan.splits;
  a.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)s.head_dim));
  a.q = q;
  a.Kc = K_c;
  a.Vc = V_c;
  a.bias = bias;
  a.lengths = lengths;
  a.k_new = k_new;
  a.v_new = v_new;
  a.out = out;
  a.flags = at<uint32_t>(workspace, 0);
  a.cnt_head = at<uint32_t>(workspace, plan.cnt_head);
  a.cnt_seq = at<uint32_t>(workspace, plan.cnt_seq);
  a.partial = at<float>(workspace, plan.partial);
  const cudaError_t e = launch_decode(a, reinterpret_cast<cudaStream_t>(stream));
  g_launches += kDecodeKernels;
  return e == cudaSuccess ? SELKV_OK : cuda_fail(e);
}

}  // extern "C"
