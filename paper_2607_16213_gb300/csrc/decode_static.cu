// selkv_decode_attn_static: the compensated decode of selkv_decode_attn for callers that
// cannot allocate device memory.
//
// Who needs it: code that runs inside a host framework which owns every device buffer and
// hands a kernel only its inputs and outputs (no allocator, no workspace), and latency-bound
// serving loops where a cudaMalloc / cudaFree (cudaFree synchronises the device) in the
// step is not acceptable and no workspace has been planned for this call.  For them the
// decode scratch (split partials and arrival counters) lives in one file-scope device array
// of a fixed size, reserved on every GPU that loads the library for as long as the process
// lives.
//
// Rules of the shared array (see include/selkv.h):
//   * It holds SELKV_STATIC_SCRATCH_BYTES; shapes that need more are rejected before launch.
//   * Every call reuses it and it keeps the previous call's contents; the counters that must
//     start at zero are cleared by each call before its kernel runs.
//   * Calls that overlap on the GPU (other streams, other host threads) race on it.
//   * Its device address is looked up on the first call made with a device current, and
//     again whenever that device's current context has changed since (after cudaDeviceReset
//     the module is loaded anew, at a new address); make the first call on a device, and the
//     first call after a reset, before any stream capture begins.
#include <cmath>
#include <mutex>

#include <cudaTypedefs.h>

#include "selkv_internal.cuh"

namespace selkv {
void note_launches(int kernels);
}

namespace {

static __device__ __align__(256) unsigned char g_decode_scratch[SELKV_STATIC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;

std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices] = {};
CUcontext g_scratch_ctx[kMaxDevices] = {};

// cuCtxGetCurrent through the runtime's driver entry point (the library does not link libcuda).
PFN_cuCtxGetCurrent_v4000 ctx_fn() {
  static PFN_cuCtxGetCurrent_v4000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(p);
  });
  return fn;
}

// Device address of g_decode_scratch on the current device: looked up on the device's first
// call and again when the thread's current context is not the one the address was taken in.
// (If the context cannot be queried, the first address is kept.)
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  auto get_ctx = ctx_fn();
  CUcontext ctx = nullptr;
  if (get_ctx != nullptr && get_ctx(&ctx) != CUDA_SUCCESS) ctx = nullptr;
  std::lock_guard<std::mutex> lock(g_mu);
  const bool known = g_scratch_ptr[dev] != nullptr && (get_ctx == nullptr || (ctx != nullptr && ctx == g_scratch_ctx[dev]));
  if (!known) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_decode_scratch);  // also makes the device's context current
    if (e != cudaSuccess) return e;
    if (get_ctx != nullptr && get_ctx(&ctx) != CUDA_SUCCESS) ctx = nullptr;
    g_scratch_ptr[dev] = p;
    g_scratch_ctx[dev] = ctx;
  }
  *out = g_scratch_ptr[dev];
  return cudaSuccess;
}

size_t round256(size_t x) { return (x + 255) & ~size_t(255); }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" SELKV_API selkv_status selkv_decode_attn_static(
    const selkv_shape* shape, const void* q, void* K_c, void* V_c, float* bias,
    int32_t* lengths, const void* k_new, const void* v_new, void* out, uint32_t* flags_out,
    selkv_stream_t stream) {
  using namespace selkv;
  if (shape == nullptr) return SELKV_ERR_INVALID_ARG;
  const selkv_shape& s = *shape;
  if (s.dtype != SELKV_BF16 && s.dtype != SELKV_FP32) return SELKV_ERR_INVALID_ARG;
  if (s.batch < 1 || s.batch > SELKV_MAX_BATCH || s.num_kv_heads < 1 || s.num_kv_heads > 32 ||
      s.num_q_heads < 1 || s.num_q_heads % s.num_kv_heads != 0 ||
      s.num_q_heads / s.num_kv_heads > 16 || s.m_cap < 1)
    return SELKV_ERR_INVALID_ARG;
  if (s.head_dim != 64 && s.head_dim != 128) return SELKV_ERR_UNSUPPORTED;
  const void* tensors[] = {q, K_c, V_c, lengths, out};
  for (const void* t : tensors)
    if (t == nullptr || !aligned16(t)) return SELKV_ERR_INVALID_ARG;
  if ((k_new == nullptr) != (v_new == nullptr)) return SELKV_ERR_INVALID_ARG;
  if (k_new != nullptr && (!aligned16(k_new) || !aligned16(v_new))) return SELKV_ERR_INVALID_ARG;
  if (bias != nullptr && !aligned16(bias)) return SELKV_ERR_INVALID_ARG;
  if (flags_out != nullptr && (reinterpret_cast<uintptr_t>(flags_out) & 3u) != 0) return SELKV_ERR_INVALID_ARG;

  // Scratch layout: error word | per-(b, kv) counters | per-b counters | split partials.
  const int splits = decode_splits(s.batch, s.num_kv_heads, s.m_cap, kPlanSMs, s.dtype == SELKV_BF16);
  const size_t off_head = 256;
  const size_t off_seq = off_head + round256((size_t)s.batch * s.num_kv_heads * 4);
  const size_t off_part = off_seq + round256((size_t)s.batch * 4);
  const size_t need = off_part + (size_t)s.batch * s.num_kv_heads *
                                     decode_record_floats(s.num_q_heads / s.num_kv_heads, splits, s.head_dim) * 4;
  if (need > (size_t)SELKV_STATIC_SCRATCH_BYTES) return SELKV_ERR_WORKSPACE;

  void* base = nullptr;
  if (const cudaError_t e = scratch_address(&base); e != cudaSuccess) return cuda_fail(e);
  char* sb = static_cast<char*>(base);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  // the counters must start at zero; the error word is cleared with them
  if (const cudaError_t e = cudaMemsetAsync(sb, 0, off_part, st); e != cudaSuccess) return cuda_fail(e);

  DecodeArgs a{};
  a.dtype = s.dtype;
  a.B = s.batch;
  a.Hq = s.num_q_heads;
  a.Hkv = s.num_kv_heads;
  a.G = s.num_q_heads / s.num_kv_heads;
  a.D = s.head_dim;
  a.m_cap = s.m_cap;
  a.splits = splits;
  a.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)s.head_dim));
  a.q = q;
  a.Kc = K_c;
  a.Vc = V_c;
  a.bias = bias;
  a.lengths = lengths;
  a.k_new = k_new;
  a.v_new = v_new;
  a.out = out;
  a.flags = flags_out != nullptr ? flags_out : reinterpret_cast<uint32_t*>(sb);
  a.cnt_head = reinterpret_cast<uint32_t*>(sb + off_head);
  a.cnt_seq = reinterpret_cast<uint32_t*>(sb + off_seq);
  a.partial = reinterpret_cast<float*>(sb + off_part);
  const cudaError_t e = launch_decode(a, st);
  note_launches(1);
  return e == cudaSuccess ? SELKV_OK : cuda_fail(e);
}
