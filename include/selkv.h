/*
 * selkv.h - C ABI of the SelKV GB300 library (sm_103a).
 *
 * SelKV compresses a prefilled KV cache once (score -> select -> route -> gate -> merge ->
 * attention ratio) and then decodes over the compressed cache with the attention-ratio
 * compensation added to the logits (arxiv 2607.16213, Algorithm 1).  Two calls carry the
 * whole path:
 *
 *   selkv_compress(K, V, Q_obs, budget, params) -> (K_c, V_c, bias, lengths)
 *   selkv_decode_attn(q, K_c, V_c, bias, lengths) -> out
 *
 * Conventions shared by every entry point
 *   - All tensors are caller-owned DEVICE memory, dense, row-major, in the layouts given
 *     below; every base pointer is 16-byte aligned.  The library never allocates: scratch
 *     space is a caller-provided workspace whose size comes from the *_workspace_size call.
 *   - Work is enqueued asynchronously on `stream`; no call synchronises the stream except
 *     selkv_workspace_error.  Host-side argument checks happen before any launch: a call
 *     that returns anything but SELKV_OK has enqueued nothing (SELKV_ERR_CUDA excepted: a
 *     launch failed).
 *   - Conditions only the device can see (a length beyond capacity, a timed-out wait) set
 *     bits in the workspace's error word (SELKV_DEVERR_*); the kernels never trap.  Read and
 *     clear them with selkv_workspace_error.
 *   - A workspace must be zeroed once before its first use (selkv_workspace_init).  Calls
 *     that share a workspace must not overlap on the GPU; calls with workspaces of their own
 *     may run concurrently on different streams (for instance the compressions of a model's
 *     layers after prefill).
 *   - Element types: dtype SELKV_BF16 (storage bf16, fp32 arithmetic) or SELKV_FP32.
 *   - Shapes: B sequences, Hq query heads, Hkv KV heads (Hkv divides Hq, G = Hq / Hkv; query
 *     head h reads KV head h / G), head dimension d in {64, 128}, observation window W.
 */
#ifndef SELKV_H
#define SELKV_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define SELKV_API __attribute__((visibility("default")))
#else
#define SELKV_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* A CUDA stream (the same handle as cudaStream_t); NULL is the legacy default stream. */
typedef struct CUstream_st* selkv_stream_t;

typedef enum selkv_status {
  SELKV_OK = 0,
  SELKV_ERR_INVALID_ARG = 1, /* a pointer, size, shape or budget violates the contract */
  SELKV_ERR_UNSUPPORTED = 2, /* a valid request the library does not implement        */
  SELKV_ERR_WORKSPACE = 3,   /* workspace NULL, misaligned or smaller than required    */
  SELKV_ERR_CUDA = 4,        /* a CUDA runtime call or launch failed                   */
  SELKV_ERR_DEVICE = 5       /* selkv_workspace_error found device error bits          */
} selkv_status;

typedef enum selkv_dtype { SELKV_BF16 = 0, SELKV_FP32 = 1 } selkv_dtype;

/* Eq. 4 gate: COSINE is the method (g = clamp(cos(v_j, v_pi(j)), 0, 1)); OPEN (g = 1) and
 * CLOSED (g = 0) are the paper's ablation end points "merge all" and "eviction only". */
typedef enum selkv_gate_mode {
  SELKV_GATE_COSINE = 0,
  SELKV_GATE_OPEN = 1,
  SELKV_GATE_CLOSED = 2
} selkv_gate_mode;

/* Evicted tokens whose bucket holds no kept token (Eq. 3 leaves this open): EXPAND looks at
 * buckets b-r and b+r for r = 1, 2, ... and takes the first ring with a kept token; DROP
 * gives them g = 0 and no target. */
typedef enum selkv_empty_bucket { SELKV_EMPTY_EXPAND = 0, SELKV_EMPTY_DROP = 1 } selkv_empty_bucket;

/* Token selection (Sec. 3.3): SHARED is the union selection of GQA models (every KV head keeps
 * the same set: each KV head's top-m_s, union, trim by the mean score); PER_HEAD is the
 * per-head selection of MHA models (each KV head keeps its own top-m_s, and its bias is
 * alpha * ln R of its own entries, without averaging across heads, Sec. 3.6). */
typedef enum selkv_select_mode { SELKV_SELECT_SHARED = 0, SELKV_SELECT_PER_HEAD = 1 } selkv_select_mode;

/* RoPE repositioning of the kept keys (Eq. 7, Sec. 3.7; off in the paper's configuration):
 * the key kept in slot s, originally at position j, becomes RoPE(RoPE^{-1}(k, j), s) for the
 * plain rotary embedding with base rope_theta, frequency f in [0, d/2) turning the pair
 * (k[f], k[f + d/2]) (HALF layout) or (k[2f], k[2f + 1]) (INTERLEAVED layout) by
 * p * rope_theta^(-2f/d).  Positions count from 0 at the first prefill token.  Decode does
 * not rotate: the caller embeds new queries and keys at positions lengths[b], ... . */
/* Attention compensation (Sec. 3.6): RATIO is SelKV's alpha * ln R (Eq. 6); COUNT is the
 * KeepKV-style alpha * ln(1 + M), M the evicted tokens merged into the kept token (routed to
 * it with g > 0), averaged over KV heads in SHARED mode (alpha = 1: KeepKV's log(1 + M)). */
typedef enum selkv_bias_mode { SELKV_BIAS_RATIO = 0, SELKV_BIAS_COUNT = 1 } selkv_bias_mode;

/* Routing of the evicted tokens (Sec. 3.4): BUCKET is the paper's bucket attention routing
 * (Eq. 3, with empty_bucket); COSINE is the full cosine routing that Sec. 3.4 sets against it
 * (cost O(|S| |E| d) per KV head): evicted j goes to the kept token i of its KV head with the
 * largest cos(v_j, v_i) over ALL kept tokens (original values; ties to the lower position; a
 * zero norm gives cosine 0).  The gate, merge and bias are the same in both. */
typedef enum selkv_routing { SELKV_ROUTE_BUCKET = 0, SELKV_ROUTE_COSINE = 1 } selkv_routing;

typedef enum selkv_rope {
  SELKV_ROPE_OFF = 0,
  SELKV_ROPE_HALF = 1,
  SELKV_ROPE_INTERLEAVED = 2
} selkv_rope;

/* Device error bits (selkv_workspace_error). */
#define SELKV_DEVERR_CAPACITY 0x1u /* decode append would pass m_cap: not appended       */
#define SELKV_DEVERR_TIMEOUT 0x2u  /* a bounded wait gave up; the launch's output is void  */
#define SELKV_DEVERR_LENGTH 0x4u   /* lengths[b] outside [0, m_cap]; clamped              */
#define SELKV_DEVERR_COUNT 0x8u    /* compress kept a count other than m_b (internal)     */

typedef struct selkv_shape {
  int32_t dtype;        /* selkv_dtype of K, V, Q_obs, q, k_new, v_new, K_c, V_c and out  */
  int32_t batch;        /* B, 1 .. SELKV_MAX_BATCH                                       */
  int32_t num_q_heads;  /* Hq                                                            */
  int32_t num_kv_heads; /* Hkv, divides Hq, at most 32                                   */
  int32_t head_dim;     /* d: 64 or 128                                                  */
  int32_t obs_window;   /* W: observation-window rows per query head (Sec. 3.1)          */
  int32_t n_cap;        /* rows per (b, kv) of K and V                                   */
  int32_t m_cap;        /* rows per (b, kv) of K_c, V_c and bias                         */
} selkv_shape;

#define SELKV_MAX_BATCH 1024

/* Hyperparameters (Sec. 3, defaults of Sec. 4.1 / App. F in the comments). */
typedef struct selkv_params {
  float alpha;          /* compensation strength, 0.5 (Sec. 3.6); 0 disables the bias  */
  int32_t pool_kernel;  /* average-pooling kernel K, odd, 5 (Sec. 3.2)                  */
  int32_t bucket;       /* routing bucket size B, 1 .. 32, 32 (Sec. 3.4)                */
  int32_t recent;       /* recent window m_r always kept, 16 (Sec. 3.1)                 */
  int32_t gate_mode;    /* selkv_gate_mode                                              */
  int32_t empty_bucket; /* selkv_empty_bucket                                           */
  int32_t select_mode;  /* selkv_select_mode, SHARED for GQA models (Sec. 4.1)            */
  int32_t rope;         /* selkv_rope, OFF (Sec. 4.1)                                     */
  float rope_theta;     /* rotary base, finite and > 0 when rope is on                    */
  int32_t bias_mode;    /* selkv_bias_mode, RATIO (Sec. 3.6)                              */
  int32_t routing;      /* selkv_routing, BUCKET (Sec. 3.4)                               */
} selkv_params;

/* Optional device outputs of selkv_compress, for inspection and testing.  Any field may be
 * NULL.  Entries for positions >= n_b (or slots >= m_b) are left untouched. */
typedef struct selkv_compress_debug {
  float* attn;       /* [B][Hkv][n_cap] a: cumulative window attention, group mean     */
  float* score;      /* [B][Hkv][n_cap] pooled contribution score; 0 past candidates   */
  uint8_t* topk;     /* [B][Hkv][n_cap] 1 where KV head kv's own top-m_s chose j       */
  int32_t* kept_idx; /* [B][m_cap] kept positions, ascending; [B][Hkv][m_cap] in the
                        PER_HEAD selection mode                                        */
  int32_t* target;   /* [B][Hkv][n_cap] merge target of evicted j; -1 for kept j and
                        for tokens left without a target                              */
  float* gate;       /* [B][Hkv][n_cap] g of evicted j (0 for kept j)                  */
  uint8_t* decision; /* [B][Hkv][n_cap] 1 = merge (g > 0), 0 = drop; 2 for kept j      */
  float* ratio;      /* [B][Hkv][m_cap] attention ratio R per kept slot (Eq. 6)        */
} selkv_compress_debug;

/* Human-readable name of a status code (static storage). */
SELKV_API const char* selkv_status_string(selkv_status status);

/* The CUDA runtime error behind the last SELKV_ERR_CUDA returned on the calling thread
 * (cudaSuccess = 0 if none), and its name in *name when name is not NULL (static storage). */
SELKV_API int selkv_last_cuda_error(const char** name);

/* Number of kernels this library has enqueued since it was loaded, over all threads and
 * devices (a diagnostic counter; a captured CUDA graph counts its kernels once, at capture). */
SELKV_API uint64_t selkv_kernel_launches(void);

/* Zero a workspace (its error word and the decode counters).  Enqueued on `stream`.
 * Returns SELKV_ERR_WORKSPACE for a NULL or misaligned workspace. */
SELKV_API selkv_status selkv_workspace_init(void* workspace, size_t workspace_bytes, selkv_stream_t stream);

/* Synchronise `stream`, copy the workspace's device error bits to *flags and clear them.
 * Returns SELKV_OK when no bit was set, SELKV_ERR_DEVICE when some were. */
SELKV_API selkv_status selkv_workspace_error(void* workspace, selkv_stream_t stream, uint32_t* flags);

/* ---------------------------------------------------------------------------------------
 * Compression (Algorithm 1; Sec. 3.1-3.6; RoPE repositioning, Eq. 7, off as in Sec. 4.1).
 *
 * For every sequence b (prefill length n_b = n_len[b]) and every KV head:
 *   a  = mean over the G query heads of the column sums of the causal observation-window
 *        attention softmax(Q_obs K^T / sqrt(d)), row i at position n_b - W + i (Sec. 3.1);
 *   c  = a * ||v|| (Eq. 1), average-pooled over the candidates [0, n_b - m_r) (Sec. 3.2);
 *   per-KV-head top-m_s of c (Eq. 2), union over KV heads, trimmed to m_s by the mean score
 *   (Sec. 3.3), plus the recent window: m_b = floor(rho * n_b) kept positions shared by
 *   every head, ties to the lower position (PER_HEAD mode: each KV head's own top-m_s plus
 *   the recent window, m_b positions per head);
 *   each evicted j routes to the kept token of its bucket with the largest a (Eq. 3, Sec. 3.4;
 *   COSINE routing: to the kept token with the largest cos(v_j, v_i)), gets
 *   g = clamp(cos(v_j, v_pi(j)), 0, 1) (Eq. 4) and is merged into V_c with weight g*a_j
 *   (Eq. 5); R = (a_i + sum g a_j) / a_i (Eq. 6); bias = alpha * ln(mean over KV heads R)
 *   (Sec. 3.6, GQA; PER_HEAD mode: alpha * ln R of each head's own entry; COUNT bias:
 *   alpha * ln(1 + M) of the merge counts instead); K_c holds the kept keys, unchanged or,
 *   with params->rope, re-embedded at their slot positions (Eq. 7).
 *
 * n_len     HOST array [B]: prefill lengths, W <= n_b <= n_cap.
 * rho       retention ratio in (0, 1]; m_b = floor(rho * n_b) (double), and
 *           m_b - recent >= 0 and m_b <= m_cap must hold for every b.
 * K, V      [B][Hkv][n_cap][d]; rows >= n_b are ignored.
 * Q_obs     [B][Hq][W][d]: the last W query rows of each sequence.
 * K_c, V_c  [B][Hkv][m_cap][d] outputs; rows >= m_b untouched.
 * bias      [B][Hkv][m_cap] fp32 output (the same row for every KV head in SHARED mode).
 * lengths   [B] int32 device output: m_b.
 * Errors: SELKV_ERR_INVALID_ARG for a NULL tensor, a bad shape, a misaligned pointer or a
 * budget outside the rules above; SELKV_ERR_UNSUPPORTED for d not in {64, 128} or a bucket
 * above 32; SELKV_ERR_WORKSPACE when workspace_bytes < selkv_compress_workspace_size.
 * ------------------------------------------------------------------------------------- */
SELKV_API size_t selkv_compress_workspace_size(const selkv_shape* shape);

SELKV_API selkv_status selkv_compress(const selkv_shape* shape, const int32_t* n_len, double rho,
                            const selkv_params* params, const void* K, const void* V,
                            const void* Q_obs, void* K_c, void* V_c, float* bias,
                            int32_t* lengths, const selkv_compress_debug* debug,
                            void* workspace, size_t workspace_bytes, selkv_stream_t stream);

/* ---------------------------------------------------------------------------------------
 * Observation-window attention alone: the scoring stage of selkv_compress (Sec. 3.1 re-pass;
 * the attention sums Eq. 1 weights by ||v|| and Eq. 5 calls a).  For every sequence b, KV
 * head kv and position j < n_b:
 *   attn[b][kv][j] = (1/G) sum over the G query heads h = kv G + g and the W window rows i
 *                    of softmax_j(Q_obs[b][h][i] . K[b][kv][j] / sqrt(d)),
 * causal: row i sits at position n_b - W + i and sees keys j <= n_b - W + i.  The values are
 * bitwise those of selkv_compress's `attn` debug output for the same inputs.
 *
 * It runs as two passes over K: the first finds each window row's softmax normaliser (the
 * maximum and the sum of the exponentials), the second sums the normalised probabilities
 * over the rows.  `passes` selects what the call runs:
 *   SELKV_SCORE_ALL       both passes: attn is written;
 *   SELKV_SCORE_ROWSTATS  the first pass only: the normalisers stay in the workspace and
 *                         attn is not touched (may be NULL);
 *   SELKV_SCORE_COLSUMS   the second pass only, from the normalisers that the previous
 *                         ROWSTATS call on this workspace left (same shape, n_len, K and
 *                         Q_obs; this call reuses that call's sequence lengths).
 *
 * n_len   HOST array [B]: prefill lengths, W <= n_b <= n_cap.
 * K       [B][Hkv][n_cap][d]; Q_obs [B][Hq][W][d]; attn [B][Hkv][n_cap] fp32 output
 *         (entries j >= n_b untouched).
 * Errors: SELKV_ERR_INVALID_ARG for a NULL or misaligned tensor, a bad shape or length or an
 * unknown `passes`; SELKV_ERR_UNSUPPORTED for d not in {64, 128}; SELKV_ERR_WORKSPACE when
 * workspace_bytes < selkv_score_workspace_size.
 * ------------------------------------------------------------------------------------- */
typedef enum selkv_score_passes {
  SELKV_SCORE_ROWSTATS = 1,
  SELKV_SCORE_COLSUMS = 2,
  SELKV_SCORE_ALL = 3
} selkv_score_passes;

SELKV_API size_t selkv_score_workspace_size(const selkv_shape* shape);

SELKV_API selkv_status selkv_score(const selkv_shape* shape, const int32_t* n_len, const void* K,
                                   const void* Q_obs, float* attn, int32_t passes, void* workspace,
                                   size_t workspace_bytes, selkv_stream_t stream);

/* ---------------------------------------------------------------------------------------
 * Compensation averaged across layers (the overview of Sec. 3 offers it next to the
 * per-layer bias of Sec. 3.6).  After the L layers of a model have been compressed with the
 * same params, every layer's bias is replaced by one value per position shared by all
 * layers: for each sequence b (and KV head in the PER_HEAD mode) and position p, the mean over
 * the L layers of the layer's per-slot quantity at p -- the R of the bias (the KV-head mean in
 * the SHARED mode) or, with the COUNT bias, M -- a layer that evicted p counting R = 1
 * (M = 0); the slot of every layer that holds p then gets alpha * ln(mean R), or
 * alpha * ln(1 + mean M).  The per-slot quantity is read back from each bias
 * (alpha * ln(1 + x), x = R - 1 or M), so call this once per compression; with alpha = 0 the
 * biases stay 0 and nothing is launched.
 *
 * params      the params given to selkv_compress (alpha, bias_mode, select_mode are read).
 * num_layers  L, 1 .. 128.
 * kept_idx    HOST array [L] of device pointers: each layer's kept positions as written to
 *             selkv_compress_debug.kept_idx ([B][m_cap]; [B][Hkv][m_cap] in PER_HEAD mode).
 * bias        HOST array [L] of device pointers: each layer's bias [B][Hkv][m_cap], read and
 *             overwritten (slots >= lengths[b] untouched).
 * lengths     [B] int32 device: the compressed lengths m_b, the same for every layer (call
 *             before decode appends).
 * The sums are taken layer by layer in order (bitwise reproducible).  Errors:
 * SELKV_ERR_INVALID_ARG for NULL or misaligned pointers, L outside 1..128 or bad params;
 * SELKV_ERR_WORKSPACE when workspace_bytes < selkv_layer_average_workspace_size (the
 * workspace is initialised once with selkv_workspace_init); a kept position outside
 * [0, n_cap) sets SELKV_DEVERR_COUNT.
 * ------------------------------------------------------------------------------------- */
SELKV_API size_t selkv_layer_average_workspace_size(const selkv_shape* shape);

SELKV_API selkv_status selkv_layer_average_bias(const selkv_shape* shape, const selkv_params* params,
                                                int32_t num_layers, const int32_t* const* kept_idx,
                                                float* const* bias, const int32_t* lengths,
                                                void* workspace, size_t workspace_bytes,
                                                selkv_stream_t stream);

/* ---------------------------------------------------------------------------------------
 * Compensated decode attention (Algorithm 1, "Decode with compressed cache + alpha log R";
 * Sec. 3.6).  For every sequence b and query head h (KV head kv = h / G):
 *   out[b][h] = sum_{i < L} softmax_i(q[b][h] . K_c[b][kv][i] / sqrt(d) + bias[b][kv][i])
 *               * V_c[b][kv][i]
 * over L = lengths[b] rows, plus, when k_new and v_new are given, the new row
 * (k_new[b][kv], v_new[b][kv]) with bias 0 (R = 1).  The new row is then written at row
 * lengths[b] of K_c / V_c (bias 0), and lengths[b] is incremented, all inside the call.
 *
 * q, out        [B][Hq][d].
 * K_c, V_c      [B][Hkv][m_cap][d]; bias [B][Hkv][m_cap] fp32 or NULL (no compensation:
 *               plain attention, e.g. over an uncompressed cache with m_cap = n_cap).
 * lengths       [B] int32 device, read (and incremented when appending).
 * k_new, v_new  [B][Hkv][d] or both NULL.
 * An empty cache with no new row gives out = 0.  An append that would pass m_cap is skipped
 * and sets SELKV_DEVERR_CAPACITY.
 *
 * Overlap with the previous kernel (bf16 caches): the decode is launched with programmatic
 * dependent launch and may start loading cache rows below lengths[b] - 1 while the kernel
 * enqueued just before it on the same stream is still running.  That kernel must therefore
 * not write those rows of K_c and V_c (it may write q, k_new, v_new, the bias, lengths, and
 * row lengths[b] - 1 onwards).  The library's own calls never do: a decode appends only at
 * lengths[b], and a compression writes K_c and V_c before its last kernel.  A caller kernel
 * that rewrites cached rows must be separated from the decode by another stream operation
 * (any other kernel, a copy or an event).  Everything the result is computed from is read
 * after the previous kernel has completed: rows loaded early are used only where the slice
 * planned from the final lengths[b] starts at the same row and covers them.
 * ------------------------------------------------------------------------------------- */
SELKV_API size_t selkv_decode_workspace_size(const selkv_shape* shape);

SELKV_API selkv_status selkv_decode_attn(const selkv_shape* shape, const void* q, void* K_c, void* V_c,
                               float* bias, int32_t* lengths, const void* k_new,
                               const void* v_new, void* out, void* workspace,
                               size_t workspace_bytes, selkv_stream_t stream);

/* ---------------------------------------------------------------------------------------
 * Decode without a workspace.  The paper has no counterpart: this is a deployment variant of
 * selkv_decode_attn for callers that cannot allocate device memory, such as code running
 * inside a host framework that owns every device buffer and passes a kernel only its inputs
 * and outputs, or a serving loop that must not call cudaMalloc / cudaFree (cudaFree
 * synchronises the device) and has no workspace planned for this call.
 *
 * It computes exactly what selkv_decode_attn computes, with the same arguments except the
 * workspace; the scratch it needs (split partials, arrival counters) lives in one static
 * device array of SELKV_STATIC_SCRATCH_BYTES inside the library, reserved on every GPU that
 * loads the library until the process exits.  The call allocates nothing.
 *   - Shapes whose scratch exceeds SELKV_STATIC_SCRATCH_BYTES return SELKV_ERR_WORKSPACE
 *     before any launch (about B * Hq * splits * (d + 2) * 4 bytes plus counters).
 *   - Every call shares the array and it keeps the last call's contents; each call clears the
 *     part that must start at zero before its kernel.  Calls that overlap on the GPU (on
 *     different streams or from different host threads) race on the array: serialise them.
 *   - The first call on a device looks up the array's device address with that device
 *     current, and a call made in another context than the one of the address it holds
 *     (after cudaDeviceReset, for instance) looks it up again; make the first call on a
 *     device, and the first call after a reset, before any stream capture.
 *   - flags_out: optional device uint32 that receives the SELKV_DEVERR_* bits (OR-ed in,
 *     never cleared); NULL drops them.
 * ------------------------------------------------------------------------------------- */
#define SELKV_STATIC_SCRATCH_BYTES (4u << 20)

SELKV_API selkv_status selkv_decode_attn_static(const selkv_shape* shape, const void* q,
                                                void* K_c, void* V_c, float* bias,
                                                int32_t* lengths, const void* k_new,
                                                const void* v_new, void* out,
                                                uint32_t* flags_out, selkv_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* SELKV_H */
