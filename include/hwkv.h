/*
 * hwkv.h -- C ABI of the per-head-window KV cache library (libhwkv.so).
 *
 * HeadWiseKV (arXiv 2609.02029) assigns every physical KV head (layer l,
 * head h) of each residual global-attention layer one history window a_{lh}
 * from a codebook {w_1 < ... < w_K, full} (Sec. 3.1). At serving time each
 * configured head reads and writes only its own K/V slice, sized to its
 * window, instead of a mask over a full cache (Sec. 3.3; App. "Runtime
 * Realization and Deployment", physical cache realization). This library is
 * that runtime's hot path on one GPU: per-head ring allocation, K/V
 * append/wrap, window-limited causal prefill attention and split-KV decode
 * attention with a log-sum-exp merge, plus exact residency accounting.
 *
 * Conventions for every call
 *  - Tensors are bf16 (2-byte) unless stated; `out` tensors are fp32.
 *    Tensor pointers are caller-owned device memory, dense, in the stated
 *    row-major layout, 16-byte aligned.
 *  - Head mapping under GQA (Sec. 3.1, groups G_{lh}): query head q reads KV
 *    head q / G with G = n_q_heads / n_kv_heads (contiguous groups).
 *  - Positions are 0-based. A query at position p with window W attends to
 *    key positions s in [max(0, p-W+1), p] (Sec. 3.2, the set J_t(w)); a full
 *    head attends to [0, p]. Any W >= max_ctx is full (Sec. 3.1).
 *  - Every call that takes `cuda_stream` (a cudaStream_t, NULL = legacy
 *    default stream) is asynchronous and stream-ordered; argument errors are
 *    returned before anything is launched and leave the cache unchanged.
 *    Calls on one cache must be issued on one stream (they share the cache's
 *    device workspace) and from one host thread at a time.
 *  - No call throws; failures return a status and set a thread-local message
 *    readable with hwkv_last_error().
 */
#ifndef HWKV_H
#define HWKV_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define HWKV_API __attribute__((visibility("default")))
#else
#define HWKV_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  HWKV_OK = 0,
  HWKV_EINVAL = 1,       /* bad argument or policy; nothing was launched */
  HWKV_ENOMEM = 2,       /* arena too small or device allocation failed */
  HWKV_ECAPACITY = 3,    /* append would exceed max_ctx on a full-history head */
  HWKV_ECUDA = 4,        /* a CUDA runtime call or launch failed */
  HWKV_EKERNEL = 5,      /* a kernel reported an internal error (see hwkv_sync_check) */
  HWKV_EUNSUPPORTED = 6, /* valid request outside the built kernel set (e.g. head_dim) */
  HWKV_ETRACE = 7        /* hwkv_calib_trace_check: the trace does not match its replay */
} hwkv_status;

/* windows[] entry meaning "full history" (Sec. 3.1: a_{lh} = full) */
#define HWKV_WINDOW_FULL 0

/*
 * Cache format p_KV (Sec. 3.1: the nominal storage of Eq. nominal-storage is
 * per format, through the effective precisions b^K, b^V).
 *   HWKV_KV_BF16:     K and V rows in bf16 (b^K = b^V = 2 bytes).
 *   HWKV_KV_FP8_E4M3: K and V rows as 8-bit E4M3 codes (1 sign, 4 exponent bits
 *     with bias 7, 3 mantissa bits, largest finite 448) with one fp32 scale per
 *     stored row (one token of one KV head): s = the smallest power of two at or
 *     above amax / 448 (amax / 448 in fp32), code = nearest E4M3 value of x / s
 *     (ties to even, saturating), value = code * s; a zero row stores s = 0. Effective precision (d + 4) / d bytes per element. Attention
 *     reads the dequantised rows (the paper: when the format changes execution,
 *     every compared output uses it), in prefill the chunk's own keys included
 *     (they are read as the append stores them). head_dim 128 or 256.
 */
#define HWKV_KV_BF16 0
#define HWKV_KV_FP8_E4M3 1

/*
 * The policy matrix a (Sec. 3.1, Eq. for a_{lh}; App. "Runtime Realization":
 * a static layer x KV-head matrix loaded once).
 *   windows[l * n_kv_heads + h] = W_{lh} in tokens (> 0), or HWKV_WINDOW_FULL.
 * A head with W >= max_ctx is stored as full. max_ctx bounds the tokens any
 * layer will ever hold (it is the ring capacity of full heads).
 *   sinks: NULL, or sinks[l * n_kv_heads + h] = S >= 0 sink tokens kept beside a
 *   finite window W (the static sink--recent policy of the paper's StreamingLLM
 *   control): a query at position p then reads positions {0..S-1} and
 *   [max(0, p-W+1), p] (both <= p), and the head retains min(S + W, t) tokens in
 *   a ring of S + W slots (positions < S in slots 0..S-1 for good, later ones in
 *   slot S + (p - S) mod W). Ignored for full heads; S + W >= max_ctx is full.
 * Supported: head_dim in {64, 128, 256}; n_q_heads / n_kv_heads <= 8;
 * batch <= 256; n_kv_heads <= 64; the policy is copied by hwkv_alloc.
 */
typedef struct {
  int32_t n_layers;
  int32_t n_kv_heads;
  int32_t n_q_heads;
  int32_t head_dim;
  int32_t batch;
  int32_t kv_format; /* HWKV_KV_BF16 or HWKV_KV_FP8_E4M3 */
  int64_t max_ctx;
  const int64_t* windows;
  const int64_t* sinks; /* NULL: no sink tokens */
} hwkv_policy;

typedef struct hwkv_cache hwkv_cache; /* opaque; owned by the library */

/*
 * Device bytes hwkv_alloc needs for `policy`: the K and V rings of every
 * (layer, KV head, batch row) -- capacity min(W, max_ctx) tokens x head_dim
 * bf16 each -- plus the decode workspace. Pure host computation.
 */
HWKV_API hwkv_status hwkv_required_bytes(const hwkv_policy* policy, size_t* arena_bytes);

/*
 * Validates `policy` (positive sizes, n_q_heads % n_kv_heads == 0, W >= 0,
 * max_ctx > 0) and lays out one ring per (layer, KV head, batch row), rings
 * of equal capacity adjacent (one cache group per window level, Sec. 3.3).
 * dev_arena: caller-owned device memory of arena_bytes >= hwkv_required_bytes
 * (the cache does not free it), or NULL to let the library cudaMalloc it.
 * The rings and workspace are zero-filled on `cuda_stream` before return
 * completes (this call synchronizes that stream). Every layer starts with
 * t = 0 tokens. On success *out owns the cache; release with hwkv_free.
 */
HWKV_API hwkv_status hwkv_alloc(const hwkv_policy* policy, void* dev_arena, size_t arena_bytes,
                       void* cuda_stream, hwkv_cache** out);

/* Releases the cache (and the arena if the library allocated it). NULL is a no-op. */
HWKV_API hwkv_status hwkv_free(hwkv_cache* cache);

/*
 * Append/wrap (Sec. 3.3: a head keeps only its latest W states). Writes the
 * n new tokens at positions t .. t+n-1 of `layer` into every KV head's ring,
 * position p going to slot p mod cap; only the last min(n, cap) of them are
 * written (earlier ones would be overwritten within the same call). Then t += n.
 *   k, v: [batch, n, n_kv_heads, head_dim] bf16, device.
 * n == 0 is a no-op. Fails with HWKV_ECAPACITY if t + n > max_ctx.
 */
HWKV_API hwkv_status hwkv_append(hwkv_cache* cache, int32_t layer, const void* k, const void* v,
                        int64_t n, void* cuda_stream);

/*
 * Window-limited causal prefill of one chunk (Sec. 3.2, Eq. conditional-
 * attention-weight and Eq. conditional-attention; the chunked prompt pass of
 * App. "Experimental Protocol"). For the chunk at positions t0 .. t0+n-1
 * (t0 = the layer's current t): query row p of query head q attends to the
 * keys of KV head q/G at positions [max(0, p-W+1), p], taken from the ring
 * (positions < t0) and from this chunk (positions >= t0), with logits
 * scale * q.k. Then the chunk's K/V are appended as by hwkv_append.
 *   q:   [batch, n, n_q_heads, head_dim] bf16
 *   k,v: [batch, n, n_kv_heads, head_dim] bf16
 *   out: [batch, n, n_q_heads, head_dim] fp32, the per-head outputs
 *        concatenated in head order (pre-gate layout, Sec. 3.3).
 * Because attention runs before the write, a ring of capacity exactly W
 * serves chunks longer than W. Fails with HWKV_ECAPACITY as hwkv_append, and
 * with HWKV_EUNSUPPORTED past 2^30 tokens of history or for chunks over
 * 1,048,560 tokens.
 * With HWKV_KV_FP8_E4M3 every key of the query's window is read as stored
 * (code x scale), the chunk's own keys as the append will store them; the call
 * allocates (stream-ordered) and frees a staging buffer of 2 * head_dim bytes
 * per held ring slot of the layer (K and V) and per chunk token and head (q, K,
 * V) (HWKV_ENOMEM if that fails): q and the dequantized K/V rows go through the
 * tensor cores in fp16, so magnitudes past +-65504 saturate there.
 */
HWKV_API hwkv_status hwkv_prefill(hwkv_cache* cache, int32_t layer, const void* q, const void* k,
                         const void* v, int64_t n, float scale, float* out, void* cuda_stream);

/*
 * Decode attention (Sec. 3.2 at the newest position; Sec. 3.3 graph routing):
 * the query at position p = t-1 (the token the caller appended last) of each
 * query head attends over every resident slot of its KV head's ring, i.e.
 * positions [max(0, t-W), t-1], with logits scale * q.k. The kernels read
 * the row lengths on the GPU and give every CTA an equal share of the layer's
 * resident keys (in 64-key stages, plus a fixed cost per ring piece), so a
 * full-history ring is split over many CTAs and short-window rings are read
 * whole; a ring split over CTAs leaves partials (max, sum, output) that a
 * log-sum-exp merge combines.
 *   q:   [batch, n_q_heads, head_dim] bf16
 *   out: [batch, n_q_heads, head_dim] fp32
 * Fails with HWKV_EINVAL if the layer holds no tokens.
 */
HWKV_API hwkv_status hwkv_decode_attn(hwkv_cache* cache, int32_t layer, const void* q, float scale,
                             float* out, void* cuda_stream);

/*
 * One decode step of a layer in a single launch (+ the combine): appends the
 * new token at position t (as hwkv_append with n = 1) and computes the decode
 * attention of its queries (as hwkv_decode_attn after that append); then t += 1.
 * The new token's K/V go straight from k_new/v_new into the attention and into
 * ring slot t mod cap, which no other part of the step reads.
 *   q:           [batch, n_q_heads, head_dim] bf16
 *   k_new, v_new:[batch, n_kv_heads, head_dim] bf16
 *   out:         [batch, n_q_heads, head_dim] fp32
 * Fails with HWKV_ECAPACITY if t + 1 > max_ctx.
 */
HWKV_API hwkv_status hwkv_decode_step(hwkv_cache* cache, int32_t layer, const void* q,
                                      const void* k_new, const void* v_new, float scale,
                                      float* out, void* cuda_stream);

/*
 * Per-row lengths (serving form of the same method; the paper's runs decode one
 * request at a time, so it defines no batching). Every (layer, batch row) holds
 * its own length t_b: rows are independent sequences, and every operation above
 * applies to each row at that row's own t_b. A row can also be idle (t_b = -1):
 * it holds nothing, takes no append, and decode writes zeros for it. The cache
 * keeps the lengths twice: on the host (read by the calls above) and in an
 * int32 [n_layers][batch] array inside the arena (read by the kernels). Every
 * call keeps both equal, except hwkv_decode_step_graph, which advances only the
 * device copy.
 *
 * Decode over ragged or idle rows: hwkv_decode_attn / hwkv_decode_step accept
 * them (the work is always planned on the GPU from the device lengths). Rows
 * with t_b = 0 give zeros in hwkv_decode_attn.
 */

/* hwkv_append for the rows [row0, row0 + n_rows) only; each appends at its own t_b.
 *   k, v: [n_rows, n, n_kv_heads, head_dim] bf16, device.
 * Fails with HWKV_EINVAL for an idle row, HWKV_ECAPACITY if a row's t_b + n > max_ctx. */
HWKV_API hwkv_status hwkv_append_rows(hwkv_cache* cache, int32_t layer, int32_t row0,
                                      int32_t n_rows, const void* k, const void* v, int64_t n,
                                      void* cuda_stream);

/* hwkv_prefill for the rows [row0, row0 + n_rows) only (e.g. a newly admitted
 * request); q, k, v and out hold n_rows rows. The rows must hold the same length
 * (HWKV_EINVAL otherwise). Other errors as hwkv_prefill. */
HWKV_API hwkv_status hwkv_prefill_rows(hwkv_cache* cache, int32_t layer, int32_t row0,
                                       int32_t n_rows, const void* q, const void* k,
                                       const void* v, int64_t n, float scale, float* out,
                                       void* cuda_stream);

/*
 * hwkv_decode_step for CUDA-graph capture and replay: the step of every active
 * row b reads t_b from the device length array at run time, appends the new
 * token at slot t_b mod cap, attends over min(t_b + 1, cap) slots, and then
 * advances the device t_b by one. Nothing on the host depends on the lengths,
 * so a captured sequence of these calls (one per layer) replays as later decode
 * steps. Idle rows get zero output and stay idle. A row already at max_ctx is
 * skipped (zero output, length kept) and sets the error word (hwkv_sync_check).
 * From the first such call on, the device owns the layer's lengths (replays
 * advance them unseen by the host): every later host call that reads them
 * (append, prefill, the other decodes, hwkv_seq_len, hwkv_row_len,
 * hwkv_residency_bytes) first waits for the device (cudaDeviceSynchronize) and
 * re-reads them; such calls cannot be captured. Arguments as hwkv_decode_step.
 * During capture, make no other call on the cache from another thread.
 */
HWKV_API hwkv_status hwkv_decode_step_graph(hwkv_cache* cache, int32_t layer, const void* q,
                                            const void* k_new, const void* v_new, float scale,
                                            float* out, void* cuda_stream);

/* Waits for cuda_stream, then copies the device lengths of every layer to the
 * host copy (the calls above do this by themselves for graph-owned layers). */
HWKV_API hwkv_status hwkv_sync_lens(hwkv_cache* cache, void* cuda_stream);

/*
 * Rows [row0, row0 + n_rows) of every layer restart empty (idle = 0: t_b = 0)
 * or become idle (idle != 0: t_b = -1), e.g. when a request finishes and its
 * batch slot is reused. Ring contents are left in place; the new length makes
 * them unreachable. Stream-ordered (a cudaMemsetAsync per layer); may be captured.
 */
HWKV_API hwkv_status hwkv_reset_rows(hwkv_cache* cache, int32_t row0, int32_t n_rows,
                                     int32_t idle, void* cuda_stream);

/* Length t_b of one row (-1 = idle). */
HWKV_API hwkv_status hwkv_row_len(const hwkv_cache* cache, int32_t layer, int32_t row, int64_t* t);

/* Size of the device array hwkv_decode_attn_static keeps its scratch in. */
#define HWKV_DECODE_STATIC_SCRATCH_BYTES (4u << 20)

/*
 * The paper has no counterpart of this call; it serves callers that cannot
 * allocate device memory. Plugins running inside another engine whose
 * allocator owns all GPU memory, code that must never synchronize the device
 * (cudaMalloc and cudaFree can), and code issued during stream capture are
 * handed their inputs and outputs but cannot create scratch buffers.
 *
 * Same result and arguments as hwkv_decode_attn, but the partial outputs and
 * the work plan live in a fixed 4 MiB array inside this library's device image
 * (present on every GPU that loads the library until the process exits)
 * instead of the cache's workspace. It calls no cudaMalloc, cudaFree or
 * allocating routine, and it does not synchronize: the kernels read the
 * layer's lengths on the device (after graph-mode steps the host copy only
 * sizes the grid, and the "holds no tokens" check is skipped; rows holding
 * nothing decode to zeros).
 * The first call on each device, with that device current, looks up the
 * array's device address (cudaGetSymbolAddress) and keeps it for the life of
 * the process (a device reset is not supported); make that first call before
 * any stream capture. The array keeps the last call's contents and nothing in
 * it needs to start at zero. All calls share it: calls whose kernels overlap
 * on the GPU (other streams, other caches) race and give wrong results.
 * It needs 2 * grid * (32 * head_dim + 64) bytes of partials (grid <= the SM
 * count) plus 16 * (2 + batch * n_kv_heads) bytes of plan, each rounded up to
 * 256 (hwkv_decode_static_scratch_bytes computes it): 2.8 MB on 152 SMs at
 * head_dim 256 with 256 batch rows and 64 KV heads, the largest valid policy.
 * A layout that does not fit fails with HWKV_EINVAL before anything is launched.
 */
HWKV_API hwkv_status hwkv_decode_attn_static(hwkv_cache* cache, int32_t layer, const void* q,
                                             float scale, float* out, void* cuda_stream);

/* Host-only: the static scratch bytes hwkv_decode_attn_static needs for `policy`
 * on a GPU of num_sms SMs (its largest grid). Returns HWKV_EINVAL (with *bytes
 * set) when that exceeds HWKV_DECODE_STATIC_SCRATCH_BYTES, as the call would. */
HWKV_API hwkv_status hwkv_decode_static_scratch_bytes(const hwkv_policy* policy, int32_t num_sms,
                                                      size_t* bytes);

/*
 * SeqCalib candidate replay (Sec. 3.2: one layer's trace, every candidate
 * window replayed from it). For query head q at sampled position t of
 * calibration sequence n, o^(w) is the attention output over the keys
 * [max(0, t-w+1), t] (Eq. conditional-attention) and
 *   cos[n][p][q][k] = cos_eval(o^(windows[k]), o^(full))   (App. A.2,
 *                     Eq. stabilized-cosine, eps = 1e-12),
 *   scores[h][k]    = mean of cos over (n, p, q in the group of KV head h)
 *                     (Eq. conditional-similarity).
 * The full candidate scores one and is not listed.
 */
typedef struct {
  int32_t n_seq;       /* calibration sequences N */
  int32_t n_pos;       /* sampled query positions per sequence P */
  int32_t n_kv_heads;
  int32_t n_q_heads;   /* multiple of n_kv_heads, group <= 8 */
  int32_t head_dim;    /* 64, 128 or 256 */
  int32_t n_windows;   /* K candidate finite windows, 1..8 */
  int64_t T;           /* trace length: positions 0..T-1 */
  const int64_t* windows;    /* [K] host, positive, increasing */
  const int64_t* positions;  /* [N][P] host, in [0, T) */
} hwkv_calib_desc;

/* Device workspace hwkv_calib_scores needs for this description (host-only). */
HWKV_API hwkv_status hwkv_calib_workspace_bytes(const hwkv_calib_desc* desc, size_t* bytes);

/*
 *   q:    [N][P][n_q_heads][head_dim] bf16, device: queries at the sampled positions
 *   k, v: [N][n_kv_heads][T][head_dim] bf16, device: the layer's trace, head-major
 *   workspace: device, >= hwkv_calib_workspace_bytes(desc), 256-byte aligned
 *   scores: host [n_kv_heads][K] double; cos_out: host [N][P][n_q_heads][K] float or NULL
 * The keys of each (sequence, position, KV head) are cut into the nested
 * suffix bands of the windows, replayed once with split-KV tiles, and merged
 * band by band. Synchronizes `cuda_stream` (results are returned on the host).
 */
HWKV_API hwkv_status hwkv_calib_scores(const hwkv_calib_desc* desc, const void* q, const void* k,
                                       const void* v, float scale, void* workspace,
                                       size_t ws_bytes, double* scores, float* cos_out,
                                       void* cuda_stream);

/*
 * Trace-compatibility check of SeqCalib (App. "Experimental Protocol" and
 * App. "Runtime Realization": before accepting a layer's trace the calibrator
 * replays the full-window attention for the sampled positions and aborts the run
 * when it does not reproduce the traced output; the paper aborts below cosine
 * 0.99). Same replay as hwkv_calib_scores; traced: device fp32
 * [N][P][n_q_heads][head_dim], the traced full-history outputs at the sampled
 * positions. *min_cos receives the smallest cos_eval(replayed full, traced)
 * (App. A.2, Eq. stabilized-cosine); trace_cos_out (host [N][P][n_q_heads] or
 * NULL) all of them. Returns HWKV_ETRACE (naming the worst row) when
 * *min_cos < threshold. Synchronizes `cuda_stream`.
 */
HWKV_API hwkv_status hwkv_calib_trace_check(const hwkv_calib_desc* desc, const void* q,
                                            const void* k, const void* v, float scale,
                                            const float* traced, double threshold,
                                            void* workspace, size_t ws_bytes, double* min_cos,
                                            float* trace_cos_out, void* cuda_stream);

/*
 * Threshold selection (Sec. 3.2, Eq. threshold-selection) for each of n_heads
 * heads: among the windows whose score is >= tau, plus full (score one), the
 * one of lowest nominal cost min(w, C); equal costs go to the earlier window in
 * the order <_W (increasing finite windows, then full). policy[h] receives the
 * window, HWKV_WINDOW_FULL for full. scores: [n_heads][n_windows]. Host-only.
 */
HWKV_API hwkv_status hwkv_calib_select(const double* scores, int32_t n_heads,
                                       const int64_t* windows, int32_t n_windows, int64_t C,
                                       double tau, int64_t* policy);

/*
 * Finite-grid budget selection (App. A.2, Eq. budget-selector): among the
 * records g with beta[g] <= budget, the largest phi[g], then the smallest
 * beta[g], then the smallest g; *chosen = g, or -1 if no record meets the
 * budget. Host-only.
 */
HWKV_API hwkv_status hwkv_budget_select(const double* beta, const double* phi, int32_t n_records,
                                        double budget, int32_t* chosen);

/*
 * Policy artifact (App. "Experimental Protocol": each calibration run stores its
 * artifact identifier, seed and final policy matrix; App. "Runtime Realization":
 * the runtime loads the layer x KV-head matrix once). Text format, one item per
 * line, '#' starts a comment:
 *   hwkv-policy 1
 *   artifact <id: 1..127 printable characters, no spaces>
 *   seed <unsigned 64-bit>
 *   shape <n_layers> <n_kv_heads>
 *   layer <l> <W_l0> <W_l1> ... <W_l(n_kv_heads-1)>     (one line per layer, in
 *                                                      order; 0 = full)
 * hwkv_policy_save writes `windows` [n_layers * n_kv_heads] to `path`.
 * hwkv_policy_load reads it: windows_out must hold capacity entries; the shape
 * and seed are returned, the id copied into artifact (NUL-terminated, artifact_cap
 * bytes). Malformed files, negative windows or a shape larger than capacity give
 * HWKV_EINVAL with the line number in hwkv_last_error(). Host-only.
 */
HWKV_API hwkv_status hwkv_policy_save(const char* path, const char* artifact, uint64_t seed,
                                      int32_t n_layers, int32_t n_kv_heads, const int64_t* windows);
HWKV_API hwkv_status hwkv_policy_load(const char* path, char* artifact, size_t artifact_cap,
                                      uint64_t* seed, int32_t* n_layers, int32_t* n_kv_heads,
                                      int64_t* windows_out, size_t capacity);

/*
 * Resident K+V bytes (Sec. 3.1, Eq. nominal-storage with C = t, per row): sum
 * over KV heads and rows b of min(cap, t_b) * (head_dim * 2 * 2) for bf16, or
 * min(cap, t_b) * (head_dim + 4) * 2 for the 8-bit format (codes and scales)
 * (idle rows hold nothing), for one layer, or summed over all layers when
 * layer == -1. Host-only.
 */
HWKV_API hwkv_status hwkv_residency_bytes(const hwkv_cache* cache, int32_t layer, uint64_t* bytes);

/* Bytes of ring storage allocated (sum of batch * cap * head_dim * 4); layer -1 = all. */
HWKV_API hwkv_status hwkv_allocated_ring_bytes(const hwkv_cache* cache, int32_t layer, uint64_t* bytes);

/* Tokens held by `layer` so far (its t) when every row holds the same number;
 * HWKV_EINVAL when rows differ or are idle (use hwkv_row_len). */
HWKV_API hwkv_status hwkv_seq_len(const hwkv_cache* cache, int32_t layer, int64_t* t);

/* Ring capacity of (layer, kv_head): min(W, max_ctx), or max_ctx for full. */
HWKV_API hwkv_status hwkv_ring_capacity(const hwkv_cache* cache, int32_t layer, int32_t kv_head,
                               int64_t* cap);

/*
 * Copies the ring of (layer, batch row b, kv_head) to host buffers
 * k_host, v_host of cap * head_dim elements each (slot-major): bf16, or E4M3
 * codes (1 byte) for HWKV_KV_FP8_E4M3. Synchronizes the device. For tests and
 * debugging.
 */
HWKV_API hwkv_status hwkv_debug_copy_ring(const hwkv_cache* cache, int32_t layer, int32_t b,
                                 int32_t kv_head, void* k_host, void* v_host);

/* HWKV_KV_FP8_E4M3 only: the cap fp32 row scales of that ring's K and V
 * (slot-major), as hwkv_debug_copy_ring. */
HWKV_API hwkv_status hwkv_debug_copy_scales(const hwkv_cache* cache, int32_t layer, int32_t b,
                                            int32_t kv_head, float* k_scales, float* v_scales);

/*
 * Synchronizes the device and reads the cache's kernel error word; returns
 * HWKV_EKERNEL (and clears the word) if a kernel gave up on a bounded wait,
 * saw an inconsistent index, or a graph-mode step skipped a row at max_ctx,
 * else HWKV_OK.
 */
HWKV_API hwkv_status hwkv_sync_check(hwkv_cache* cache);

/*
 * Test of the failure path of every kernel wait (no paper counterpart): launches
 * one CTA whose thread waits, with the bounded mbarrier wait the kernels use, on
 * an mbarrier that nothing arrives at; after limit_ns nanoseconds (1e6 .. 2e9)
 * of the GPU's global timer it gives up and sets the wait-timeout bit of the
 * cache's error word, exactly as a kernel whose wait ran out would, and ends. No
 * copy or tensor-core operation is in flight, so the context stays usable; the
 * next hwkv_sync_check returns HWKV_EKERNEL and clears the word.
 */
HWKV_API hwkv_status hwkv_debug_wait_probe(hwkv_cache* cache, int64_t limit_ns, void* cuda_stream);

/* Message of the last failure on this thread ("" if none). */
HWKV_API const char* hwkv_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* HWKV_H */
