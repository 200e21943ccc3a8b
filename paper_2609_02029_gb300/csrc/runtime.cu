// runtime.cu -- host side of libhwkv: the C ABI of include/hwkv.h.
//
// Policy -> physical layout (HeadWiseKV Sec. 3.3 and App. "Runtime
// Realization": storage partitioned into (window, KV head) groups; each
// configured head owns a slice sized to its window, disjoint per layer).
// Here every (layer, KV head, batch row) owns one K ring and one V ring of
// cap = min(W, max_ctx) rows of head_dim bf16; rings of the same capacity
// (one window level) are adjacent in one arena, K region first, then the V
// region in the same order, then the decode workspace.
#include <algorithm>
#include <cerrno>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include <cudaTypedefs.h>

#include "../../include/hwkv.h"
#include "hwkv_internal.cuh"

using namespace hwkv;

namespace {

thread_local std::string g_last_error;

hwkv_status fail(hwkv_status st, const char* fmt, ...) __attribute__((format(printf, 2, 3)));
hwkv_status fail(hwkv_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return st;
}

hwkv_status ok() {
  g_last_error.clear();
  return HWKV_OK;
}

constexpr size_t kAlign = 256;
size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

struct Unit {
  int64_t window;  // effective: 0 = full
  int64_t cap;
  int64_t stride;  // rows per batch row: cap, rounded up to 64 in the 8-bit format
  int64_t sink;    // sink slots (sink + recent policy), 0 otherwise
  int64_t k_row0, v_row0;
};

struct Layout {
  std::vector<Unit> units;  // [layer * n_kv_heads + h]
  int64_t rows = 0;         // K rows (= V rows)
  size_t ring_bytes = 0;    // K + V
  size_t scale_off = 0;     // 8-bit format: fp32 row scales [2 * rows + 64]
  size_t part_o_off = 0, part_ml_off = 0, err_off = 0, lens_off = 0, plan_off = 0, total = 0;
  int slots = 0;  // decode partial slots: two per CTA of a split launch
};

hwkv_status validate(const hwkv_policy* p) {
  if (!p) return fail(HWKV_EINVAL, "policy is NULL");
  if (p->n_layers <= 0 || p->n_kv_heads <= 0 || p->n_q_heads <= 0 || p->batch <= 0 ||
      p->head_dim <= 0 || p->max_ctx <= 0)
    return fail(HWKV_EINVAL, "policy sizes must be positive");
  if (p->n_q_heads % p->n_kv_heads != 0)
    return fail(HWKV_EINVAL, "n_q_heads (%d) must be a multiple of n_kv_heads (%d)",
                p->n_q_heads, p->n_kv_heads);
  if (!p->windows) return fail(HWKV_EINVAL, "policy windows is NULL");
  for (int64_t i = 0; i < (int64_t)p->n_layers * p->n_kv_heads; ++i) {
    if (p->windows[i] < 0)
      return fail(HWKV_EINVAL, "window of (layer %lld, kv head %lld) is negative",
                  (long long)(i / p->n_kv_heads), (long long)(i % p->n_kv_heads));
    if (p->sinks && p->sinks[i] < 0)
      return fail(HWKV_EINVAL, "sink count of (layer %lld, kv head %lld) is negative",
                  (long long)(i / p->n_kv_heads), (long long)(i % p->n_kv_heads));
  }
  if (p->head_dim != 64 && p->head_dim != 128 && p->head_dim != 256)
    return fail(HWKV_EUNSUPPORTED, "head_dim %d not built (64, 128, 256)", p->head_dim);
  if (p->n_q_heads / p->n_kv_heads > kMaxGroup)
    return fail(HWKV_EUNSUPPORTED, "GQA group %d > %d", p->n_q_heads / p->n_kv_heads, kMaxGroup);
  if (p->n_kv_heads > kMaxKvHeads)
    return fail(HWKV_EUNSUPPORTED, "n_kv_heads %d > %d", p->n_kv_heads, kMaxKvHeads);
  if (p->batch > 256) return fail(HWKV_EUNSUPPORTED, "batch %d > 256", p->batch);
  if (p->kv_format != HWKV_KV_BF16 && p->kv_format != HWKV_KV_FP8_E4M3)
    return fail(HWKV_EINVAL, "unknown kv_format %d", p->kv_format);
  if (p->kv_format == HWKV_KV_FP8_E4M3 && p->head_dim != 128 && p->head_dim != 256)
    return fail(HWKV_EUNSUPPORTED, "the 8-bit format is built for head_dim 128 and 256");
  return HWKV_OK;
}

Layout make_layout(const hwkv_policy* p) {
  Layout L;
  const int nu = p->n_layers * p->n_kv_heads;
  L.units.resize(nu);
  for (int i = 0; i < nu; ++i) {
    const int64_t W = p->windows[i];
    const int64_t S = p->sinks ? p->sinks[i] : 0;
    Unit& u = L.units[i];
    // w >= C is full (Sec. 3.1); so is a sink + window that covers max_ctx
    u.window = (W == HWKV_WINDOW_FULL || W >= p->max_ctx || S + W >= p->max_ctx) ? 0 : W;
    u.sink = u.window == 0 ? 0 : S;
    u.cap = u.window == 0 ? p->max_ctx : u.sink + u.window;
    // 8-bit rings start on 64-row boundaries: a stage's 64 scales are one aligned run
    u.stride = p->kv_format == HWKV_KV_FP8_E4M3 ? (u.cap + 63) / 64 * 64 : u.cap;
  }
  // group by level: larger capacity first, then layer, then head
  std::vector<int> order(nu);
  for (int i = 0; i < nu; ++i) order[i] = i;
  std::stable_sort(order.begin(), order.end(),
                   [&](int a, int b) { return L.units[a].cap > L.units[b].cap; });
  int64_t row = 0;
  for (int i : order) {
    L.units[i].k_row0 = row;
    row += L.units[i].stride * p->batch;
  }
  L.rows = row;
  for (auto& u : L.units) u.v_row0 = u.k_row0 + L.rows;
  const bool fp8 = p->kv_format == HWKV_KV_FP8_E4M3;
  const size_t row_bytes = (size_t)p->head_dim * (fp8 ? 1 : 2);
  L.ring_bytes = (size_t)(2 * L.rows) * row_bytes;
  L.scale_off = align_up(L.ring_bytes, kAlign);
  const size_t scale_bytes = fp8 ? (size_t)(2 * L.rows + kStageTokens) * 4 : 0;
  L.slots = kDecodeSlots;
  L.part_o_off = align_up(L.scale_off + scale_bytes, kAlign);
  L.part_ml_off = align_up(L.part_o_off + (size_t)L.slots * kMaxGroup * p->head_dim * 4, kAlign);
  L.err_off = align_up(L.part_ml_off + (size_t)L.slots * kMaxGroup * 8, kAlign);
  // per-row lengths on the device, [layer][batch] int32, then the decode plan
  // table (int64): the cost line's length, the CTAs, the segment cost, and per
  // ring its place on the line and its keys
  L.lens_off = align_up(L.err_off + 64, kAlign);
  L.plan_off = align_up(L.lens_off + (size_t)p->n_layers * p->batch * 4, kAlign);
  L.total = align_up(L.plan_off + (size_t)(4 + 2 * p->batch * p->n_kv_heads) * 8, kAlign);
  return L;
}

PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static bool tried = false;
  if (!tried) {
    tried = true;
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  }
  return fn;
}

}  // namespace

struct hwkv_cache {
  hwkv_policy pol;
  std::vector<int64_t> windows, sinks;
  Layout lay;
  // tokens held per (layer, row), -1 = idle row: the host copy of the device
  // length array. A layer that has had a graph-mode step is advanced on the
  // device without the host knowing (graph replays), so its copy is re-read
  // before every use (dev_owned).
  mutable std::vector<int64_t> t;
  std::vector<char> dev_owned;  // per layer
  uint8_t* arena = nullptr;
  bool owns_arena = false;
  int num_sms = 0;
  CUtensorMap kv_map;  // 2-D view of the K and V regions: [2 * rows][head_dim] elements
  bool fp8() const { return pol.kv_format == HWKV_KV_FP8_E4M3; }
  size_t elem_bytes() const { return fp8() ? 1 : 2; }
  // bytes one resident token of one KV head occupies (K and V, with scales)
  size_t token_bytes() const { return fp8() ? 2 * ((size_t)pol.head_dim + 4) : 4 * (size_t)pol.head_dim; }
  __nv_bfloat16* k_base() const { return reinterpret_cast<__nv_bfloat16*>(arena); }
  float* scales() const { return fp8() ? reinterpret_cast<float*>(arena + lay.scale_off) : nullptr; }
  float* part_o() const { return reinterpret_cast<float*>(arena + lay.part_o_off); }
  float2* part_ml() const { return reinterpret_cast<float2*>(arena + lay.part_ml_off); }
  int* err() const { return reinterpret_cast<int*>(arena + lay.err_off); }
  int32_t* lens(int layer) const {
    return reinterpret_cast<int32_t*>(arena + lay.lens_off) + (size_t)layer * pol.batch;
  }
  int64_t* plan() const { return reinterpret_cast<int64_t*>(arena + lay.plan_off); }
  int64_t& row_t(int layer, int b) { return t[(size_t)layer * pol.batch + b]; }
  int64_t row_t(int layer, int b) const { return t[(size_t)layer * pol.batch + b]; }
  // true (and the length) when every row of the layer holds the same number of tokens
  bool uniform(int layer, int64_t* len) const {
    const int64_t t0 = row_t(layer, 0);
    for (int b = 1; b < pol.batch; ++b)
      if (row_t(layer, b) != t0) return false;
    if (t0 < 0) return false;
    *len = t0;
    return true;
  }
};

extern "C" {

const char* hwkv_last_error(void) { return g_last_error.c_str(); }

hwkv_status hwkv_required_bytes(const hwkv_policy* policy, size_t* arena_bytes) {
  if (!arena_bytes) return fail(HWKV_EINVAL, "arena_bytes is NULL");
  hwkv_status st = validate(policy);
  if (st != HWKV_OK) return st;
  *arena_bytes = make_layout(policy).total;
  return ok();
}

hwkv_status hwkv_alloc(const hwkv_policy* policy, void* dev_arena, size_t arena_bytes,
                       void* cuda_stream, hwkv_cache** out) {
  if (!out) return fail(HWKV_EINVAL, "out is NULL");
  *out = nullptr;
  hwkv_status st = validate(policy);
  if (st != HWKV_OK) return st;
  Layout lay = make_layout(policy);
  if (2 * lay.rows + kStageTokens >= (int64_t)INT32_MAX)
    return fail(HWKV_EUNSUPPORTED, "ring rows %lld exceed the 2^31 TMA coordinate range",
                (long long)(2 * lay.rows));
  if (dev_arena && arena_bytes < lay.total)
    return fail(HWKV_ENOMEM, "arena of %zu bytes < required %zu", arena_bytes, lay.total);
  if (dev_arena && (reinterpret_cast<uintptr_t>(dev_arena) % kAlign) != 0)
    return fail(HWKV_EINVAL, "dev_arena must be %zu-byte aligned", kAlign);
  auto encode = get_encode();
  if (!encode) return fail(HWKV_ECUDA, "cuTensorMapEncodeTiled entry point unavailable");
  {
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return fail(HWKV_ECUDA, "device query failed");
    if (2 * sms > kDecodeSlots)
      return fail(HWKV_EUNSUPPORTED, "%d SMs need more than the %d decode partial slots", sms,
                  kDecodeSlots);
  }

  hwkv_cache* c = new hwkv_cache();
  c->pol = *policy;
  c->windows.assign(policy->windows, policy->windows + (size_t)policy->n_layers * policy->n_kv_heads);
  c->pol.windows = c->windows.data();
  if (policy->sinks) {
    c->sinks.assign(policy->sinks, policy->sinks + (size_t)policy->n_layers * policy->n_kv_heads);
    c->pol.sinks = c->sinks.data();
  }
  c->lay = std::move(lay);
  c->t.assign((size_t)policy->n_layers * policy->batch, 0);
  c->dev_owned.assign(policy->n_layers, 0);
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) {
    delete c;
    return fail(HWKV_ECUDA, "device query failed: %s", cudaGetErrorString(e));
  }
  if (dev_arena) {
    c->arena = static_cast<uint8_t*>(dev_arena);
  } else {
    e = cudaMalloc(reinterpret_cast<void**>(&c->arena), c->lay.total);
    if (e != cudaSuccess) {
      delete c;
      return fail(HWKV_ENOMEM, "cudaMalloc(%zu) failed: %s", c->lay.total, cudaGetErrorString(e));
    }
    c->owns_arena = true;
  }
  e = decode_prepare_device();
  if (e != cudaSuccess) {
    if (c->owns_arena) cudaFree(c->arena);
    delete c;
    return fail(HWKV_ECUDA, "decode kernel attributes: %s", cudaGetErrorString(e));
  }
  e = cudaMemsetAsync(c->arena, 0, c->lay.total, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) {
    if (c->owns_arena) cudaFree(c->arena);
    delete c;
    return fail(HWKV_ECUDA, "zero-fill failed: %s", cudaGetErrorString(e));
  }
  // one tensor map over both regions: rows of head_dim bf16, boxes of 64 rows x 64 channels
  // (128-byte rows of boxes: 64 bf16 or 128 E4M3 channels)
  const cuuint64_t gdim[2] = {(cuuint64_t)c->pol.head_dim, (cuuint64_t)(2 * c->lay.rows)};
  const cuuint64_t gstride[1] = {(cuuint64_t)c->pol.head_dim * c->elem_bytes()};
  const cuuint32_t box[2] = {c->fp8() ? 128u : 64u, (cuuint32_t)kStageTokens};
  const cuuint32_t estride[2] = {1, 1};
  CUresult r = encode(&c->kv_map, c->fp8() ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16,
                      2, c->arena, gdim, gstride,
                      box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                      CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    if (c->owns_arena) cudaFree(c->arena);
    delete c;
    return fail(HWKV_ECUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
  }
  *out = c;
  return ok();
}

hwkv_status hwkv_free(hwkv_cache* c) {
  if (!c) return ok();
  if (c->owns_arena) cudaFree(c->arena);
  delete c;
  return ok();
}

static hwkv_status check_layer(const hwkv_cache* c, int32_t layer) {
  if (!c) return fail(HWKV_EINVAL, "cache is NULL");
  if (layer < 0 || layer >= c->pol.n_layers)
    return fail(HWKV_EINVAL, "layer %d out of range [0, %d)", layer, c->pol.n_layers);
  return HWKV_OK;
}

// Host calls that read the host copy of a layer's lengths: if graph-mode steps
// own the layer, wait for the device and re-read its lengths first.
static hwkv_status refresh_lens(const hwkv_cache* c, int32_t layer) {
  if (!c->dev_owned[layer]) return HWKV_OK;
  std::vector<int32_t> host(c->pol.batch);
  cudaError_t e = cudaDeviceSynchronize();
  if (e == cudaSuccess)
    e = cudaMemcpy(host.data(), c->lens(layer), host.size() * 4, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "length copy: %s", cudaGetErrorString(e));
  for (int b = 0; b < c->pol.batch; ++b) c->t[(size_t)layer * c->pol.batch + b] = host[b] < 0 ? -1 : host[b];
  return HWKV_OK;
}

static hwkv_status check_fresh(const hwkv_cache* c, int32_t layer) {
  hwkv_status st = check_layer(c, layer);
  if (st != HWKV_OK) return st;
  return refresh_lens(c, layer);
}

static hwkv_status check_rows(const hwkv_cache* c, int32_t row0, int32_t n_rows) {
  if (row0 < 0 || n_rows <= 0 || (int64_t)row0 + n_rows > c->pol.batch)
    return fail(HWKV_EINVAL, "rows [%d, %d + %d) outside the batch of %d", row0, row0, n_rows,
                c->pol.batch);
  return HWKV_OK;
}

static AppendParams append_params(const hwkv_cache* c, int32_t layer, int32_t row0,
                                  int32_t n_rows, const void* k, const void* v, int64_t n) {
  AppendParams p{};
  p.n_units = c->pol.n_kv_heads;
  p.batch = n_rows;
  p.row0 = row0;
  p.lens = c->lens(layer);
  for (int b = 0; b < n_rows; ++b) p.t0[b] = (int32_t)c->row_t(layer, row0 + b);
  p.n = n;
  p.d = c->pol.head_dim;
  p.k = static_cast<const __nv_bfloat16*>(k);
  p.v = static_cast<const __nv_bfloat16*>(v);
  p.k_arena = c->k_base();
  p.v_arena = c->k_base();  // V rows are addressed by v_row0, which already includes the K region
  p.scales = c->scales();
  for (int h = 0; h < p.n_units; ++h) {
    const Unit& u = c->lay.units[(size_t)layer * p.n_units + h];
    p.u[h] = AppendUnit{u.k_row0, u.v_row0, u.cap, u.stride, u.sink};
  }
  return p;
}

// rows [row0, row0 + n_rows) may each append n tokens: active, and within max_ctx
static hwkv_status check_room(const hwkv_cache* c, int32_t layer, int32_t row0, int32_t n_rows,
                              int64_t n) {
  for (int b = row0; b < row0 + n_rows; ++b) {
    const int64_t t = c->row_t(layer, b);
    if (t < 0) return fail(HWKV_EINVAL, "layer %d row %d is idle (hwkv_reset_rows makes it active)", layer, b);
    if (t + n > c->pol.max_ctx)
      return fail(HWKV_ECAPACITY, "layer %d row %d: t=%lld + n=%lld exceeds max_ctx=%lld", layer, b,
                  (long long)t, (long long)n, (long long)c->pol.max_ctx);
  }
  return HWKV_OK;
}

hwkv_status hwkv_append_rows(hwkv_cache* c, int32_t layer, int32_t row0, int32_t n_rows,
                             const void* k, const void* v, int64_t n, void* cuda_stream) {
  hwkv_status st = check_fresh(c, layer);
  if (st != HWKV_OK) return st;
  if ((st = check_rows(c, row0, n_rows)) != HWKV_OK) return st;
  if (n < 0) return fail(HWKV_EINVAL, "n must be >= 0");
  if (n == 0) return ok();
  if (!k || !v) return fail(HWKV_EINVAL, "k/v is NULL");
  if ((st = check_room(c, layer, row0, n_rows, n)) != HWKV_OK) return st;
  const AppendParams p = append_params(c, layer, row0, n_rows, k, v, n);
  cudaError_t e = launch_append(p, c->fp8(), static_cast<cudaStream_t>(cuda_stream));
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "append launch: %s", cudaGetErrorString(e));
  for (int b = row0; b < row0 + n_rows; ++b) c->row_t(layer, b) += n;
  return ok();
}

hwkv_status hwkv_append(hwkv_cache* c, int32_t layer, const void* k, const void* v, int64_t n,
                        void* cuda_stream) {
  if (!c) return fail(HWKV_EINVAL, "cache is NULL");
  return hwkv_append_rows(c, layer, 0, c->pol.batch, k, v, n, cuda_stream);
}

hwkv_status hwkv_prefill_rows(hwkv_cache* c, int32_t layer, int32_t row0, int32_t n_rows,
                              const void* q, const void* k, const void* v, int64_t n, float scale,
                              float* out, void* cuda_stream) {
  hwkv_status st = check_fresh(c, layer);
  if (st != HWKV_OK) return st;
  if ((st = check_rows(c, row0, n_rows)) != HWKV_OK) return st;
  if (n < 0) return fail(HWKV_EINVAL, "n must be >= 0");
  if (n == 0) return ok();
  if (!q || !k || !v || !out) return fail(HWKV_EINVAL, "q/k/v/out is NULL");
  if ((st = check_room(c, layer, row0, n_rows, n)) != HWKV_OK) return st;
  const int64_t t_rows = c->row_t(layer, row0);
  for (int b = row0 + 1; b < row0 + n_rows; ++b)
    if (c->row_t(layer, b) != t_rows)
      return fail(HWKV_EINVAL, "prefill rows must hold the same length (row %d: %lld, row %d: %lld)",
                  row0, (long long)t_rows, b, (long long)c->row_t(layer, b));
  if (!(scale > 0.f) || scale == INFINITY) return fail(HWKV_EINVAL, "scale must be positive and finite");
  if (n > (int64_t)65535 * 16) return fail(HWKV_EUNSUPPORTED, "chunk of %lld tokens too long", (long long)n);
  // the prefill kernel walks positions and ring slots in 32-bit arithmetic
  if (t_rows + n >= ((int64_t)1 << 30))
    return fail(HWKV_EUNSUPPORTED, "prefill past 2^30 tokens of history");
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  PrefillParams p{};
  p.n_units = c->pol.n_kv_heads;
  p.batch = n_rows;
  p.row0 = row0;
  p.group = c->pol.n_q_heads / c->pol.n_kv_heads;
  p.n_q_heads = c->pol.n_q_heads;
  p.t0 = t_rows;
  p.n = n;
  p.scale_log2 = scale * 1.4426950408889634f;
  p.q = static_cast<const __nv_bfloat16*>(q);
  p.k = static_cast<const __nv_bfloat16*>(k);
  p.v = static_cast<const __nv_bfloat16*>(v);
  p.k_arena = c->k_base();
  p.v_arena = c->k_base();
  p.out = out;
  p.err = c->err();
  for (int h = 0; h < p.n_units; ++h) {
    const Unit& u = c->lay.units[(size_t)layer * p.n_units + h];
    if (u.cap >= ((int64_t)1 << 30)) return fail(HWKV_EUNSUPPORTED, "prefill into a ring of 2^30 slots or more");
    // a window that reaches past every position the kernel can see is the full history
    p.u[h] = PrefillUnit{u.k_row0, u.v_row0, u.cap, u.window >= ((int64_t)1 << 30) ? 0 : u.window,
                         u.stride, u.sink};
  }
  // tensor maps of this call's q and chunk K/V: 3-D views {d, heads, batch * n}
  auto encode = get_encode();
  const int d = c->pol.head_dim, G = p.group, QP = 128 / G;
  const cuuint32_t estr[3] = {1, 1, 1};
  CUtensorMap q_map, ck_map, cv_map;
  {
    const cuuint64_t dim[3] = {(cuuint64_t)d, (cuuint64_t)c->pol.n_q_heads,
                               (cuuint64_t)n_rows * (cuuint64_t)n};
    const cuuint64_t str[2] = {(cuuint64_t)d * 2, (cuuint64_t)c->pol.n_q_heads * d * 2};
    const cuuint32_t box[3] = {64, (cuuint32_t)G, (cuuint32_t)QP};
    CUresult r = encode(&q_map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(q), dim, str,
                        box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(HWKV_EINVAL, "q tensor map rejected (%d): q must be 16-byte aligned", (int)r);
  }
  if ((int64_t)n_rows * n + 128 >= (int64_t)INT32_MAX)
    return fail(HWKV_EUNSUPPORTED, "batch x chunk exceeds the TMA coordinate range");
  const int H = c->pol.n_kv_heads;
  auto encode_chunk = [&](CUtensorMap* m, const void* base) -> CUresult {
    const cuuint64_t dim[3] = {(cuuint64_t)d, (cuuint64_t)H, (cuuint64_t)n_rows * (cuuint64_t)n};
    const cuuint64_t str[2] = {(cuuint64_t)d * 2, (cuuint64_t)H * d * 2};
    const cuuint32_t box[3] = {64, 1, 64};
    return encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dim, str, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  };
  cudaError_t e = cudaSuccess;
  if (!c->fp8()) {
    CUresult r = encode_chunk(&ck_map, k);
    if (r == CUDA_SUCCESS) r = encode_chunk(&cv_map, v);
    if (r != CUDA_SUCCESS) return fail(HWKV_EINVAL, "k/v tensor map rejected (%d): k/v must be 16-byte aligned", (int)r);
    e = launch_prefill_tc(p, d, q_map, ck_map, cv_map, c->kv_map, s);
    if (e != cudaSuccess) return fail(HWKV_ECUDA, "prefill launch: %s", cudaGetErrorString(e));
  } else {
    // 8-bit cache: attention reads every key as stored (code x row scale), the
    // chunk's own rows included. The held ring rows are staged dequantized and the
    // chunk quantized as the append will store it, then dequantized; with q they
    // go through the tensor cores in fp16 (11 significant bits).
    if (d != 128 && d != 256) return fail(HWKV_EUNSUPPORTED, "8-bit prefill needs head_dim 128 or 256");
    Fp8StageParams sp{};
    sp.n_units = H;
    sp.batch = n_rows;
    sp.row0 = row0;
    sp.n_q_heads = c->pol.n_q_heads;
    sp.t0 = t_rows;
    sp.n = n;
    sp.arena = reinterpret_cast<const uint8_t*>(c->k_base());
    sp.arena_scales = c->scales();
    sp.q = static_cast<const __nv_bfloat16*>(q);
    sp.k = static_cast<const __nv_bfloat16*>(k);
    sp.v = static_cast<const __nv_bfloat16*>(v);
    int64_t rows = 0;
    for (int h = 0; h < H; ++h) {
      const Unit& u = c->lay.units[(size_t)layer * H + h];
      sp.u[h] = Fp8StageUnit{u.k_row0, u.v_row0, u.cap, u.stride, u.sink, rows, rows + (int64_t)n_rows * u.cap};
      rows += 2 * (int64_t)n_rows * u.cap;
    }
    const size_t ring_bytes = align_up((size_t)rows * d * 2, 1024);
    const size_t kv_bytes = align_up((size_t)n_rows * n * H * d * 2, 1024);
    const size_t q_bytes = align_up((size_t)n_rows * n * c->pol.n_q_heads * d * 2, 1024);
    const size_t total = ring_bytes + 2 * kv_bytes + q_bytes;
    uint8_t* buf = nullptr;
    e = cudaMallocAsync(reinterpret_cast<void**>(&buf), total, s);
    if (e != cudaSuccess) return fail(HWKV_ENOMEM, "8-bit prefill staging (%zu bytes): %s", total, cudaGetErrorString(e));
    sp.ring = reinterpret_cast<uint16_t*>(buf);
    sp.k16 = reinterpret_cast<uint16_t*>(buf + ring_bytes);
    sp.v16 = reinterpret_cast<uint16_t*>(buf + ring_bytes + kv_bytes);
    sp.q16 = reinterpret_cast<uint16_t*>(buf + ring_bytes + 2 * kv_bytes);
    e = launch_fp8_stage(sp, d, s);
    CUtensorMap ring_map, q16_map;
    CUresult r = CUDA_SUCCESS;
    if (e == cudaSuccess) {
      const cuuint64_t gdim[2] = {(cuuint64_t)d, (cuuint64_t)rows};
      const cuuint64_t gstride[1] = {(cuuint64_t)d * 2};
      const cuuint32_t box[2] = {64u, (cuuint32_t)kStageTokens};
      const cuuint32_t es2[2] = {1, 1};
      r = encode(&ring_map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, sp.ring, gdim, gstride, box, es2,
                 CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                 CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
      // the staged copies have the input layouts; the maps only move 2-byte elements
      if (r == CUDA_SUCCESS) r = encode_chunk(&ck_map, sp.k16);
      if (r == CUDA_SUCCESS) r = encode_chunk(&cv_map, sp.v16);
      if (r == CUDA_SUCCESS) {
        const cuuint64_t dim[3] = {(cuuint64_t)d, (cuuint64_t)c->pol.n_q_heads,
                                   (cuuint64_t)n_rows * (cuuint64_t)n};
        const cuuint64_t str[2] = {(cuuint64_t)d * 2, (cuuint64_t)c->pol.n_q_heads * d * 2};
        const cuuint32_t qbox[3] = {64, (cuuint32_t)G, (cuuint32_t)QP};
        r = encode(&q16_map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, sp.q16, dim, str, qbox, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
      }
    }
    if (e == cudaSuccess && r == CUDA_SUCCESS) {
      for (int h = 0; h < H; ++h) {
        p.u[h].k_row0 = sp.u[h].sk_row0;
        p.u[h].v_row0 = sp.u[h].sv_row0;
        p.u[h].stride = sp.u[h].cap;
      }
      p.row0 = 0;
      e = launch_prefill_tc(p, d, q16_map, ck_map, cv_map, ring_map, s, true);
    }
    const cudaError_t ef = cudaFreeAsync(buf, s);
    if (r != CUDA_SUCCESS) return fail(HWKV_ECUDA, "8-bit prefill tensor maps rejected (%d)", (int)r);
    if (e != cudaSuccess) return fail(HWKV_ECUDA, "8-bit prefill launch: %s", cudaGetErrorString(e));
    if (ef != cudaSuccess) return fail(HWKV_ECUDA, "8-bit prefill staging free: %s", cudaGetErrorString(ef));
  }
  // attend first, then write the chunk's retained tokens (stream order)
  const AppendParams ap = append_params(c, layer, row0, n_rows, k, v, n);
  e = launch_append(ap, c->fp8(), s);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "append launch: %s", cudaGetErrorString(e));
  for (int b = row0; b < row0 + n_rows; ++b) c->row_t(layer, b) += n;
  return ok();
}

hwkv_status hwkv_prefill(hwkv_cache* c, int32_t layer, const void* q, const void* k,
                         const void* v, int64_t n, float scale, float* out, void* cuda_stream) {
  if (!c) return fail(HWKV_EINVAL, "cache is NULL");
  return hwkv_prefill_rows(c, layer, 0, c->pol.batch, q, k, v, n, scale, out, cuda_stream);
}

// CTAs of a decode split launch. A grid of one (shared-memory-filling) CTA on
// every SM cannot start until every SM is free, and leaves no room for the
// combine kernel's CTAs to become resident ahead of time; measured on GB300 that
// costs ~7 us per launch, more than 8 extra SMs gain below ~1 GB of K/V per
// layer-step. So small steps leave 8 SMs free. `tokens` = resident K/V rows the
// step reads (an estimate is enough: it changes speed, not results).
static int decode_grid_cap(const hwkv_cache* c, int64_t tokens) {
  const int sms = std::max(1, c->num_sms);
  const int64_t bytes = tokens * (int64_t)c->token_bytes();
  constexpr int64_t kFullGridBytes = 1LL << 30;
  return (bytes >= kFullGridBytes || sms <= 16) ? sms : sms - 8;
}

// resident K/V rows a step of `layer` reads, from the host copy of the lengths
static int64_t step_tokens(const hwkv_cache* c, int32_t layer, int add) {
  const int H = c->pol.n_kv_heads;
  int64_t n = 0;
  for (int b = 0; b < c->pol.batch; ++b) {
    const int64_t t = c->row_t(layer, b);
    if (t < 0) continue;
    for (int h = 0; h < H; ++h) n += std::min(t + add, c->lay.units[(size_t)layer * H + h].cap);
  }
  return n;
}

enum DecodeMode { kPlain = 0, kFused = 1, kFusedGraph = 2 };

// the fields of a ring-mode decode launch that do not depend on the call's tensors
static void ring_params(const hwkv_cache* c, int32_t layer, DecodeParams& p, int lens_inc) {
  p.n_units = c->pol.n_kv_heads;
  p.batch = c->pol.batch;
  p.group = c->pol.n_q_heads / c->pol.n_kv_heads;
  p.n_q_heads = c->pol.n_q_heads;
  p.err = c->err();
  p.lens = c->lens(layer);
  p.lens_inc = lens_inc;
  p.max_ctx = c->pol.max_ctx;
  p.scales = c->scales();
  // a segment's fixed cost (query load, merge, partial write) ~ the time to stream
  // 256 KB of K/V at one CTA's share of HBM bandwidth, in 64-key stages
  p.seg_cost = std::max(1, (int)((256 << 10) / c->token_bytes() / kStageTokens));
  for (int h = 0; h < p.n_units; ++h) {
    const Unit& u = c->lay.units[(size_t)layer * p.n_units + h];
    p.u[h] = DecodeUnit{u.k_row0, u.v_row0, u.cap, u.stride, u.sink};
  }
}

// One decode call of a layer: the split kernel plans its work on the GPU from
// the device lengths (so one launch serves uniform, ragged and idle rows, and
// replays correctly from a CUDA graph), then the combine kernel merges.
static hwkv_status decode_call(hwkv_cache* c, int32_t layer, const void* q, const void* k_new,
                               const void* v_new, float scale, float* out, void* cuda_stream,
                               DecodeMode mode) {
  hwkv_status st = mode == kFusedGraph ? check_layer(c, layer) : check_fresh(c, layer);
  if (st != HWKV_OK) return st;
  if (!q || !out) return fail(HWKV_EINVAL, "q/out is NULL");
  if (mode != kPlain && (!k_new || !v_new)) return fail(HWKV_EINVAL, "k_new/v_new is NULL");
  if (!(scale > 0.f) || scale == INFINITY) return fail(HWKV_EINVAL, "scale must be positive and finite");
  const int B = c->pol.batch;
  if (mode == kPlain) {
    bool any = false;
    for (int b = 0; b < B; ++b) any |= c->row_t(layer, b) > 0;
    if (!any) return fail(HWKV_EINVAL, "layer %d holds no tokens", layer);
  } else if (mode == kFused) {
    for (int b = 0; b < B; ++b)
      if (c->row_t(layer, b) + 1 > c->pol.max_ctx)
        return fail(HWKV_ECAPACITY, "layer %d row %d: t=%lld + 1 exceeds max_ctx=%lld", layer, b,
                    (long long)c->row_t(layer, b), (long long)c->pol.max_ctx);
  }
  DecodeParams p{};
  ring_params(c, layer, p, mode == kPlain ? 0 : 1);
  p.scale_log2 = scale * 1.4426950408889634f;
  p.q = static_cast<const __nv_bfloat16*>(q);
  p.part_o = c->part_o();
  p.part_ml = c->part_ml();
  p.out = out;
  p.plan = c->plan();
  if (mode != kPlain) {
    p.k_new = static_cast<const __nv_bfloat16*>(k_new);
    p.v_new = static_cast<const __nv_bfloat16*>(v_new);
    p.arena = c->k_base();
  }
  // the host copy of the lengths sizes the grid (stale under graph capture: an estimate)
  const int grid = decode_grid_cap(c, step_tokens(c, layer, mode == kPlain ? 0 : 1));
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  cudaError_t e = launch_decode(p, c->kv_map, c->kv_map, c->pol.head_dim, grid, s, c->fp8());
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "decode launch: %s", cudaGetErrorString(e));
  e = launch_decode_combine(p, c->pol.head_dim, c->num_sms, s);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "combine launch: %s", cudaGetErrorString(e));
  if (mode == kFused)
    for (int b = 0; b < B; ++b)
      if (c->row_t(layer, b) >= 0) c->row_t(layer, b) += 1;
  if (mode == kFusedGraph) c->dev_owned[layer] = 1;
  return ok();
}

hwkv_status hwkv_decode_attn(hwkv_cache* c, int32_t layer, const void* q, float scale, float* out,
                             void* cuda_stream) {
  return decode_call(c, layer, q, nullptr, nullptr, scale, out, cuda_stream, kPlain);
}

hwkv_status hwkv_decode_step(hwkv_cache* c, int32_t layer, const void* q, const void* k_new,
                             const void* v_new, float scale, float* out, void* cuda_stream) {
  return decode_call(c, layer, q, k_new, v_new, scale, out, cuda_stream, kFused);
}

hwkv_status hwkv_decode_step_graph(hwkv_cache* c, int32_t layer, const void* q, const void* k_new,
                                   const void* v_new, float scale, float* out, void* cuda_stream) {
  return decode_call(c, layer, q, k_new, v_new, scale, out, cuda_stream, kFusedGraph);
}

hwkv_status hwkv_sync_lens(hwkv_cache* c, void* cuda_stream) {
  if (!c) return fail(HWKV_EINVAL, "cache is NULL");
  const size_t n = (size_t)c->pol.n_layers * c->pol.batch;
  std::vector<int32_t> host(n);
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  cudaError_t e = cudaStreamSynchronize(s);
  if (e == cudaSuccess) e = cudaMemcpy(host.data(), c->lens(0), n * 4, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "length copy: %s", cudaGetErrorString(e));
  for (size_t i = 0; i < n; ++i) c->t[i] = host[i] < 0 ? -1 : host[i];
  return ok();
}

hwkv_status hwkv_reset_rows(hwkv_cache* c, int32_t row0, int32_t n_rows, int32_t idle,
                            void* cuda_stream) {
  if (!c) return fail(HWKV_EINVAL, "cache is NULL");
  hwkv_status st = check_rows(c, row0, n_rows);
  if (st != HWKV_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  for (int l = 0; l < c->pol.n_layers; ++l) {
    cudaError_t e = cudaMemsetAsync(c->lens(l) + row0, idle ? 0xFF : 0, (size_t)n_rows * 4, s);
    if (e != cudaSuccess) return fail(HWKV_ECUDA, "length reset: %s", cudaGetErrorString(e));
    for (int b = row0; b < row0 + n_rows; ++b) c->row_t(l, b) = idle ? -1 : 0;
  }
  return ok();
}

hwkv_status hwkv_row_len(const hwkv_cache* c, int32_t layer, int32_t row, int64_t* t) {
  hwkv_status st = check_fresh(c, layer);
  if (st != HWKV_OK) return st;
  if (row < 0 || row >= c->pol.batch || !t) return fail(HWKV_EINVAL, "bad row or NULL t");
  *t = c->row_t(layer, row);
  return ok();
}

hwkv_status hwkv_residency_bytes(const hwkv_cache* c, int32_t layer, uint64_t* bytes) {
  if (!c || !bytes) return fail(HWKV_EINVAL, "NULL argument");
  if (layer < -1 || layer >= c->pol.n_layers) return fail(HWKV_EINVAL, "layer out of range");
  const int H = c->pol.n_kv_heads;
  // d^K b^K + d^V b^V: bf16, or E4M3 codes plus a 4-byte scale per row
  const uint64_t per_token = c->token_bytes();
  uint64_t total = 0;
  for (int l = 0; l < c->pol.n_layers; ++l) {
    if (layer >= 0 && l != layer) continue;
    hwkv_status st = refresh_lens(c, l);
    if (st != HWKV_OK) return st;
    for (int h = 0; h < H; ++h) {
      const Unit& u = c->lay.units[(size_t)l * H + h];
      for (int b = 0; b < c->pol.batch; ++b)  // idle rows (-1) hold nothing
        total += (uint64_t)std::min(std::max<int64_t>(c->row_t(l, b), 0), u.cap) * per_token;
    }
  }
  *bytes = total;
  return ok();
}

hwkv_status hwkv_allocated_ring_bytes(const hwkv_cache* c, int32_t layer, uint64_t* bytes) {
  if (!c || !bytes) return fail(HWKV_EINVAL, "NULL argument");
  if (layer < -1 || layer >= c->pol.n_layers) return fail(HWKV_EINVAL, "layer out of range");
  const int H = c->pol.n_kv_heads;
  uint64_t total = 0;
  for (int l = 0; l < c->pol.n_layers; ++l) {
    if (layer >= 0 && l != layer) continue;
    for (int h = 0; h < H; ++h)  // rows held for the ring (codes and scales in 8 bits)
      total += (uint64_t)c->lay.units[(size_t)l * H + h].stride * c->token_bytes() *
               (uint64_t)c->pol.batch;
  }
  *bytes = total;
  return ok();
}

hwkv_status hwkv_seq_len(const hwkv_cache* c, int32_t layer, int64_t* t) {
  hwkv_status st = check_fresh(c, layer);
  if (st != HWKV_OK) return st;
  if (!t) return fail(HWKV_EINVAL, "t is NULL");
  if (!c->uniform(layer, t))
    return fail(HWKV_EINVAL, "layer %d rows hold different lengths (or are idle): use hwkv_row_len",
                layer);
  return ok();
}

hwkv_status hwkv_ring_capacity(const hwkv_cache* c, int32_t layer, int32_t kv_head, int64_t* cap) {
  hwkv_status st = check_layer(c, layer);
  if (st != HWKV_OK) return st;
  if (kv_head < 0 || kv_head >= c->pol.n_kv_heads || !cap)
    return fail(HWKV_EINVAL, "bad kv_head or NULL cap");
  *cap = c->lay.units[(size_t)layer * c->pol.n_kv_heads + kv_head].cap;
  return ok();
}

hwkv_status hwkv_debug_copy_ring(const hwkv_cache* c, int32_t layer, int32_t b, int32_t kv_head,
                                 void* k_host, void* v_host) {
  hwkv_status st = check_layer(c, layer);
  if (st != HWKV_OK) return st;
  if (b < 0 || b >= c->pol.batch || kv_head < 0 || kv_head >= c->pol.n_kv_heads || !k_host ||
      !v_host)
    return fail(HWKV_EINVAL, "bad ring coordinates or NULL buffer");
  const Unit& u = c->lay.units[(size_t)layer * c->pol.n_kv_heads + kv_head];
  const size_t row = (size_t)c->pol.head_dim * c->elem_bytes();
  const uint8_t* kb = c->arena + (size_t)(u.k_row0 + (int64_t)b * u.stride) * row;
  const uint8_t* vb = c->arena + (size_t)(u.v_row0 + (int64_t)b * u.stride) * row;
  cudaError_t e = cudaDeviceSynchronize();
  if (e == cudaSuccess) e = cudaMemcpy(k_host, kb, (size_t)u.cap * row, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess) e = cudaMemcpy(v_host, vb, (size_t)u.cap * row, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "ring copy: %s", cudaGetErrorString(e));
  return ok();
}

hwkv_status hwkv_debug_copy_scales(const hwkv_cache* c, int32_t layer, int32_t b, int32_t kv_head,
                                   float* k_scales, float* v_scales) {
  hwkv_status st = check_layer(c, layer);
  if (st != HWKV_OK) return st;
  if (!c->fp8()) return fail(HWKV_EINVAL, "the cache is not in the 8-bit format");
  if (b < 0 || b >= c->pol.batch || kv_head < 0 || kv_head >= c->pol.n_kv_heads || !k_scales ||
      !v_scales)
    return fail(HWKV_EINVAL, "bad ring coordinates or NULL buffer");
  const Unit& u = c->lay.units[(size_t)layer * c->pol.n_kv_heads + kv_head];
  const float* ks = c->scales() + u.k_row0 + (int64_t)b * u.stride;
  const float* vs = c->scales() + u.v_row0 + (int64_t)b * u.stride;
  cudaError_t e = cudaDeviceSynchronize();
  if (e == cudaSuccess) e = cudaMemcpy(k_scales, ks, (size_t)u.cap * 4, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess) e = cudaMemcpy(v_scales, vs, (size_t)u.cap * 4, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "scale copy: %s", cudaGetErrorString(e));
  return ok();
}

hwkv_status hwkv_sync_check(hwkv_cache* c) {
  if (!c) return fail(HWKV_EINVAL, "cache is NULL");
  int word = 0;
  cudaError_t e = cudaDeviceSynchronize();
  if (e == cudaSuccess) e = cudaMemcpy(&word, c->err(), sizeof word, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "sync: %s", cudaGetErrorString(e));
  if (word != 0) {
    cudaMemset(c->err(), 0, sizeof(int));
    return fail(HWKV_EKERNEL, "kernel error word 0x%x (1 = bounded wait gave up, 2 = bad index, "
                "4 = a graph-mode step skipped a row at max_ctx)",
                word);
  }
  return ok();
}

hwkv_status hwkv_debug_wait_probe(hwkv_cache* c, int64_t limit_ns, void* cuda_stream) {
  if (!c) return fail(HWKV_EINVAL, "cache is NULL");
  if (limit_ns < 1000000 || limit_ns > 2000000000)
    return fail(HWKV_EINVAL, "limit_ns %lld outside [1e6, 2e9]", (long long)limit_ns);
  cudaError_t e = launch_wait_probe(c->err(), (uint64_t)limit_ns, static_cast<cudaStream_t>(cuda_stream));
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "wait probe launch: %s", cudaGetErrorString(e));
  return ok();
}

// ---------------------------------------------------------------------------
// Decode without any device allocation. Some callers cannot allocate device
// memory at all: code embedded in another engine whose allocator owns every
// byte of the GPU, code that must never synchronize the device (cudaMalloc and
// cudaFree can), and code issued while a stream is being captured. They own
// the cache arena and the q/out tensors, but cannot provide scratch. This
// entry point keeps the decode tile partials in a fixed array that lives in
// the library's own device image instead of the cache's workspace.
//
// The array is HWKV_DECODE_STATIC_SCRATCH_BYTES (4 MiB) on every GPU that
// loads this library, held until the process exits. Host code cannot use the
// array's name as a device address (on the host it is only a stand-in), so
// the first call on each device, with that device current, looks the address
// up with cudaGetSymbolAddress and keeps it; that first call should come
// before any stream capture. Every call shares the array and it keeps the
// last call's contents; nothing in it has to start at zero (each tile partial
// is written before it is read). Calls whose kernels overlap on the GPU (two
// streams, or two caches, at once) race on it.
static __device__ __align__(256) uint8_t g_decode_static_scratch[HWKV_DECODE_STATIC_SCRATCH_BYTES];

// Byte layout of the static scratch for a decode launch of `grid` CTAs: two
// partial slots per CTA (outputs, then (max, sum) pairs), then the plan table.
struct StaticScratch {
  size_t o_bytes, ml_bytes, plan_bytes;
  size_t total() const { return o_bytes + ml_bytes + plan_bytes; }
};
static StaticScratch static_scratch_layout(int grid, int head_dim, int batch, int n_kv_heads) {
  StaticScratch s;
  s.o_bytes = align_up((size_t)2 * grid * kMaxGroup * head_dim * 4, kAlign);
  s.ml_bytes = align_up((size_t)2 * grid * kMaxGroup * 8, kAlign);
  s.plan_bytes = align_up((size_t)(4 + 2 * (size_t)batch * n_kv_heads) * 8, kAlign);
  return s;
}

hwkv_status hwkv_decode_static_scratch_bytes(const hwkv_policy* policy, int32_t num_sms,
                                             size_t* bytes) {
  if (!bytes) return fail(HWKV_EINVAL, "bytes is NULL");
  hwkv_status st = validate(policy);
  if (st != HWKV_OK) return st;
  if (num_sms <= 0) return fail(HWKV_EINVAL, "num_sms must be positive");
  const StaticScratch s =
      static_scratch_layout(num_sms, policy->head_dim, policy->batch, policy->n_kv_heads);
  *bytes = s.total();
  if (s.total() > HWKV_DECODE_STATIC_SCRATCH_BYTES)
    return fail(HWKV_EINVAL, "static decode needs %zu scratch bytes > %u", s.total(),
                (unsigned)HWKV_DECODE_STATIC_SCRATCH_BYTES);
  return ok();
}

// The array's device address per device ordinal, looked up once and kept for
// the life of the process (a device reset would leave it stale; not supported).
static void* static_scratch_address(int device, cudaError_t* err) {
  constexpr int kMaxDevices = 64;
  static std::mutex mu;
  static void* addr[kMaxDevices] = {};
  std::lock_guard<std::mutex> lock(mu);
  *err = cudaSuccess;
  if (device < 0 || device >= kMaxDevices) {
    *err = cudaErrorInvalidDevice;
    return nullptr;
  }
  if (!addr[device]) {
    void* ptr = nullptr;
    *err = cudaGetSymbolAddress(&ptr, g_decode_static_scratch);
    if (*err != cudaSuccess) return nullptr;
    addr[device] = ptr;
  }
  return addr[device];
}

hwkv_status hwkv_decode_attn_static(hwkv_cache* c, int32_t layer, const void* q, float scale,
                                    float* out, void* cuda_stream) {
  // no length refresh here: that would synchronize the device. The kernels plan
  // from the device lengths; the host copy only sizes the grid (an estimate when
  // graph-mode steps own the layer), and rows holding nothing decode to zeros.
  hwkv_status st = check_layer(c, layer);
  if (st != HWKV_OK) return st;
  if (!q || !out) return fail(HWKV_EINVAL, "q/out is NULL");
  if (!(scale > 0.f) || scale == INFINITY) return fail(HWKV_EINVAL, "scale must be positive and finite");
  if (!c->dev_owned[layer]) {
    bool any = false;
    for (int b = 0; b < c->pol.batch; ++b) any |= c->row_t(layer, b) > 0;
    if (!any) return fail(HWKV_EINVAL, "layer %d holds no tokens", layer);
  }
  const int d = c->pol.head_dim;
  const int grid = decode_grid_cap(c, step_tokens(c, layer, 0));
  const StaticScratch sl = static_scratch_layout(grid, d, c->pol.batch, c->pol.n_kv_heads);
  if (sl.total() > HWKV_DECODE_STATIC_SCRATCH_BYTES)
    return fail(HWKV_EINVAL, "static decode needs %zu scratch bytes > %u", sl.total(),
                (unsigned)HWKV_DECODE_STATIC_SCRATCH_BYTES);
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "cudaGetDevice: %s", cudaGetErrorString(e));
  uint8_t* scratch = static_cast<uint8_t*>(static_scratch_address(dev, &e));
  if (!scratch)
    return fail(HWKV_ECUDA, "cudaGetSymbolAddress(static decode scratch) on device %d: %s", dev,
                cudaGetErrorString(e));
  DecodeParams p{};
  ring_params(c, layer, p, 0);
  p.scale_log2 = scale * 1.4426950408889634f;
  p.q = static_cast<const __nv_bfloat16*>(q);
  p.part_o = reinterpret_cast<float*>(scratch);
  p.part_ml = reinterpret_cast<float2*>(scratch + sl.o_bytes);
  p.plan = reinterpret_cast<int64_t*>(scratch + sl.o_bytes + sl.ml_bytes);
  p.out = out;
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  e = launch_decode(p, c->kv_map, c->kv_map, d, grid, s, c->fp8());
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "decode launch: %s", cudaGetErrorString(e));
  e = launch_decode_combine(p, d, c->num_sms, s);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "combine launch: %s", cudaGetErrorString(e));
  return ok();
}

// ---------------------------------------------------------------------------
// SeqCalib candidate replay and selection (Sec. 3.2, Eq. conditional-similarity
// and Eq. threshold-selection; App. A.2, Eq. stabilized-cosine and
// Eq. budget-selector).

static hwkv_status calib_validate(const hwkv_calib_desc* d) {
  if (!d) return fail(HWKV_EINVAL, "calib desc is NULL");
  if (d->n_seq <= 0 || d->n_pos <= 0 || d->n_kv_heads <= 0 || d->n_q_heads <= 0 || d->T <= 0)
    return fail(HWKV_EINVAL, "calib sizes must be positive");
  if (d->n_q_heads % d->n_kv_heads != 0) return fail(HWKV_EINVAL, "n_q_heads must be a multiple of n_kv_heads");
  if (d->n_q_heads / d->n_kv_heads > kMaxGroup) return fail(HWKV_EUNSUPPORTED, "GQA group > 8");
  if (d->head_dim != 64 && d->head_dim != 128 && d->head_dim != 256)
    return fail(HWKV_EUNSUPPORTED, "head_dim %d not built", d->head_dim);
  if (d->n_windows < 1 || d->n_windows > 8) return fail(HWKV_EUNSUPPORTED, "1..8 candidate windows");
  if (!d->windows || !d->positions) return fail(HWKV_EINVAL, "windows/positions is NULL");
  for (int k = 0; k < d->n_windows; ++k)
    if (d->windows[k] <= 0 || (k > 0 && d->windows[k] <= d->windows[k - 1]))
      return fail(HWKV_EINVAL, "candidate windows must be positive and increasing");
  for (int64_t i = 0; i < (int64_t)d->n_seq * d->n_pos; ++i)
    if (d->positions[i] < 0 || d->positions[i] >= d->T)
      return fail(HWKV_EINVAL, "position %lld outside [0, T)", (long long)d->positions[i]);
  if ((int64_t)d->n_seq * d->n_kv_heads * d->T + kStageTokens >= (int64_t)INT32_MAX)
    return fail(HWKV_EUNSUPPORTED, "trace rows exceed the TMA coordinate range");
  return HWKV_OK;
}

struct CalibPlan {
  std::vector<CalibTile> tiles;
  std::vector<int32_t> band_begin;  // [units][K + 2]
  int64_t units = 0;
  size_t off_tiles = 0, off_bands = 0, off_o = 0, off_ml = 0, off_cos = 0, off_tcos = 0;
  size_t off_err = 0, total = 0;
};

// Nested-suffix bands of position t for increasing windows W[0..K-1]: band 0 =
// [t-W0+1, t], band k = [t-Wk+1, t-W(k-1)], band K = [0, t-W(K-1)] (clipped at 0),
// each cut into tiles of at most tile_len keys.
static CalibPlan calib_plan(const hwkv_calib_desc* d) {
  CalibPlan P;
  const int K = d->n_windows, H = d->n_kv_heads, G = d->n_q_heads / d->n_kv_heads;
  P.units = (int64_t)d->n_seq * d->n_pos * H;
  int64_t total_keys = 0;
  for (int64_t i = 0; i < (int64_t)d->n_seq * d->n_pos; ++i) total_keys += (d->positions[i] + 1) * H;
  int64_t tile_len = (total_keys / 1216 + 63) / 64 * 64;  // about 8 tiles per SM of 152
  tile_len = std::min<int64_t>(8192, std::max<int64_t>(512, tile_len));
  P.band_begin.reserve(P.units * (K + 2));
  for (int n = 0; n < d->n_seq; ++n)
    for (int pp = 0; pp < d->n_pos; ++pp)
      for (int h = 0; h < H; ++h) {
        const int64_t t = d->positions[(int64_t)n * d->n_pos + pp];
        const int64_t row0 = ((int64_t)n * H + h) * d->T;
        for (int k = 0; k <= K; ++k) {
          const int64_t hi = k == 0 ? t : t - d->windows[k - 1];
          const int64_t lo = k == K ? 0 : std::max<int64_t>(0, t - d->windows[k] + 1);
          P.band_begin.push_back((int32_t)P.tiles.size());
          for (int64_t s0 = lo; s0 <= hi; s0 += tile_len) {
            CalibTile ct{};
            ct.k_row = row0 + s0;
            ct.v_row = row0 + s0;
            ct.len = (int32_t)std::min<int64_t>(tile_len, hi - s0 + 1);
            ct.q_row = n * d->n_pos + pp;
            ct.h = h;
            P.tiles.push_back(ct);
          }
        }
        P.band_begin.push_back((int32_t)P.tiles.size());
      }
  const size_t nt = std::max<size_t>(P.tiles.size(), 1);
  P.off_tiles = 0;
  P.off_bands = align_up(nt * sizeof(CalibTile), kAlign);
  P.off_o = align_up(P.off_bands + P.band_begin.size() * 4, kAlign);
  P.off_ml = align_up(P.off_o + nt * kMaxGroup * d->head_dim * 4, kAlign);
  P.off_cos = align_up(P.off_ml + nt * kMaxGroup * 8, kAlign);
  P.off_tcos = align_up(P.off_cos + (size_t)P.units * G * K * 4, kAlign);
  P.off_err = align_up(P.off_tcos + (size_t)P.units * G * 4, kAlign);
  P.total = align_up(P.off_err + 64, kAlign);
  return P;
}

hwkv_status hwkv_calib_workspace_bytes(const hwkv_calib_desc* d, size_t* bytes) {
  if (!bytes) return fail(HWKV_EINVAL, "bytes is NULL");
  hwkv_status st = calib_validate(d);
  if (st != HWKV_OK) return st;
  *bytes = calib_plan(d).total;
  return ok();
}

// The replay shared by hwkv_calib_scores and hwkv_calib_trace_check: fills cosv
// [units][G][K] and, with traced, tcos [units][G]; synchronizes the stream.
static hwkv_status calib_run(const hwkv_calib_desc* d, const void* q, const void* k,
                             const void* v, float scale, void* workspace, size_t ws_bytes,
                             const float* traced, std::vector<float>& cosv,
                             std::vector<float>& tcos, void* cuda_stream) {
  hwkv_status st = calib_validate(d);
  if (st != HWKV_OK) return st;
  if (!q || !k || !v || !workspace) return fail(HWKV_EINVAL, "NULL argument");
  if (!(scale > 0.f) || scale == INFINITY) return fail(HWKV_EINVAL, "scale must be positive and finite");
  const CalibPlan P = calib_plan(d);
  if (ws_bytes < P.total) return fail(HWKV_ENOMEM, "workspace %zu < required %zu", ws_bytes, P.total);
  auto encode = get_encode();
  if (!encode) return fail(HWKV_ECUDA, "cuTensorMapEncodeTiled entry point unavailable");
  const int D = d->head_dim, H = d->n_kv_heads, G = d->n_q_heads / d->n_kv_heads, K = d->n_windows;
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  // trace maps: head-major [n_seq][n_kv_heads][T][D] seen as rows of D bf16
  CUtensorMap kmap, vmap;
  const cuuint64_t gdim[2] = {(cuuint64_t)D, (cuuint64_t)d->n_seq * H * d->T};
  const cuuint64_t gstr[1] = {(cuuint64_t)D * 2};
  const cuuint32_t box[2] = {64, (cuuint32_t)kStageTokens};
  const cuuint32_t est[2] = {1, 1};
  CUresult r = encode(&kmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(k), gdim, gstr,
                      box, est, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                      CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r == CUDA_SUCCESS)
    r = encode(&vmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(v), gdim, gstr, box,
               est, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(HWKV_EINVAL, "trace tensor map rejected (%d): k/v must be 16-byte aligned", (int)r);
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess && !P.tiles.empty())
    e = cudaMemcpyAsync(ws + P.off_tiles, P.tiles.data(), P.tiles.size() * sizeof(CalibTile),
                        cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(ws + P.off_bands, P.band_begin.data(), P.band_begin.size() * 4,
                        cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = cudaMemsetAsync(ws + P.off_err, 0, 64, s);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "calib setup: %s", cudaGetErrorString(e));
  DecodeParams p{};
  p.n_units = H;
  p.batch = 1;
  p.group = G;
  p.n_q_heads = d->n_q_heads;
  p.scale_log2 = scale * 1.4426950408889634f;
  p.q = static_cast<const __nv_bfloat16*>(q);
  p.part_o = reinterpret_cast<float*>(ws + P.off_o);
  p.part_ml = reinterpret_cast<float2*>(ws + P.off_ml);
  p.err = reinterpret_cast<int*>(ws + P.off_err);
  p.tiles = reinterpret_cast<const CalibTile*>(ws + P.off_tiles);
  p.n_tiles = (int32_t)P.tiles.size();
  if (p.n_tiles > 0) {
    e = launch_decode(p, kmap, vmap, D, std::min(p.n_tiles, std::max(1, sms)), s);
    if (e != cudaSuccess) return fail(HWKV_ECUDA, "calib tile launch: %s", cudaGetErrorString(e));
  }
  CalibCombineParams cp{};
  cp.n_units = (int32_t)P.units;
  cp.group = G;
  cp.n_windows = K;
  cp.scale_log2 = p.scale_log2;
  cp.band_begin = reinterpret_cast<const int32_t*>(ws + P.off_bands);
  cp.part_o = p.part_o;
  cp.part_ml = p.part_ml;
  cp.cos = reinterpret_cast<float*>(ws + P.off_cos);
  cp.traced = traced;
  cp.trace_cos = reinterpret_cast<float*>(ws + P.off_tcos);
  e = launch_calib_combine(cp, D, s);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "calib combine launch: %s", cudaGetErrorString(e));
  cosv.assign((size_t)P.units * G * K, 0.f);
  tcos.assign(traced ? (size_t)P.units * G : 0, 0.f);
  int err_word = 0;
  e = cudaMemcpyAsync(cosv.data(), cp.cos, cosv.size() * 4, cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess && traced)
    e = cudaMemcpyAsync(tcos.data(), cp.trace_cos, tcos.size() * 4, cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaMemcpyAsync(&err_word, p.err, sizeof(int), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "calib readback: %s", cudaGetErrorString(e));
  if (err_word != 0) return fail(HWKV_EKERNEL, "calib kernel error word 0x%x", err_word);
  return HWKV_OK;
}

hwkv_status hwkv_calib_scores(const hwkv_calib_desc* d, const void* q, const void* k,
                              const void* v, float scale, void* workspace, size_t ws_bytes,
                              double* scores, float* cos_out, void* cuda_stream) {
  if (!scores) return fail(HWKV_EINVAL, "scores is NULL");
  std::vector<float> cosv, tcos;
  hwkv_status st = calib_run(d, q, k, v, scale, workspace, ws_bytes, nullptr, cosv, tcos, cuda_stream);
  if (st != HWKV_OK) return st;
  const int H = d->n_kv_heads, G = d->n_q_heads / d->n_kv_heads, K = d->n_windows;
  // Eq. conditional-similarity: mean over (sequence, position, query head), fixed order
  const double inv = 1.0 / ((double)d->n_seq * d->n_pos * G);
  for (int h = 0; h < H; ++h)
    for (int kk = 0; kk < K; ++kk) {
      double acc = 0.0;
      for (int64_t np = 0; np < (int64_t)d->n_seq * d->n_pos; ++np)
        for (int g = 0; g < G; ++g) acc += cosv[((np * H + h) * G + g) * K + kk];
      scores[h * K + kk] = acc * inv;
    }
  if (cos_out)  // [n_seq][n_pos][n_q_heads][K]
    for (int64_t np = 0; np < (int64_t)d->n_seq * d->n_pos; ++np)
      for (int h = 0; h < H; ++h)
        for (int g = 0; g < G; ++g)
          for (int kk = 0; kk < K; ++kk)
            cos_out[((np * d->n_q_heads) + h * G + g) * K + kk] = cosv[((np * H + h) * G + g) * K + kk];
  return ok();
}

hwkv_status hwkv_calib_trace_check(const hwkv_calib_desc* d, const void* q, const void* k,
                                   const void* v, float scale, const float* traced,
                                   double threshold, void* workspace, size_t ws_bytes,
                                   double* min_cos, float* trace_cos_out, void* cuda_stream) {
  if (!traced || !min_cos) return fail(HWKV_EINVAL, "traced/min_cos is NULL");
  std::vector<float> cosv, tcos;
  hwkv_status st = calib_run(d, q, k, v, scale, workspace, ws_bytes, traced, cosv, tcos, cuda_stream);
  if (st != HWKV_OK) return st;
  double m = 1.0;
  int64_t worst = 0;
  for (size_t i = 0; i < tcos.size(); ++i)
    if ((double)tcos[i] < m) {
      m = tcos[i];
      worst = (int64_t)i;
    }
  *min_cos = m;
  if (trace_cos_out) std::copy(tcos.begin(), tcos.end(), trace_cos_out);  // [N][P][n_q_heads]
  if (m < threshold) {
    const int64_t Hq = d->n_q_heads;
    return fail(HWKV_ETRACE,
                "trace check failed: replayed full-window output of (sequence %lld, position "
                "index %lld, query head %lld) has cosine %.6f < %.3f against the trace",
                (long long)(worst / Hq / d->n_pos), (long long)(worst / Hq % d->n_pos),
                (long long)(worst % Hq), m, threshold);
  }
  return ok();
}

hwkv_status hwkv_calib_select(const double* scores, int32_t n_heads, const int64_t* windows,
                              int32_t n_windows, int64_t C, double tau, int64_t* policy) {
  if (!scores || !windows || !policy || n_heads <= 0 || n_windows < 0 || C <= 0)
    return fail(HWKV_EINVAL, "bad selection arguments");
  for (int k = 1; k < n_windows; ++k)
    if (windows[k] <= windows[k - 1]) return fail(HWKV_EINVAL, "windows must be increasing");
  for (int h = 0; h < n_heads; ++h) {
    // candidates in <_W order: finite windows increasing, then full (score one)
    int64_t pick = HWKV_WINDOW_FULL, pick_cost = C;
    for (int k = n_windows - 1; k >= 0; --k) {  // scan backwards: the earliest minimum wins
      if (!(scores[(int64_t)h * n_windows + k] >= tau)) continue;
      const int64_t cost = std::min(windows[k], C);
      if (cost <= pick_cost) {
        pick = windows[k];
        pick_cost = cost;
      }
    }
    policy[h] = pick;
  }
  return ok();
}

hwkv_status hwkv_budget_select(const double* beta, const double* phi, int32_t n_records,
                               double budget, int32_t* chosen) {
  if (!beta || !phi || !chosen || n_records < 0) return fail(HWKV_EINVAL, "bad selector arguments");
  int32_t best = -1;
  for (int32_t g = 0; g < n_records; ++g) {
    if (!(beta[g] <= budget)) continue;
    const bool better = best < 0 || phi[g] > phi[best] || (phi[g] == phi[best] && beta[g] < beta[best]);
    if (better) best = g;
  }
  *chosen = best;
  return ok();
}

// ---------------------------------------------------------------------------
// Policy artifact I/O (App. "Experimental Protocol" / "Runtime Realization").

static bool artifact_id_ok(const char* a) {
  if (!a) return false;
  size_t n = strlen(a);
  if (n == 0 || n > 127) return false;
  for (size_t i = 0; i < n; ++i)
    if (a[i] <= ' ' || a[i] > '~') return false;
  return true;
}

hwkv_status hwkv_policy_save(const char* path, const char* artifact, uint64_t seed,
                             int32_t n_layers, int32_t n_kv_heads, const int64_t* windows) {
  if (!path || !windows || n_layers <= 0 || n_kv_heads <= 0)
    return fail(HWKV_EINVAL, "bad policy save arguments");
  if (!artifact_id_ok(artifact))
    return fail(HWKV_EINVAL, "artifact id must be 1..127 printable characters without spaces");
  for (int64_t i = 0; i < (int64_t)n_layers * n_kv_heads; ++i)
    if (windows[i] < 0) return fail(HWKV_EINVAL, "negative window at entry %lld", (long long)i);
  FILE* f = fopen(path, "w");
  if (!f) return fail(HWKV_EINVAL, "cannot open %s for writing", path);
  fprintf(f, "hwkv-policy 1\nartifact %s\nseed %llu\nshape %d %d\n", artifact,
          (unsigned long long)seed, n_layers, n_kv_heads);
  for (int l = 0; l < n_layers; ++l) {
    fprintf(f, "layer %d", l);
    for (int h = 0; h < n_kv_heads; ++h) fprintf(f, " %lld", (long long)windows[(int64_t)l * n_kv_heads + h]);
    fputc('\n', f);
  }
  const bool bad = ferror(f) != 0;
  if (fclose(f) != 0 || bad) return fail(HWKV_EINVAL, "write to %s failed", path);
  return ok();
}

hwkv_status hwkv_policy_load(const char* path, char* artifact, size_t artifact_cap, uint64_t* seed,
                             int32_t* n_layers, int32_t* n_kv_heads, int64_t* windows_out,
                             size_t capacity) {
  if (!path || !artifact || artifact_cap == 0 || !seed || !n_layers || !n_kv_heads || !windows_out)
    return fail(HWKV_EINVAL, "bad policy load arguments");
  FILE* f = fopen(path, "r");
  if (!f) return fail(HWKV_EINVAL, "cannot open %s", path);
  char line[1 << 16];
  int lineno = 0, stage = 0, next_layer = 0;
  int32_t L = 0, H = 0;
  hwkv_status st = HWKV_OK;
  auto bad = [&](const char* what) {
    st = fail(HWKV_EINVAL, "%s:%d: %s", path, lineno, what);
    return false;
  };
  while (st == HWKV_OK && fgets(line, sizeof line, f)) {
    ++lineno;
    if (!strchr(line, '\n') && !feof(f)) { bad("line too long"); break; }
    char* hash = strchr(line, '#');
    if (hash) *hash = '\0';
    char* tok = strtok(line, " \t\r\n");
    if (!tok) continue;  // blank or comment-only line
    const bool header = stage < 4;
    if (stage == 0) {
      char* v = strtok(nullptr, " \t\r\n");
      if (strcmp(tok, "hwkv-policy") != 0 || !v || strcmp(v, "1") != 0) { bad("expected 'hwkv-policy 1'"); break; }
      stage = 1;
    } else if (stage == 1) {
      char* v = strtok(nullptr, " \t\r\n");
      if (strcmp(tok, "artifact") != 0 || !v || !artifact_id_ok(v) || strlen(v) + 1 > artifact_cap) {
        bad("expected 'artifact <id>' fitting the buffer");
        break;
      }
      strcpy(artifact, v);
      stage = 2;
    } else if (stage == 2) {
      char* v = strtok(nullptr, " \t\r\n");
      char* end = nullptr;
      if (strcmp(tok, "seed") != 0 || !v || v[0] == '-') { bad("expected 'seed <n>'"); break; }
      errno = 0;
      unsigned long long sv = strtoull(v, &end, 10);
      if (errno != 0 || !end || *end != '\0') { bad("bad seed"); break; }
      *seed = (uint64_t)sv;
      stage = 3;
    } else if (stage == 3) {
      char* a = strtok(nullptr, " \t\r\n");
      char* b = strtok(nullptr, " \t\r\n");
      char *ea = nullptr, *eb = nullptr;
      long la = a ? strtol(a, &ea, 10) : 0, lb = b ? strtol(b, &eb, 10) : 0;
      if (strcmp(tok, "shape") != 0 || !a || !b || *ea || *eb || la <= 0 || lb <= 0 ||
          la > 4096 || lb > 4096) { bad("expected 'shape <n_layers> <n_kv_heads>'"); break; }
      L = (int32_t)la;
      H = (int32_t)lb;
      if ((size_t)L * (size_t)H > capacity) { bad("policy larger than the output capacity"); break; }
      stage = 4;
    } else {
      char* ls = strtok(nullptr, " \t\r\n");
      char* e = nullptr;
      long li = ls ? strtol(ls, &e, 10) : -1;
      if (strcmp(tok, "layer") != 0 || !ls || *e || li != next_layer || next_layer >= L) {
        bad("expected the next 'layer <l> ...' line");
        break;
      }
      for (int h = 0; h < H; ++h) {
        char* w = strtok(nullptr, " \t\r\n");
        char* ew = nullptr;
        errno = 0;
        long long wv = w ? strtoll(w, &ew, 10) : -1;
        if (!w || *ew || errno != 0 || wv < 0) { bad("expected a non-negative window per KV head"); break; }
        windows_out[(size_t)next_layer * H + h] = (int64_t)wv;
      }
      if (st != HWKV_OK) break;
      if (strtok(nullptr, " \t\r\n")) { bad("more windows than KV heads"); break; }
      ++next_layer;
    }
    if (header && strtok(nullptr, " \t\r\n")) { bad("unexpected extra field"); break; }
  }
  fclose(f);
  if (st != HWKV_OK) return st;
  if (stage < 4 || next_layer != L) return fail(HWKV_EINVAL, "%s: incomplete policy (%d of %d layers)", path, next_layer, L);
  *n_layers = L;
  *n_kv_heads = H;
  return ok();
}

}  // extern "C"
