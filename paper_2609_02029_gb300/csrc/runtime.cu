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
  int64_t k_row0, v_row0;
};

struct Layout {
  std::vector<Unit> units;  // [layer * n_kv_heads + h]
  int64_t rows = 0;         // K rows (= V rows)
  size_t ring_bytes = 0;    // K + V
  size_t part_o_off = 0, part_ml_off = 0, err_off = 0, total = 0;
  int max_tiles = 0;
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
  for (int64_t i = 0; i < (int64_t)p->n_layers * p->n_kv_heads; ++i)
    if (p->windows[i] < 0)
      return fail(HWKV_EINVAL, "window of (layer %lld, kv head %lld) is negative",
                  (long long)(i / p->n_kv_heads), (long long)(i % p->n_kv_heads));
  if (p->head_dim != 64 && p->head_dim != 128 && p->head_dim != 256)
    return fail(HWKV_EUNSUPPORTED, "head_dim %d not built (64, 128, 256)", p->head_dim);
  if (p->n_q_heads / p->n_kv_heads > kMaxGroup)
    return fail(HWKV_EUNSUPPORTED, "GQA group %d > %d", p->n_q_heads / p->n_kv_heads, kMaxGroup);
  if (p->n_kv_heads > kMaxKvHeads)
    return fail(HWKV_EUNSUPPORTED, "n_kv_heads %d > %d", p->n_kv_heads, kMaxKvHeads);
  if (p->batch > 256) return fail(HWKV_EUNSUPPORTED, "batch %d > 256", p->batch);
  return HWKV_OK;
}

Layout make_layout(const hwkv_policy* p) {
  Layout L;
  const int nu = p->n_layers * p->n_kv_heads;
  L.units.resize(nu);
  for (int i = 0; i < nu; ++i) {
    const int64_t W = p->windows[i];
    Unit& u = L.units[i];
    u.window = (W == HWKV_WINDOW_FULL || W >= p->max_ctx) ? 0 : W;  // w >= C is full (Sec. 3.1)
    u.cap = u.window == 0 ? p->max_ctx : u.window;
  }
  // group by level: larger capacity first, then layer, then head
  std::vector<int> order(nu);
  for (int i = 0; i < nu; ++i) order[i] = i;
  std::stable_sort(order.begin(), order.end(),
                   [&](int a, int b) { return L.units[a].cap > L.units[b].cap; });
  int64_t row = 0;
  for (int i : order) {
    L.units[i].k_row0 = row;
    row += L.units[i].cap * p->batch;
  }
  L.rows = row;
  for (auto& u : L.units) u.v_row0 = u.k_row0 + L.rows;
  const size_t row_bytes = (size_t)p->head_dim * 2;
  L.ring_bytes = (size_t)(2 * L.rows) * row_bytes;
  L.max_tiles = std::max(2048, 2 * p->batch * p->n_kv_heads);
  L.part_o_off = align_up(L.ring_bytes, kAlign);
  L.part_ml_off =
      align_up(L.part_o_off + (size_t)L.max_tiles * kMaxGroup * p->head_dim * 4, kAlign);
  L.err_off = align_up(L.part_ml_off + (size_t)L.max_tiles * kMaxGroup * 8, kAlign);
  L.total = align_up(L.err_off + 64, kAlign);
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
  std::vector<int64_t> windows;
  Layout lay;
  std::vector<int64_t> t;  // tokens held, per layer
  uint8_t* arena = nullptr;
  bool owns_arena = false;
  int num_sms = 0;
  CUtensorMap kv_map;  // 2-D view of the K and V regions: [2 * rows][head_dim] bf16
  __nv_bfloat16* k_base() const { return reinterpret_cast<__nv_bfloat16*>(arena); }
  __nv_bfloat16* v_base() const { return k_base() + lay.rows * pol.head_dim; }
  float* part_o() const { return reinterpret_cast<float*>(arena + lay.part_o_off); }
  float2* part_ml() const { return reinterpret_cast<float2*>(arena + lay.part_ml_off); }
  int* err() const { return reinterpret_cast<int*>(arena + lay.err_off); }
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

  hwkv_cache* c = new hwkv_cache();
  c->pol = *policy;
  c->windows.assign(policy->windows, policy->windows + (size_t)policy->n_layers * policy->n_kv_heads);
  c->pol.windows = c->windows.data();
  c->lay = std::move(lay);
  c->t.assign(policy->n_layers, 0);
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
  e = cudaMemsetAsync(c->arena, 0, c->lay.total, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) {
    if (c->owns_arena) cudaFree(c->arena);
    delete c;
    return fail(HWKV_ECUDA, "zero-fill failed: %s", cudaGetErrorString(e));
  }
  // one tensor map over both regions: rows of head_dim bf16, boxes of 64 rows x 64 channels
  const cuuint64_t gdim[2] = {(cuuint64_t)c->pol.head_dim, (cuuint64_t)(2 * c->lay.rows)};
  const cuuint64_t gstride[1] = {(cuuint64_t)c->pol.head_dim * 2};
  const cuuint32_t box[2] = {64, (cuuint32_t)kStageTokens};
  const cuuint32_t estride[2] = {1, 1};
  CUresult r = encode(&c->kv_map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, c->arena, gdim, gstride,
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

static AppendParams append_params(const hwkv_cache* c, int32_t layer, const void* k,
                                  const void* v, int64_t n) {
  AppendParams p{};
  p.n_units = c->pol.n_kv_heads;
  p.batch = c->pol.batch;
  p.t0 = c->t[layer];
  p.n = n;
  p.d = c->pol.head_dim;
  p.k = static_cast<const __nv_bfloat16*>(k);
  p.v = static_cast<const __nv_bfloat16*>(v);
  p.k_arena = c->k_base();
  p.v_arena = c->k_base();  // V rows are addressed by v_row0, which already includes the K region
  for (int h = 0; h < p.n_units; ++h) {
    const Unit& u = c->lay.units[(size_t)layer * p.n_units + h];
    p.u[h] = AppendUnit{u.k_row0, u.v_row0, u.cap};
  }
  return p;
}

hwkv_status hwkv_append(hwkv_cache* c, int32_t layer, const void* k, const void* v, int64_t n,
                        void* cuda_stream) {
  hwkv_status st = check_layer(c, layer);
  if (st != HWKV_OK) return st;
  if (n < 0) return fail(HWKV_EINVAL, "n must be >= 0");
  if (n == 0) return ok();
  if (!k || !v) return fail(HWKV_EINVAL, "k/v is NULL");
  if (c->t[layer] + n > c->pol.max_ctx)
    return fail(HWKV_ECAPACITY, "layer %d: t=%lld + n=%lld exceeds max_ctx=%lld", layer,
                (long long)c->t[layer], (long long)n, (long long)c->pol.max_ctx);
  const AppendParams p = append_params(c, layer, k, v, n);
  cudaError_t e = launch_append(p, static_cast<cudaStream_t>(cuda_stream));
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "append launch: %s", cudaGetErrorString(e));
  c->t[layer] += n;
  return ok();
}

hwkv_status hwkv_prefill(hwkv_cache* c, int32_t layer, const void* q, const void* k,
                         const void* v, int64_t n, float scale, float* out, void* cuda_stream) {
  hwkv_status st = check_layer(c, layer);
  if (st != HWKV_OK) return st;
  if (n < 0) return fail(HWKV_EINVAL, "n must be >= 0");
  if (n == 0) return ok();
  if (!q || !k || !v || !out) return fail(HWKV_EINVAL, "q/k/v/out is NULL");
  if (c->t[layer] + n > c->pol.max_ctx)
    return fail(HWKV_ECAPACITY, "layer %d: t=%lld + n=%lld exceeds max_ctx=%lld", layer,
                (long long)c->t[layer], (long long)n, (long long)c->pol.max_ctx);
  if (!(scale > 0.f) || scale == INFINITY) return fail(HWKV_EINVAL, "scale must be positive and finite");
  if (n > (int64_t)65535 * 16) return fail(HWKV_EUNSUPPORTED, "chunk of %lld tokens too long", (long long)n);
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  PrefillParams p{};
  p.n_units = c->pol.n_kv_heads;
  p.batch = c->pol.batch;
  p.group = c->pol.n_q_heads / c->pol.n_kv_heads;
  p.n_q_heads = c->pol.n_q_heads;
  p.t0 = c->t[layer];
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
    p.u[h] = PrefillUnit{u.k_row0, u.v_row0, u.cap, u.window};
  }
  // tensor maps of this call's q and chunk K/V: 3-D views {d, heads, batch * n}
  auto encode = get_encode();
  const int d = c->pol.head_dim, G = p.group, QP = 128 / G;
  const cuuint32_t estr[3] = {1, 1, 1};
  CUtensorMap q_map, ck_map, cv_map;
  {
    const cuuint64_t dim[3] = {(cuuint64_t)d, (cuuint64_t)c->pol.n_q_heads,
                               (cuuint64_t)c->pol.batch * (cuuint64_t)n};
    const cuuint64_t str[2] = {(cuuint64_t)d * 2, (cuuint64_t)c->pol.n_q_heads * d * 2};
    const cuuint32_t box[3] = {64, (cuuint32_t)G, (cuuint32_t)QP};
    CUresult r = encode(&q_map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(q), dim, str,
                        box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(HWKV_EINVAL, "q tensor map rejected (%d): q must be 16-byte aligned", (int)r);
  }
  {
    const cuuint64_t dim[3] = {(cuuint64_t)d, (cuuint64_t)c->pol.n_kv_heads,
                               (cuuint64_t)c->pol.batch * (cuuint64_t)n};
    const cuuint64_t str[2] = {(cuuint64_t)d * 2, (cuuint64_t)c->pol.n_kv_heads * d * 2};
    const cuuint32_t box[3] = {64, 1, 64};
    CUresult r = encode(&ck_map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(k), dim,
                        str, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r == CUDA_SUCCESS)
      r = encode(&cv_map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(v), dim, str,
                 box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                 CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(HWKV_EINVAL, "k/v tensor map rejected (%d): k/v must be 16-byte aligned", (int)r);
  }
  if ((int64_t)c->pol.batch * n + 128 >= (int64_t)INT32_MAX)
    return fail(HWKV_EUNSUPPORTED, "batch x chunk exceeds the TMA coordinate range");
  cudaError_t e = launch_prefill_tc(p, d, q_map, ck_map, cv_map, c->kv_map, s);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "prefill launch: %s", cudaGetErrorString(e));
  // attend first, then write the chunk's retained tokens (stream order)
  const AppendParams ap = append_params(c, layer, k, v, n);
  e = launch_append(ap, s);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "append launch: %s", cudaGetErrorString(e));
  c->t[layer] += n;
  return ok();
}

// Decode tile plan: equal-length tiles (multiple of 64 tokens) over every
// (batch row, KV head) ring. The length is chosen to balance the persistent
// grid: minimise (tiles per CTA) x (tile length + a fixed per-tile cost).
static void plan_decode(const hwkv_cache* c, int32_t layer, int max_tiles, DecodeParams& p,
                        int& grid, int64_t t) {
  const int H = c->pol.n_kv_heads, B = c->pol.batch;
  int64_t n_valid[kMaxKvHeads];
  int64_t longest = 0;
  for (int h = 0; h < H; ++h) {
    const Unit& u = c->lay.units[(size_t)layer * H + h];
    n_valid[h] = std::min(t, u.cap);
    longest = std::max(longest, n_valid[h]);
  }
  const int sms = std::max(1, c->num_sms);
  auto count = [&](int64_t len) {
    int64_t n = 0;
    for (int h = 0; h < H; ++h) n += (n_valid[h] + len - 1) / len;
    return n * B;
  };
  const int64_t per_tile_cost = 96;  // tokens-equivalent of a tile's fixed cost
  int64_t best_len = 0;
  double best = 0;
  const int64_t max_len = std::max<int64_t>(64, (longest + 63) / 64 * 64);
  for (int64_t len = 128; ; len = len < 1024 ? len + 64 : len + len / 8 / 64 * 64) {
    const int64_t L = std::min(len, max_len);
    const int64_t nt = count(L);
    if (nt <= max_tiles) {
      const int64_t g = std::min<int64_t>(nt, sms);
      const double cost = (double)((nt + g - 1) / g) * (double)(L + per_tile_cost);
      if (best_len == 0 || cost < best) {
        best = cost;
        best_len = L;
      }
    }
    if (L >= max_len) break;
  }
  if (best_len == 0) best_len = max_len;
  p.tile_len = (int32_t)best_len;
  int32_t begin = 0;
  for (int h = 0; h < H; ++h) {
    const Unit& u = c->lay.units[(size_t)layer * H + h];
    DecodeUnit& du = p.u[h];
    du.k_row0 = u.k_row0;
    du.v_row0 = u.v_row0;
    du.cap = u.cap;
    du.n_valid = (int32_t)n_valid[h];
    du.n_tiles = (int32_t)((n_valid[h] + best_len - 1) / best_len);
    du.tile_begin = begin;
    du.s_new = (int32_t)((t - 1) % u.cap);  // slot of the newest token (fused step)
    begin += du.n_tiles;
  }
  p.tiles_per_b = begin;
  p.n_tiles = begin * B;
  // per-ring tiles are bounded by max_tiles / batch <= max(2048, 2 * n_kv_heads) < kCombineMaxTiles
  grid = std::min(p.n_tiles, sms);
}

hwkv_status hwkv_decode_attn(hwkv_cache* c, int32_t layer, const void* q, float scale, float* out,
                             void* cuda_stream) {
  hwkv_status st = check_layer(c, layer);
  if (st != HWKV_OK) return st;
  if (!q || !out) return fail(HWKV_EINVAL, "q/out is NULL");
  if (!(scale > 0.f) || scale == INFINITY) return fail(HWKV_EINVAL, "scale must be positive and finite");
  if (c->t[layer] <= 0) return fail(HWKV_EINVAL, "layer %d holds no tokens", layer);
  if (c->t[layer] > INT32_MAX) return fail(HWKV_EUNSUPPORTED, "ring longer than 2^31");
  DecodeParams p{};
  p.n_units = c->pol.n_kv_heads;
  p.batch = c->pol.batch;
  p.group = c->pol.n_q_heads / c->pol.n_kv_heads;
  p.n_q_heads = c->pol.n_q_heads;
  p.scale_log2 = scale * 1.4426950408889634f;
  p.q = static_cast<const __nv_bfloat16*>(q);
  p.part_o = c->part_o();
  p.part_ml = c->part_ml();
  p.out = out;
  p.err = c->err();
  int grid = 0;
  plan_decode(c, layer, c->lay.max_tiles, p, grid, c->t[layer]);
  if (p.n_tiles > c->lay.max_tiles)
    return fail(HWKV_EUNSUPPORTED, "decode plan needs %d tiles > %d", p.n_tiles, c->lay.max_tiles);
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  cudaError_t e = launch_decode(p, c->kv_map, c->kv_map, c->pol.head_dim, grid, s);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "decode launch: %s", cudaGetErrorString(e));
  e = launch_decode_combine(p, c->pol.head_dim, s);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "combine launch: %s", cudaGetErrorString(e));
  return ok();
}

hwkv_status hwkv_decode_step(hwkv_cache* c, int32_t layer, const void* q, const void* k_new,
                             const void* v_new, float scale, float* out, void* cuda_stream) {
  hwkv_status st = check_layer(c, layer);
  if (st != HWKV_OK) return st;
  if (!q || !out || !k_new || !v_new) return fail(HWKV_EINVAL, "q/k_new/v_new/out is NULL");
  if (!(scale > 0.f) || scale == INFINITY) return fail(HWKV_EINVAL, "scale must be positive and finite");
  if (c->t[layer] + 1 > c->pol.max_ctx)
    return fail(HWKV_ECAPACITY, "layer %d: t=%lld + 1 exceeds max_ctx=%lld", layer,
                (long long)c->t[layer], (long long)c->pol.max_ctx);
  if (c->t[layer] + 1 > INT32_MAX) return fail(HWKV_EUNSUPPORTED, "ring longer than 2^31");
  DecodeParams p{};
  p.n_units = c->pol.n_kv_heads;
  p.batch = c->pol.batch;
  p.group = c->pol.n_q_heads / c->pol.n_kv_heads;
  p.n_q_heads = c->pol.n_q_heads;
  p.scale_log2 = scale * 1.4426950408889634f;
  p.q = static_cast<const __nv_bfloat16*>(q);
  p.part_o = c->part_o();
  p.part_ml = c->part_ml();
  p.out = out;
  p.err = c->err();
  p.k_new = static_cast<const __nv_bfloat16*>(k_new);
  p.v_new = static_cast<const __nv_bfloat16*>(v_new);
  p.arena = c->k_base();
  int grid = 0;
  plan_decode(c, layer, c->lay.max_tiles, p, grid, c->t[layer] + 1);  // state after the append
  if (p.n_tiles > c->lay.max_tiles)
    return fail(HWKV_EUNSUPPORTED, "decode plan needs %d tiles > %d", p.n_tiles, c->lay.max_tiles);
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  cudaError_t e = launch_decode(p, c->kv_map, c->kv_map, c->pol.head_dim, grid, s);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "decode launch: %s", cudaGetErrorString(e));
  e = launch_decode_combine(p, c->pol.head_dim, s);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "combine launch: %s", cudaGetErrorString(e));
  c->t[layer] += 1;
  return ok();
}

hwkv_status hwkv_residency_bytes(const hwkv_cache* c, int32_t layer, uint64_t* bytes) {
  if (!c || !bytes) return fail(HWKV_EINVAL, "NULL argument");
  if (layer < -1 || layer >= c->pol.n_layers) return fail(HWKV_EINVAL, "layer out of range");
  const int H = c->pol.n_kv_heads;
  const uint64_t per_token = (uint64_t)c->pol.head_dim * 2 * 2;  // d^K b^K + d^V b^V, bf16
  uint64_t total = 0;
  for (int l = 0; l < c->pol.n_layers; ++l) {
    if (layer >= 0 && l != layer) continue;
    for (int h = 0; h < H; ++h) {
      const Unit& u = c->lay.units[(size_t)l * H + h];
      total += (uint64_t)std::min(c->t[l], u.cap) * per_token * (uint64_t)c->pol.batch;
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
    for (int h = 0; h < H; ++h)
      total += (uint64_t)c->lay.units[(size_t)l * H + h].cap * c->pol.head_dim * 4 *
               (uint64_t)c->pol.batch;
  }
  *bytes = total;
  return ok();
}

hwkv_status hwkv_seq_len(const hwkv_cache* c, int32_t layer, int64_t* t) {
  hwkv_status st = check_layer(c, layer);
  if (st != HWKV_OK) return st;
  if (!t) return fail(HWKV_EINVAL, "t is NULL");
  *t = c->t[layer];
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
  const size_t row = (size_t)c->pol.head_dim * 2;
  const uint8_t* kb = c->arena + (size_t)(u.k_row0 + (int64_t)b * u.cap) * row;
  const uint8_t* vb = c->arena + (size_t)(u.v_row0 + (int64_t)b * u.cap) * row;
  cudaError_t e = cudaDeviceSynchronize();
  if (e == cudaSuccess) e = cudaMemcpy(k_host, kb, (size_t)u.cap * row, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess) e = cudaMemcpy(v_host, vb, (size_t)u.cap * row, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "ring copy: %s", cudaGetErrorString(e));
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
    return fail(HWKV_EKERNEL, "kernel error word 0x%x (1 = bounded wait gave up, 2 = bad index)",
                word);
  }
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
  hwkv_status st = check_layer(c, layer);
  if (st != HWKV_OK) return st;
  if (!q || !out) return fail(HWKV_EINVAL, "q/out is NULL");
  if (c->t[layer] <= 0) return fail(HWKV_EINVAL, "layer %d holds no tokens", layer);
  if (c->t[layer] > INT32_MAX) return fail(HWKV_EUNSUPPORTED, "ring longer than 2^31");
  const int d = c->pol.head_dim;
  const size_t o_bytes_per_tile = (size_t)kMaxGroup * d * 4;
  const size_t ml_bytes_per_tile = (size_t)kMaxGroup * 8;
  const int cap_tiles =
      (int)((HWKV_DECODE_STATIC_SCRATCH_BYTES - kAlign) / (o_bytes_per_tile + ml_bytes_per_tile));
  const int min_tiles = c->pol.batch * c->pol.n_kv_heads;  // one tile per (batch row, KV head)
  if (min_tiles > cap_tiles)
    return fail(HWKV_EINVAL,
                "batch x n_kv_heads = %d exceeds the %d tiles the %d-byte static decode scratch "
                "holds at head_dim %d",
                min_tiles, cap_tiles, (int)HWKV_DECODE_STATIC_SCRATCH_BYTES, d);
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "cudaGetDevice: %s", cudaGetErrorString(e));
  uint8_t* scratch = static_cast<uint8_t*>(static_scratch_address(dev, &e));
  if (!scratch)
    return fail(HWKV_ECUDA, "cudaGetSymbolAddress(static decode scratch) on device %d: %s", dev,
                cudaGetErrorString(e));
  DecodeParams p{};
  p.n_units = c->pol.n_kv_heads;
  p.batch = c->pol.batch;
  p.group = c->pol.n_q_heads / c->pol.n_kv_heads;
  p.n_q_heads = c->pol.n_q_heads;
  p.scale_log2 = scale * 1.4426950408889634f;
  p.q = static_cast<const __nv_bfloat16*>(q);
  p.part_o = reinterpret_cast<float*>(scratch);
  p.part_ml = reinterpret_cast<float2*>(scratch + align_up((size_t)cap_tiles * o_bytes_per_tile, kAlign));
  p.out = out;
  p.err = c->err();
  int grid = 0;
  plan_decode(c, layer, cap_tiles, p, grid, c->t[layer]);
  if (p.n_tiles > cap_tiles)
    return fail(HWKV_EINVAL, "decode plan needs %d tiles > %d in the static scratch", p.n_tiles,
                cap_tiles);
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  e = launch_decode(p, c->kv_map, c->kv_map, d, grid, s);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "decode launch: %s", cudaGetErrorString(e));
  e = launch_decode_combine(p, d, s);
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
  size_t off_tiles = 0, off_bands = 0, off_o = 0, off_ml = 0, off_cos = 0, off_err = 0, total = 0;
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
  P.off_err = align_up(P.off_cos + (size_t)P.units * G * K * 4, kAlign);
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

hwkv_status hwkv_calib_scores(const hwkv_calib_desc* d, const void* q, const void* k,
                              const void* v, float scale, void* workspace, size_t ws_bytes,
                              double* scores, float* cos_out, void* cuda_stream) {
  hwkv_status st = calib_validate(d);
  if (st != HWKV_OK) return st;
  if (!q || !k || !v || !workspace || !scores) return fail(HWKV_EINVAL, "NULL argument");
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
  p.tiles_per_b = p.n_tiles;
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
  e = launch_calib_combine(cp, D, s);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "calib combine launch: %s", cudaGetErrorString(e));
  std::vector<float> cosv((size_t)P.units * G * K);
  int err_word = 0;
  e = cudaMemcpyAsync(cosv.data(), cp.cos, cosv.size() * 4, cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaMemcpyAsync(&err_word, p.err, sizeof(int), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return fail(HWKV_ECUDA, "calib readback: %s", cudaGetErrorString(e));
  if (err_word != 0) return fail(HWKV_EKERNEL, "calib kernel error word 0x%x", err_word);
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
