// hwkv_internal.cuh -- shared device helpers and launch parameter blocks of libhwkv.
//
// Inline PTX for sm_103a: mbarrier (with bounded waits that report through an
// error word instead of spinning forever), TMA tensor loads, ldmatrix, warp-level
// bf16 mma and movmatrix.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

namespace hwkv {

constexpr int kMaxKvHeads = 64;
constexpr int kMaxGroup = 8;          // query heads per KV head handled by one mma n-tile
constexpr int kDecodeWarps = 4;       // consumer warps per decode CTA
constexpr int kStageTokens = 64;      // tokens per pipeline stage (16 per consumer warp)
constexpr int kSlabBytes = 64 * 128;  // one TMA box: 64 rows x 128 B (64 bf16)

// error word bits (set with atomicOr, read by hwkv_sync_check)
constexpr int kErrWaitTimeout = 1;
constexpr int kErrBadIndex = 2;
constexpr int kErrCapacity = 4;  // a device-length step found a row at max_ctx (row skipped)

constexpr int kMaxBatch = 256;
constexpr int kDecodeSlots = 512;  // decode partial slots in the cache workspace (2 per CTA)

// ------------------------------------------------------------------ decode
struct DecodeUnit {
  int64_t k_row0;   // arena row of (this KV head, batch row 0) in the K region
  int64_t v_row0;   // same in the V region
  int64_t cap;      // ring capacity (slots)
  int64_t stride;   // rows between batch rows: batch row b starts at row0 + b * stride
  int64_t sink;     // sink slots: positions < sink stay in slots 0..sink-1
};

// ring slot of position p: sinks first, then the window region of cap - sink slots
__host__ __device__ __forceinline__ int64_t ring_slot(int64_t p, int64_t cap, int64_t sink) {
  return p < sink ? p : sink + (p - sink) % (cap - sink);
}

// a tile of explicit key rows (SeqCalib replay): rows k_row.. / v_row.. of the trace
// maps, queries of row q_row of q, KV head h
struct CalibTile {
  int64_t k_row, v_row;
  int32_t len, q_row, h, pad;
};

// Ring mode (tiles == nullptr): the rings of one layer, planned on the GPU from the
// per-row lengths. Table mode: an explicit tile list (SeqCalib replay).
struct DecodeParams {
  int32_t n_units;      // KV heads of the layer
  int32_t batch;
  int32_t group;        // G = n_q_heads / n_kv_heads
  int32_t n_q_heads;
  int32_t n_tiles;      // table mode: tiles in `tiles`
  float scale_log2;     // scale * log2(e)
  const __nv_bfloat16* q;  // [batch][n_q_heads][D]
  float* part_o;           // [slots][kMaxGroup][D]: unnormalised partial outputs
  float2* part_ml;         // [slots][kMaxGroup]: (max logit, sum of weights)
  float* out;              // [batch][n_q_heads][D]
  int* err;
  // fused step (append the new token, then attend): k_new/v_new [batch][n_units][D];
  // the new token's row is patched into the staged tile and written to the ring
  const __nv_bfloat16* k_new;  // null: plain decode over the current ring contents
  const __nv_bfloat16* v_new;
  __nv_bfloat16* arena;        // K/V rows: row r at arena + r * D (bytes r * D for 8-bit)
  float* scales;               // 8-bit format: fp32 scale of K/V row r at scales[r]
  const CalibTile* tiles;      // table mode: tiles[n_tiles]; every tile leaves a partial
  // ring mode: per-row lengths of this layer on the device, [batch]: tokens held by
  // row b before this call, -1 = idle row. With lens_inc = 1 (fused step) the new
  // token counts and the combine kernel advances every active row by one.
  int32_t* lens;
  int32_t lens_inc;
  int64_t max_ctx;      // rows whose step would pass max_ctx are skipped (kErrCapacity)
  int32_t seg_cost;     // fixed cost of a segment, in 64-key stages (F of the plan)
  int64_t* plan;        // [4 + 2 * batch * n_units]: Lt, G, F, -, then (L_u, n_u) per ring
  DecodeUnit u[kMaxKvHeads];
};

struct CalibCombineParams {
  int32_t n_units;      // (sequence, position, KV head) units
  int32_t group;        // G
  int32_t n_windows;    // K candidate windows (bands K + 1)
  float scale_log2;
  const int32_t* band_begin;  // [n_units][K + 2]: first tile of each band, then the end
  const float* part_o;        // [tiles][kMaxGroup][D]
  const float2* part_ml;      // [tiles][kMaxGroup]
  float* cos;                 // [n_units][G][K]
  const float* traced;        // NULL, or [n_units][G][D]: traced full-history outputs
  float* trace_cos;           // with traced: [n_units][G] cos_eval(replayed full, traced)
};

// ------------------------------------------------------------------ append
struct AppendUnit {
  int64_t k_row0, v_row0, cap, stride, sink;
};

struct AppendParams {
  int32_t n_units, batch;  // batch = rows of this call, cache rows row0 .. row0 + batch - 1
  int32_t row0;
  int32_t* lens;   // the layer's per-row lengths on the device; row r gets t0[r - row0] + n
  int32_t t0[kMaxBatch];  // position of the first new token, per row of the call
  int64_t n;       // new tokens
  int64_t d;       // head_dim
  const __nv_bfloat16* k;  // [batch][n][n_units][d]
  const __nv_bfloat16* v;
  __nv_bfloat16* k_arena;  // row r at k_arena + r * d (bytes r * d for 8-bit)
  __nv_bfloat16* v_arena;
  float* scales;           // 8-bit format: scale of row r at scales[r]
  AppendUnit u[kMaxKvHeads];
  // grid x of one batch row: KV head h owns blocks [blk0[h], blk0[h + 1]), sized for its
  // own landing rows (at most min(n, cap))
  int32_t blk0[kMaxKvHeads + 1];
};

// KV head whose block range [blk0[h], blk0[h + 1]) holds block x (x < blk0[n_units])
__device__ __forceinline__ int append_block_head(const AppendParams& p, int32_t x) {
  int lo = 0, hi = p.n_units - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (p.blk0[mid] <= x) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// ------------------------------------------------------------------ prefill
struct PrefillUnit {
  int64_t k_row0, v_row0, cap;
  int64_t window;  // 0 = full
  int64_t stride;  // rows between batch rows
  int64_t sink;    // sink slots before the window region
};

struct PrefillParams {
  int32_t n_units, batch, group, n_q_heads;  // batch = rows of this call
  int32_t row0;                              // first cache row of the call
  int64_t t0;  // first chunk position (tokens already in the cache)
  int64_t n;   // chunk length
  float scale_log2;
  const __nv_bfloat16* q;   // [batch][n][n_q_heads][D]
  const __nv_bfloat16* k;   // [batch][n][n_units][D]
  const __nv_bfloat16* v;
  const __nv_bfloat16* k_arena;
  const __nv_bfloat16* v_arena;
  float* out;               // [batch][n][n_q_heads][D]
  int* err;
  PrefillUnit u[kMaxKvHeads];
};

// Staging of an 8-bit cache for prefill, everything in fp16 for an fp16 tensor-core
// pass: the visible ring rows of one layer dequantized (code x scale), the chunk's
// K/V rows quantized exactly as the append stores them and dequantized, and q.
struct Fp8StageUnit {
  int64_t k_row0, v_row0, cap, stride, sink;  // arena rows
  int64_t sk_row0, sv_row0;                   // staging rows (batch row b at + b * cap)
};
struct Fp8StageParams {
  int32_t n_units, batch, row0, n_q_heads;
  int64_t t0, n;
  const uint8_t* arena;           // E4M3 codes, one row of D bytes per arena row
  const float* arena_scales;      // per arena row
  uint16_t* ring;                 // staging rows x D, fp16
  const __nv_bfloat16* q;         // chunk input [batch][n][n_q_heads][D]
  const __nv_bfloat16* k;         // chunk input [batch][n][n_units][D]
  const __nv_bfloat16* v;
  uint16_t* q16;                  // the same layouts, fp16
  uint16_t* k16;
  uint16_t* v16;
  Fp8StageUnit u[kMaxKvHeads];
};

// launchers (defined in the kernel translation units); return cudaGetLastError()
cudaError_t launch_append(const AppendParams& p, bool fp8, cudaStream_t s);
cudaError_t launch_fp8_stage(const Fp8StageParams& p, int head_dim, cudaStream_t s);
cudaError_t launch_decode(const DecodeParams& p, const CUtensorMap& k_map,
                          const CUtensorMap& v_map, int head_dim, int grid, cudaStream_t s,
                          bool fp8 = false);
cudaError_t launch_calib_combine(const CalibCombineParams& p, int head_dim, cudaStream_t s);
cudaError_t launch_decode_combine(const DecodeParams& p, int head_dim, int num_sms, cudaStream_t s);
// fp8: q and the K/V tiles are staged 8-bit-cache rows in fp16 (fp16 mmas)
cudaError_t launch_prefill_tc(const PrefillParams& p, int head_dim, const CUtensorMap& q_map,
                              const CUtensorMap& ck_map, const CUtensorMap& cv_map,
                              const CUtensorMap& ring_map, cudaStream_t s, bool fp8 = false);
int decode_smem_bytes(int head_dim);
// one CTA waiting, with the kernels' bounded wait, on an mbarrier nothing arrives at
cudaError_t launch_wait_probe(int* err, uint64_t limit_ns, cudaStream_t s);
cudaError_t decode_prepare_device();  // one-time kernel attributes on the current device

// ------------------------------------------------------------ device PTX
#if defined(__CUDACC__)

// Launch with programmatic dependent launch: the kernel may start while the
// previous kernel of the stream finishes; it must call grid_dep_wait() before
// touching memory that kernel wrote (and before overwriting memory it reads).
template <typename... KArgs, typename... Args>
static inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                                     cudaStream_t s, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// wait until the grids this launch depends on have completed and their writes are visible
__device__ __forceinline__ void grid_dep_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}
// allow the next programmatically dependent launch to begin launching
__device__ __forceinline__ void grid_dep_launch() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}

__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
  return t;
}

constexpr uint64_t kWaitLimitNs = 2000000000ull;  // every kernel wait gives up after 2 s

// Waits for the phase of `parity` to complete, giving up after limit_ns of
// %globaltimer. Returns false (and sets the error word) on timeout.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity, int* err,
                                                  uint64_t limit_ns = kWaitLimitNs) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 255u) == 0u && globaltimer_ns() - t0 > limit_ns) {
      atomicOr(err, kErrWaitTimeout);
      return false;
    }
  }
}

// 2-D TMA tile load (x = column in elements, y = row) completing on `bar`
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int32_t x,
                                            int32_t y, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes "
      "[%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

// plain bulk copy global -> shared (both 16-byte aligned, bytes a multiple of 16)
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes,
                                          uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(smem_u32(dst)), "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes),
      "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void prefetch_tensormap(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

// D = A(16x16, row) * B(16x8, col) + D, bf16 inputs, fp32 accumulate
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], uint32_t a0, uint32_t a1,
                                               uint32_t a2, uint32_t a3, uint32_t b0,
                                               uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, "
      "{%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void mma_f16_16816(float (&d)[4], uint32_t a0, uint32_t a1,
                                              uint32_t a2, uint32_t a3, uint32_t b0,
                                              uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, "
      "{%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// four E4M3 codes (bytes 0..3 of x) -> f16 pairs: lo = bytes 0, 1; hi = bytes 2, 3
__device__ __forceinline__ void e4m3x4_to_f16x2(uint32_t x, uint32_t& lo, uint32_t& hi) {
  asm("{\n\t.reg .b16 l, h;\n\t"
      "mov.b32 {l, h}, %2;\n\t"
      "cvt.rn.f16x2.e4m3x2 %0, l;\n\t"
      "cvt.rn.f16x2.e4m3x2 %1, h;\n\t}"
      : "=r"(lo), "=r"(hi)
      : "r"(x));
}

// two floats -> two E4M3 codes (round to nearest even, saturating): byte 0 = lo
__device__ __forceinline__ uint32_t f32x2_to_e4m3x2(float lo, float hi) {
  uint16_t d;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(d) : "f"(hi), "f"(lo));
  return d;
}

// Smallest power of two >= r, for a finite r > 0 below 2^127 (from the fp32 bits:
// a normal r with a zero mantissa is a power of two already; otherwise the next
// exponent; a subnormal r rounds its integer mantissa up to a power of two).
__device__ __forceinline__ float pow2_ceil(float r) {
  const uint32_t b = __float_as_uint(r);
  const uint32_t ex = b >> 23, man = b & 0x7FFFFFu;
  if (ex != 0) return man == 0 ? r : __uint_as_float((ex + 1u) << 23);
  return __uint_as_float(man <= 1u ? man : 1u << (32 - __clz(man - 1u)));
}

// packed fp32 pair product (sm_100+), each lane rounded to nearest even
__device__ __forceinline__ float2 mul2(float2 a, float2 b) {
  uint64_t d;
  asm("mul.rn.f32x2 %0, %1, %2;"
      : "=l"(d)
      : "l"(*reinterpret_cast<uint64_t*>(&a)), "l"(*reinterpret_cast<uint64_t*>(&b)));
  return *reinterpret_cast<float2*>(&d);
}

// Larger magnitude of two bf16 pairs, lane by lane (exact; the sign bits carry the
// xor of the operands' signs, which callers drop)
__device__ __forceinline__ uint32_t bf16x2_absmax(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("max.xorsign.abs.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

// One row of bf16 values quantized to the 8-bit format by LANES lanes (a warp, or
// each half of one with LANES = 16), each lane holding PER of them as PER / 2 packed
// pairs (element 2i in the low half of raw[i]): amax = max |x| over the row; s = the
// smallest power of two >= amax / 448 (amax / 448 rounded to fp32, as the format
// defines it); code = E4M3 of x / s (round to nearest even, saturating), where x / s is
// an exact scaling, taken as x times the exact reciprocal of s (a division when that
// reciprocal would not be a normal float); amax = 0 gives s = 0 and zero codes.
// Returns s; w[i] packs the codes of elements 4i .. 4i+3.
//
// s comes from amax's bits without a division. Write amax = (1 + f) 2^e with f in
// [0, 1) and 448 = 1.75 2^8. If 1 + f <= 1.75, amax / 448 lies in (2^(e-9), 2^(e-8)]
// and s = 2^(e-8); otherwise it lies in (2^(e-8), 2^(e-7)) and s = 2^(e-7). Rounding
// amax / 448 to fp32 cannot cross those powers of two: amax is a bf16 value (7 fraction
// bits), so unless 1 + f = 1.75 exactly (quotient exactly 2^(e-8)) the quotient is at
// least a factor 1.0044 away from each of them, far beyond fp32 rounding.
//
// The maximum is taken on the packed pairs and the scaling on fp32 pairs: both are
// exact, so the codes are those of the elementwise definition.
template <int PER, int LANES = 32>
__device__ __forceinline__ float e4m3_quantize_row_warp(const uint32_t (&raw)[PER / 2], uint32_t (&w)[PER / 4]) {
  static_assert(LANES == 32 || LANES == 16, "a warp or half a warp per row");
  static_assert(PER % 4 == 0, "codes are packed four to a word");
  uint32_t mw[PER / 2];
#pragma unroll
  for (int i = 0; i < PER / 2; ++i) mw[i] = raw[i];
#pragma unroll
  for (int span = PER / 4; span > 0; span >>= 1)  // pairwise tree over the words
#pragma unroll
    for (int i = 0; i < span; ++i) mw[i] = bf16x2_absmax(mw[i], mw[i + span]);
  float amax = fmaxf(fabsf(__uint_as_float(mw[0] << 16)), fabsf(__uint_as_float(mw[0] & 0xffff0000u)));
#pragma unroll
  for (int off = LANES / 2; off > 0; off >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, off));
  const uint32_t ab = __float_as_uint(amax), aex = ab >> 23;
  float sc = 0.f;
  if (aex > 8u)  // s = 2^(e-8) or 2^(e-7) is a normal float
    sc = __uint_as_float(((ab & 0x7FFFFFu) <= 0x600000u ? aex - 8u : aex - 7u) << 23);
  else if (amax > 0.f)
    sc = pow2_ceil(__fdiv_rn(amax, 448.f));
  const uint32_t sex = __float_as_uint(sc) >> 23;  // exponent field of s
  const bool mul = sex >= 1u && sex <= 253u;       // 1 / s is then a normal float
  const float inv = __uint_as_float((254u - sex) << 23);
  const float2 inv2 = make_float2(inv, inv);
#pragma unroll
  for (int i = 0; i < PER / 2; i += 2) {
    float2 x01 = make_float2(__uint_as_float(raw[i] << 16), __uint_as_float(raw[i] & 0xffff0000u));
    float2 x23 = make_float2(__uint_as_float(raw[i + 1] << 16), __uint_as_float(raw[i + 1] & 0xffff0000u));
    uint32_t c01 = 0, c23 = 0;
    if (amax > 0.f) {
      if (mul) {
        x01 = mul2(x01, inv2);
        x23 = mul2(x23, inv2);
      } else {
        x01 = make_float2(__fdiv_rn(x01.x, sc), __fdiv_rn(x01.y, sc));
        x23 = make_float2(__fdiv_rn(x23.x, sc), __fdiv_rn(x23.y, sc));
      }
      c01 = f32x2_to_e4m3x2(x01.x, x01.y);
      c23 = f32x2_to_e4m3x2(x23.x, x23.y);
    }
    w[i / 2] = c01 | (c23 << 16);
  }
  return sc;
}

__device__ __forceinline__ uint32_t pack_f16(float lo, float hi) {
  uint32_t d;
  asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
  return d;
}
// as pack_f16, magnitudes past the fp16 range saturating to +-65504
__device__ __forceinline__ uint32_t pack_f16_sat(float lo, float hi) {
  uint32_t d;
  asm("cvt.rn.satfinite.f16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
  return d;
}

__device__ __forceinline__ uint32_t movmatrix_trans(uint32_t a) {
  uint32_t d;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(d) : "r"(a));
  return d;
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// packed fp32 pairs (sm_100+): d = a * b + c and d = a + b on two lanes at once
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;"
      : "=l"(d)
      : "l"(*reinterpret_cast<uint64_t*>(&a)), "l"(*reinterpret_cast<uint64_t*>(&b)),
        "l"(*reinterpret_cast<uint64_t*>(&c)));
  return *reinterpret_cast<float2*>(&d);
}
__device__ __forceinline__ float2 add2(float2 a, float2 b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;"
      : "=l"(d)
      : "l"(*reinterpret_cast<uint64_t*>(&a)), "l"(*reinterpret_cast<uint64_t*>(&b)));
  return *reinterpret_cast<float2*>(&d);
}

// (lo, hi) -> bf16x2 with lo in the low half, round to nearest even
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

// byte offset of 16-byte chunk `c` (0..7) of row `r` inside a 128B-swizzled slab
__device__ __forceinline__ uint32_t swz128(int r, int c) {
  return static_cast<uint32_t>(r * 128 + ((c ^ (r & 7)) << 4));
}


// ------------------------------------------------------------ tcgen05 (5th-gen tensor cores)
__device__ __forceinline__ void tmem_alloc(uint32_t* smem_dst, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(smem_dst)),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// generic-proxy shared-memory writes made visible to the async proxy (tensor core, TMA)
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// D[tmem] (+)= A[smem desc] * B[smem desc], bf16 in, fp32 accumulate; issued by one thread
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                          uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// D[tmem] (+)= A[tmem] * B[smem desc]: A (M rows = TMEM lanes, K bf16 packed two per
// 32-bit column) read from tensor memory
__device__ __forceinline__ void umma_bf16_tmem_a(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc,
                                                 uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// arrive once on `bar` when every tcgen05.mma issued so far by this thread has completed
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

// 32 lanes x 32 columns of 32-bit from TMEM (lane quarter of the calling warp)
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
               : "r"(taddr));
}
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
               : "memory");
}
__device__ __forceinline__ void tmem_ld_wait() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_st_wait() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// Shared-memory matrix descriptor, 128-byte swizzle, atoms 1024-byte aligned.
// K-major operand: rows of 128 B (64 bf16 of K), 8-row groups `sbo` bytes apart.
// MN-major operand: `lbo` = bytes between 64-element MN blocks, `sbo` = bytes
// between 8-row K groups.
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1 << 46;  // descriptor version
  d |= (uint64_t)2 << 61;  // 128-byte swizzle
  return d;
}

// Instruction descriptor, kind::f16: bf16 A and B, fp32 D, dense, A K-major.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N, bool b_mn_major) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((b_mn_major ? 1u : 0u) << 16) |
         ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}
// The same with fp16 A and B (both operands of one mma share the type).
__host__ __device__ constexpr uint32_t idesc_f16_f32(int M, int N, bool b_mn_major) {
  return (1u << 4) | ((b_mn_major ? 1u : 0u) << 16) | ((uint32_t)(N >> 3) << 17) |
         ((uint32_t)(M >> 4) << 24);
}

#endif  // __CUDACC__

}  // namespace hwkv
