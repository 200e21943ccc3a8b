// decode.cu -- split-KV decode attention over per-head rings, and its
// log-sum-exp combine (HeadWiseKV Sec. 3.2, Eq. conditional-attention-weight
// and Eq. conditional-attention, evaluated at the newest position; Sec. 3.3:
// each GQA query-head group reads its KV head's own slice).
//
// Work decomposition. For one layer, every (batch row b, KV head h) ring holds
// n = min(t_b, cap_h) resident slots; after the append of token t_b - 1 these
// are exactly the positions J_{t_b - 1}(W_h), so the softmax runs over all of
// them and slot order does not matter. The rings are laid end to end and every
// CTA of the persistent grid takes an equal share of their tokens, cut at ring
// boundaries into segments (the plan is made on the GPU from the per-row
// lengths, see make_device_plan): a full-history ring is split over many CTAs,
// short-window rings are read whole by one, and all window levels share one
// launch.
//
// Inside a CTA: warp 4 is the producer -- one lane issues 2-D TMA loads of
// 64-token stages of K and V (128-byte swizzle, one box per 64 channels) into
// a STAGES-deep shared-memory ring guarded by full/empty mbarriers. Warps 0-3
// consume 16 tokens of each stage:
//   S^T[16 tok x 8 heads]  = K[16 x D] . Q^T[D x 8]        (mma m16n8k16, K as A)
//   online softmax per head column (max / sum over warp shuffles)
//   O^T[D x 8 heads]      += V^T[D x 16] . P^T[16 x 8]     (mma m16n8k16, V^T via ldmatrix.trans)
// where P^T reaches the B-operand layout through movmatrix.trans. Up to 8 query
// heads of a GQA group share every K/V byte read. Each warp leaves a partial
// (max, sum, unnormalised output); the four warps merge theirs in shared memory
// into one partial per tile, and the combine kernel merges the tiles of a head.
#include <mutex>

#include "hwkv_internal.cuh"

namespace hwkv {

namespace {

struct TileInfo {
  int b, h;
  int64_t start;  // first slot of the tile
  int len;        // slots in the tile (>= 1)
  int64_t k_row, v_row;
  int tile;       // partial slot of the tile
  int64_t s_new;  // fused step: ring slot that receives the new token
  bool single;    // the tile covers the whole ring: its output is final
};

// ---- device-side plan (per-row lengths read on the GPU)
//
// Ring u (unit order u = b * n_units + h) holds n_u = min(len_b + lens_inc,
// cap_h) keys (0 for an idle row or a row whose step would pass max_ctx), read in
// q_u = ceil(n_u / 64) stages (a partial last stage is loaded whole). A segment
// (a piece of one ring read by one CTA) also has a fixed cost of F stages (the
// query load, the cross-warp merge and the partial write). The rings are laid
// end to end on a cost line in stage units, ring u taking F + q_u from L_u =
// sum_{v<u} w_v (w_v = q_v + F for a ring with keys, 0 otherwise), total Lt. CTA
// c takes the line [floor(c Lt / G'), floor((c + 1) Lt / G')), G' = min(gridDim.x,
// Lt), and reads the stages it covers (a point in a ring's F-stretch maps to the
// ring's first stage). So every CTA gets the same cost to one stage, a CTA that
// starts more rings reads fewer keys, cuts fall on stage boundaries (neighbouring
// CTAs never load the same stage), and no CTA below G' is empty. Only a CTA's
// first and last segment can belong to a ring other CTAs also read; every other
// segment is a whole ring and gives that ring's output at once. A partial needs
// two slots per CTA: 2c for the first segment, 2c + 1 for the last.
//
// Every warp derives the plan in registers (no block barrier): the rings are
// spread over the lanes (u = 32 r + lane), the first 256 kept in registers and
// further ones re-read. Warp 0 of CTA 0 also stores Lt, G', F and every ring's
// (L_u, n_u) for the combine kernel.
constexpr int kPlanRegs = 8;

struct DevPlan {
  int64_t count;  // keys of this CTA (0: idle)
  int64_t off0;   // first slot of the first segment, within ring u0
  int u0;
};

__device__ __forceinline__ int dev_unit_len(const DecodeParams& p, int u, int32_t& len_b) {
  const int b = u / p.n_units;
  const int h = u - b * p.n_units;
  len_b = p.lens[b];
  if (len_b < 0 || (int64_t)len_b + p.lens_inc > p.max_ctx) return 0;
  const int64_t n = (int64_t)len_b + p.lens_inc;
  return (int)(n < p.u[h].cap ? n : p.u[h].cap);
}

__device__ __forceinline__ int warp_incl_scan(int v, int lane) {
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int x = __shfl_up_sync(0xffffffffu, v, off);
    if (lane >= off) v += x;
  }
  return v;
}

__device__ __forceinline__ int stages_of(int n) { return (n + kStageTokens - 1) / kStageTokens; }

// Called by whole warps; every lane returns the same plan. Every count fits in 32
// bits: a layer's keys are at most the arena's ring rows (below 2^30, which
// hwkv_alloc checks), so its stages and the cost line stay below 2^26, and
// c Lt / G is split as c (Lt / G) + c (Lt mod G) / G to stay in range.
__device__ DevPlan make_device_plan(const DecodeParams& p, bool write_table) {
  const int lane = threadIdx.x & 31;
  const int U = p.batch * p.n_units;
  const int R = (U + 31) / 32;
  const int F = p.seg_cost;  // stages
  int nreg[kPlanRegs];
  int Lt = 0, N = 0;
#pragma unroll
  for (int r = 0; r < kPlanRegs; ++r) {
    const int u = r * 32 + lane;
    int n = 0;
    if (r < R && u < U) {
      int32_t L;
      n = dev_unit_len(p, u, L);
      if (write_table && u % p.n_units == 0 && L >= 0 && (int64_t)L + p.lens_inc > p.max_ctx)
        atomicOr(p.err, kErrCapacity);
    }
    nreg[r] = n;
    Lt += n > 0 ? stages_of(n) + F : 0;
    N += n;
  }
  for (int r = kPlanRegs; r < R; ++r) {  // rings beyond the register cache
    const int u = r * 32 + lane;
    if (u < U) {
      int32_t L;
      const int n = dev_unit_len(p, u, L);
      Lt += n > 0 ? stages_of(n) + F : 0;
      N += n;
      if (write_table && u % p.n_units == 0 && L >= 0 && (int64_t)L + p.lens_inc > p.max_ctx)
        atomicOr(p.err, kErrCapacity);
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    Lt += __shfl_xor_sync(0xffffffffu, Lt, off);
    N += __shfl_xor_sync(0xffffffffu, N, off);
  }

  const int G = min((int)gridDim.x, max(Lt, 1));
  const int c = (int)blockIdx.x;
  const bool mine = c < G && Lt > 0;
  const int qL = Lt / G, rL = Lt - qL * G;
  const int A0 = mine ? c * qL + (c * rL) / G : 0;                    // floor(c Lt / G)
  const int A1 = mine ? (c + 1) * qL + ((c + 1) * rL) / G : 0;        // floor((c + 1) Lt / G)
  // line point -> key: the ring whose stretch [L_u, L_u + F + q_u) holds the point
  int a = -1, b = mine && A1 >= Lt ? N : -1;  // A1 = Lt: up to the last key
  int sa = 0, ua = 0;
  int carry_w = 0, carry_n = 0;
  for (int r = 0; r < R && ((mine && (a < 0 || b == -1)) || write_table); ++r) {
    int n = 0;
#pragma unroll
    for (int i = 0; i < kPlanRegs; ++i)
      if (i == r) n = nreg[i];
    const int u = r * 32 + lane;
    if (r >= kPlanRegs && u < U) {
      int32_t L;
      n = dev_unit_len(p, u, L);
    }
    const int w = n > 0 ? stages_of(n) + F : 0;
    const int iw = warp_incl_scan(w, lane), in = warp_incl_scan(n, lane);
    const int Lu = carry_w + iw - w, su = carry_n + in - n;
    if (write_table && u < U) {
      p.plan[4 + 2 * u] = Lu;
      p.plan[5 + 2 * u] = n;
    }
    if (mine && a < 0) {
      const unsigned hit = __ballot_sync(0xffffffffu, w > 0 && Lu <= A0 && A0 < Lu + w);
      if (hit) {
        const int src = __ffs(hit) - 1;
        const int lu = __shfl_sync(0xffffffffu, Lu, src);
        const int s0 = __shfl_sync(0xffffffffu, su, src);
        a = s0 + max(0, A0 - lu - F) * kStageTokens;
        sa = s0;
        ua = r * 32 + src;
      }
    }
    if (mine && b == -1) {
      const unsigned hit = __ballot_sync(0xffffffffu, w > 0 && Lu <= A1 && A1 < Lu + w);
      if (hit) {
        const int src = __ffs(hit) - 1;
        const int lu = __shfl_sync(0xffffffffu, Lu, src);
        const int s1 = __shfl_sync(0xffffffffu, su, src);
        b = s1 + max(0, A1 - lu - F) * kStageTokens;
      }
    }
    carry_w += __shfl_sync(0xffffffffu, iw, 31);
    carry_n += __shfl_sync(0xffffffffu, in, 31);
  }
  DevPlan dp;
  dp.count = mine && a >= 0 && b > a ? b - a : 0;
  dp.u0 = ua;
  dp.off0 = a - sa;  // key a lies in ring ua
  if (write_table && lane == 0) {
    p.plan[0] = Lt;
    p.plan[1] = G;
    p.plan[2] = F;
  }
  return dp;
}

// The tiles of one CTA, in order. Ring mode: the CTA's segments (above). Table
// mode: tiles blockIdx.x, + gridDim.x, ... of the explicit tile list.
struct TileWalker {
  int j = 0, count = 0;  // table mode
  // ring mode cursor
  int64_t rem = 0, start = 0;
  int u = 0, n = 0;
  int32_t len_b = 0;
  bool first = true, advance = false;

  __device__ void init(const DecodeParams& p, const DevPlan& dp) {
    if (p.tiles != nullptr) {
      count = blockIdx.x < p.n_tiles ? (p.n_tiles - blockIdx.x + gridDim.x - 1) / gridDim.x : 0;
      return;
    }
    rem = dp.count;
    if (rem > 0) {
      u = dp.u0;
      start = dp.off0;
      n = dev_unit_len(p, u, len_b);
    }
  }

  __device__ bool next(const DecodeParams& p, TileInfo& ti) {
    if (p.tiles != nullptr) {
      if (j >= count) return false;
      table_tile(p, blockIdx.x + j * gridDim.x, ti);
      ++j;
      return true;
    }
    if (rem <= 0) return false;
    if (advance) {  // the next ring that holds anything
      const int U = p.batch * p.n_units;
      do {
        if (++u >= U) {  // the plan promised more tokens: lengths changed under the kernel
          atomicOr(p.err, kErrBadIndex);
          rem = 0;
          return false;
        }
        n = dev_unit_len(p, u, len_b);
      } while (n == 0);
      start = 0;
    }
    ti.b = u / p.n_units;
    ti.h = u - ti.b * p.n_units;
    const DecodeUnit& du = p.u[ti.h];
    const int64_t len = min((int64_t)n - start, rem);
    ti.start = start;
    ti.len = (int)len;
    ti.k_row = du.k_row0 + (int64_t)ti.b * du.stride + start;
    ti.v_row = du.v_row0 + (int64_t)ti.b * du.stride + start;
    ti.s_new = ring_slot(len_b, du.cap, du.sink);
    ti.single = start == 0 && len == n;
    ti.tile = 2 * (int)blockIdx.x + (first ? 0 : 1);
    rem -= len;
    first = false;
    advance = true;
    return true;
  }

  __device__ static void table_tile(const DecodeParams& p, int tile, TileInfo& ti) {
    const CalibTile ct = p.tiles[tile];
    ti.tile = tile;
    ti.b = ct.q_row;
    ti.h = ct.h;
    ti.start = 0;
    ti.len = ct.len;
    ti.k_row = ct.k_row;
    ti.v_row = ct.v_row;
    ti.s_new = -1;
    ti.single = false;
  }
};

// named barrier of the four consumer warps (the producer warp does not take part)
__device__ __forceinline__ void consumer_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(kDecodeWarps * 32) : "memory");
}

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

// FP8: K/V stages hold E4M3 codes (one byte per channel, 128 channels per
// 128-byte slab) and each stage's 64 K and 64 V row scales arrive beside it.
template <int D, bool FP8>
struct DecodeCfg {
  static constexpr int kChanPerSlab = FP8 ? 128 : 64;
  static constexpr int kSlabs = D / kChanPerSlab;
  static constexpr int kTileBytes = kSlabs * kSlabBytes;  // 64 tokens of K (or V)
  static constexpr int kStageBytes = 2 * kTileBytes;
  static constexpr int kStages = FP8 ? (D == 256 ? 5 : 10) : (D == 256 ? 3 : (D == 128 ? 6 : 8));
  static constexpr int kScaleBytes = FP8 ? kStages * 2 * kStageTokens * 4 : 0;
  static constexpr int kScratchBytes = 0;
  static constexpr int kRedLd = D + 4;  // padded row of the cross-warp merge area (floats)
  static constexpr int kRedBytes = kDecodeWarps * kMaxGroup * kRedLd * 4;
  static constexpr int kMlBytes = kDecodeWarps * kMaxGroup * 8;
  static constexpr int kSmem = kStages * kStageBytes + kScratchBytes + kScaleBytes + kRedBytes +
                               kMlBytes + 2 * kStages * 8 + 1024;
};

}  // namespace

template <int D, bool FP8>
__global__ void __launch_bounds__((kDecodeWarps + 1) * 32, 1)
    decode_split_kernel(const __grid_constant__ CUtensorMap k_map,
                        const __grid_constant__ CUtensorMap v_map, const DecodeParams p) {
  using C = DecodeCfg<D, FP8>;
  constexpr int STAGES = C::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  float* stage_scales = reinterpret_cast<float*>(smem + STAGES * C::kStageBytes);  // FP8: [stage][K|V][64]
  uint8_t* tail = smem + STAGES * C::kStageBytes + C::kScaleBytes;
  float* red_o = reinterpret_cast<float*>(tail);
  float2* red_ml = reinterpret_cast<float2*>(tail + C::kRedBytes);
  uint64_t* full = reinterpret_cast<uint64_t*>(tail + C::kRedBytes + C::kMlBytes);
  uint64_t* empty = full + STAGES;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kDecodeWarps);
    }
    fence_barrier_init();
  }
  // Before waiting for the kernel launched before (this launch may start while it
  // runs): the unit table and the tensor maps do not depend on it, so bring them
  // into the constant cache now
  if (p.tiles == nullptr && lane < p.n_units) {
    const DecodeUnit& du = p.u[lane];
    asm volatile("" ::"l"(du.k_row0), "l"(du.v_row0), "l"(du.cap), "l"(du.stride), "l"(du.sink));
  }
  if (warp == kDecodeWarps && lane == 0) {
    prefetch_tensormap(&k_map);
    prefetch_tensormap(&v_map);
  }
  __syncthreads();
  grid_dep_wait();    // the ring append, q and the lengths come from kernels launched before
  grid_dep_launch();  // the combine kernel may start launching
  DevPlan dplan{};
  if (p.tiles == nullptr)  // each warp plans for itself; warp 0 of CTA 0 leaves the table
    dplan = make_device_plan(p, blockIdx.x == 0 && warp == 0);

  if (warp == kDecodeWarps) {
    // ------------------------------------------------------------ producer
    if (lane != 0) return;
    prefetch_tensormap(&k_map);
    prefetch_tensormap(&v_map);
    uint32_t it = 0;
    bool ok = true;
    TileWalker wk;
    wk.init(p, dplan);
    TileInfo ti;
    while (ok && wk.next(p, ti)) {
      const int n_st = (ti.len + kStageTokens - 1) / kStageTokens;
      for (int st = 0; st < n_st; ++st, ++it) {
        const int s = it % STAGES;
        const uint32_t ph = (it / STAGES) & 1u;
        if (!mbar_wait_bounded(&empty[s], ph ^ 1u, p.err)) {
          ok = false;
          break;
        }
        uint8_t* kdst = smem + s * C::kStageBytes;
        uint8_t* vdst = kdst + C::kTileBytes;
        mbar_arrive_expect_tx(&full[s], C::kStageBytes + (FP8 ? 2 * kStageTokens * 4 : 0));
        const int32_t krow = (int32_t)(ti.k_row + (int64_t)st * kStageTokens);
        const int32_t vrow = (int32_t)(ti.v_row + (int64_t)st * kStageTokens);
#pragma unroll
        for (int sl = 0; sl < C::kSlabs; ++sl)
          tma_load_2d(kdst + sl * kSlabBytes, &k_map, sl * C::kChanPerSlab, krow, &full[s]);
#pragma unroll
        for (int sl = 0; sl < C::kSlabs; ++sl)
          tma_load_2d(vdst + sl * kSlabBytes, &v_map, sl * C::kChanPerSlab, vrow, &full[s]);
        if constexpr (FP8) {  // rows are 64-aligned, so each 256-byte scale run is too
          float* sdst = stage_scales + s * 2 * kStageTokens;
          bulk_load(sdst, p.scales + krow, kStageTokens * 4, &full[s]);
          bulk_load(sdst + kStageTokens, p.scales + vrow, kStageTokens * 4, &full[s]);
        }
      }
    }
    if (!ok) {
      // let the copies already issued land before the CTA's shared memory goes away
      const uint32_t first = it > (uint32_t)STAGES ? it - STAGES : 0u;
      for (uint32_t j = first; j < it; ++j)
        mbar_wait_bounded(&full[j % STAGES], (j / STAGES) & 1u, p.err);
    }
    return;
  }

  // -------------------------------------------------------------- consumers
  const int w = warp;
  const int qn = lane >> 2;        // query head of this lane's Q^T fragment column
  const int qk = (lane & 3) * 2;   // channel pair within a 16-channel step
  const float c = p.scale_log2;
  uint32_t it = 0;
  // Once a bounded wait gives up, this warp stops waiting and computing but
  // keeps walking the same tile/stage sequence, so every consumer warp still
  // reaches the same named barriers.
  bool aborted = false;

  TileWalker wk;
  wk.init(p, dplan);
  TileInfo ti;
  while (wk.next(p, ti)) {
    const int n_st = (ti.len + kStageTokens - 1) / kStageTokens;

    // Q^T as mma B fragments, column = head qn. bf16: b0 = channels 16kk + qk +
    // {0,1}, b1 = +8. FP8 (f16 mma): the E4M3 A fragments of 32 channels arrive as
    // 4 consecutive channels per lane, so mma m of step kk contracts over channels
    // 32kk + 4(lane&3) + 2m + {0,1} (b0) and the same + 16 (b1); Q follows that order
    uint32_t qf[D / 16][2];
    {
      const bool qv = qn < p.group;
      const __nv_bfloat16* qrow =
          p.q + ((int64_t)ti.b * p.n_q_heads + (int64_t)ti.h * p.group + (qv ? qn : 0)) * D;
      if constexpr (!FP8) {
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          qf[kk][0] = qv ? *reinterpret_cast<const uint32_t*>(qrow + kk * 16 + qk) : 0u;
          qf[kk][1] = qv ? *reinterpret_cast<const uint32_t*>(qrow + kk * 16 + 8 + qk) : 0u;
        }
      } else {
        auto f16pair = [&](int ch) -> uint32_t {
          const uint32_t x = *reinterpret_cast<const uint32_t*>(qrow + ch);
          return pack_f16(__uint_as_float(x << 16), __uint_as_float(x & 0xffff0000u));
        };
#pragma unroll
        for (int kk = 0; kk < D / 32; ++kk)
#pragma unroll
          for (int m = 0; m < 2; ++m) {
            const int ch = kk * 32 + (lane & 3) * 4 + 2 * m;
            qf[2 * kk + m][0] = qv ? f16pair(ch) : 0u;
            qf[2 * kk + m][1] = qv ? f16pair(ch + 16) : 0u;
          }
      }
    }

    float o[D / 16][4];
#pragma unroll
    for (int mt = 0; mt < D / 16; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
    float mA = -INFINITY, mB = -INFINITY, lA = 0.f, lB = 0.f;

    for (int st = 0; st < n_st; ++st, ++it) {
      const int s = it % STAGES;
      const uint32_t ph = (it / STAGES) & 1u;
      if (!aborted && !mbar_wait_bounded(&full[s], ph, p.err)) aborted = true;
      if (aborted) {
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[s]);
        continue;
      }
      const uint32_t kbase = smem_u32(smem + s * C::kStageBytes);
      const uint32_t vbase = kbase + C::kTileBytes;
      float* ksc = stage_scales + s * 2 * kStageTokens;  // FP8: this stage's row scales
      float* vsc = ksc + kStageTokens;
      if (p.k_new != nullptr) {
        // fused step: the new token's slot may lie in this stage; the warp owning that
        // row replaces the staged (stale) row with the new K/V and writes the ring row
        const int64_t row_in = ti.s_new - (ti.start + (int64_t)st * kStageTokens);
        if constexpr (FP8) {
         if (row_in >= w * 16 && row_in < w * 16 + 16) {
          // quantise as the append does (the same row helper)
          constexpr int PER = D / 32;
          const int r = (int)row_in;
#pragma unroll
          for (int kv = 0; kv < 2; ++kv) {
            const __nv_bfloat16* src =
                (kv ? p.v_new : p.k_new) + ((int64_t)ti.b * p.n_units + ti.h) * D + lane * PER;
            uint32_t raw[PER / 2];
            if constexpr (PER == 8) {
              const uint4 v = *reinterpret_cast<const uint4*>(src);
              raw[0] = v.x; raw[1] = v.y; raw[2] = v.z; raw[3] = v.w;
            } else {
              const uint2 v = *reinterpret_cast<const uint2*>(src);
              raw[0] = v.x; raw[1] = v.y;
            }
            uint32_t cw[PER / 4];
            const float sc = e4m3_quantize_row_warp<PER>(raw, cw);
            const int64_t ring = (kv ? ti.v_row : ti.k_row) - ti.start + ti.s_new;
            uint8_t* g = reinterpret_cast<uint8_t*>(p.arena) + ring * D + lane * PER;
            const int c0 = lane * PER;  // first channel of this lane
            const uint32_t a = (kv ? vbase : kbase) + (c0 >> 7) * kSlabBytes +
                               swz128(r, (c0 & 127) >> 4) + (c0 & 15);
            if constexpr (PER == 8) {
              *reinterpret_cast<uint2*>(g) = make_uint2(cw[0], cw[1]);
              asm volatile("st.shared.v2.b32 [%0], {%1, %2};" ::"r"(a), "r"(cw[0]), "r"(cw[1])
                           : "memory");
            } else {
              *reinterpret_cast<uint32_t*>(g) = cw[0];
              asm volatile("st.shared.b32 [%0], %1;" ::"r"(a), "r"(cw[0]) : "memory");
            }
            if (lane == 0) {
              p.scales[ring] = sc;
              (kv ? vsc : ksc)[r] = sc;
            }
          }
          fence_proxy_async_smem();  // these generic writes precede the next copy into the stage
          __syncwarp();
         }
        } else if (row_in >= w * 16 && row_in < w * 16 + 16) {
          const int r = (int)row_in;
          const __nv_bfloat16* src_k = p.k_new + ((int64_t)ti.b * p.n_units + ti.h) * D;
          const __nv_bfloat16* src_v = p.v_new + ((int64_t)ti.b * p.n_units + ti.h) * D;
          const int64_t ring_row = ti.k_row - ti.start + ti.s_new;  // K region row
          const int64_t vring_row = ti.v_row - ti.start + ti.s_new;
          for (int idx = lane; idx < 2 * (D / 8); idx += 32) {
            const int isv = idx >= D / 8;
            const int ch = isv ? idx - D / 8 : idx;  // 16-byte chunk of the row
            const uint4 val = *reinterpret_cast<const uint4*>((isv ? src_v : src_k) + ch * 8);
            const uint32_t dst = (isv ? vbase : kbase) + (ch >> 3) * kSlabBytes + swz128(r, ch & 7);
            asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(dst), "r"(val.x),
                         "r"(val.y), "r"(val.z), "r"(val.w)
                         : "memory");
            *reinterpret_cast<uint4*>(p.arena + (isv ? vring_row : ring_row) * D + ch * 8) = val;
          }
          fence_proxy_async_smem();  // this generic write precedes the next TMA into the stage
          __syncwarp();
        }
      }

      // S^T = K . Q^T  (two accumulators to shorten the dependent mma chain)
      float sa[4] = {0.f, 0.f, 0.f, 0.f}, sb[4] = {0.f, 0.f, 0.f, 0.f};
      {
        const int r = w * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
        const int csel = lane >> 4;
        if constexpr (!FP8) {
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            uint32_t a0, a1, a2, a3;
            ldsm_x4(kbase + (kk >> 2) * kSlabBytes + swz128(r, (kk & 3) * 2 + csel), a0, a1, a2,
                    a3);
            if (kk & 1)
              mma_bf16_16816(sb, a0, a1, a2, a3, qf[kk][0], qf[kk][1]);
            else
              mma_bf16_16816(sa, a0, a1, a2, a3, qf[kk][0], qf[kk][1]);
          }
        } else {
          // 32 channels per step: the x4 load gives every lane 4 consecutive E4M3
          // channels of two rows, split into the two f16 mmas of Q's channel order
#pragma unroll
          for (int kk = 0; kk < D / 32; ++kk) {
            uint32_t a0, a1, a2, a3, l0, l1, l2, l3, h0, h1, h2, h3;
            ldsm_x4(kbase + (kk >> 2) * kSlabBytes + swz128(r, (kk & 3) * 2 + csel), a0, a1, a2,
                    a3);
            e4m3x4_to_f16x2(a0, l0, h0);
            e4m3x4_to_f16x2(a1, l1, h1);
            e4m3x4_to_f16x2(a2, l2, h2);
            e4m3x4_to_f16x2(a3, l3, h3);
            mma_f16_16816(sa, l0, l1, l2, l3, qf[2 * kk][0], qf[2 * kk][1]);
            mma_f16_16816(sb, h0, h1, h2, h3, qf[2 * kk + 1][0], qf[2 * kk + 1][1]);
          }
        }
      }
      float s0 = sa[0] + sb[0], s1 = sa[1] + sb[1], s2 = sa[2] + sb[2], s3 = sa[3] + sb[3];
      float vsA = 1.f, vsB = 1.f;  // FP8: V row scales of this lane's two tokens
      if constexpr (FP8) {
        const int tA = w * 16 + (lane >> 2);
        const float ksA = ksc[tA], ksB = ksc[tA + 8];
        vsA = vsc[tA];
        vsB = vsc[tA + 8];
        s0 *= ksA;
        s1 *= ksA;
        s2 *= ksB;
        s3 *= ksB;
      }
      const int tok = st * kStageTokens + w * 16 + (lane >> 2);
      if (tok >= ti.len) s0 = s1 = -INFINITY;
      if (tok + 8 >= ti.len) s2 = s3 = -INFINITY;

      // online softmax; this lane owns head columns qk (A) and qk+1 (B)
      float xA = fmaxf(s0, s2), xB = fmaxf(s1, s3);
#pragma unroll
      for (int off = 4; off < 32; off <<= 1) {
        xA = fmaxf(xA, __shfl_xor_sync(0xffffffffu, xA, off));
        xB = fmaxf(xB, __shfl_xor_sync(0xffffffffu, xB, off));
      }
      const float nA = fmaxf(mA, xA), nB = fmaxf(mB, xB);
      const float uA = nA == -INFINITY ? 0.f : nA;
      const float uB = nB == -INFINITY ? 0.f : nB;
      const float alA = ex2((mA - uA) * c), alB = ex2((mB - uB) * c);
      const float p0 = ex2((s0 - uA) * c), p1 = ex2((s1 - uB) * c);
      const float p2 = ex2((s2 - uA) * c), p3 = ex2((s3 - uB) * c);
      lA = lA * alA + p0 + p2;
      lB = lB * alB + p1 + p3;
      mA = nA;
      mB = nB;
      if (__any_sync(0xffffffffu, alA != 1.f || alB != 1.f)) {
#pragma unroll
        for (int mt = 0; mt < D / 16; ++mt) {
          o[mt][0] *= alA;
          o[mt][1] *= alB;
          o[mt][2] *= alA;
          o[mt][3] *= alB;
        }
      }
      // O^T += V^T . P^T  (FP8: the V row scales ride on P; the sums l do not)
      const uint32_t pb0 = movmatrix_trans(FP8 ? pack_f16(p0 * vsA, p1 * vsA) : pack_bf16(p0, p1));
      const uint32_t pb1 = movmatrix_trans(FP8 ? pack_f16(p2 * vsB, p3 * vsB) : pack_bf16(p2, p3));
      {
        const int mi = lane >> 3;
        const int csel = mi & 1;
        if constexpr (!FP8) {
          const int r = w * 16 + (lane & 7) + (mi >> 1) * 8;
#pragma unroll
          for (int mt = 0; mt < D / 16; ++mt) {
            uint32_t a0, a1, a2, a3;
            ldsm_x4_t(vbase + (mt >> 2) * kSlabBytes + swz128(r, (mt & 3) * 2 + csel), a0, a1,
                      a2, a3);
            mma_bf16_16816(o[mt], a0, a1, a2, a3, pb0, pb1);
          }
        } else {
          // V^T fragments straight from the E4M3 stage: the transposing x4 load of
          // byte pairs gives each lane tokens (2q, 2q+1) x channels (2g, 2g+1) of 16
          // tokens x 32 channels; a byte permute splits them into the even- and
          // odd-channel token pairs, which feed two f16 mmas (o[2kk]: channels
          // 32kk + 2g (+16), o[2kk + 1]: the odd ones)
          const int tr = w * 16 + (mi >> 1) * 8 + (lane & 7);
#pragma unroll
          for (int kk = 0; kk < D / 32; ++kk) {
            const int ch = kk * 32 + (mi & 1) * 16;
            uint32_t r[4], lo[4], hi[4];
            ldsm_x4_t(vbase + (ch >> 7) * kSlabBytes + swz128(tr, (ch & 127) >> 4), r[0], r[1],
                      r[2], r[3]);
#pragma unroll
            for (int j = 0; j < 4; ++j) e4m3x4_to_f16x2(__byte_perm(r[j], 0, 0x3120), lo[j], hi[j]);
            mma_f16_16816(o[2 * kk], lo[0], lo[1], lo[2], lo[3], pb0, pb1);
            mma_f16_16816(o[2 * kk + 1], hi[0], hi[1], hi[2], hi[3], pb0, pb1);
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[s]);
    }

    // ---- merge the four warps' partials of this tile in shared memory
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
      lA += __shfl_xor_sync(0xffffffffu, lA, off);
      lB += __shfl_xor_sync(0xffffffffu, lB, off);
    }
    consumer_sync();  // previous tile's merge has been read
    {
      float* ro = red_o + (size_t)w * kMaxGroup * C::kRedLd;
#pragma unroll
      for (int mt = 0; mt < D / 16; ++mt) {
        // bf16: o[mt] rows are channels 16 mt + g and + 8; FP8: 32 (mt / 2) + 2g + (mt & 1)
        // and + 16 (the channel order of the V^T fragments)
        const int dim = FP8 ? (mt >> 1) * 32 + 2 * (lane >> 2) + (mt & 1) : mt * 16 + (lane >> 2);
        const int dim2 = dim + (FP8 ? 16 : 8);
        ro[qk * C::kRedLd + dim] = o[mt][0];
        ro[(qk + 1) * C::kRedLd + dim] = o[mt][1];
        ro[qk * C::kRedLd + dim2] = o[mt][2];
        ro[(qk + 1) * C::kRedLd + dim2] = o[mt][3];
      }
      if (lane < 4) {
        red_ml[w * kMaxGroup + qk] = make_float2(mA, lA);
        red_ml[w * kMaxGroup + qk + 1] = make_float2(mB, lB);
      }
    }
    consumer_sync();
    {
      // one tile covers the whole ring: this is the final output, normalised here;
      // otherwise leave the tile's partial for the combine kernel
      const bool single = ti.single;
      float* po = p.part_o + (int64_t)ti.tile * kMaxGroup * D;
      float* fo = p.out + ((int64_t)ti.b * p.n_q_heads + (int64_t)ti.h * p.group) * D;
      for (int n = 0; n < p.group; ++n) {
        float M = -INFINITY;
#pragma unroll
        for (int ww = 0; ww < kDecodeWarps; ++ww) M = fmaxf(M, red_ml[ww * kMaxGroup + n].x);
        float e[kDecodeWarps], L = 0.f;
#pragma unroll
        for (int ww = 0; ww < kDecodeWarps; ++ww) {
          const float2 ml = red_ml[ww * kMaxGroup + n];
          e[ww] = ml.x == -INFINITY ? 0.f : ex2((ml.x - M) * c);
          L += e[ww] * ml.y;
        }
        const float scale_out = single ? 1.f / L : 1.f;
        float* dst = single ? fo + (int64_t)n * D : po + (int64_t)n * D;
        for (int i = w * (D / kDecodeWarps) + lane; i < (w + 1) * (D / kDecodeWarps); i += 32) {
          float acc = 0.f;
#pragma unroll
          for (int ww = 0; ww < kDecodeWarps; ++ww)
            acc += e[ww] * red_o[((size_t)ww * kMaxGroup + n) * C::kRedLd + i];
          dst[i] = acc * scale_out;
        }
        if (!single && w == 0 && lane == 0)
          p.part_ml[(int64_t)ti.tile * kMaxGroup + n] = make_float2(M, L);
      }
    }
  }
}

// Log-sum-exp merge of the segment partials of one (batch row, query head):
// o = sum_j 2^{(m_j - M) c} o_j / sum_j 2^{(m_j - M) c} l_j, M = max_j m_j.
// CH CTAs of 8 warps per (batch row, query head), each over D / CH consecutive
// channels (CH > 1 for small steps, with few (batch row, query head) pairs: the merge
// is spread over more SMs and each warp takes more partials per round). Warp w merges
// partials w, w + 8, w + 16, ... in that order with a running maximum (each lane
// D / (32 CH) consecutive channels), loading a batch of partials (32 floats per lane)
// before using any of them, so a ring split over many CTAs costs a few rounds of L2
// latency rather than one per partial; the eight warps' results are then merged in
// warp order (deterministic). Rings read whole by one CTA were written by the split
// kernel.
constexpr int kCombineWarps = 8;

template <int D, int CH>
__global__ void __launch_bounds__(kCombineWarps * 32) decode_combine_kernel(const DecodeParams p) {
  constexpr int DC = D / CH;    // channels of this CTA
  constexpr int PER = DC / 32;  // channels per lane
  static_assert(PER >= 2 && PER % 2 == 0, "channel pairs per lane");
  // partials loaded together; the registers stay low enough for a combine CTA to
  // sit beside a split CTA on one SM (it launches early and waits there)
  constexpr int kCombineBatch = 32 / PER;
  __shared__ float s_num[kCombineWarps][DC];
  __shared__ float2 s_ml[kCombineWarps];
  grid_dep_wait();  // partials come from the split kernel launched before
  const int bq = blockIdx.x / CH;
  const int c0 = (blockIdx.x - bq * CH) * DC;  // first channel of this CTA
  const int b = bq / p.n_q_heads;
  const int qh = bq - b * p.n_q_heads;
  const int h = qh / p.group;
  const int n = qh - h * p.group;
  // the ring's segments: its stages span the cost line [L + F, L + F + q), read
  // by CTAs c1 .. c2 of the split launch; the first segment's partial sits in
  // slot 2 c1 (the ring starts that CTA's range) or 2 c1 + 1 (it is that CTA's
  // last segment), every later one in slot 2 c (the ring starts that CTA's range)
  const int u = b * p.n_units + h;
  const long long Lt = p.plan[0], G = p.plan[1], F = p.plan[2];
  const long long Lu = p.plan[4 + 2 * u], nu = p.plan[5 + 2 * u];
  // every ring of an active row holds >= 1 key; the split kernel has finished
  // reading the lengths, so the row can advance now
  if (p.lens_inc && qh == 0 && c0 == 0 && threadIdx.x == 0 && p.plan[5 + 2 * (b * p.n_units)] > 0)
    p.lens[b] += 1;
  if (nu == 0) {  // idle row (or a row at max_ctx): zero output
    for (int i = threadIdx.x; i < DC; i += blockDim.x)
      p.out[((int64_t)b * p.n_q_heads + qh) * D + c0 + i] = 0.f;
    return;
  }
  const long long qu = (nu + kStageTokens - 1) / kStageTokens;
  const long long c1 = ((Lu + F + 1) * G - 1) / Lt;   // the CTA with the first stage
  const long long c2 = ((Lu + F + qu) * G - 1) / Lt;  // the CTA with the last stage
  if (c1 == c2) return;  // one CTA read the whole ring and wrote the output
  const int n_t = (int)(c2 - c1 + 1);
  const int64_t slot0 = 2 * c1 + (c1 * Lt / G >= Lu ? 0 : 1);
  auto slot = [&](int j) -> int64_t { return j == 0 ? slot0 : 2 * (c1 + j); };
  const float c = p.scale_log2;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;

  float m = -INFINITY, den = 0.f;
  float acc[PER];
#pragma unroll
  for (int e = 0; e < PER; ++e) acc[e] = 0.f;
  for (int j0 = w; j0 < n_t; j0 += kCombineBatch * kCombineWarps) {
    float2 ml[kCombineBatch];
    float v[kCombineBatch][PER];
#pragma unroll
    for (int k = 0; k < kCombineBatch; ++k) {
      const int j = j0 + k * kCombineWarps;
      if (j < n_t) {
        const int64_t sl = slot(j);
        ml[k] = p.part_ml[sl * kMaxGroup + n];
        const float* src = p.part_o + (sl * kMaxGroup + n) * D + c0 + lane * PER;
#pragma unroll
        for (int e = 0; e < PER; e += 2) {
          const float2 x = *reinterpret_cast<const float2*>(src + e);
          v[k][e] = x.x;
          v[k][e + 1] = x.y;
        }
      } else {
        ml[k] = make_float2(-INFINITY, 0.f);
#pragma unroll
        for (int e = 0; e < PER; ++e) v[k][e] = 0.f;
      }
    }
    float mn = m;
#pragma unroll
    for (int k = 0; k < kCombineBatch; ++k) mn = fmaxf(mn, ml[k].x);
    if (mn == -INFINITY) continue;  // nothing but empty partials so far
    const float a = m == -INFINITY ? 0.f : ex2((m - mn) * c);
    den *= a;
#pragma unroll
    for (int e = 0; e < PER; ++e) acc[e] *= a;
#pragma unroll
    for (int k = 0; k < kCombineBatch; ++k) {
      const float wk = ml[k].x == -INFINITY ? 0.f : ex2((ml[k].x - mn) * c);
      den += wk * ml[k].y;
#pragma unroll
      for (int e = 0; e < PER; ++e) acc[e] += wk * v[k][e];
    }
    m = mn;
  }
#pragma unroll
  for (int e = 0; e < PER; ++e) s_num[w][lane * PER + e] = acc[e];
  if (lane == 0) s_ml[w] = make_float2(m, den);
  __syncthreads();
  float M = -INFINITY;
#pragma unroll
  for (int k = 0; k < kCombineWarps; ++k) M = fmaxf(M, s_ml[k].x);
  float wk[kCombineWarps], dsum = 0.f;
#pragma unroll
  for (int k = 0; k < kCombineWarps; ++k) {
    wk[k] = s_ml[k].x == -INFINITY ? 0.f : ex2((s_ml[k].x - M) * c);
    dsum += wk[k] * s_ml[k].y;
  }
  for (int i = threadIdx.x; i < DC; i += blockDim.x) {
    float num = 0.f;
#pragma unroll
    for (int k = 0; k < kCombineWarps; ++k) num += wk[k] * s_num[k][i];
    p.out[((int64_t)b * p.n_q_heads + qh) * D + c0 + i] = num / dsum;
  }
}

int decode_smem_bytes(int head_dim) {
  switch (head_dim) {
    case 64: return DecodeCfg<64, false>::kSmem;
    case 128: return DecodeCfg<128, false>::kSmem;
    case 256: return DecodeCfg<256, false>::kSmem;
    default: return -1;
  }
}

template <int D, bool FP8>
static cudaError_t opt_in() {
  return cudaFuncSetAttribute(decode_split_kernel<D, FP8>,
                              cudaFuncAttributeMaxDynamicSharedMemorySize, DecodeCfg<D, FP8>::kSmem);
}

// The shared-memory opt-in of the split kernels, once per device (host calls
// made before any stream capture, e.g. hwkv_alloc, take care of it).
cudaError_t decode_prepare_device() {
  constexpr int kMaxDevices = 64;
  static std::mutex mu;
  static bool done[kMaxDevices] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(mu);
  if (done[dev]) return cudaSuccess;
  e = opt_in<64, false>();
  if (e == cudaSuccess) e = opt_in<128, false>();
  if (e == cudaSuccess) e = opt_in<256, false>();
  if (e == cudaSuccess) e = opt_in<128, true>();
  if (e == cudaSuccess) e = opt_in<256, true>();
  if (e == cudaSuccess) done[dev] = true;
  return e;
}

template <int D, bool FP8>
static cudaError_t launch_decode_t(const DecodeParams& p, const CUtensorMap& kmap,
                                   const CUtensorMap& vmap, int grid, cudaStream_t s) {
  cudaError_t e = decode_prepare_device();
  if (e != cudaSuccess) return e;
  return launch_pdl(decode_split_kernel<D, FP8>, dim3(grid), dim3((kDecodeWarps + 1) * 32),
                    DecodeCfg<D, FP8>::kSmem, s, kmap, vmap, p);
}

cudaError_t launch_decode(const DecodeParams& p, const CUtensorMap& kmap, const CUtensorMap& vmap,
                          int head_dim, int grid, cudaStream_t s, bool fp8) {
  if (fp8) {
    switch (head_dim) {
      case 128: return launch_decode_t<128, true>(p, kmap, vmap, grid, s);
      case 256: return launch_decode_t<256, true>(p, kmap, vmap, grid, s);
      default: return cudaErrorInvalidValue;
    }
  }
  switch (head_dim) {
    case 64: return launch_decode_t<64, false>(p, kmap, vmap, grid, s);
    case 128: return launch_decode_t<128, false>(p, kmap, vmap, grid, s);
    case 256: return launch_decode_t<256, false>(p, kmap, vmap, grid, s);
    default: return cudaErrorInvalidValue;
  }
}

// SeqCalib candidate replay (Sec. 3.2, Eq. conditional-similarity; App. A.2,
// Eq. stabilized-cosine). For one unit (sequence, sampled position, KV head)
// the keys were split into nested-suffix bands: band 0 = the newest W_0 keys,
// band k = keys between W_{k-1} and W_k back, band K = everything older. Warp g
// merges the band partials of query head g in band order; after band k (< K)
// the running output is o^(W_k), after the last band it is o^(full). Each
// candidate is scored against full with the stabilized cosine (eps = 1e-12:
// a vector of norm <= eps counts as zero; both zero -> 1, one zero -> 0); with
// a traced output given, o^(full) is scored against it the same way (the
// calibrator's trace-compatibility check, App. "Experimental Protocol").
constexpr int kCalibMaxWindows = 8;

template <int D>
__global__ void __launch_bounds__(kMaxGroup * 32) calib_combine_kernel(const CalibCombineParams p) {
  constexpr int PER = D / 32;
  grid_dep_wait();
  const int u = blockIdx.x;
  const int g = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (g >= p.group) return;
  const int K = p.n_windows;
  const float c = p.scale_log2;
  const int32_t* bb = p.band_begin + (int64_t)u * (K + 2);
  float M = -INFINITY, L = 0.f;
  float O[PER];
#pragma unroll
  for (int e = 0; e < PER; ++e) O[e] = 0.f;
  float snap[kCalibMaxWindows][PER];
  float snap_l[kCalibMaxWindows];
#pragma unroll
  for (int k = 0; k < kCalibMaxWindows; ++k) {
    snap_l[k] = 0.f;
#pragma unroll
    for (int e = 0; e < PER; ++e) snap[k][e] = 0.f;
  }
  for (int k = 0; k <= K; ++k) {
    for (int j = bb[k]; j < bb[k + 1]; ++j) {
      const float2 ml = p.part_ml[(int64_t)j * kMaxGroup + g];
      if (ml.x == -INFINITY) continue;
      const float nm = fmaxf(M, ml.x);
      const float a = M == -INFINITY ? 0.f : ex2((M - nm) * c);
      const float bw = ex2((ml.x - nm) * c);
      const float* src = p.part_o + ((int64_t)j * kMaxGroup + g) * D + lane * PER;
#pragma unroll
      for (int e = 0; e < PER; ++e) O[e] = O[e] * a + src[e] * bw;
      L = L * a + ml.y * bw;
      M = nm;
    }
    if (k < K) {  // o^(W_k) up to the common factor 2^{-M c}, normalised below
#pragma unroll
      for (int kk = 0; kk < kCalibMaxWindows; ++kk)
        if (kk == k) {
          snap_l[kk] = L;
#pragma unroll
          for (int e = 0; e < PER; ++e) snap[kk][e] = O[e];
        }
      // later bands rescale O by 2^{(M_old - M_new) c}; keep the snapshots' reference
      // by storing them normalised now
#pragma unroll
      for (int kk = 0; kk < kCalibMaxWindows; ++kk)
        if (kk == k) {
          const float inv = snap_l[kk] > 0.f ? 1.f / snap_l[kk] : 0.f;
#pragma unroll
          for (int e = 0; e < PER; ++e) snap[kk][e] *= inv;
        }
    }
  }
  const float invL = L > 0.f ? 1.f / L : 0.f;
  float full[PER];
  float ff = 0.f;
#pragma unroll
  for (int e = 0; e < PER; ++e) {
    full[e] = O[e] * invL;
    ff += full[e] * full[e];
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) ff += __shfl_xor_sync(0xffffffffu, ff, off);
  const float nf = sqrtf(ff);
#pragma unroll
  for (int k = 0; k < kCalibMaxWindows; ++k) {
    if (k >= K) break;
    float uu = 0.f, uv = 0.f;
#pragma unroll
    for (int e = 0; e < PER; ++e) {
      uu += snap[k][e] * snap[k][e];
      uv += snap[k][e] * full[e];
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      uu += __shfl_xor_sync(0xffffffffu, uu, off);
      uv += __shfl_xor_sync(0xffffffffu, uv, off);
    }
    const float nu = sqrtf(uu);
    const bool zu = nu <= 1e-12f, zf = nf <= 1e-12f;
    const float cv = (zu && zf) ? 1.f : ((zu || zf) ? 0.f : uv / (nu * nf));
    if (lane == 0) p.cos[((int64_t)u * p.group + g) * K + k] = cv;
  }
  if (p.traced != nullptr) {
    // trace check: the replayed full-window output against the traced one
    const float* tr = p.traced + ((int64_t)u * p.group + g) * D + lane * PER;
    float tt = 0.f, ft = 0.f;
#pragma unroll
    for (int e = 0; e < PER; ++e) {
      tt += tr[e] * tr[e];
      ft += tr[e] * full[e];
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      tt += __shfl_xor_sync(0xffffffffu, tt, off);
      ft += __shfl_xor_sync(0xffffffffu, ft, off);
    }
    const float nt = sqrtf(tt);
    const bool zt = nt <= 1e-12f, zf = nf <= 1e-12f;
    const float cv = (zt && zf) ? 1.f : ((zt || zf) ? 0.f : ft / (nt * nf));
    if (lane == 0) p.trace_cos[(int64_t)u * p.group + g] = cv;
  }
}

cudaError_t launch_calib_combine(const CalibCombineParams& p, int head_dim, cudaStream_t s) {
  if (p.n_windows > kCalibMaxWindows || p.n_units == 0) return cudaErrorInvalidValue;
  const dim3 grid(p.n_units), block(kMaxGroup * 32);
  switch (head_dim) {
    case 64: return launch_pdl(calib_combine_kernel<64>, grid, block, 0, s, p);
    case 128: return launch_pdl(calib_combine_kernel<128>, grid, block, 0, s, p);
    case 256: return launch_pdl(calib_combine_kernel<256>, grid, block, 0, s, p);
    default: return cudaErrorInvalidValue;
  }
}

// The bounded wait on its own: thread 0 waits for phase 0 of a freshly initialised
// mbarrier that no thread and no copy will ever arrive at, so the wait runs out after
// limit_ns and sets kErrWaitTimeout, as a kernel wait that gives up would. Nothing
// asynchronous is in flight and nothing else waits, so the CTA then simply ends.
__global__ void wait_probe_kernel(int* err, uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_barrier_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) mbar_wait_bounded(&bar, 0u, err, limit_ns);
}

cudaError_t launch_wait_probe(int* err, uint64_t limit_ns, cudaStream_t s) {
  wait_probe_kernel<<<1, 32, 0, s>>>(err, limit_ns);
  return cudaGetLastError();
}

cudaError_t launch_decode_combine(const DecodeParams& p, int head_dim, int num_sms, cudaStream_t s) {
  // at most a quarter as many (batch row, query head) pairs as SMs (a small step, whose
  // rings are cut into many segments): each pair's channels over D / 64 CTAs; with more
  // pairs the extra CTAs measured slower (batch 4 at 161K: 1-2% per step)
  const int pairs = p.batch * p.n_q_heads;
  const bool split = 4 * pairs <= num_sms && head_dim >= 128;
  const dim3 block(kCombineWarps * 32);
  switch (head_dim) {
    case 64: return launch_pdl(decode_combine_kernel<64, 1>, dim3(pairs), block, 0, s, p);
    case 128:
      return split ? launch_pdl(decode_combine_kernel<128, 2>, dim3(pairs * 2), block, 0, s, p)
                   : launch_pdl(decode_combine_kernel<128, 1>, dim3(pairs), block, 0, s, p);
    case 256:
      return split ? launch_pdl(decode_combine_kernel<256, 4>, dim3(pairs * 4), block, 0, s, p)
                   : launch_pdl(decode_combine_kernel<256, 1>, dim3(pairs), block, 0, s, p);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace hwkv
