// decode.cu -- split-KV decode attention over per-head rings, and its
// log-sum-exp combine (HeadWiseKV Sec. 3.2, Eq. conditional-attention-weight
// and Eq. conditional-attention, evaluated at the newest position; Sec. 3.3:
// each GQA query-head group reads its KV head's own slice).
//
// Work decomposition. For one layer, every (batch row b, KV head h) ring holds
// n_h = min(t, cap_h) resident slots; after the append of token t-1 these are
// exactly the positions J_{t-1}(W_h), so the softmax runs over all of them and
// slot order does not matter. Rings are cut into tiles of equal length
// (tile_len tokens, a multiple of 64), so a full-history head gets many tiles
// and a short-window head few: the split count follows the resident length and
// all window levels share one launch. A persistent grid walks the tile list.
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
#include "hwkv_internal.cuh"

namespace hwkv {

namespace {

struct TileInfo {
  int b, h;
  int64_t start;  // first slot of the tile
  int len;        // slots in the tile (>= 1)
  int64_t k_row, v_row;
};

__device__ __forceinline__ TileInfo locate_tile(const DecodeParams& p, int tile) {
  TileInfo ti;
  if (p.tiles != nullptr) {  // explicit tile table
    const CalibTile ct = p.tiles[tile];
    ti.b = ct.q_row;
    ti.h = ct.h;
    ti.start = 0;
    ti.len = ct.len;
    ti.k_row = ct.k_row;
    ti.v_row = ct.v_row;
    return ti;
  }
  ti.b = tile / p.tiles_per_b;
  const int lt = tile - ti.b * p.tiles_per_b;
  int h = 0;
  while (h + 1 < p.n_units && lt >= p.u[h].tile_begin + p.u[h].n_tiles) ++h;
  ti.h = h;
  const DecodeUnit& u = p.u[h];
  const int i = lt - u.tile_begin;
  ti.start = (int64_t)i * p.tile_len;
  const int64_t rem = (int64_t)u.n_valid - ti.start;
  ti.len = (int)(rem < p.tile_len ? rem : p.tile_len);
  ti.k_row = u.k_row0 + (int64_t)ti.b * u.cap + ti.start;
  ti.v_row = u.v_row0 + (int64_t)ti.b * u.cap + ti.start;
  return ti;
}

// named barrier of the four consumer warps (the producer warp does not take part)
__device__ __forceinline__ void consumer_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(kDecodeWarps * 32) : "memory");
}

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

template <int D>
struct DecodeCfg {
  static constexpr int kSlabs = D / 64;
  static constexpr int kTileBytes = kSlabs * kSlabBytes;  // 64 tokens of K (or V)
  static constexpr int kStageBytes = 2 * kTileBytes;
  static constexpr int kStages = D == 256 ? 3 : (D == 128 ? 6 : 8);
  static constexpr int kRedLd = D + 4;  // padded row of the cross-warp merge area (floats)
  static constexpr int kRedBytes = kDecodeWarps * kMaxGroup * kRedLd * 4;
  static constexpr int kMlBytes = kDecodeWarps * kMaxGroup * 8;
  static constexpr int kSmem = kStages * kStageBytes + kRedBytes + kMlBytes + 2 * kStages * 8 + 1024;
};

}  // namespace

template <int D>
__global__ void __launch_bounds__((kDecodeWarps + 1) * 32, 1)
    decode_split_kernel(const __grid_constant__ CUtensorMap k_map,
                        const __grid_constant__ CUtensorMap v_map, const DecodeParams p) {
  using C = DecodeCfg<D>;
  constexpr int STAGES = C::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  float* red_o = reinterpret_cast<float*>(smem + STAGES * C::kStageBytes);
  float2* red_ml = reinterpret_cast<float2*>(smem + STAGES * C::kStageBytes + C::kRedBytes);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * C::kStageBytes + C::kRedBytes +
                                               C::kMlBytes);
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
  __syncthreads();
  grid_dep_wait();    // the ring append and q come from kernels launched before
  grid_dep_launch();  // the combine kernel may start launching

  if (warp == kDecodeWarps) {
    // ------------------------------------------------------------ producer
    if (lane != 0) return;
    prefetch_tensormap(&k_map);
    prefetch_tensormap(&v_map);
    uint32_t it = 0;
    bool ok = true;
    for (int tile = blockIdx.x; ok && tile < p.n_tiles; tile += gridDim.x) {
      const TileInfo ti = locate_tile(p, tile);
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
        mbar_arrive_expect_tx(&full[s], C::kStageBytes);
        const int32_t krow = (int32_t)(ti.k_row + (int64_t)st * kStageTokens);
        const int32_t vrow = (int32_t)(ti.v_row + (int64_t)st * kStageTokens);
#pragma unroll
        for (int sl = 0; sl < C::kSlabs; ++sl)
          tma_load_2d(kdst + sl * kSlabBytes, &k_map, sl * 64, krow, &full[s]);
#pragma unroll
        for (int sl = 0; sl < C::kSlabs; ++sl)
          tma_load_2d(vdst + sl * kSlabBytes, &v_map, sl * 64, vrow, &full[s]);
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

  for (int tile = blockIdx.x; tile < p.n_tiles; tile += gridDim.x) {
    const TileInfo ti = locate_tile(p, tile);
    const int n_st = (ti.len + kStageTokens - 1) / kStageTokens;

    // Q^T as mma B fragments: b0 = channels 16kk + qk + {0,1}, b1 = +8; column = head qn
    uint32_t qf[D / 16][2];
    {
      const bool qv = qn < p.group;
      const __nv_bfloat16* qrow =
          p.q + ((int64_t)ti.b * p.n_q_heads + (int64_t)ti.h * p.group + (qv ? qn : 0)) * D;
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        qf[kk][0] = qv ? *reinterpret_cast<const uint32_t*>(qrow + kk * 16 + qk) : 0u;
        qf[kk][1] = qv ? *reinterpret_cast<const uint32_t*>(qrow + kk * 16 + 8 + qk) : 0u;
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
      if (p.k_new != nullptr) {
        // fused step: the new token's slot may lie in this stage; the warp owning that
        // row replaces the staged (stale) row with the new K/V and writes the ring row
        const int64_t row_in = (int64_t)p.u[ti.h].s_new - (ti.start + (int64_t)st * kStageTokens);
        if (row_in >= w * 16 && row_in < w * 16 + 16) {
          const int r = (int)row_in;
          const __nv_bfloat16* src_k = p.k_new + ((int64_t)ti.b * p.n_units + ti.h) * D;
          const __nv_bfloat16* src_v = p.v_new + ((int64_t)ti.b * p.n_units + ti.h) * D;
          const int64_t ring_row = ti.k_row - ti.start + p.u[ti.h].s_new;  // K region row
          const int64_t vring_row = ti.v_row - ti.start + p.u[ti.h].s_new;
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
      }
      float s0 = sa[0] + sb[0], s1 = sa[1] + sb[1], s2 = sa[2] + sb[2], s3 = sa[3] + sb[3];
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
      const uint32_t pb0 = movmatrix_trans(pack_bf16(p0, p1));
      const uint32_t pb1 = movmatrix_trans(pack_bf16(p2, p3));

      // O^T += V^T . P^T
      {
        const int mi = lane >> 3;
        const int r = w * 16 + (lane & 7) + (mi >> 1) * 8;
        const int csel = mi & 1;
#pragma unroll
        for (int mt = 0; mt < D / 16; ++mt) {
          uint32_t a0, a1, a2, a3;
          ldsm_x4_t(vbase + (mt >> 2) * kSlabBytes + swz128(r, (mt & 3) * 2 + csel), a0, a1, a2,
                    a3);
          mma_bf16_16816(o[mt], a0, a1, a2, a3, pb0, pb1);
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
        const int dim = mt * 16 + (lane >> 2);
        ro[qk * C::kRedLd + dim] = o[mt][0];
        ro[(qk + 1) * C::kRedLd + dim] = o[mt][1];
        ro[qk * C::kRedLd + dim + 8] = o[mt][2];
        ro[(qk + 1) * C::kRedLd + dim + 8] = o[mt][3];
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
      const bool single = p.tiles == nullptr && p.u[ti.h].n_tiles == 1;
      float* po = p.part_o + (int64_t)tile * kMaxGroup * D;
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
          p.part_ml[(int64_t)tile * kMaxGroup + n] = make_float2(M, L);
      }
    }
  }
}

// Log-sum-exp merge of the tile partials of one (batch row, query head):
// o = sum_j 2^{(m_j - M) c} o_j / sum_j 2^{(m_j - M) c} l_j, M = max_j m_j.
// One CTA of 8 warps per (batch row, query head): warp w sums tiles w, w+8, ...
// over all channels (each lane D/32 consecutive channels, vector loads); the
// eight partial sums are added in shared memory in warp order (deterministic).
// Heads whose ring is a single tile were written by the split kernel.
constexpr int kCombineWarps = 8;

template <int D>
__global__ void __launch_bounds__(kCombineWarps * 32) decode_combine_kernel(const DecodeParams p) {
  constexpr int PER = D / 32;  // channels per lane
  __shared__ float s_num[kCombineWarps][D];
  __shared__ float s_den[kCombineWarps];
  __shared__ float s_max[kCombineWarps];
  grid_dep_wait();  // partials come from the split kernel launched before
  const int bq = blockIdx.x;
  const int b = bq / p.n_q_heads;
  const int qh = bq - b * p.n_q_heads;
  const int h = qh / p.group;
  const int n = qh - h * p.group;
  const DecodeUnit& u = p.u[h];
  const int n_t = u.n_tiles;
  if (n_t <= 1) return;
  const int64_t tile0 = (int64_t)b * p.tiles_per_b + u.tile_begin;
  const float c = p.scale_log2;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;

  float mx = -INFINITY;
  for (int j = threadIdx.x; j < n_t; j += blockDim.x)
    mx = fmaxf(mx, p.part_ml[(tile0 + j) * kMaxGroup + n].x);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
  if (lane == 0) s_max[w] = mx;
  __syncthreads();
  float M = s_max[0];
#pragma unroll
  for (int k = 1; k < kCombineWarps; ++k) M = fmaxf(M, s_max[k]);

  float acc[PER];
#pragma unroll
  for (int e = 0; e < PER; ++e) acc[e] = 0.f;
  float den = 0.f;
  for (int j = w; j < n_t; j += kCombineWarps) {
    const float2 ml = p.part_ml[(tile0 + j) * kMaxGroup + n];
    const float wgt = ml.x == -INFINITY ? 0.f : ex2((ml.x - M) * c);
    den += wgt * ml.y;
    const float* src = p.part_o + ((tile0 + j) * kMaxGroup + n) * D + lane * PER;
#pragma unroll
    for (int e = 0; e < PER; e += 2) {
      const float2 v = *reinterpret_cast<const float2*>(src + e);
      acc[e] += wgt * v.x;
      acc[e + 1] += wgt * v.y;
    }
  }
#pragma unroll
  for (int e = 0; e < PER; ++e) s_num[w][lane * PER + e] = acc[e];
  if (lane == 0) s_den[w] = den;
  __syncthreads();
  float dsum = 0.f;
#pragma unroll
  for (int k = 0; k < kCombineWarps; ++k) dsum += s_den[k];
  for (int i = threadIdx.x; i < D; i += blockDim.x) {
    float num = 0.f;
#pragma unroll
    for (int k = 0; k < kCombineWarps; ++k) num += s_num[k][i];
    p.out[((int64_t)b * p.n_q_heads + qh) * D + i] = num / dsum;
  }
}

int decode_smem_bytes(int head_dim) {
  switch (head_dim) {
    case 64: return DecodeCfg<64>::kSmem;
    case 128: return DecodeCfg<128>::kSmem;
    case 256: return DecodeCfg<256>::kSmem;
    default: return -1;
  }
}

template <int D>
static cudaError_t launch_decode_t(const DecodeParams& p, const CUtensorMap& kmap,
                                   const CUtensorMap& vmap, int grid, cudaStream_t s) {
  const int smem = DecodeCfg<D>::kSmem;
  cudaError_t e = cudaFuncSetAttribute(decode_split_kernel<D>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(decode_split_kernel<D>, dim3(grid), dim3((kDecodeWarps + 1) * 32), smem, s,
                    kmap, vmap, p);
}

cudaError_t launch_decode(const DecodeParams& p, const CUtensorMap& kmap, const CUtensorMap& vmap,
                          int head_dim, int grid, cudaStream_t s) {
  switch (head_dim) {
    case 64: return launch_decode_t<64>(p, kmap, vmap, grid, s);
    case 128: return launch_decode_t<128>(p, kmap, vmap, grid, s);
    case 256: return launch_decode_t<256>(p, kmap, vmap, grid, s);
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
// a vector of norm <= eps counts as zero; both zero -> 1, one zero -> 0).
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

cudaError_t launch_decode_combine(const DecodeParams& p, int head_dim, cudaStream_t s) {
  bool any = false;  // nothing to merge when every ring is a single tile
  for (int h = 0; h < p.n_units; ++h) any |= p.u[h].n_tiles > 1;
  if (!any) return cudaSuccess;
  const dim3 grid(p.batch * p.n_q_heads), block(kCombineWarps * 32);
  switch (head_dim) {
    case 64: return launch_pdl(decode_combine_kernel<64>, grid, block, 0, s, p);
    case 128: return launch_pdl(decode_combine_kernel<128>, grid, block, 0, s, p);
    case 256: return launch_pdl(decode_combine_kernel<256>, grid, block, 0, s, p);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace hwkv
