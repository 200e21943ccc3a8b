// prefill.cu -- window-limited causal prefill attention of one chunk
// (HeadWiseKV Sec. 3.2, Eq. conditional-attention-weight and
// Eq. conditional-attention for every prompt position; Sec. 3.3 / App.
// "Runtime Realization": the head reads only its own K/V slice).
//
// Query p in [t0, t0+n) of query head q attends to KV head q/G at positions
// [max(0, p-W+1), p]. Positions < t0 come from the head's ring, > = t0 from
// the chunk's own K/V input. The ring is walked in slot order: slot j holds
// the unique retained position congruent to j mod cap, so every key column
// carries its position and the window/causal mask is applied per element
// (softmax does not depend on key order). Tiles that no query of the block
// can see are skipped, so a short-window head does window-sized work.
//
// CTA = 64 query rows of one query head, 4 warps x 16 rows; key tiles of 64
// double-buffered through cp.async into 128-byte-swizzled shared memory;
// S = Q K^T and O += P V on mma.sync m16n8k16 (bf16 in, fp32 accumulate) with
// an online softmax per row.
#include "hwkv_internal.cuh"

namespace hwkv {

namespace {

constexpr int BM = 64;  // query rows per CTA
constexpr int BN = 64;  // keys per tile

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool valid) {
  const int sz = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(sz)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// a key tile: either ring slots [j0, j0+64) or chunk rows [i0, i0+64)
struct KeyTile {
  int hist;     // 1 = ring, 0 = chunk
  int64_t j0;   // first slot (ring) or first chunk row
};

}  // namespace

template <int D>
__global__ void __launch_bounds__(128) prefill_kernel(const PrefillParams p) {
  constexpr int SLAB_ROWS_BYTES = 64 * 128;  // 64 rows x 128 B
  constexpr int TILE_BYTES = (D / 64) * SLAB_ROWS_BYTES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* sQ = smem;
  uint8_t* sK[2] = {smem + TILE_BYTES, smem + 2 * TILE_BYTES};
  uint8_t* sV[2] = {smem + 3 * TILE_BYTES, smem + 4 * TILE_BYTES};

  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  const int n_qblocks = (int)((p.n + BM - 1) / BM);
  const int qb = n_qblocks - 1 - (int)blockIdx.x;  // longest rows first
  const int qh = blockIdx.y;
  const int b = blockIdx.z;
  const int h = qh / p.group;
  const PrefillUnit& u = p.u[h];
  const int64_t t0 = p.t0;
  const int64_t W = u.window;
  const int64_t p0 = t0 + (int64_t)qb * BM;                        // first query position
  const int64_t p_last = min(p0 + BM, t0 + p.n) - 1;               // last valid query position
  const int64_t lo_need = W == 0 ? 0 : max((int64_t)0, p0 - W + 1);  // lowest key any row needs
  const int64_t n_hist = min(t0, u.cap);
  const int64_t r0 = t0 % u.cap;
  const int64_t ld_in = (int64_t)p.n_units * D;  // chunk K/V row stride (elements)
  const int64_t ld_q = (int64_t)p.n_q_heads * D;

  // position held by ring slot j (valid only for j < n_hist)
  auto slot_pos = [&](int64_t j) -> int64_t {
    if (t0 <= u.cap) return j;
    return j < r0 ? t0 - r0 + j : t0 - r0 - u.cap + j;
  };

  // ---- the key tiles this block needs
  // ring: slot tiles whose largest held position reaches lo_need
  // chunk: rows [max(t0, lo_need), p_last] - t0
  const int64_t n_hist_tiles = (n_hist + BN - 1) / BN;
  const int64_t c_lo = max(t0, lo_need) - t0;
  const int64_t c_first = (c_lo / BN) * BN;
  const int64_t c_hi = p_last - t0;  // inclusive
  const int64_t n_chunk_tiles = c_hi >= c_first ? (c_hi - c_first) / BN + 1 : 0;
  const bool hist_needed = n_hist > 0 && (W == 0 || p0 - W + 1 < t0);

  auto tile_needed = [&](int64_t jt) -> bool {  // ring tile index
    if (!hist_needed) return false;
    if (W == 0) return true;
    const int64_t j0 = jt * BN, j1 = min(j0 + BN, n_hist) - 1;
    int64_t mx = slot_pos(j1);
    if (t0 > u.cap && r0 > j0 && r0 <= j1) mx = max(mx, slot_pos(r0 - 1));
    return mx >= lo_need;
  };
  auto next_hist = [&](int64_t jt) -> int64_t {  // first needed ring tile >= jt, or -1
    for (; jt < n_hist_tiles; ++jt)
      if (tile_needed(jt)) return jt;
    return -1;
  };

  // ---- loaders
  const __nv_bfloat16* ring_k = p.k_arena + (u.k_row0 + (int64_t)b * u.cap) * D;
  const __nv_bfloat16* ring_v = p.v_arena + (u.v_row0 + (int64_t)b * u.cap) * D;
  const __nv_bfloat16* in_k = p.k + ((int64_t)b * p.n * p.n_units + h) * D;
  const __nv_bfloat16* in_v = p.v + ((int64_t)b * p.n * p.n_units + h) * D;

  auto load_tile = [&](const KeyTile& kt, int buf) {
    const uint32_t kd = smem_u32(sK[buf]), vd = smem_u32(sV[buf]);
    constexpr int CHUNKS = BN * D / 8;
#pragma unroll 4
    for (int e = tid; e < CHUNKS; e += 128) {
      const int r = e / (D / 8), cc = e % (D / 8);
      const uint32_t off = (cc >> 3) * SLAB_ROWS_BYTES + swz128(r, cc & 7);
      const int64_t row = kt.j0 + r;
      if (kt.hist) {
        const bool ok = row < n_hist;
        const int64_t rr = ok ? row : 0;
        cp_async16(kd + off, ring_k + rr * D + cc * 8, ok);
        cp_async16(vd + off, ring_v + rr * D + cc * 8, ok);
      } else {
        const bool ok = row < p.n;
        const int64_t rr = ok ? row : 0;
        cp_async16(kd + off, in_k + rr * ld_in + cc * 8, ok);
        cp_async16(vd + off, in_v + rr * ld_in + cc * 8, ok);
      }
    }
  };

  // Q tile
  {
    const __nv_bfloat16* qsrc = p.q + ((int64_t)b * p.n * p.n_q_heads + qh) * D;
    const uint32_t qd = smem_u32(sQ);
    constexpr int CHUNKS = BM * D / 8;
    for (int e = tid; e < CHUNKS; e += 128) {
      const int r = e / (D / 8), cc = e % (D / 8);
      const int64_t row = (int64_t)qb * BM + r;
      const bool ok = row < p.n;
      cp_async16(qd + (cc >> 3) * SLAB_ROWS_BYTES + swz128(r, cc & 7),
                 qsrc + (ok ? row : 0) * ld_q + cc * 8, ok);
    }
  }

  // tile sequence: needed ring tiles, then chunk tiles
  int64_t hist_cur = next_hist(0);
  int64_t chunk_cur = 0;
  auto fetch_next = [&](KeyTile& kt) -> bool {
    if (hist_cur >= 0) {
      kt.hist = 1;
      kt.j0 = hist_cur * BN;
      hist_cur = next_hist(hist_cur + 1);
      return true;
    }
    if (chunk_cur < n_chunk_tiles) {
      kt.hist = 0;
      kt.j0 = c_first + chunk_cur * BN;
      ++chunk_cur;
      return true;
    }
    return false;
  };

  KeyTile cur, nxt;
  bool have_cur = fetch_next(cur);
  if (have_cur) load_tile(cur, 0);
  cp_async_commit();

  const float c = p.scale_log2;
  float o[D / 8][4];
#pragma unroll
  for (int i = 0; i < D / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  const int64_t prow0 = p0 + warp * 16 + (lane >> 2);  // query positions of this lane's rows
  const int64_t prow1 = prow0 + 8;

  int buf = 0;
  while (have_cur) {
    const bool have_nxt = fetch_next(nxt);
    if (have_nxt) load_tile(nxt, buf ^ 1);
    cp_async_commit();
    cp_async_wait<1>();
    __syncthreads();

    // S = Q K^T : 16 rows x 64 keys per warp
    float s[BN / 8][4];
#pragma unroll
    for (int i = 0; i < BN / 8; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
    {
      const uint32_t qbase = smem_u32(sQ), kbase = smem_u32(sK[buf]);
      const int qr = warp * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
      const int qc = lane >> 4;
      const int kr = (lane & 7) + (lane >> 4) * 8;
      const int kc = (lane >> 3) & 1;
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        uint32_t a0, a1, a2, a3;
        ldsm_x4(qbase + (kk >> 2) * SLAB_ROWS_BYTES + swz128(qr, (kk & 3) * 2 + qc), a0, a1, a2,
                a3);
#pragma unroll
        for (int nt = 0; nt < BN / 8; nt += 2) {
          uint32_t b0, b1, b2, b3;
          ldsm_x4(kbase + (kk >> 2) * SLAB_ROWS_BYTES + swz128(nt * 8 + kr, (kk & 3) * 2 + kc),
                  b0, b1, b2, b3);
          mma_bf16_16816(s[nt], a0, a1, a2, a3, b0, b1);
          mma_bf16_16816(s[nt + 1], a0, a1, a2, a3, b2, b3);
        }
      }
    }

    // mask by position: key visible to row p iff pos <= p and p - pos < W (and held)
#pragma unroll
    for (int nt = 0; nt < BN / 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int64_t col = cur.j0 + nt * 8 + (lane & 3) * 2 + e;
        int64_t pos;
        bool held;
        if (cur.hist) {
          held = col < n_hist;
          pos = held ? slot_pos(col) : 0;
        } else {
          held = col < p.n;
          pos = t0 + col;
        }
        const bool v0 = held && pos <= prow0 && (W == 0 || prow0 - pos < W);
        const bool v1 = held && pos <= prow1 && (W == 0 || prow1 - pos < W);
        if (!v0) s[nt][e] = -INFINITY;
        if (!v1) s[nt][2 + e] = -INFINITY;
      }
    }

    // online softmax (rows prow0 -> elements 0,1; prow1 -> elements 2,3)
    float x0 = -INFINITY, x1 = -INFINITY;
#pragma unroll
    for (int nt = 0; nt < BN / 8; ++nt) {
      x0 = fmaxf(x0, fmaxf(s[nt][0], s[nt][1]));
      x1 = fmaxf(x1, fmaxf(s[nt][2], s[nt][3]));
    }
    x0 = fmaxf(x0, __shfl_xor_sync(0xffffffffu, x0, 1));
    x0 = fmaxf(x0, __shfl_xor_sync(0xffffffffu, x0, 2));
    x1 = fmaxf(x1, __shfl_xor_sync(0xffffffffu, x1, 1));
    x1 = fmaxf(x1, __shfl_xor_sync(0xffffffffu, x1, 2));
    const float n0 = fmaxf(m0, x0), n1 = fmaxf(m1, x1);
    const float u0 = n0 == -INFINITY ? 0.f : n0, u1 = n1 == -INFINITY ? 0.f : n1;
    const float al0 = ex2((m0 - u0) * c), al1 = ex2((m1 - u1) * c);
    m0 = n0;
    m1 = n1;
    float rs0 = 0.f, rs1 = 0.f;
#pragma unroll
    for (int nt = 0; nt < BN / 8; ++nt) {
      s[nt][0] = ex2((s[nt][0] - u0) * c);
      s[nt][1] = ex2((s[nt][1] - u0) * c);
      s[nt][2] = ex2((s[nt][2] - u1) * c);
      s[nt][3] = ex2((s[nt][3] - u1) * c);
      rs0 += s[nt][0] + s[nt][1];
      rs1 += s[nt][2] + s[nt][3];
    }
    l0 = l0 * al0 + rs0;
    l1 = l1 * al1 + rs1;
#pragma unroll
    for (int i = 0; i < D / 8; ++i) {
      o[i][0] *= al0;
      o[i][1] *= al0;
      o[i][2] *= al1;
      o[i][3] *= al1;
    }

    // O += P V
    {
      const uint32_t vbase = smem_u32(sV[buf]);
      const int vr = (lane & 7) + ((lane >> 3) & 1) * 8;
      const int vc = lane >> 4;
#pragma unroll
      for (int ks = 0; ks < BN / 16; ++ks) {
        const uint32_t a0 = pack_bf16(s[2 * ks][0], s[2 * ks][1]);
        const uint32_t a1 = pack_bf16(s[2 * ks][2], s[2 * ks][3]);
        const uint32_t a2 = pack_bf16(s[2 * ks + 1][0], s[2 * ks + 1][1]);
        const uint32_t a3 = pack_bf16(s[2 * ks + 1][2], s[2 * ks + 1][3]);
#pragma unroll
        for (int dt = 0; dt < D / 8; dt += 2) {
          uint32_t b0, b1, b2, b3;
          ldsm_x4_t(vbase + (dt >> 3) * SLAB_ROWS_BYTES + swz128(ks * 16 + vr, (dt & 7) + vc), b0,
                    b1, b2, b3);
          mma_bf16_16816(o[dt], a0, a1, a2, a3, b0, b1);
          mma_bf16_16816(o[dt + 1], a0, a1, a2, a3, b2, b3);
        }
      }
    }
    __syncthreads();  // everyone done with buf before it is refilled
    cur = nxt;
    have_cur = have_nxt;
    buf ^= 1;
  }
  cp_async_wait<0>();

  // normalise and store rows that exist
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  const float inv0 = l0 > 0.f ? 1.f / l0 : 0.f, inv1 = l1 > 0.f ? 1.f / l1 : 0.f;
  const int64_t i0 = prow0 - t0, i1 = prow1 - t0;
  float* out0 = p.out + (((int64_t)b * p.n + i0) * p.n_q_heads + qh) * D;
  float* out1 = p.out + (((int64_t)b * p.n + i1) * p.n_q_heads + qh) * D;
#pragma unroll
  for (int dt = 0; dt < D / 8; ++dt) {
    const int col = dt * 8 + (lane & 3) * 2;
    if (i0 < p.n) *reinterpret_cast<float2*>(out0 + col) = make_float2(o[dt][0] * inv0, o[dt][1] * inv0);
    if (i1 < p.n) *reinterpret_cast<float2*>(out1 + col) = make_float2(o[dt][2] * inv1, o[dt][3] * inv1);
  }
}

template <int D>
static cudaError_t launch_prefill_t(const PrefillParams& p, cudaStream_t s) {
  const int smem = 5 * (D / 64) * 64 * 128 + 1024;
  cudaError_t e =
      cudaFuncSetAttribute(prefill_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  dim3 grid((unsigned)((p.n + BM - 1) / BM), (unsigned)p.n_q_heads, (unsigned)p.batch);
  prefill_kernel<D><<<grid, 128, smem, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_prefill(const PrefillParams& p, int head_dim, cudaStream_t s) {
  if (p.n == 0) return cudaSuccess;
  switch (head_dim) {
    case 64: return launch_prefill_t<64>(p, s);
    case 128: return launch_prefill_t<128>(p, s);
    case 256: return launch_prefill_t<256>(p, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace hwkv
