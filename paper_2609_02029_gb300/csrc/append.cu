// append.cu -- K/V append with ring wrap (HeadWiseKV Sec. 3.3: each KV head keeps
// only its latest W states; App. "Runtime Realization": a head writes only its
// own slice).
//
// Position p of KV head u goes to slot p mod cap_u (with S sink slots: p < S
// to slot p, later ones to slot S + (p - S) mod (cap_u - S)); every row has its
// own first position t0 (ragged rows). A new token whose window slot a later
// token of the same call takes is not written (nor read). Block 0 also stores the
// rows' new lengths in the device length array. One launch covers every KV head
// and batch row of a layer: grid z is the batch row, grid x is laid out head by head,
// each head's range sized for the rows it can keep (min(n, cap)). Each thread moves
// 16-byte vectors of the rows that land, reads coalesced within each input row and
// writes over the ring rows.
#include <algorithm>

#include "hwkv_internal.cuh"

namespace hwkv {

__global__ void __launch_bounds__(256) append_kernel(const AppendParams p) {
  grid_dep_launch();  // the next kernel may start its prologue (it waits for this one)
  grid_dep_wait();  // k/v may come from the kernel launched before; the previous
                    // decode of this ring must be done reading before slots are reused
  if (blockIdx.x == 0 && blockIdx.z == 0 && p.lens != nullptr)
    for (int b = threadIdx.x; b < p.batch; b += blockDim.x)  // nothing in this grid reads them
      p.lens[p.row0 + b] = (int32_t)(p.t0[b] + p.n);
  // block (x, b): a block of KV head h's range of batch row b. Of the n new tokens only
  // these land: the ns that are sink positions (< sink, slot = position) and, of the
  // rest, the last wr (window-region slots), whose slots follow each other from one base
  // mod wr
  const int h = append_block_head(p, (int32_t)blockIdx.x), b = blockIdx.z;
  const int64_t xb = (int64_t)blockIdx.x - p.blk0[h];    // block within the head's range
  const int64_t nb = (int64_t)p.blk0[h + 1] - p.blk0[h];  // blocks of the head's range
  const AppendUnit& u = p.u[h];
  const int64_t n = p.n, t0 = p.t0[b];
  const int64_t wr = u.cap - u.sink;
  const int64_t ns = u.sink - t0 <= 0 ? 0 : (u.sink - t0 < n ? u.sink - t0 : n);
  const int64_t iw = n - wr > ns ? n - wr : ns;  // first new token kept in the window region
  const int64_t count = ns + (n - iw);
  const int64_t base = iw < n ? (t0 + iw - u.sink) % wr : 0;  // window slot of token iw
  const int vpr_log2 = __ffs((int)(p.d / 8)) - 1;  // 16-byte vectors per row: 8, 16 or 32
  const int64_t vmask = (1 << vpr_log2) - 1;
  const int64_t krow0 = u.k_row0 + (int64_t)(p.row0 + b) * u.stride;
  const int64_t vrow0 = u.v_row0 + (int64_t)(p.row0 + b) * u.stride;
  for (int64_t e = xb * blockDim.x + threadIdx.x; e < (count << vpr_log2); e += nb * blockDim.x) {
    const int64_t j = e >> vpr_log2, vec = e & vmask;
    int64_t i, slot;
    if (j < ns) {
      i = j;
      slot = t0 + j;
    } else {
      i = iw + (j - ns);
      const int64_t q = base + (j - ns);  // < 2 wr
      slot = u.sink + (q >= wr ? q - wr : q);
    }
    const int64_t src = ((((int64_t)b * n + i) * p.n_units + h) * p.d) + vec * 8;
    const uint4 kv = *reinterpret_cast<const uint4*>(p.k + src);
    const uint4 vv = *reinterpret_cast<const uint4*>(p.v + src);
    *reinterpret_cast<uint4*>(p.k_arena + (krow0 + slot) * p.d + vec * 8) = kv;
    *reinterpret_cast<uint4*>(p.v_arena + (vrow0 + slot) * p.d + vec * 8) = vv;
  }
}

// The 8-bit format (E4M3 codes, one fp32 scale per stored row), laid out as the
// bf16 kernel: the blocks of head h's range in grid x and row b in grid z take the
// landing tokens of KV head h of batch row b; each half warp quantizes one token row
// (K and V), each lane D/16 consecutive
// channels (a half-warp row needs one shuffle step less per value than a warp row
// and spreads each row's index arithmetic over twice the values).
// amax = max |x|; s = the smallest power of two >= amax / 448; code = E4M3 of x / s
// (an exact scaling; round to nearest even, saturating); amax = 0 stores s = 0 and
// zeros (the shared row helper e4m3_quantize_row_warp).
template <int D>
__global__ void __launch_bounds__(256) append_fp8_kernel(const AppendParams p) {
  constexpr int PER = D / 16;  // values per lane
  grid_dep_launch();
  grid_dep_wait();
  if (blockIdx.x == 0 && blockIdx.z == 0 && p.lens != nullptr)
    for (int b = threadIdx.x; b < p.batch; b += blockDim.x)
      p.lens[p.row0 + b] = (int32_t)(p.t0[b] + p.n);
  const int h = append_block_head(p, (int32_t)blockIdx.x), b = blockIdx.z;
  const int64_t xb = (int64_t)blockIdx.x - p.blk0[h];    // block within the head's range
  const int64_t nb = (int64_t)p.blk0[h + 1] - p.blk0[h];  // blocks of the head's range
  const int hl = threadIdx.x & 15;  // lane within the half warp
  const AppendUnit& u = p.u[h];
  const int64_t n = p.n, t0 = p.t0[b];
  const int64_t wr = u.cap - u.sink;
  const int64_t ns = u.sink - t0 <= 0 ? 0 : (u.sink - t0 < n ? u.sink - t0 : n);
  const int64_t iw = n - wr > ns ? n - wr : ns;  // first new token kept in the window region
  const int64_t count = ns + (n - iw);
  const int64_t base = iw < n ? (t0 + iw - u.sink) % wr : 0;  // window slot of token iw
  const int64_t krow0 = u.k_row0 + (int64_t)(p.row0 + b) * u.stride;
  const int64_t vrow0 = u.v_row0 + (int64_t)(p.row0 + b) * u.stride;
  // half warp g takes rows g, g + H, ... (H = the half warps of the grid's x slice); both
  // halves of a warp make the same trips (a row past the end is read clamped and not
  // stored) so the shuffles of the row maximum stay converged
  const int64_t hstride = nb * (blockDim.x / 16);
  const int half = (threadIdx.x >> 4) & 1;
  constexpr int ROWS = 2;  // rows per half warp and trip, all their loads in flight at once
  for (int64_t jw = xb * (blockDim.x / 16) + (threadIdx.x >> 4) - half; jw < count;
       jw += ROWS * hstride) {
    bool valid[ROWS];
    int64_t slot[ROWS];
    // K and V loads of every row before any arithmetic: the stores below go through
    // the arena pointer, which the compiler cannot tell apart from p.k and p.v
    uint32_t raw[ROWS][2][PER / 2];
#pragma unroll
    for (int r = 0; r < ROWS; ++r) {
      const int64_t j0 = jw + r * hstride + half;
      valid[r] = j0 < count;
      const int64_t j = valid[r] ? j0 : count - 1;
      int64_t i;
      if (j < ns) {
        i = j;
        slot[r] = t0 + j;
      } else {
        i = iw + (j - ns);
        const int64_t q = base + (j - ns);  // < 2 wr
        slot[r] = u.sink + (q >= wr ? q - wr : q);
      }
      const int64_t src = ((((int64_t)b * n + i) * p.n_units + h) * D) + hl * PER;
#pragma unroll
      for (int kv = 0; kv < 2; ++kv)
#pragma unroll
        for (int c = 0; c < PER / 8; ++c) {
          const uint4 v4 = *reinterpret_cast<const uint4*>((kv ? p.v : p.k) + src + c * 8);
          raw[r][kv][4 * c] = v4.x; raw[r][kv][4 * c + 1] = v4.y;
          raw[r][kv][4 * c + 2] = v4.z; raw[r][kv][4 * c + 3] = v4.w;
        }
    }
#pragma unroll
    for (int r = 0; r < ROWS; ++r)
#pragma unroll
      for (int kv = 0; kv < 2; ++kv) {
        uint32_t w[PER / 4];
        const float sc = e4m3_quantize_row_warp<PER, 16>(raw[r][kv], w);
        if (valid[r]) {
          const int64_t row = (kv ? vrow0 : krow0) + slot[r];
          uint8_t* dst = reinterpret_cast<uint8_t*>(p.k_arena) + row * D + hl * PER;
          if constexpr (PER == 16)
            *reinterpret_cast<uint4*>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
          else
            *reinterpret_cast<uint2*>(dst) = make_uint2(w[0], w[1]);
          if (hl == 0) p.scales[row] = sc;
        }
      }
  }
}

// Prefill staging for the 8-bit format, one warp per row, everything in fp16 for
// an fp16 tensor-core pass. Ring rows: the held slots of (unit, batch row), below
// min(t0, cap), dequantized (code x scale), and zeros for the next 128 slots, which
// a key tile may read past them. Chunk K/V rows: quantized as append_fp8_kernel
// stores them (same helper), then dequantized. q rows: converted. A code has at
// most 4 significant bits and the row scale is a power of two, so code x scale is
// exact in fp16 whenever it lies in fp16's range (at least 2^-24 for the smallest
// code step, at most 65504); q in fp16 is exact for bf16 values of magnitude 2^-14
// to 65504. Magnitudes past the fp16 range saturate to +-65504.
__device__ __forceinline__ void e4m3_words_to_f16(const uint32_t* words, int nwords, float sc,
                                                  uint32_t* out) {
  for (int i = 0; i < nwords; ++i) {
    uint32_t lo, hi;
    e4m3x4_to_f16x2(words[i], lo, hi);
    const __half2 l2 = *reinterpret_cast<const __half2*>(&lo);
    const __half2 h2 = *reinterpret_cast<const __half2*>(&hi);
    out[2 * i] = pack_f16_sat(__low2float(l2) * sc, __high2float(l2) * sc);
    out[2 * i + 1] = pack_f16_sat(__low2float(h2) * sc, __high2float(h2) * sc);
  }
}
template <int PER>
__device__ __forceinline__ void store_row16(uint16_t* dst, const uint32_t (&w)[PER / 2]) {
  if constexpr (PER == 8)
    *reinterpret_cast<uint4*>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
  else
    *reinterpret_cast<uint2*>(dst) = make_uint2(w[0], w[1]);
}
template <int PER>
__device__ __forceinline__ void load_row_bf16(const __nv_bfloat16* src, uint32_t (&raw)[PER / 2]) {
  if constexpr (PER == 8) {
    const uint4 v = *reinterpret_cast<const uint4*>(src);
    raw[0] = v.x; raw[1] = v.y; raw[2] = v.z; raw[3] = v.w;
  } else {
    const uint2 v = *reinterpret_cast<const uint2*>(src);
    raw[0] = v.x; raw[1] = v.y;
  }
}

template <int D>
__global__ void __launch_bounds__(256) fp8_stage_kernel(const Fp8StageParams p) {
  constexpr int PER = D / 32;
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x / 32);
  const int64_t warp0 = (int64_t)blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5);
  // ring rows: index over (unit, kv, batch row, slot < span)
  int64_t max_cap = 0;
  for (int h = 0; h < p.n_units; ++h) max_cap = p.u[h].cap > max_cap ? p.u[h].cap : max_cap;
  const int64_t span = min(max_cap, p.t0 + 128);
  const int64_t ring_items = (int64_t)p.n_units * 2 * p.batch * span;
  for (int64_t e = warp0; e < ring_items; e += warps) {
    const int64_t slot = e % span;
    int64_t r = e / span;
    const int b = (int)(r % p.batch);
    r /= p.batch;
    const int kv = (int)(r % 2);
    const int h = (int)(r / 2);
    const Fp8StageUnit& u = p.u[h];
    if (slot >= u.cap) continue;
    const int64_t src = (kv ? u.v_row0 : u.k_row0) + (int64_t)(p.row0 + b) * u.stride + slot;
    const int64_t dst = (kv ? u.sv_row0 : u.sk_row0) + (int64_t)b * u.cap + slot;
    uint32_t out[PER / 2];
    if (slot >= p.t0) {  // not held
#pragma unroll
      for (int i = 0; i < PER / 2; ++i) out[i] = 0u;
    } else {
      const uint8_t* c = p.arena + src * D + lane * PER;
      uint32_t words[PER / 4];
      if constexpr (PER == 8) {
        const uint2 w2 = *reinterpret_cast<const uint2*>(c);
        words[0] = w2.x;
        words[1] = w2.y;
      } else {
        words[0] = *reinterpret_cast<const uint32_t*>(c);
      }
      e4m3_words_to_f16(words, PER / 4, p.arena_scales[src], out);
    }
    store_row16<PER>(p.ring + dst * D + lane * PER, out);
  }
  // chunk rows: index over (batch row, token, KV head)
  const int64_t chunk_items = (int64_t)p.batch * p.n * p.n_units;
  for (int64_t e = warp0; e < chunk_items; e += warps) {
    const int64_t off = e * D + lane * PER;
#pragma unroll
    for (int kv = 0; kv < 2; ++kv) {
      uint32_t raw[PER / 2];
      load_row_bf16<PER>((kv ? p.v : p.k) + off, raw);
      uint32_t w[PER / 4];
      const float sc = e4m3_quantize_row_warp<PER>(raw, w);
      uint32_t out[PER / 2];
      e4m3_words_to_f16(w, PER / 4, sc, out);
      store_row16<PER>((kv ? p.v16 : p.k16) + off, out);
    }
  }
  // q rows: index over (batch row, token, query head)
  const int64_t q_items = (int64_t)p.batch * p.n * p.n_q_heads;
  for (int64_t e = warp0; e < q_items; e += warps) {
    const int64_t off = e * D + lane * PER;
    uint32_t raw[PER / 2];
    load_row_bf16<PER>(p.q + off, raw);
    uint32_t out[PER / 2];
#pragma unroll
    for (int i = 0; i < PER / 2; ++i)
      out[i] = pack_f16_sat(__uint_as_float(raw[i] << 16), __uint_as_float(raw[i] & 0xffff0000u));
    store_row16<PER>(p.q16 + off, out);
  }
}

cudaError_t launch_fp8_stage(const Fp8StageParams& p, int head_dim, cudaStream_t s) {
  int64_t max_cap = 0;
  for (int h = 0; h < p.n_units; ++h) max_cap = p.u[h].cap > max_cap ? p.u[h].cap : max_cap;
  const int64_t span = min(max_cap, p.t0 + 128);
  const int64_t rows = (int64_t)p.n_units * 2 * p.batch * span +
                       (int64_t)p.batch * p.n * (p.n_units + p.n_q_heads);
  if (rows == 0) return cudaSuccess;
  int64_t blocks = (rows + 7) / 8;  // 8 warps per block
  const int64_t cap_blocks = 152 * 16;
  if (blocks > cap_blocks) blocks = cap_blocks;
  switch (head_dim) {
    case 128: fp8_stage_kernel<128><<<(unsigned)blocks, 256, 0, s>>>(p); break;
    case 256: fp8_stage_kernel<256><<<(unsigned)blocks, 256, 0, s>>>(p); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

cudaError_t launch_append(const AppendParams& p0, bool fp8, cudaStream_t s) {
  // grid x of a batch row is laid out head by head, each head sized for the most rows it
  // can take (min(n, cap)); a block past its row's own landing count exits at once.
  // bf16: up to 4 16-byte vectors per thread. 8-bit: 16 half warps per block, up to
  // kFp8RowsPerHalfWarp rows each (fewer, longer-lived blocks measured faster than one or
  // two trips per half warp).
  constexpr int64_t kFp8RowsPerHalfWarp = 8;
  AppendParams p = p0;
  int64_t total = 0;
  for (int h = 0; h < p.n_units; ++h) {
    const int64_t rows = std::min(p.n, p.u[h].cap);
    p.blk0[h] = (int32_t)total;
    total += fp8 ? (rows + 16 * kFp8RowsPerHalfWarp - 1) / (16 * kFp8RowsPerHalfWarp)
                 : (rows * (p.d / 8) + 1023) / 1024;
    if (total >= (int64_t)INT32_MAX) return cudaErrorInvalidValue;
  }
  p.blk0[p.n_units] = (int32_t)total;
  if (total == 0 || p.batch == 0) return cudaSuccess;
  const dim3 grid((unsigned)total, 1, (unsigned)p.batch);
  if (fp8) {
    switch (p.d) {
      case 128: return launch_pdl(append_fp8_kernel<128>, grid, dim3(256), 0, s, p);
      case 256: return launch_pdl(append_fp8_kernel<256>, grid, dim3(256), 0, s, p);
      default: return cudaErrorInvalidValue;
    }
  }
  return launch_pdl(append_kernel, grid, dim3(256), 0, s, p);
}

}  // namespace hwkv
