// append.cu -- K/V append with ring wrap (HeadWiseKV Sec. 3.3: each KV head keeps
// only its latest W states; App. "Runtime Realization": a head writes only its
// own slice).
//
// Position p of KV head u goes to slot p mod cap_u (with S sink slots: p < S
// to slot p, later ones to slot S + (p - S) mod (cap_u - S)); every row has its
// own first position t0 (ragged rows). A new token whose window slot a later
// token of the same call takes is not written. Block 0 also stores the rows' new lengths in the device length array. One launch covers every KV head and batch row of a layer;
// each thread moves one 16-byte vector, reads are coalesced over the input
// [batch][n][heads][d] and writes over the ring rows.
#include "hwkv_internal.cuh"

namespace hwkv {

__global__ void __launch_bounds__(256) append_kernel(const AppendParams p) {
  grid_dep_wait();  // k/v may come from the kernel launched before; the previous
                    // decode of this ring must be done reading before slots are reused
  if (blockIdx.x == 0 && p.lens != nullptr)  // nothing in this grid reads the lengths
    for (int b = threadIdx.x; b < p.batch; b += blockDim.x)
      p.lens[p.row0 + b] = (int32_t)(p.t0[b] + p.n);
  const int64_t vec_per_row = p.d / 8;
  const int64_t total = (int64_t)p.batch * p.n * p.n_units * vec_per_row;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t vec = e % vec_per_row;
    int64_t r = e / vec_per_row;
    const int h = (int)(r % p.n_units);
    r /= p.n_units;
    const int64_t i = r % p.n;
    const int b = (int)(r / p.n);
    const AppendUnit& u = p.u[h];
    const int64_t pos = (int64_t)p.t0[b] + i;
    // a window slot is overwritten within this call if position pos + (cap - sink) comes too
    if (pos >= u.sink && pos < (int64_t)p.t0[b] + p.n - (u.cap - u.sink)) continue;
    const int64_t slot = ring_slot(pos, u.cap, u.sink);
    const int64_t src = ((((int64_t)b * p.n + i) * p.n_units + h) * p.d) + vec * 8;
    const int64_t krow = u.k_row0 + (int64_t)(p.row0 + b) * u.stride + slot;
    const int64_t vrow = u.v_row0 + (int64_t)(p.row0 + b) * u.stride + slot;
    const uint4 kv = *reinterpret_cast<const uint4*>(p.k + src);
    const uint4 vv = *reinterpret_cast<const uint4*>(p.v + src);
    *reinterpret_cast<uint4*>(p.k_arena + krow * p.d + vec * 8) = kv;
    *reinterpret_cast<uint4*>(p.v_arena + vrow * p.d + vec * 8) = vv;
  }
}

// The 8-bit format (E4M3 codes, one fp32 scale per stored row): one warp per
// (batch row, token, KV head) row, each lane D/32 consecutive channels.
// amax = max |x|; s = amax / 448 (IEEE division); code = E4M3 of x / s (IEEE
// division, round to nearest even, saturating); amax = 0 stores s = 0 and zeros.
template <int D>
__global__ void __launch_bounds__(256) append_fp8_kernel(const AppendParams p) {
  constexpr int PER = D / 32;
  grid_dep_wait();
  if (blockIdx.x == 0 && p.lens != nullptr)
    for (int b = threadIdx.x; b < p.batch; b += blockDim.x)
      p.lens[p.row0 + b] = (int32_t)(p.t0[b] + p.n);
  const int lane = threadIdx.x & 31;
  const int64_t total = (int64_t)p.batch * p.n * p.n_units;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x / 32);
  for (int64_t e = (int64_t)blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5); e < total;
       e += warps) {
    const int h = (int)(e % p.n_units);
    const int64_t r = e / p.n_units;
    const int64_t i = r % p.n;
    const int b = (int)(r / p.n);
    const AppendUnit& u = p.u[h];
    const int64_t pos = (int64_t)p.t0[b] + i;
    if (pos >= u.sink && pos < (int64_t)p.t0[b] + p.n - (u.cap - u.sink)) continue;
    const int64_t slot = ring_slot(pos, u.cap, u.sink);
    const int64_t src = ((((int64_t)b * p.n + i) * p.n_units + h) * D) + lane * PER;
    const int64_t rows[2] = {u.k_row0 + (int64_t)(p.row0 + b) * u.stride + slot,
                             u.v_row0 + (int64_t)(p.row0 + b) * u.stride + slot};
    const __nv_bfloat16* in[2] = {p.k, p.v};
#pragma unroll
    for (int kv = 0; kv < 2; ++kv) {
      float x[PER];
      uint32_t raw[PER / 2];
      if constexpr (PER == 8) {
        const uint4 v = *reinterpret_cast<const uint4*>(in[kv] + src);
        raw[0] = v.x; raw[1] = v.y; raw[2] = v.z; raw[3] = v.w;
      } else {
        const uint2 v = *reinterpret_cast<const uint2*>(in[kv] + src);
        raw[0] = v.x; raw[1] = v.y;
      }
      float amax = 0.f;
#pragma unroll
      for (int j = 0; j < PER; ++j) {
        x[j] = __uint_as_float((j & 1 ? raw[j / 2] >> 16 : raw[j / 2] & 0xffffu) << 16);
        amax = fmaxf(amax, fabsf(x[j]));
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, off));
      const float sc = amax > 0.f ? __fdiv_rn(amax, 448.f) : 0.f;
      uint32_t w[PER / 4];
#pragma unroll
      for (int j = 0; j < PER; j += 4) {
        uint32_t c01 = 0, c23 = 0;
        if (amax > 0.f) {
          c01 = f32x2_to_e4m3x2(__fdiv_rn(x[j], sc), __fdiv_rn(x[j + 1], sc));
          c23 = f32x2_to_e4m3x2(__fdiv_rn(x[j + 2], sc), __fdiv_rn(x[j + 3], sc));
        }
        w[j / 4] = c01 | (c23 << 16);
      }
      uint8_t* dst = reinterpret_cast<uint8_t*>(p.k_arena) + rows[kv] * D + lane * PER;
      if constexpr (PER == 8)
        *reinterpret_cast<uint2*>(dst) = make_uint2(w[0], w[1]);
      else
        *reinterpret_cast<uint32_t*>(dst) = w[0];
      if (lane == 0) p.scales[rows[kv]] = sc;
    }
  }
}

cudaError_t launch_append(const AppendParams& p, bool fp8, cudaStream_t s) {
  if (fp8) {
    const int64_t rows = (int64_t)p.batch * p.n * p.n_units;
    if (rows == 0) return cudaSuccess;
    int64_t blocks = (rows + 7) / 8;  // 8 warps per block, one row each
    const int64_t cap_blocks = 152 * 16;
    if (blocks > cap_blocks) blocks = cap_blocks;
    switch (p.d) {
      case 128: return launch_pdl(append_fp8_kernel<128>, dim3((unsigned)blocks), dim3(256), 0, s, p);
      case 256: return launch_pdl(append_fp8_kernel<256>, dim3((unsigned)blocks), dim3(256), 0, s, p);
      default: return cudaErrorInvalidValue;
    }
  }
  const int64_t total = (int64_t)p.batch * p.n * p.n_units * (p.d / 8);
  if (total == 0) return cudaSuccess;
  int64_t blocks = (total + 255) / 256;
  const int64_t cap_blocks = 152 * 16;
  if (blocks > cap_blocks) blocks = cap_blocks;
  return launch_pdl(append_kernel, dim3((unsigned)blocks), dim3(256), 0, s, p);
}

}  // namespace hwkv
