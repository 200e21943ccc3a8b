// append.cu -- K/V append with ring wrap (HeadWiseKV Sec. 3.3: each KV head keeps
// only its latest W states; App. "Runtime Realization": a head writes only its
// own slice).
//
// Position p of KV head u goes to slot p mod cap_u; every row has its own
// first position t0 (ragged rows). Of the n new tokens only the last
// min(n, cap_u) are written: an earlier one would be overwritten in the same
// call. Block 0 also stores the rows' new lengths in the device length array. One launch covers every KV head and batch row of a layer;
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
    const int64_t keep = p.n < u.cap ? p.n : u.cap;
    if (i < p.n - keep) continue;  // overwritten within this call
    const int64_t slot = ((int64_t)p.t0[b] + i) % u.cap;
    const int64_t src = ((((int64_t)b * p.n + i) * p.n_units + h) * p.d) + vec * 8;
    const int64_t krow = u.k_row0 + (int64_t)(p.row0 + b) * u.cap + slot;
    const int64_t vrow = u.v_row0 + (int64_t)(p.row0 + b) * u.cap + slot;
    const uint4 kv = *reinterpret_cast<const uint4*>(p.k + src);
    const uint4 vv = *reinterpret_cast<const uint4*>(p.v + src);
    *reinterpret_cast<uint4*>(p.k_arena + krow * p.d + vec * 8) = kv;
    *reinterpret_cast<uint4*>(p.v_arena + vrow * p.d + vec * 8) = vv;
  }
}

cudaError_t launch_append(const AppendParams& p, cudaStream_t s) {
  const int64_t total = (int64_t)p.batch * p.n * p.n_units * (p.d / 8);
  if (total == 0) return cudaSuccess;
  int64_t blocks = (total + 255) / 256;
  const int64_t cap_blocks = 152 * 16;
  if (blocks > cap_blocks) blocks = cap_blocks;
  return launch_pdl(append_kernel, dim3((unsigned)blocks), dim3(256), 0, s, p);
}

}  // namespace hwkv
