/*
 * gen_device.cu -- device fill of seeded synthetic inputs (definition in hwkv_gen.h).
 * Bit-identical to gen_host.c. Test and bench infrastructure: it fills input
 * tensors; it is not part of the attention path.
 */
#include <cuda_runtime.h>
#include "hwkv_gen.h"

__global__ void hwkv_gen_fill_kernel(hwkv_gen_desc g, uint32_t tensor, uint32_t layer, int32_t B,
                                     int64_t pos0, int64_t n, int32_t H, int32_t d,
                                     uint16_t* __restrict__ out) {
  const int64_t total = (int64_t)B * n * H * d;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int32_t c = (int32_t)(e % d);
    const int64_t r = e / d;
    const int32_t h = (int32_t)(r % H);
    const int64_t bi = r / H;
    const int64_t i = bi % n;
    const int32_t b = (int32_t)(bi / n);
    const float s = hwkv_gen_head_scale(&g, tensor, layer, (uint32_t)h);
    out[e] = hwkv_gen_elem(&g, tensor, layer, (uint32_t)b, (uint32_t)h, (uint64_t)(pos0 + i),
                           (uint32_t)c, s);
  }
}

extern "C" int hwkv_gen_fill_device(const hwkv_gen_desc* g, uint32_t tensor, uint32_t layer,
                                    int32_t B, int64_t pos0, int64_t n, int32_t H, int32_t d,
                                    void* out, void* stream) {
  if (!g || (!out && (int64_t)B * n * H * d > 0) || B < 0 || n < 0 || H < 0 || d < 0) return 1;
  if (B > HWKV_GEN_MAX_BATCH || H > HWKV_GEN_MAX_HEADS || d > HWKV_GEN_MAX_DIM ||
      layer >= HWKV_GEN_MAX_LAYERS || pos0 < 0 || pos0 + n > HWKV_GEN_MAX_POS)
    return 1;
  const int64_t total = (int64_t)B * n * H * d;
  if (total == 0) return 0;
  int64_t blocks = (total + 255) / 256;
  if (blocks > 152 * 64) blocks = 152 * 64;
  hwkv_gen_fill_kernel<<<(unsigned)blocks, 256, 0, (cudaStream_t)stream>>>(
      *g, tensor, layer, B, pos0, n, H, d, (uint16_t*)out);
  return cudaGetLastError() == cudaSuccess ? 0 : 2;
}
