/*
 * gen_host.c -- host fill of seeded synthetic inputs (definition in hwkv_gen.h).
 * Output layout matches the tensors the library takes: [B][n][H][d] bf16 bits,
 * positions pos0 .. pos0+n-1.
 */
#include "hwkv_gen.h"

int hwkv_gen_fill_host(const hwkv_gen_desc* g, uint32_t tensor, uint32_t layer, int32_t B,
                       int64_t pos0, int64_t n, int32_t H, int32_t d, uint16_t* out) {
  if (!g || !out || B < 0 || n < 0 || H < 0 || d < 0) return 1;
  if (B > HWKV_GEN_MAX_BATCH || H > HWKV_GEN_MAX_HEADS || d > HWKV_GEN_MAX_DIM ||
      layer >= HWKV_GEN_MAX_LAYERS || pos0 < 0 || pos0 + n > HWKV_GEN_MAX_POS)
    return 1;
  for (int32_t h = 0; h < H; ++h) {
    float s = hwkv_gen_head_scale(g, tensor, layer, (uint32_t)h);
    for (int32_t b = 0; b < B; ++b)
      for (int64_t i = 0; i < n; ++i)
        for (int32_t c = 0; c < d; ++c)
          out[(((int64_t)b * n + i) * H + h) * d + c] =
              hwkv_gen_elem(g, tensor, layer, (uint32_t)b, (uint32_t)h, (uint64_t)(pos0 + i),
                            (uint32_t)c, s);
  }
  return 0;
}

/* batch rows b0 .. b0+B-1 and heads head0 .. head0+H-1 only: out is [B][n][H][d] */
int hwkv_gen_fill_host_sub(const hwkv_gen_desc* g, uint32_t tensor, uint32_t layer, int32_t b0,
                           int32_t B, int64_t pos0, int64_t n, int32_t head0, int32_t H, int32_t d,
                           uint16_t* out) {
  if (!g || !out || b0 < 0 || B < 0 || n < 0 || H < 0 || d < 0 || head0 < 0) return 1;
  if (b0 + B > HWKV_GEN_MAX_BATCH || head0 + H > HWKV_GEN_MAX_HEADS || d > HWKV_GEN_MAX_DIM ||
      layer >= HWKV_GEN_MAX_LAYERS || pos0 < 0 || pos0 + n > HWKV_GEN_MAX_POS)
    return 1;
  for (int32_t h = 0; h < H; ++h) {
    float s = hwkv_gen_head_scale(g, tensor, layer, (uint32_t)(head0 + h));
    for (int32_t b = 0; b < B; ++b)
      for (int64_t i = 0; i < n; ++i)
        for (int32_t c = 0; c < d; ++c)
          out[(((int64_t)b * n + i) * H + h) * d + c] =
              hwkv_gen_elem(g, tensor, layer, (uint32_t)(b0 + b), (uint32_t)(head0 + h),
                            (uint64_t)(pos0 + i), (uint32_t)c, s);
  }
  return 0;
}

/* one element, for spot checks */
uint16_t hwkv_gen_one(const hwkv_gen_desc* g, uint32_t tensor, uint32_t layer, uint32_t b,
                      uint32_t head, int64_t pos, uint32_t dim) {
  return hwkv_gen_elem(g, tensor, layer, b, head, (uint64_t)pos, dim,
                       hwkv_gen_head_scale(g, tensor, layer, head));
}

float hwkv_gen_scale(const hwkv_gen_desc* g, uint32_t tensor, uint32_t layer, uint32_t head) {
  return hwkv_gen_head_scale(g, tensor, layer, head);
}

/* j-th output (j >= 1) of splitmix64 seeded with `state`, for checking against published vectors */
uint64_t hwkv_gen_splitmix64_out(uint64_t state, uint32_t j) {
  return hwkv_gen_mix(state + (uint64_t)j * HWKV_GEN_GAMMA);
}
