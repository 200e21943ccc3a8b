/*
 * hwkv_gen.h -- seeded, counter-based synthetic input generator.
 *
 * This module only maps the coordinates of one input element (which tensor,
 * layer, batch row, head, token position, channel) to a bf16 value. It holds
 * none of the attention arithmetic. It is the one piece of code that both the
 * CUDA path's tests/bench (device fill kernels) and the CPU oracle (host
 * regeneration of any element on demand) use, so that both sides see the same
 * inputs without storing tens of GB of K/V on the host.
 *
 * Definition (host and device give bit-identical results):
 *   c   = element counter, the coordinates packed with fixed radices
 *         (tensor:4 | layer:8 | b:8 | head:8 | pos:26 | dim:10 bits, high->low)
 *   r_j = j-th output (j = 1, 2, 3) of the splitmix64 generator
 *         (Steele, Lea & Flood, OOPSLA 2014) seeded with (seed XOR c)
 *   S   = sum of the twelve 16-bit words of r_1, r_2, r_3     (integer)
 *   z   = (S - 393210) * 2^-16   -- Irwin-Hall(12) of discrete uniforms:
 *         mean 0, variance (2^32 - 1) / 2^32, exact in fp32
 *   x   = bf16_rne(s * z) with s = 1, or, with per-head scaling, the
 *         per-(tensor, layer, head) factor s = (2^21 + 3 u) * 2^-22 in
 *         [0.5, 2), u = top 21 bits of the first splitmix64 output seeded with
 *         (seed XOR c(scale tensor, layer, 0, head, 0, 0)); s is exact in fp32,
 *         s * z is one IEEE fp32 multiply (round to nearest even).
 *
 * Plain C99 for gcc; `__host__ __device__` under nvcc.
 */
#ifndef HWKV_GEN_H
#define HWKV_GEN_H

#include <stdint.h>

#if defined(__CUDACC__)
#define HWKV_GEN_FN __host__ __device__ __forceinline__
#else
#define HWKV_GEN_FN static inline
#endif

/* tensor ids (4 bits) */
#define HWKV_GEN_Q 1u
#define HWKV_GEN_K 2u
#define HWKV_GEN_V 3u
#define HWKV_GEN_SCALE_OF(tensor) ((tensor) + 8u)

/* radix limits of the counter packing */
#define HWKV_GEN_MAX_LAYERS 256
#define HWKV_GEN_MAX_BATCH 256
#define HWKV_GEN_MAX_HEADS 256
#define HWKV_GEN_MAX_POS (1ll << 26)
#define HWKV_GEN_MAX_DIM 1024

typedef struct {
  uint64_t seed;
  int32_t per_head_scale; /* 0: s = 1;  1: K and V of each (layer, kv head) get s ~ U[0.5, 2) */
  int32_t reserved;
} hwkv_gen_desc;

HWKV_GEN_FN uint64_t hwkv_gen_counter(uint32_t tensor, uint32_t layer, uint32_t b,
                                      uint32_t head, uint64_t pos, uint32_t dim) {
  return ((uint64_t)(tensor & 0xFu) << 60) | ((uint64_t)(layer & 0xFFu) << 52) |
         ((uint64_t)(b & 0xFFu) << 44) | ((uint64_t)(head & 0xFFu) << 36) |
         ((pos & 0x3FFFFFFull) << 10) | (uint64_t)(dim & 0x3FFu);
}

/* splitmix64 output function applied to a state that has already been advanced */
HWKV_GEN_FN uint64_t hwkv_gen_mix(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

#define HWKV_GEN_GAMMA 0x9E3779B97F4A7C15ull

/* sum of the twelve 16-bit words of the first three splitmix64 outputs from state x */
HWKV_GEN_FN uint32_t hwkv_gen_irwin_hall_sum(uint64_t x) {
  uint32_t s = 0;
  for (int j = 1; j <= 3; ++j) {
    uint64_t r = hwkv_gen_mix(x + (uint64_t)j * HWKV_GEN_GAMMA);
    s += (uint32_t)(r & 0xFFFFu) + (uint32_t)((r >> 16) & 0xFFFFu) +
         (uint32_t)((r >> 32) & 0xFFFFu) + (uint32_t)(r >> 48);
  }
  return s;
}

/* float -> bf16 bits, round to nearest even (finite inputs) */
HWKV_GEN_FN uint16_t hwkv_gen_bf16_rne(float f) {
  union { float f; uint32_t u; } cvt;
  cvt.f = f;
  uint32_t u = cvt.u;
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

HWKV_GEN_FN float hwkv_gen_mul_rn(float a, float b) {
#if defined(__CUDA_ARCH__)
  return __fmul_rn(a, b);
#else
  volatile float p = a * b; /* one IEEE binary32 multiply, never contracted */
  return p;
#endif
}

/* per-(tensor, layer, head) scale in [0.5, 2), exact in fp32 */
HWKV_GEN_FN float hwkv_gen_head_scale(const hwkv_gen_desc* g, uint32_t tensor, uint32_t layer,
                                      uint32_t head) {
  if (!g->per_head_scale || tensor == HWKV_GEN_Q) return 1.0f;
  uint64_t c = hwkv_gen_counter(HWKV_GEN_SCALE_OF(tensor), layer, 0u, head, 0ull, 0u);
  uint64_t r = hwkv_gen_mix((g->seed ^ c) + HWKV_GEN_GAMMA);
  uint32_t u = (uint32_t)(r >> 43); /* 21 bits */
  return (float)((1u << 21) + 3u * u) * (1.0f / 4194304.0f);
}

/* standard-normal-like value before scaling, exact in fp32 */
HWKV_GEN_FN float hwkv_gen_z(uint64_t seed, uint64_t counter) {
  uint32_t s = hwkv_gen_irwin_hall_sum(seed ^ counter);
  return (float)((int32_t)s - 393210) * (1.0f / 65536.0f);
}

/* the bf16 bits of one element; `scale` is hwkv_gen_head_scale(...) for its (tensor, layer, head) */
HWKV_GEN_FN uint16_t hwkv_gen_elem(const hwkv_gen_desc* g, uint32_t tensor, uint32_t layer,
                                   uint32_t b, uint32_t head, uint64_t pos, uint32_t dim,
                                   float scale) {
  float z = hwkv_gen_z(g->seed, hwkv_gen_counter(tensor, layer, b, head, pos, dim));
  return hwkv_gen_bf16_rne(hwkv_gen_mul_rn(scale, z));
}

#endif /* HWKV_GEN_H */
