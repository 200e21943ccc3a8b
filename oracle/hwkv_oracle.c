/*
 * hwkv_oracle.c -- TEST INFRASTRUCTURE. A plain, slow, fp64 CPU statement of
 * what the per-head-window KV path computes, written from the HeadWiseKV
 * paper. Only the test suite, the smoke check and the benchmark's CPU-baseline
 * leg load it; the library never does, and it shares no code with the CUDA
 * path (its only include besides libc is the seeded input generator).
 *
 * Everything here is the definition written out, with no blocking, splitting,
 * fusion or reordering:
 *   - retained window   J_t(w) = {max(1, t-w+1), ..., t}, J_t(full) = {1..t}
 *                       (Sec. 3.2, definition above Eq. conditional-attention-weight),
 *                       used 0-based: s in [max(0, p-W+1), p];
 *   - attention         pi_s = exp(z_s) / sum_{j in J} exp(z_j),  z_s = gamma q.k_s,
 *                       o = sum_{s in J} pi_s v_s
 *                       (Sec. 3.2, Eq. conditional-attention-weight and
 *                       Eq. conditional-attention; exp(z - M) / sum exp(z - M)
 *                       with M = max z is the same quotient);
 *   - retained count    r_C(w) = min(w, C), r_C(full) = C (Sec. 3.1);
 *   - nominal storage   n = r_C(w) (d^K b^K + d^V b^V), N_C = sum over units
 *                       (Sec. 3.1, Eq. nominal-storage);
 *   - normalized rate   R_C = N_C(a) / N_C(all full) (Sec. 3.1, Eq. normalized-rate);
 *   - physical residency: each head keeps only its latest r_t(w) K/V states
 *                       (Sec. 3.3); stored as a ring with slot(p) = p mod cap;
 *   - SeqCalib scoring and selection: stabilized cosine (App. A.2,
 *                       Eq. stabilized-cosine), conditional similarity
 *                       (Eq. conditional-similarity), threshold selection
 *                       (Eq. threshold-selection), budget selector (App. A.2,
 *                       Eq. budget-selector).
 *
 *   - 8-bit cache format (p_KV of Sec. 3.1; the paper names no 8-bit format, so
 *                       this is a reading): E4M3 codes (1 sign bit, 4 exponent bits
 *                       with bias 7, 3 mantissa bits, no infinities, S.1111.111 =
 *                       NaN, largest finite 448) with one fp32 scale per stored row
 *                       (one token of one KV head): s = the smallest power of two
 *                       >= amax / 448 (the shared power-of-two scale of the OCP
 *                       microscaling formats, here per row), code = nearest E4M3
 *                       value of x / s (ties to even, beyond 448 clamped to 448),
 *                       dequantised value decode(code) * s. Attention over such a
 *                       cache reads the dequantised rows (Sec. 3.1: when the format
 *                       changes execution, every compared output uses it).
 *
 *   - sink + recent window (the static sink--recent policy of the StreamingLLM
 *                       control the paper compares against, App. baseline controls:
 *                       S sink tokens and a W-token recent window): a query at p
 *                       reads J = {0..S-1} U [max(0, p-W+1), p], both limited to
 *                       <= p; it retains min(S + W, C) tokens; held in a ring of
 *                       S + W slots: positions < S in slots 0..S-1 for good, later
 *                       ones in slot S + (p - S) mod W.
 *
 * Windows are int64: 0 (HWKV_WINDOW_FULL) means full history; any W >= the
 * context is equivalent to full (Sec. 3.1). bf16 inputs are widened exactly to
 * double. Row loops may run under OpenMP; each row is computed independently.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#include "../hwkv_gen/hwkv_gen.h"

#define ORACLE_FULL 0

int oracle_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

void oracle_set_threads(int n) {
#ifdef _OPENMP
  if (n > 0) omp_set_num_threads(n);
#else
  (void)n;
#endif
}

/* exact bf16 -> double */
static double bf16_to_double(uint16_t h) {
  union { uint32_t u; float f; } c;
  c.u = (uint32_t)h << 16;
  return (double)c.f;
}

/* ---------------------------------------------------------------- windows */

/* lower end of J_p(W), 0-based (Sec. 3.2); the upper end is p itself */
int64_t oracle_window_lo(int64_t p, int64_t W) {
  if (W == ORACLE_FULL) return 0;
  int64_t lo = p - W + 1;
  return lo > 0 ? lo : 0;
}

/* ------------------------------------------------------------- attention */

/*
 * Softmax attention of one query over an explicit key/value set of n rows
 * (Eq. conditional-attention-weight, Eq. conditional-attention).
 * q[d], K[n][d], V[n][d]; writes o[d]; returns sum of pi (1 up to rounding).
 * pi_out, if non-NULL, receives the n weights.
 */
double oracle_attend(const double* q, const double* K, const double* V, int64_t n, int64_t d,
                     double gamma, double* o, double* pi_out) {
  double* z = (double*)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
  double M = -INFINITY;
  for (int64_t s = 0; s < n; ++s) {
    double dot = 0.0;
    for (int64_t i = 0; i < d; ++i) dot += q[i] * K[s * d + i];
    z[s] = gamma * dot;
    if (z[s] > M) M = z[s];
  }
  double Z = 0.0;
  for (int64_t s = 0; s < n; ++s) Z += exp(z[s] - M);
  for (int64_t i = 0; i < d; ++i) o[i] = 0.0;
  double sum_pi = 0.0;
  for (int64_t s = 0; s < n; ++s) {
    double pi = exp(z[s] - M) / Z;
    sum_pi += pi;
    if (pi_out) pi_out[s] = pi;
    for (int64_t i = 0; i < d; ++i) o[i] += pi * V[s * d + i];
  }
  free(z);
  return sum_pi;
}

/*
 * Window-limited attention over bf16 arrays indexed by absolute position.
 * Kp, Vp: history of one (batch row, KV head), row s at Kp + s*ld (positions
 * 0..T-1, T > max pos). Queries: R rows, q row r at Q + r*ldq, position pos[r].
 * Window W (0 = full). Writes O[r][d] and sum_pi[r].
 */
int oracle_window_attention_bf16(const uint16_t* Q, int64_t ldq, const int64_t* pos, int64_t R,
                                 const uint16_t* Kp, const uint16_t* Vp, int64_t ld, int64_t T,
                                 int64_t d, int64_t W, double gamma, double* O, double* sum_pi) {
  if (R < 0 || d <= 0 || W < 0) return 1;
  for (int64_t r = 0; r < R; ++r)
    if (pos[r] < 0 || pos[r] >= T) return 1;
  int bad = 0;
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t r = 0; r < R; ++r) {
    const int64_t p = pos[r];
    const int64_t lo = oracle_window_lo(p, W);
    const int64_t n = p - lo + 1;
    double* q = (double*)malloc(sizeof(double) * (size_t)d);
    double* K = (double*)malloc(sizeof(double) * (size_t)(n * d));
    double* V = (double*)malloc(sizeof(double) * (size_t)(n * d));
    if (!q || !K || !V) {
      bad = 1;
    } else {
      for (int64_t i = 0; i < d; ++i) q[i] = bf16_to_double(Q[r * ldq + i]);
      for (int64_t s = lo; s <= p; ++s)
        for (int64_t i = 0; i < d; ++i) {
          K[(s - lo) * d + i] = bf16_to_double(Kp[s * ld + i]);
          V[(s - lo) * d + i] = bf16_to_double(Vp[s * ld + i]);
        }
      double sp = oracle_attend(q, K, V, n, d, gamma, O + r * d, NULL);
      if (sum_pi) sum_pi[r] = sp;
    }
    free(q);
    free(K);
    free(V);
  }
  return bad ? 2 : 0;
}

/*
 * The same definition, with q, K and V regenerated from the seeded generator
 * instead of read from arrays (for contexts too large to hold on the host).
 * Query rows: (batch row b, query head qh, position pos[r]) for r < R; the
 * query head reads KV head kvh (its GQA group). Writes O[r][d].
 * Two passes over J (logits, then weights and values) so no |J| x d buffer
 * is needed.
 */
int oracle_window_attention_gen(const hwkv_gen_desc* g, int32_t layer, int32_t b, int32_t kvh,
                                const int32_t* qh, const int64_t* pos, int64_t R, int32_t d,
                                int64_t W, double gamma, double* O, double* sum_pi) {
  if (!g || R < 0 || d <= 0 || W < 0) return 1;
  int bad = 0;
  const float sk = hwkv_gen_head_scale(g, HWKV_GEN_K, (uint32_t)layer, (uint32_t)kvh);
  const float sv = hwkv_gen_head_scale(g, HWKV_GEN_V, (uint32_t)layer, (uint32_t)kvh);
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t r = 0; r < R; ++r) {
    const int64_t p = pos[r];
    const int64_t lo = oracle_window_lo(p, W);
    const int64_t n = p - lo + 1;
    double* q = (double*)malloc(sizeof(double) * (size_t)d);
    double* kv = (double*)malloc(sizeof(double) * (size_t)d);
    double* z = (double*)malloc(sizeof(double) * (size_t)n);
    if (!q || !kv || !z || p < 0) {
      bad = 1;
    } else {
      const float sq = hwkv_gen_head_scale(g, HWKV_GEN_Q, (uint32_t)layer, (uint32_t)qh[r]);
      for (int32_t i = 0; i < d; ++i)
        q[i] = bf16_to_double(hwkv_gen_elem(g, HWKV_GEN_Q, (uint32_t)layer, (uint32_t)b,
                                            (uint32_t)qh[r], (uint64_t)p, (uint32_t)i, sq));
      double M = -INFINITY;
      for (int64_t s = lo; s <= p; ++s) {
        for (int32_t i = 0; i < d; ++i)
          kv[i] = bf16_to_double(hwkv_gen_elem(g, HWKV_GEN_K, (uint32_t)layer, (uint32_t)b,
                                               (uint32_t)kvh, (uint64_t)s, (uint32_t)i, sk));
        double dot = 0.0;
        for (int32_t i = 0; i < d; ++i) dot += q[i] * kv[i];
        z[s - lo] = gamma * dot;
        if (z[s - lo] > M) M = z[s - lo];
      }
      double Z = 0.0;
      for (int64_t s = lo; s <= p; ++s) Z += exp(z[s - lo] - M);
      double* o = O + r * d;
      for (int32_t i = 0; i < d; ++i) o[i] = 0.0;
      double sp = 0.0;
      for (int64_t s = lo; s <= p; ++s) {
        const double pi = exp(z[s - lo] - M) / Z;
        sp += pi;
        for (int32_t i = 0; i < d; ++i)
          o[i] += pi * bf16_to_double(hwkv_gen_elem(g, HWKV_GEN_V, (uint32_t)layer, (uint32_t)b,
                                                    (uint32_t)kvh, (uint64_t)s, (uint32_t)i, sv));
      }
      if (sum_pi) sum_pi[r] = sp;
    }
    free(q);
    free(kv);
    free(z);
  }
  return bad ? 2 : 0;
}

/* ------------------------------------------------------------------ rings */

/*
 * Physical residency as a ring of capacity cap: position p lives in slot
 * p mod cap, and after t tokens the ring holds exactly the latest min(t, cap)
 * positions (Sec. 3.3: a head retains only its latest r_t(w) states).
 * pos_of_slot[j] = the position held by slot j, or -1 if never written.
 */
int oracle_ring_positions(int64_t t, int64_t cap, int64_t* pos_of_slot) {
  if (cap <= 0 || t < 0) return 1;
  for (int64_t j = 0; j < cap; ++j) pos_of_slot[j] = -1;
  const int64_t first = t > cap ? t - cap : 0;
  for (int64_t p = first; p < t; ++p) pos_of_slot[p % cap] = p;
  return 0;
}

/*
 * Expected ring bytes for one (layer, batch row, KV head) after positions
 * 0..t-1 have been fed in order: ring[j][:] = the generated K (or V) row of
 * the position slot j holds, zero where no position is held.
 */
int oracle_ring_expected_gen(const hwkv_gen_desc* g, uint32_t tensor, int32_t layer, int32_t b,
                             int32_t kvh, int32_t d, int64_t t, int64_t cap, uint16_t* ring) {
  if (!g || cap <= 0 || t < 0 || d <= 0) return 1;
  int64_t* pos = (int64_t*)malloc(sizeof(int64_t) * (size_t)cap);
  if (!pos) return 2;
  oracle_ring_positions(t, cap, pos);
  const float s = hwkv_gen_head_scale(g, tensor, (uint32_t)layer, (uint32_t)kvh);
  for (int64_t j = 0; j < cap; ++j)
    for (int32_t i = 0; i < d; ++i)
      ring[j * d + i] = pos[j] < 0 ? (uint16_t)0
                                   : hwkv_gen_elem(g, tensor, (uint32_t)layer, (uint32_t)b,
                                                   (uint32_t)kvh, (uint64_t)pos[j], (uint32_t)i, s);
  free(pos);
  return 0;
}

/* ------------------------------------------------------ sink + recent window */

/* 1 if a query at position p reads key position k under window W (0 = full) with
 * S sink tokens: k <= p and (k < S or k >= p - W + 1) */
int oracle_sink_visible(int64_t k, int64_t p, int64_t W, int64_t S) {
  if (k < 0 || k > p) return 0;
  if (W == ORACLE_FULL) return 1;
  return k < S || k >= p - W + 1;
}

/* the positions of J in increasing order: [0, min(S, p+1)) then [max(S, lo), p];
 * returns their count (out may be NULL) */
int64_t oracle_sink_positions(int64_t p, int64_t W, int64_t S, int64_t* out) {
  if (p < 0) return 0;
  const int64_t lo = oracle_window_lo(p, W);
  const int64_t s_end = S < p + 1 ? S : p + 1;
  int64_t n = 0;
  for (int64_t k = 0; k < s_end; ++k) {
    if (out) out[n] = k;
    ++n;
  }
  for (int64_t k = (lo > s_end ? lo : s_end); k <= p; ++k) {
    if (out) out[n] = k;
    ++n;
  }
  return n;
}

/*
 * Attention (Eq. conditional-attention-weight, Eq. conditional-attention) over J
 * of the sink + recent policy, with q, K, V regenerated from the seeded generator:
 * query rows (batch row b, query head qh[r], position pos[r]) reading KV head kvh.
 */
int oracle_sink_attention_gen(const hwkv_gen_desc* g, int32_t layer, int32_t b, int32_t kvh,
                              const int32_t* qh, const int64_t* pos, int64_t R, int32_t d,
                              int64_t W, int64_t S, double gamma, double* O, double* sum_pi) {
  if (!g || R < 0 || d <= 0 || W < 0 || S < 0) return 1;
  int bad = 0;
  const float sk = hwkv_gen_head_scale(g, HWKV_GEN_K, (uint32_t)layer, (uint32_t)kvh);
  const float sv = hwkv_gen_head_scale(g, HWKV_GEN_V, (uint32_t)layer, (uint32_t)kvh);
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t r = 0; r < R; ++r) {
    const int64_t p = pos[r];
    const int64_t n = oracle_sink_positions(p, W, S, NULL);
    int64_t* J = (int64_t*)malloc(sizeof(int64_t) * (size_t)(n > 0 ? n : 1));
    double* q = (double*)malloc(sizeof(double) * (size_t)d);
    double* K = (double*)malloc(sizeof(double) * (size_t)(n * d + 1));
    double* V = (double*)malloc(sizeof(double) * (size_t)(n * d + 1));
    if (!J || !q || !K || !V || p < 0) {
      bad = 1;
    } else {
      oracle_sink_positions(p, W, S, J);
      const float sq = hwkv_gen_head_scale(g, HWKV_GEN_Q, (uint32_t)layer, (uint32_t)qh[r]);
      for (int32_t i = 0; i < d; ++i)
        q[i] = bf16_to_double(hwkv_gen_elem(g, HWKV_GEN_Q, (uint32_t)layer, (uint32_t)b,
                                            (uint32_t)qh[r], (uint64_t)p, (uint32_t)i, sq));
      for (int64_t j = 0; j < n; ++j)
        for (int32_t i = 0; i < d; ++i) {
          K[j * d + i] = bf16_to_double(hwkv_gen_elem(g, HWKV_GEN_K, (uint32_t)layer, (uint32_t)b,
                                                      (uint32_t)kvh, (uint64_t)J[j], (uint32_t)i, sk));
          V[j * d + i] = bf16_to_double(hwkv_gen_elem(g, HWKV_GEN_V, (uint32_t)layer, (uint32_t)b,
                                                      (uint32_t)kvh, (uint64_t)J[j], (uint32_t)i, sv));
        }
      const double sp = oracle_attend(q, K, V, n, d, gamma, O + r * d, NULL);
      if (sum_pi) sum_pi[r] = sp;
    }
    free(J);
    free(q);
    free(K);
    free(V);
  }
  return bad ? 2 : 0;
}

/* The same over bf16 arrays indexed by absolute position (as
 * oracle_window_attention_bf16). */
int oracle_sink_attention_bf16(const uint16_t* Q, int64_t ldq, const int64_t* pos, int64_t R,
                               const uint16_t* Kp, const uint16_t* Vp, int64_t ld, int64_t T,
                               int64_t d, int64_t W, int64_t S, double gamma, double* O,
                               double* sum_pi) {
  if (R < 0 || d <= 0 || W < 0 || S < 0) return 1;
  for (int64_t r = 0; r < R; ++r)
    if (pos[r] < 0 || pos[r] >= T) return 1;
  int bad = 0;
  for (int64_t r = 0; r < R; ++r) {
    const int64_t p = pos[r];
    const int64_t n = oracle_sink_positions(p, W, S, NULL);
    int64_t* J = (int64_t*)malloc(sizeof(int64_t) * (size_t)n);
    double* q = (double*)malloc(sizeof(double) * (size_t)d);
    double* K = (double*)malloc(sizeof(double) * (size_t)(n * d));
    double* V = (double*)malloc(sizeof(double) * (size_t)(n * d));
    if (!J || !q || !K || !V) {
      bad = 1;
    } else {
      oracle_sink_positions(p, W, S, J);
      for (int64_t i = 0; i < d; ++i) q[i] = bf16_to_double(Q[r * ldq + i]);
      for (int64_t j = 0; j < n; ++j)
        for (int64_t i = 0; i < d; ++i) {
          K[j * d + i] = bf16_to_double(Kp[J[j] * ld + i]);
          V[j * d + i] = bf16_to_double(Vp[J[j] * ld + i]);
        }
      const double sp = oracle_attend(q, K, V, n, d, gamma, O + r * d, NULL);
      if (sum_pi) sum_pi[r] = sp;
    }
    free(J);
    free(q);
    free(K);
    free(V);
  }
  return bad ? 2 : 0;
}

/*
 * The ring of the sink + recent policy after positions 0..t-1 (cap = S + W
 * slots, W > 0, S > 0): slot j < S holds position j once written; the window
 * slots hold the latest W positions >= S, position p in slot S + (p - S) mod W.
 * pos_of_slot[j] = the position held, or -1.
 */
int oracle_sink_ring_positions(int64_t t, int64_t W, int64_t S, int64_t* pos_of_slot) {
  if (W <= 0 || S < 0 || t < 0) return 1;
  for (int64_t j = 0; j < S + W; ++j) pos_of_slot[j] = -1;
  for (int64_t p = 0; p < t && p < S; ++p) pos_of_slot[p] = p;
  const int64_t first = t - W > S ? t - W : S;
  for (int64_t p = first; p < t; ++p) pos_of_slot[S + (p - S) % W] = p;
  return 0;
}

int oracle_sink_ring_expected_gen(const hwkv_gen_desc* g, uint32_t tensor, int32_t layer,
                                  int32_t b, int32_t kvh, int32_t d, int64_t t, int64_t W,
                                  int64_t S, uint16_t* ring) {
  if (!g || W <= 0 || S < 0 || t < 0 || d <= 0) return 1;
  const int64_t cap = S + W;
  int64_t* pos = (int64_t*)malloc(sizeof(int64_t) * (size_t)cap);
  if (!pos) return 2;
  oracle_sink_ring_positions(t, W, S, pos);
  const float s = hwkv_gen_head_scale(g, tensor, (uint32_t)layer, (uint32_t)kvh);
  for (int64_t j = 0; j < cap; ++j)
    for (int32_t i = 0; i < d; ++i)
      ring[j * d + i] = pos[j] < 0 ? (uint16_t)0
                                   : hwkv_gen_elem(g, tensor, (uint32_t)layer, (uint32_t)b,
                                                   (uint32_t)kvh, (uint64_t)pos[j], (uint32_t)i, s);
  free(pos);
  return 0;
}

/* retained tokens of the sink + recent policy at context C: min(S + W, C); full: C */
int64_t oracle_sink_retained_tokens(int64_t W, int64_t S, int64_t C) {
  if (W == ORACLE_FULL) return C;
  return S + W < C ? S + W : C;
}

/* ------------------------------------------------------- 8-bit KV format */

/* value of an E4M3 code, from its bit fields (exact; NaN for S.1111.111) */
double oracle_e4m3_decode(uint8_t c) {
  const int sign = c >> 7, e = (c >> 3) & 15, m = c & 7;
  if (e == 15 && m == 7) return NAN;
  const double mag = e == 0 ? ldexp((double)m / 8.0, -6)               /* subnormal */
                            : ldexp(1.0 + (double)m / 8.0, e - 7);     /* normal */
  return sign ? -mag : mag;
}

/*
 * Nearest E4M3 code of x: the finite magnitudes (codes 0x00 .. 0x7E, increasing
 * with the code) are searched for the two that bracket |x|; the nearer one wins,
 * a tie goes to the even code (mantissa lsb 0); |x| above 448, including
 * infinity, clamps to 448; NaN gives 0x7F. The sign bit is x's sign bit.
 */
uint8_t oracle_e4m3_encode(float x) {
  if (isnan(x)) return 0x7F;
  const uint8_t sign = signbit(x) ? 0x80 : 0x00;
  const double a = fabs((double)x);
  if (a >= 448.0) return (uint8_t)(sign | 0x7E);
  uint8_t lo = 0;
  for (uint8_t c = 1; c <= 0x7E; ++c)
    if (oracle_e4m3_decode(c) <= a) lo = c;
  /* a < 448 here, so lo < 0x7E and lo + 1 is the next larger magnitude */
  const uint8_t hi = (uint8_t)(lo + 1);
  const double dlo = a - oracle_e4m3_decode(lo), dhi = oracle_e4m3_decode(hi) - a;
  uint8_t c;
  if (dlo < dhi) c = lo;
  else if (dhi < dlo) c = hi;
  else c = (lo & 1) ? hi : lo;
  return (uint8_t)(sign | c);
}

/*
 * One stored row in the 8-bit format: x[d] (bf16 bits) -> codes[d], *scale.
 * amax = max |x_i|; r = amax / 448 in float arithmetic; s = the smallest power
 * of two >= r (frexp: r = m 2^e with 1/2 <= m < 1, so s = r when m = 1/2, else
 * 2^e); code_i = encode(x_i / s) with x_i / s a float division (exact, s being a
 * power of two, up to the one rounding of a subnormal quotient); amax = 0 gives
 * s = 0 and all-zero codes.
 */
int oracle_quantize_row_e4m3(const uint16_t* x, int64_t d, uint8_t* codes, float* scale) {
  if (d <= 0) return 1;
  float amax = 0.0f;
  for (int64_t i = 0; i < d; ++i) {
    const float v = (float)fabs(bf16_to_double(x[i]));
    if (v > amax) amax = v;
  }
  if (amax == 0.0f) {
    for (int64_t i = 0; i < d; ++i) codes[i] = 0;
    *scale = 0.0f;
    return 0;
  }
  const volatile float r = amax / 448.0f;
  int e = 0;
  const float m = frexpf(r, &e);
  const volatile float s = m == 0.5f ? r : ldexpf(1.0f, e);
  for (int64_t i = 0; i < d; ++i) {
    const volatile float y = (float)bf16_to_double(x[i]) / s;
    codes[i] = oracle_e4m3_encode(y);
  }
  *scale = s;
  return 0;
}

static double dequant(uint8_t c, float s) { return oracle_e4m3_decode(c) * (double)s; }

/*
 * oracle_window_attention_bf16 over a cache in the 8-bit format: key/value row
 * s of the history is decode(codes[s][i]) * scale[s]. Kc/Vc [T][d] codes,
 * Ks/Vs [T] scales, indexed by absolute position.
 */
int oracle_window_attention_fp8(const uint16_t* Q, int64_t ldq, const int64_t* pos, int64_t R,
                                const uint8_t* Kc, const float* Ks, const uint8_t* Vc,
                                const float* Vs, int64_t T, int64_t d, int64_t W, double gamma,
                                double* O, double* sum_pi) {
  if (R < 0 || d <= 0 || W < 0) return 1;
  for (int64_t r = 0; r < R; ++r)
    if (pos[r] < 0 || pos[r] >= T) return 1;
  int bad = 0;
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t r = 0; r < R; ++r) {
    const int64_t p = pos[r];
    const int64_t lo = oracle_window_lo(p, W);
    const int64_t n = p - lo + 1;
    double* q = (double*)malloc(sizeof(double) * (size_t)d);
    double* K = (double*)malloc(sizeof(double) * (size_t)(n * d));
    double* V = (double*)malloc(sizeof(double) * (size_t)(n * d));
    if (!q || !K || !V) {
      bad = 1;
    } else {
      for (int64_t i = 0; i < d; ++i) q[i] = bf16_to_double(Q[r * ldq + i]);
      for (int64_t s = lo; s <= p; ++s)
        for (int64_t i = 0; i < d; ++i) {
          K[(s - lo) * d + i] = dequant(Kc[s * d + i], Ks[s]);
          V[(s - lo) * d + i] = dequant(Vc[s * d + i], Vs[s]);
        }
      double sp = oracle_attend(q, K, V, n, d, gamma, O + r * d, NULL);
      if (sum_pi) sum_pi[r] = sp;
    }
    free(q);
    free(K);
    free(V);
  }
  return bad ? 2 : 0;
}

/*
 * Expected ring in the 8-bit format for one (layer, batch row, KV head) after
 * positions 0..t-1: slot j holds the quantised generated row of the position
 * it holds (codes[j][d], scale[j]); zeros where no position is held.
 */
int oracle_ring_expected_fp8_gen(const hwkv_gen_desc* g, uint32_t tensor, int32_t layer,
                                 int32_t b, int32_t kvh, int32_t d, int64_t t, int64_t cap,
                                 uint8_t* codes, float* scales) {
  if (!g || cap <= 0 || t < 0 || d <= 0) return 1;
  int64_t* pos = (int64_t*)malloc(sizeof(int64_t) * (size_t)cap);
  uint16_t* row = (uint16_t*)malloc(sizeof(uint16_t) * (size_t)d);
  if (!pos || !row) {
    free(pos);
    free(row);
    return 2;
  }
  oracle_ring_positions(t, cap, pos);
  const float hs = hwkv_gen_head_scale(g, tensor, (uint32_t)layer, (uint32_t)kvh);
  for (int64_t j = 0; j < cap; ++j) {
    if (pos[j] < 0) {
      memset(codes + j * d, 0, (size_t)d);
      scales[j] = 0.0f;
      continue;
    }
    for (int32_t i = 0; i < d; ++i)
      row[i] = hwkv_gen_elem(g, tensor, (uint32_t)layer, (uint32_t)b, (uint32_t)kvh,
                             (uint64_t)pos[j], (uint32_t)i, hs);
    oracle_quantize_row_e4m3(row, d, codes + j * d, scales + j);
  }
  free(pos);
  free(row);
  return 0;
}

/* ------------------------------------------------------------- accounting */

/* r_C(w) = min(w, C); r_C(full) = C  (Sec. 3.1) */
int64_t oracle_retained_tokens(int64_t W, int64_t C) {
  if (W == ORACLE_FULL) return C;
  return W < C ? W : C;
}

/*
 * N_C(a) of Eq. nominal-storage: sum over decision units of
 * r_C(w_u) (d^K b^K + d^V b^V), in bytes, times `batch` independent sequences.
 */
uint64_t oracle_nominal_storage(const int64_t* W, int64_t n_units, int64_t C, int64_t dK,
                                int64_t dV, int64_t bK, int64_t bV, int64_t batch) {
  uint64_t total = 0;
  for (int64_t u = 0; u < n_units; ++u)
    total += (uint64_t)oracle_retained_tokens(W[u], C) * (uint64_t)(dK * bK + dV * bV);
  return total * (uint64_t)batch;
}

/* R_C(a) of Eq. normalized-rate */
double oracle_normalized_rate(const int64_t* W, int64_t n_units, int64_t C, int64_t dK,
                              int64_t dV, int64_t bK, int64_t bV) {
  uint64_t num = oracle_nominal_storage(W, n_units, C, dK, dV, bK, bV, 1);
  uint64_t den = 0;
  for (int64_t u = 0; u < n_units; ++u) den += (uint64_t)C * (uint64_t)(dK * bK + dV * bV);
  return den ? (double)num / (double)den : 0.0;
}

/* ------------------------------------------------------ SeqCalib (App. A.2) */

/*
 * Stabilized cosine, App. "Calibration Score and Fixed-Prefix Selection",
 * Eq. stabilized-cosine: a vector of norm <= eps counts as zero; both zero
 * gives 1, exactly one zero gives 0, otherwise the plain cosine.
 */
double oracle_cos_eval(const double* u, const double* v, int64_t d, double eps) {
  double uu = 0.0, vv = 0.0, uv = 0.0;
  for (int64_t i = 0; i < d; ++i) {
    uu += u[i] * u[i];
    vv += v[i] * v[i];
    uv += u[i] * v[i];
  }
  const double nu = sqrt(uu), nv = sqrt(vv);
  const int zu = nu <= eps, zv = nv <= eps;
  if (zu && zv) return 1.0;
  if (zu || zv) return 0.0;
  return uv / (nu * nv);
}

/*
 * Conditional similarity of one KV head (Sec. 3.2, Eq. conditional-similarity):
 * for every candidate window W[k] (k < n_w, finite), the mean over the rows
 * (sampled position, query head) of cos_eval(o^(W[k]), o^(full)), where o^(w)
 * is Eq. conditional-attention over J_p(w). Rows: q row r at Q + r*d with
 * position pos[r]; K, V [T][d] hold positions 0..T-1 of this head.
 * scores[k] receives the means; cos_out (optional) [R][n_w] the individual scores.
 */
int oracle_conditional_similarity_bf16(const uint16_t* Q, const int64_t* pos, int64_t R,
                                       const uint16_t* Kp, const uint16_t* Vp, int64_t T,
                                       int64_t d, const int64_t* W, int64_t n_w, double gamma,
                                       double eps, double* scores, double* cos_out) {
  if (R <= 0 || d <= 0 || n_w < 0) return 1;
  double* of = (double*)malloc(sizeof(double) * (size_t)(R * d));
  double* ow = (double*)malloc(sizeof(double) * (size_t)(R * d));
  double* c = (double*)malloc(sizeof(double) * (size_t)(R * (n_w > 0 ? n_w : 1)));
  if (!of || !ow || !c) {
    free(of);
    free(ow);
    free(c);
    return 2;
  }
  int rc = oracle_window_attention_bf16(Q, d, pos, R, Kp, Vp, d, T, d, ORACLE_FULL, gamma, of, NULL);
  for (int64_t k = 0; rc == 0 && k < n_w; ++k) {
    rc = oracle_window_attention_bf16(Q, d, pos, R, Kp, Vp, d, T, d, W[k], gamma, ow, NULL);
    double sum = 0.0;
    for (int64_t r = 0; rc == 0 && r < R; ++r) {
      c[r * n_w + k] = oracle_cos_eval(ow + r * d, of + r * d, d, eps);
      sum += c[r * n_w + k];
    }
    scores[k] = sum / (double)R;
  }
  if (rc == 0 && cos_out) memcpy(cos_out, c, sizeof(double) * (size_t)(R * n_w));
  free(of);
  free(ow);
  free(c);
  return rc;
}

/*
 * Threshold selection of one head (Sec. 3.2, Eq. threshold-selection): among
 * the candidates {W[0..n_w-1] finite, full} whose score is >= tau (full always
 * scores 1), the lowest nominal cost r_C(w) = min(w, C); equal costs go to the
 * earlier candidate in the order <_W (finite windows increasing, then full).
 * Returns the chosen window, 0 for full.
 */
int64_t oracle_select_window(const double* scores, const int64_t* W, int64_t n_w, int64_t C,
                             double tau) {
  int64_t best = ORACLE_FULL;
  int64_t best_cost = C;
  int64_t best_rank = n_w;  /* full is last in <_W */
  for (int64_t k = 0; k < n_w; ++k) {
    if (!(scores[k] >= tau)) continue;
    const int64_t cost = oracle_retained_tokens(W[k], C);
    /* rank in <_W: finite windows by value */
    int64_t rank = 0;
    for (int64_t j = 0; j < n_w; ++j)
      if (W[j] < W[k]) ++rank;
    if (cost < best_cost || (cost == best_cost && rank < best_rank)) {
      best = W[k];
      best_cost = cost;
      best_rank = rank;
    }
  }
  return best;
}

/*
 * Finite-grid budget selection (App. "Finite-grid budget selection",
 * Eq. budget-selector): among records g with beta[g] <= budget, maximise
 * phi[g], then minimise beta[g], then take the smallest g. Returns g (0-based)
 * or -1 when no record meets the budget.
 */
int64_t oracle_budget_select(const double* beta, const double* phi, int64_t G, double budget) {
  int64_t best = -1;
  for (int64_t g = 0; g < G; ++g) {
    if (!(beta[g] <= budget)) continue;
    if (best < 0 || phi[g] > phi[best] || (phi[g] == phi[best] && beta[g] < beta[best])) best = g;
  }
  return best;
}
