/*
 * Plain fp64 CPU oracle for Dynamic Memory Sparsification (DMS) decode.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may include, link or
 * call this file: only the test suite, the smoke check and the CPU-baseline /
 * reference leg of the benchmark use it.  It shares no code, header, table or
 * helper with the CUDA library; the only thing both sides share is the seeded
 * input generator (which holds none of the method's arithmetic).
 *
 * What it computes (arXiv 2506.05345):
 *   - Sec. 3.2 (Inference): the binary decision alpha_t = round(sigmoid(logit_t)).
 *     sigmoid is strictly increasing with sigmoid(0) = 1/2, so alpha_t = 1 exactly
 *     when logit_t > 0.  The tie logit = 0 (sigmoid = 1/2) is read as "keep";
 *     NaN compares false and therefore keeps.
 *   - Sec. 3.1 "Delayed Eviction via Sliding Window" and Fig. 1b: a token flagged
 *     at step i stays visible while it is inside the window and disappears once it
 *     leaves it.  Reading used here: key i is visible to the query at step j iff
 *     i <= j and (alpha_i == 0 or j - i <= w).  With w = 3 this reproduces the
 *     pattern printed in Fig. 1b (q_4 loses k_0, q_5 loses k_0 and k_1 but still
 *     sees k_2).
 *   - Sec. 3.2 / Sec. 4 (GQA): plain softmax attention of each query head over
 *     the retained set of its KV head, scale 1/sqrt(D) unless given.
 *
 *   - Sec. 5 (Ablations), immediate eviction: the eviction of past token t at time
 *     t + w is decided by alpha_{t+w} instead of alpha_t.  Reading used here (the
 *     timing kept, only the deciding variable changed): key i is visible to the
 *     query at step j iff i <= j and (j - i <= w or alpha_{i+w} == 0).  With
 *     w = 0 the two policies coincide.
 *
 * The retained set R_j is built by scanning the decisions directly from the
 * definition above; there is no ring, slot or page logic here.  All arithmetic
 * is fp64 with plain sequential sums in index order.  bf16 inputs are widened
 * exactly (a bf16 value is the upper half of an IEEE binary32).
 *
 *   - Related work (KV cache reduction): quantisation of the cache is orthogonal to
 *     DMS and can be combined with it.  The quantised page format checked here is
 *     fp8 E4M3 (the OCP "E4M3FN" encoding: 1 sign, 4 exponent bits with bias 7,
 *     3 mantissa bits, no infinities, S.1111.111 = NaN, largest finite 448, smallest
 *     normal 2^-6, subnormals m * 2^-9) with one fp32 scale per row: scale =
 *     fl32(amax / 448), code = e4m3(fl32(x / scale)) rounded to nearest even and
 *     saturated to +-448; a row of zeros has scale 0 and zero codes.  These roundings
 *     decide integer codes, so both sides take them in fp32.  The attention then runs
 *     in fp64 over the dequantised rows code * scale.
 *
 * Parity pins (tests, no GPU): Fig. 1b pattern, brute-force dense masked
 * softmax with the training mask M_alpha of Sec. 3.1, dense causal attention
 * when nothing is evicted, w = 0 with all-evict, the closed-form retained count;
 * for fp8: every code against PyTorch's float8_e4m3fn, round-to-nearest-even at
 * midpoints, exact rows (values already on the e4m3 grid times a power of two).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* Exact widening of a bf16 bit pattern to double. */
double dms_oracle_bf16_to_double(uint16_t bits) {
  uint32_t u = ((uint32_t)bits) << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

/* Sec. 3.2: alpha_bin = round(sigmoid(logit)) == [logit > 0] (tie keeps). */
int dms_oracle_alpha(uint16_t logit_bits) {
  double x = dms_oracle_bf16_to_double(logit_bits);
  return x > 0.0 ? 1 : 0;
}

/* Sec. 3.1 delayed eviction: is key i visible to the query at step j? */
static int visible(const uint16_t* logits, int64_t logit_stride, int64_t i,
                   int64_t j, int64_t w) {
  if (i > j) return 0;                 /* causal */
  if (j - i <= w) return 1;            /* still inside the sliding window */
  return dms_oracle_alpha(logits[i * logit_stride]) ? 0 : 1;
}

/* Sec. 5 immediate eviction: key i is decided by the token at position i + w. */
static int visible_immediate(const uint16_t* logits, int64_t logit_stride, int64_t i,
                             int64_t j, int64_t w) {
  if (i > j) return 0;                 /* causal */
  if (j - i <= w) return 1;            /* still inside the sliding window */
  /* j - i > w, so the deciding token i + w < j has already been seen */
  return dms_oracle_alpha(logits[(i + w) * logit_stride]) ? 0 : 1;
}

/*
 * Retained set R_j of one (layer, sequence, KV head) after the token at
 * position j has been appended.  logits[i * logit_stride] is the bf16 decision
 * logit of position i.  Writes the sorted positions to pos_out (may be NULL)
 * and returns |R_j|.  Returns 0 for j < 0.
 */
int64_t dms_oracle_retained_policy(const uint16_t* logits, int64_t logit_stride,
                                   int64_t j, int64_t w, int immediate, int32_t* pos_out) {
  int64_t n = 0;
  for (int64_t i = 0; i <= j; ++i) {
    if (immediate ? visible_immediate(logits, logit_stride, i, j, w)
                  : visible(logits, logit_stride, i, j, w)) {
      if (pos_out) pos_out[n] = (int32_t)i;
      ++n;
    }
  }
  return n;
}

/*
 * Decode attention for the G query heads sharing one KV head, at step j.
 *   q:      [G][D] bf16 bits, row stride D
 *   k, v:   row i at k + i * kv_stride (bf16 bits, D contiguous), i = 0..j
 *   logits: logits[i * logit_stride], i = 0..j
 *   scale:  softmax scale (<= 0 means 1/sqrt(D))
 *   out:    [G][D] fp64
 * Softmax over R_j of s_i = scale * <q, k_i>; out = sum_i p_i v_i.
 * An empty retained set (j < 0) yields zeros.
 */
/* Delayed eviction (Sec. 3.1), the method's policy. */
int64_t dms_oracle_retained(const uint16_t* logits, int64_t logit_stride,
                            int64_t j, int64_t w, int32_t* pos_out) {
  return dms_oracle_retained_policy(logits, logit_stride, j, w, 0, pos_out);
}

/*
 * Softmax attention at step j of the G query heads q[G][D] of one group over
 * the retained set of their KV head (k, v rows at k + i * kv_stride), under the
 * delayed (immediate = 0) or immediate (1) eviction policy; out[G][D].
 */
void dms_oracle_decode_policy(const uint16_t* q, int32_t G, int32_t D,
                              const uint16_t* k, const uint16_t* v, int64_t kv_stride,
                              const uint16_t* logits, int64_t logit_stride, int64_t j,
                              int64_t w, int immediate, double scale, double* out) {
  if (scale <= 0.0) scale = 1.0 / sqrt((double)D);
  int64_t cap = j + 1 > 0 ? j + 1 : 0;
  int32_t* pos = (int32_t*)malloc(sizeof(int32_t) * (size_t)(cap > 0 ? cap : 1));
  double* s = (double*)malloc(sizeof(double) * (size_t)(cap > 0 ? cap : 1));
  int64_t n = dms_oracle_retained_policy(logits, logit_stride, j, w, immediate, pos);
  for (int32_t g = 0; g < G; ++g) {
    double* o = out + (int64_t)g * D;
    for (int32_t d = 0; d < D; ++d) o[d] = 0.0;
    if (n == 0) continue;
    const uint16_t* qg = q + (int64_t)g * D;
    double m = -INFINITY;
    for (int64_t r = 0; r < n; ++r) {
      const uint16_t* kr = k + (int64_t)pos[r] * kv_stride;
      double dot = 0.0;
      for (int32_t d = 0; d < D; ++d)
        dot += dms_oracle_bf16_to_double(qg[d]) * dms_oracle_bf16_to_double(kr[d]);
      s[r] = scale * dot;
      if (s[r] > m) m = s[r];
    }
    double den = 0.0;
    for (int64_t r = 0; r < n; ++r) {
      s[r] = exp(s[r] - m);
      den += s[r];
    }
    for (int64_t r = 0; r < n; ++r) {
      const uint16_t* vr = v + (int64_t)pos[r] * kv_stride;
      double p = s[r] / den;
      for (int32_t d = 0; d < D; ++d) o[d] += p * dms_oracle_bf16_to_double(vr[d]);
    }
  }
  free(pos);
  free(s);
}

void dms_oracle_decode(const uint16_t* q, int32_t G, int32_t D,
                       const uint16_t* k, const uint16_t* v, int64_t kv_stride,
                       const uint16_t* logits, int64_t logit_stride, int64_t j,
                       int64_t w, double scale, double* out) {
  dms_oracle_decode_policy(q, G, D, k, v, kv_stride, logits, logit_stride, j, w, 0, scale, out);
}

/* ------------------------------------------------------------------ fp8 E4M3 page format */

/* Value of an E4M3FN code (exact in double); NaN for S.1111.111. */
double dms_oracle_e4m3_to_double(uint8_t code) {
  const int sign = code >> 7, e = (code >> 3) & 15, m = code & 7;
  if (e == 15 && m == 7) return NAN;
  double mag = e == 0 ? ldexp((double)m, -9) : ldexp((double)(8 + m), e - 10);
  return sign ? -mag : mag;
}

/*
 * Nearest E4M3FN code of x, ties to even, magnitudes above 448 saturated to 448,
 * NaN -> 0x7f.  The non-negative codes are ordered like their values: code
 * 8 (e - 1) + k holds k * 2^(e - 10) for e >= 1 and k = 8..15 (k = 16 rolls over to
 * the next binade), code k holds k * 2^-9 for k = 0..8.
 */
uint8_t dms_oracle_e4m3_from_float(float x) {
  if (x != x) return 0x7f;
  const uint8_t sign = signbit(x) ? 0x80 : 0x00;
  const double a = fabs((double)x);
  if (a >= 448.0) return sign | 0x7e;
  int code;
  if (a < ldexp(1.0, -6)) {
    code = (int)rint(a / ldexp(1.0, -9)); /* 0 .. 8, exact quotient */
  } else {
    int e2;
    frexp(a, &e2);                          /* a in [2^(e2-1), 2^e2) */
    const int e = e2 + 6;                   /* binade exponent field, 1 .. 15 */
    const int k = (int)rint(a / ldexp(1.0, e - 10)); /* 8 .. 16 */
    code = 8 * (e - 1) + k;
  }
  if (code > 0x7e) code = 0x7e;
  return sign | (uint8_t)code;
}

/* One row of D bf16 values to E4M3 codes and its fp32 scale (see the header). */
void dms_oracle_quantize_row_e4m3(const uint16_t* x, int32_t D, uint8_t* codes, float* scale) {
  float amax = 0.0f;
  for (int32_t d = 0; d < D; ++d) {
    const float a = fabsf((float)dms_oracle_bf16_to_double(x[d]));
    if (a > amax) amax = a;
  }
  if (amax == 0.0f) {
    *scale = 0.0f;
    for (int32_t d = 0; d < D; ++d) codes[d] = 0;
    return;
  }
  const float s = amax / 448.0f;
  *scale = s;
  for (int32_t d = 0; d < D; ++d) {
    const float q = (float)dms_oracle_bf16_to_double(x[d]) / s;
    codes[d] = dms_oracle_e4m3_from_float(q);
  }
}

/*
 * Decode attention as dms_oracle_decode_policy, over fp64 key / value rows (row i at
 * k + i * kv_stride): the dequantised rows of a quantised cache.
 */
void dms_oracle_decode_kv64(const uint16_t* q, int32_t G, int32_t D, const double* k,
                            const double* v, int64_t kv_stride, const uint16_t* logits,
                            int64_t logit_stride, int64_t j, int64_t w, int immediate,
                            double scale, double* out) {
  if (scale <= 0.0) scale = 1.0 / sqrt((double)D);
  int64_t cap = j + 1 > 0 ? j + 1 : 0;
  int32_t* pos = (int32_t*)malloc(sizeof(int32_t) * (size_t)(cap > 0 ? cap : 1));
  double* s = (double*)malloc(sizeof(double) * (size_t)(cap > 0 ? cap : 1));
  int64_t n = dms_oracle_retained_policy(logits, logit_stride, j, w, immediate, pos);
  for (int32_t g = 0; g < G; ++g) {
    double* o = out + (int64_t)g * D;
    for (int32_t d = 0; d < D; ++d) o[d] = 0.0;
    if (n == 0) continue;
    const uint16_t* qg = q + (int64_t)g * D;
    double m = -INFINITY;
    for (int64_t r = 0; r < n; ++r) {
      const double* kr = k + (int64_t)pos[r] * kv_stride;
      double dot = 0.0;
      for (int32_t d = 0; d < D; ++d) dot += dms_oracle_bf16_to_double(qg[d]) * kr[d];
      s[r] = scale * dot;
      if (s[r] > m) m = s[r];
    }
    double den = 0.0;
    for (int64_t r = 0; r < n; ++r) {
      s[r] = exp(s[r] - m);
      den += s[r];
    }
    for (int64_t r = 0; r < n; ++r) {
      const double* vr = v + (int64_t)pos[r] * kv_stride;
      double p = s[r] / den;
      for (int32_t d = 0; d < D; ++d) o[d] += p * vr[d];
    }
  }
  free(pos);
  free(s);
}
