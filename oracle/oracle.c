/*
 * oracle.c — plain, slow, single-threaded CPU oracle for the error-feedback
 * (EF) sparsification step of "Rethinking gradient sparsification as total
 * error minimization" (arXiv:2108.00951).
 *
 * TEST INFRASTRUCTURE ONLY. Nothing in the product path may call, link or
 * load this file or the library built from it; only the tests, the smoke
 * check and the CPU-baseline leg of the benchmark use it. It shares no code,
 * header, table or helper with the CUDA library: every line here is written
 * from the paper's definitions, in the paper's order, for a reader to check
 * by eye.
 *
 * Build: gcc -O2 -std=c11 -ffp-contract=off -fno-fast-math -fPIC -shared
 * (no contraction: the only fused operation is the explicit fmaf below).
 *
 * Readings of the paper taken here (the same ones the CUDA library follows):
 *   R1 gamma placement: the threshold applies to a = e + gamma*g directly and
 *      the value sent is a itself (Algorithm 1 with Delta = C(p), which
 *      Remark 1 states is the same for the sparsifiers considered).
 *   R2 rounding: a is one fused multiply-add, fmaf(gamma, g, e).
 *   R3 the hard-threshold support uses >= (Sec. 1; Sec. 4.2).
 *   R4 a coordinate equal to +-0 is never sent (it adds nothing to C(a) and
 *      ||C(a)||_0 does not count it).
 *   R5 Top-k ties go to the lowest index; exactly k pairs are sent.
 *   R6 NaN (the paper is silent on it): a NaN carries no value, so every
 *      NaN is the same magnitude, above +inf (equal magnitudes tie by index
 *      as in R5); the hard-threshold test |a| >= lambda is false for NaN.
 *      NaN results keep whatever encoding the host arithmetic gives them;
 *      results are compared with any NaN equal to any other NaN.
 *   R7 the residual of a sent coordinate is +0.0f.
 *   R9 aggregation returns the sum (the 1/n of Algorithm 1 is the caller's),
 *      accumulated from +0.0f in ascending worker order.
 *   R14 scaled integer rounding (Sec. 5 names it an absolute compressor):
 *      q_j = round-half-to-even(a_j 2^m) as int32, C(a)_j = q_j 2^-m, e'_j =
 *      a_j - C(a)_j (exact); a coordinate whose a_j 2^m has magnitude at least
 *      2^31 (or is NaN) is not sent: q_j = 0, e'_j = a_j, and it is counted. The integer messages are summed exactly and the sum
 *      decompressed with one rounding: RN(S_j) 2^-m.
 *   R12 model update after aggregation (the paper is silent on rounding):
 *      Delta'_j = alpha * s_j rounded once (alpha = 1/n gives the mean);
 *      without momentum x_j <- x_j - Delta'_j; with momentum
 *      m_j <- fmaf(mu, m_j, Delta'_j) and x_j <- fmaf(-lr, Delta'_j + m_j, x_j),
 *      the sum Delta'_j + m_j rounded once.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* Widen a bfloat16 bit pattern to the fp32 value it denotes: the 16 stored
 * bits are the high half of the fp32 encoding, the low half is zero. */
static float bf16_bits_to_float(uint16_t bits) {
  uint32_t w = ((uint32_t)bits) << 16;
  float f;
  memcpy(&f, &w, sizeof f);
  return f;
}

/* ------------------------------------------------------------------------
 * Hard-threshold (Algorithm 1 with C = C_lambda).
 *   p_{i,t} = e_{i,t} + gamma g_{i,t}             (Algorithm 1, first step)
 *   S_lambda(p) = { j : |p[j]| >= lambda }         (Sec. 1; Sec. 4.2)
 *   Delta = sum_{j in S} p[j] u_j, sent as pairs   (Sec. 4.2 sparsifier form)
 *   e_{i,t+1} = p - Delta                          (Algorithm 1, error update)
 * ------------------------------------------------------------------------ */
static int hard_threshold_core(const float* g_f32, const uint16_t* g_bf16,
                               float* e, float gamma, float lambda, uint64_t d,
                               uint32_t* idx, float* val, uint32_t* count) {
  uint64_t c = 0;
  for (uint64_t j = 0; j < d; ++j) {
    float gj = g_f32 ? g_f32[j] : bf16_bits_to_float(g_bf16[j]);
    float a = fmaf(gamma, gj, e[j]);                       /* R2 */
    int in_support = (fabsf(a) >= lambda) && (a != 0.0f); /* R3, R4, R6 */
    if (in_support) {
      idx[c] = (uint32_t)j;
      val[c] = a;
      ++c;
      e[j] = 0.0f;                                       /* R7 */
    } else {
      e[j] = a;
    }
  }
  *count = (uint32_t)c;
  return 0;
}

int oracle_ef_hard_threshold(const float* g, float* e, float gamma,
                             float lambda, uint64_t d, uint32_t* idx,
                             float* val, uint32_t* count) {
  return hard_threshold_core(g, NULL, e, gamma, lambda, d, idx, val, count);
}

int oracle_ef_hard_threshold_bf16(const uint16_t* g, float* e, float gamma,
                                  float lambda, uint64_t d, uint32_t* idx,
                                  float* val, uint32_t* count) {
  return hard_threshold_core(NULL, g, e, gamma, lambda, d, idx, val, count);
}

/* ------------------------------------------------------------------------
 * Top-k (Algorithm 1 with C = Top-k; Lemma 1 / Lemma 2: keeping the k
 * largest-magnitude entries minimises ||p - C(p)||^2 under ||C(p)||_0 <= k).
 * ------------------------------------------------------------------------ */

/* Magnitude order of R6: the ordinary order of fabsf for numbers; every NaN
 * ranks above +inf, and two NaNs are equal. Returns -1, 0 or +1. */
static int magnitude_cmp(float x, float y) {
  float ax = fabsf(x), ay = fabsf(y);
  int nx = isnan(ax), ny = isnan(ay);
  if (nx || ny) {
    if (nx && ny) return 0;
    return nx ? 1 : -1;
  }
  return (ax > ay) - (ax < ay);
}

static const float* g_sort_keys; /* single-threaded oracle: qsort context */

/* Sort order for the Top-k selection: larger magnitude first; equal
 * magnitudes by ascending index (R5). */
static int topk_order(const void* pa, const void* pb) {
  uint32_t ia = *(const uint32_t*)pa, ib = *(const uint32_t*)pb;
  int m = magnitude_cmp(g_sort_keys[ia], g_sort_keys[ib]);
  if (m != 0) return -m;
  return (ia > ib) - (ia < ib);
}

static int ascending_u32(const void* pa, const void* pb) {
  uint32_t a = *(const uint32_t*)pa, b = *(const uint32_t*)pb;
  return (a > b) - (a < b);
}

static int topk_core(const float* g_f32, const uint16_t* g_bf16, float* e,
                     float gamma, uint64_t k, uint64_t d, uint32_t* idx,
                     float* val, uint32_t* count) {
  if (k > d) return 1;
  float* a = (float*)malloc((d ? d : 1) * sizeof(float));
  uint32_t* order = (uint32_t*)malloc((d ? d : 1) * sizeof(uint32_t));
  if (!a || !order) { free(a); free(order); return 2; }
  /* corrected update p = e + gamma g (Algorithm 1), one fma each (R2) */
  for (uint64_t j = 0; j < d; ++j) {
    float gj = g_f32 ? g_f32[j] : bf16_bits_to_float(g_bf16[j]);
    a[j] = fmaf(gamma, gj, e[j]);
    order[j] = (uint32_t)j;
  }
  /* S = the first k coordinates in decreasing magnitude, ties by index */
  g_sort_keys = a;
  qsort(order, d, sizeof(uint32_t), topk_order);
  /* emit S in ascending index order */
  qsort(order, k, sizeof(uint32_t), ascending_u32);
  for (uint64_t j = 0; j < d; ++j) e[j] = a[j];      /* e' = p on j not in S */
  for (uint64_t p = 0; p < k; ++p) {
    uint32_t j = order[p];
    idx[p] = j;
    val[p] = a[j];
    e[j] = 0.0f;                                      /* R7 */
  }
  *count = (uint32_t)k;
  free(a);
  free(order);
  return 0;
}

int oracle_ef_topk(const float* g, float* e, float gamma, uint64_t k,
                   uint64_t d, uint32_t* idx, float* val, uint32_t* count) {
  return topk_core(g, NULL, e, gamma, k, d, idx, val, count);
}

int oracle_ef_topk_bf16(const uint16_t* g, float* e, float gamma, uint64_t k,
                        uint64_t d, uint32_t* idx, float* val,
                        uint32_t* count) {
  return topk_core(NULL, g, e, gamma, k, d, idx, val, count);
}

/* ------------------------------------------------------------------------
 * Layer-wise Top-k (Appendix, "layer-wise or entire-model" sparsification:
 * in layer-wise sparsification the sparsifier is invoked on each layer's
 * tensor separately; the experiments use it for Top-k). The vector is the
 * concatenation of n_seg tensors; segment s covers [seg_end[s-1], seg_end[s])
 * (seg_end[-1] = 0, seg_end[n_seg-1] = d) and sends its k_s = seg_k[s]
 * largest-magnitude coordinates under the Top-k rules above (R5, R6, R7).
 * The pairs of all segments are emitted in ascending index order, so the
 * message is the concatenation of the per-segment messages.
 * ------------------------------------------------------------------------ */
static int topk_layerwise_core(const float* g_f32, const uint16_t* g_bf16, float* e,
                               float gamma, uint32_t n_seg, const uint64_t* seg_end,
                               const uint64_t* seg_k, uint64_t d, uint32_t* idx,
                               float* val, uint32_t* count) {
  uint64_t lo = 0, sent = 0;
  for (uint32_t s = 0; s < n_seg; ++s) {
    uint64_t hi = seg_end[s];
    if (hi < lo || hi > d || seg_k[s] > hi - lo) return 1;
    uint32_t c = 0;
    /* the Top-k sparsifier on this tensor alone: indices come out local */
    int rc = topk_core(g_f32 ? g_f32 + lo : NULL, g_bf16 ? g_bf16 + lo : NULL, e + lo, gamma,
                       seg_k[s], hi - lo, idx + sent, val + sent, &c);
    if (rc != 0) return rc;
    for (uint32_t p = 0; p < c; ++p) idx[sent + p] += (uint32_t)lo; /* to global indices */
    sent += c;
    lo = hi;
  }
  if (lo != d) return 1;
  *count = (uint32_t)sent;
  return 0;
}

int oracle_ef_topk_layerwise(const float* g, float* e, float gamma, uint32_t n_seg,
                             const uint64_t* seg_end, const uint64_t* seg_k, uint64_t d,
                             uint32_t* idx, float* val, uint32_t* count) {
  return topk_layerwise_core(g, NULL, e, gamma, n_seg, seg_end, seg_k, d, idx, val, count);
}

int oracle_ef_topk_layerwise_bf16(const uint16_t* g, float* e, float gamma, uint32_t n_seg,
                                  const uint64_t* seg_end, const uint64_t* seg_k, uint64_t d,
                                  uint32_t* idx, float* val, uint32_t* count) {
  return topk_layerwise_core(NULL, g, e, gamma, n_seg, seg_end, seg_k, d, idx, val, count);
}

/* ------------------------------------------------------------------------
 * Aggregation (Algorithm 1, exchange step): sum_i Delta_{i,t}, decompressed
 * into a dense vector. Sum, not mean (R9); from +0.0f; workers in order.
 * ------------------------------------------------------------------------ */
int oracle_sparse_aggregate(uint32_t n, const uint32_t* const* idx,
                            const float* const* val, const uint32_t* counts,
                            uint64_t d, float* dense) {
  for (uint64_t j = 0; j < d; ++j) dense[j] = 0.0f;
  for (uint32_t i = 0; i < n; ++i) {
    for (uint32_t p = 0; p < counts[i]; ++p) {
      uint32_t j = idx[i][p];
      if ((uint64_t)j >= d) return 1;
      dense[j] = dense[j] + val[i][p];
    }
  }
  return 0;
}

/* ------------------------------------------------------------------------
 * Model update after the exchange step (R12).
 *   Algorithm 1:  Delta_bar_t = (1/n) sum_i Delta_{i,t};  x_{t+1} = x_t - Delta_bar_t.
 *   Appendix, distributed EF SGD with momentum by gradient compression (the
 *   EF strategy of the experiments): Delta' = the aggregated compressed
 *   vectors; m <- lambda m + Delta'; x <- x - gamma (Delta' + m), with the
 *   momentum factor called mu and the learning rate lr here.
 * m == NULL selects Algorithm 1's update; otherwise the momentum one.
 * ------------------------------------------------------------------------ */
int oracle_sparse_aggregate_apply(uint32_t n, const uint32_t* const* idx,
                                  const float* const* val, const uint32_t* counts,
                                  uint64_t d, float alpha, float* x, float* m, float mu,
                                  float lr) {
  float* s = (float*)malloc((d ? d : 1) * sizeof(float));
  if (!s) return 2;
  int rc = oracle_sparse_aggregate(n, idx, val, counts, d, s);
  if (rc == 0) {
    for (uint64_t j = 0; j < d; ++j) {
      float delta = alpha * s[j];                    /* Delta'_j */
      if (m) {
        m[j] = fmaf(mu, m[j], delta);                /* m <- mu m + Delta' */
        float u = delta + m[j];                      /* Delta' + m */
        x[j] = fmaf(-lr, u, x[j]);                   /* x <- x - lr (Delta' + m) */
      } else {
        x[j] = x[j] - delta;                         /* x <- x - Delta_bar */
      }
    }
  }
  free(s);
  return rc;
}

/* ------------------------------------------------------------------------
 * Squared error norm of one step, ||e_{t+1}||^2 = sum_j e'_j^2: the term
 * whose sum over iterations is the total error (Sec. 1; the remark after
 * the EF convergence theorem). Plain fp64: every fp32 square is exact in
 * fp64, summed in index order.
 * ------------------------------------------------------------------------ */
double oracle_error_norm_sq(const float* e, uint64_t d) {
  double s = 0.0;
  for (uint64_t j = 0; j < d; ++j) s += (double)e[j] * (double)e[j];
  return s;
}

/* ------------------------------------------------------------------------
 * Scaled integer rounding (Sec. 5: any rounding with error bounded by eps
 * is an absolute compressor with kappa^2 = d eps^2, the scaled integer
 * rounding of in-network aggregation among them), under error feedback
 * (Algorithm 1):
 *   a_j = fmaf(gamma, g_j, e_j); q_j = RNE(a_j 2^m);
 *   C(a)_j = q_j 2^-m; e'_j = a_j - C(a)_j, |e'_j| <= 2^(-m-1)  (R14)
 * ------------------------------------------------------------------------ */
static int scaled_round_core(const float* g_f32, const uint16_t* g_bf16, float* e, float gamma,
                             int m, uint64_t d, int32_t* q, uint32_t* unsent) {
  uint32_t u = 0;
  for (uint64_t j = 0; j < d; ++j) {
    float gj = g_f32 ? g_f32[j] : bf16_bits_to_float(g_bf16[j]);
    float a = fmaf(gamma, gj, e[j]);                           /* R2 */
    float s = ldexpf(a, m);                                    /* a 2^m (exact scaling) */
    if (!(fabsf(s) < 2147483648.0f)) {                         /* |a 2^m| >= 2^31, or NaN */
      q[j] = 0;                                                /* not representable: */
      e[j] = a;                                                /* kept in e (R14) */
      ++u;
      continue;
    }
    float r = rintf(s);                                        /* round half to even */
    q[j] = (int32_t)r;
    float c = ldexpf((float)q[j], -m);                         /* C(a)_j */
    e[j] = a - c;                                              /* e'_j = a_j - C(a)_j */
  }
  *unsent = u;
  return 0;
}

int oracle_ef_scaled_round(const float* g, float* e, float gamma, int m, uint64_t d, int32_t* q,
                           uint32_t* unsent) {
  return scaled_round_core(g, NULL, e, gamma, m, d, q, unsent);
}

int oracle_ef_scaled_round_bf16(const uint16_t* g, float* e, float gamma, int m, uint64_t d,
                                int32_t* q, uint32_t* unsent) {
  return scaled_round_core(NULL, g, e, gamma, m, d, q, unsent);
}

/* Exchange of the integer messages: S_j = sum_i q_i[j] exactly (int64, any
 * order gives the same sum), decompressed as RN(S_j) 2^-m (R14). */
int oracle_int_aggregate(uint32_t n, const int32_t* const* q, uint64_t d, int m, float* dense) {
  for (uint64_t j = 0; j < d; ++j) {
    int64_t s = 0;
    for (uint32_t i = 0; i < n; ++i) s += q[i][j];
    dense[j] = ldexpf((float)s, -m);
  }
  return 0;
}
