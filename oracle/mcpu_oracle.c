/*
 * CPU oracle for the paged-attention hot path.
 *
 * TEST INFRASTRUCTURE ONLY. Nothing in the product path links, loads or calls
 * this file: only the tests, the smoke check and the bench's CPU-baseline leg
 * use it. It shares no code, header or constant with the CUDA library.
 *
 * What it computes. The paper (§3.2) names generation -- autoregressive
 * decoding of hundreds of concurrent multi-turn trajectories, with tool
 * observations appended between turns -- as the GPU-bound stage of a rollout
 * step; the G = 8 samples of a GRPO task (§4, App. B Tab. "hparams") share
 * their prompt. The paper prints no attention formula, so the operation is the
 * textbook one, written out exactly as defined and in the most direct order:
 *
 *   1. kv append:  for row r with L_r new tokens and post-append length S_r,
 *      new token i (0 <= i < L_r) lands at position pos = S_r - L_r + i, i.e.
 *      physical page block_table[r][pos / page] at slot pos % page, for K and
 *      for V, bit for bit.
 *   2. attention:  query i of row r sits at position p = S_r - L_r + i. Key j
 *      of the row is gathered from page block_table[r][j / page], slot
 *      j % page. Key j is visible iff j <= p (causal) and, when the sliding
 *      window W > 0, p - j < W. With q head h reading kv head h / (H_q/H_kv):
 *         s_j  = scale * sum_d q[d] * K[j][d]
 *         m    = max_j s_j,   l = sum_j exp(s_j - m)
 *         out  = sum_j exp(s_j - m) / l * V[j]          (rounded to bf16)
 *         lse  = m + ln(l)    (natural log of sum_j exp(s_j))
 *      A query with no visible key has out = 0 and lse = -inf.
 *   3. attention sinks (optional; gpt-oss's per-head sink logits, from the
 *      public model card, not from the paper): q head h has a logit sigma_h
 *      that joins the normaliser but carries no value,
 *         Z    = sum_j exp(s_j) + exp(sigma_h)
 *         out  = sum_j exp(s_j) / Z * V[j],   lse = ln Z,
 *      evaluated as above with m = max(max_j s_j, sigma_h). sigma_h = -inf
 *      (or no sinks array) is step 2 exactly.
 *   4. rotary position embedding (optional, before step 1; the rotation of
 *      q and k that gpt-oss applies, with its angles given as a table): a
 *      vector x of length D at position p becomes, for i < D/2,
 *         y_i       = x_i cos_i(p) - x_{i+D/2} sin_i(p)
 *         y_{i+D/2} = x_{i+D/2} cos_i(p) + x_i sin_i(p)
 *      with cos_i(p) = table[p][i], sin_i(p) = table[p][D/2 + i] (float),
 *      products and sums in double, y rounded once to bf16.
 *   5. fp8 KV pages (optional; a storage variant, not in the paper): each new
 *      (token, kv head) row x of 64 bf16 values is stored as 64 e4m3 codes
 *      and one float scale. In float arithmetic: a = max_i |x_i|; if a = 0
 *      the codes and the scale are 0, else inv = 448 / a, scale = a / 448
 *      and code_i = e4m3(x_i * inv), the nearest e4m3 value (ties to even,
 *      saturating at +-448). e4m3 here is the "fn" format: 1 sign, 4
 *      exponent (bias 7), 3 mantissa bits, subnormals down to 2^-9, largest
 *      448, no infinities. Attention then reads K[j][d] = e4m3value(code) *
 *      scale (in double) in place of the bf16 value.
 *
 * Precision: bf16 inputs are widened exactly; every sum and product is taken
 * in double; out is rounded once, double -> bf16, to nearest-even.
 *
 * Layouts (all row-major, bf16 passed as its uint16 bit pattern):
 *   q        [T_q, H_q, D]            k_new, v_new [T_q, H_kv, D]
 *   k_cache  [num_pages, H_kv, page, D]   (same for v_cache)
 *   block_table [num_seqs, max_pages_per_seq] int32
 *   seq_lens [num_seqs] int32,  query_start_loc [num_seqs + 1] int32
 *   out [T_q, H_q, D] bf16 bits,  lse [T_q, H_q] float
 *   sinks [H_q] float or NULL (step 3)
 *
 * Return value: 0 on success, otherwise a positive code naming the first
 * problem found (see ORACLE_ERR_*); nothing is written past a failed check.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORACLE_OK 0
#define ORACLE_ERR_SHAPE 1     /* bad dims, or query_start_loc not monotone */
#define ORACLE_ERR_LENGTH 2    /* L_r > S_r, S_r < 0, or S_r beyond the table */
#define ORACLE_ERR_PAGE 3      /* a page that must be read or written is out of range */
#define ORACLE_ERR_NOMEM 4

static double bf16_to_double(uint16_t b) {
  uint32_t u = (uint32_t)b << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

/* Round a double to the nearest bf16 (8 significant bits, exponent range of
 * float), ties to even. Written from the definition: pick the quantum of the
 * binade (or the subnormal quantum 2^-133), round the scaled value with rint
 * (nearest-even in the default rounding mode), scale back. */
uint16_t oracle_double_to_bf16(double x) {
  if (isnan(x)) return 0x7FC0;
  double ax = fabs(x);
  double r;
  if (ax == 0.0) {
    r = 0.0;
  } else {
    int e;
    frexp(ax, &e);          /* ax = m * 2^e, 0.5 <= m < 1 */
    int qexp = e - 8;       /* 8 significant bits -> quantum 2^(e-8) */
    if (qexp < -133) qexp = -133;
    r = ldexp(rint(ldexp(ax, -qexp)), qexp);
  }
  float f = (float)r; /* exact (or +inf on overflow) */
  if (x < 0) f = -f;
  uint32_t u;
  memcpy(&u, &f, sizeof u);
  return (uint16_t)(u >> 16);
}

static int check_common(const int32_t* seq_lens, const int32_t* qsl, int32_t num_seqs,
                        int32_t max_pages_per_seq, int32_t num_q_heads, int32_t num_kv_heads,
                        int32_t head_dim, int32_t page_size) {
  if (num_seqs < 0 || max_pages_per_seq < 0 || num_kv_heads <= 0 || num_q_heads <= 0 ||
      head_dim <= 0 || page_size <= 0 || num_q_heads % num_kv_heads != 0)
    return ORACLE_ERR_SHAPE;
  if (num_seqs > 0 && qsl[0] != 0) return ORACLE_ERR_SHAPE;
  for (int32_t r = 0; r < num_seqs; ++r) {
    int64_t L = (int64_t)qsl[r + 1] - qsl[r];
    int64_t S = seq_lens[r];
    if (L < 0) return ORACLE_ERR_SHAPE;
    if (S < 0 || L > S) return ORACLE_ERR_LENGTH;
    if (S > (int64_t)max_pages_per_seq * page_size) return ORACLE_ERR_LENGTH;
  }
  return ORACLE_OK;
}

/* Step 1: scatter the new K/V rows of every query token into the pools. */
int oracle_kv_append(const uint16_t* k_new, const uint16_t* v_new, uint16_t* k_cache,
                     uint16_t* v_cache, const int32_t* block_table, const int32_t* seq_lens,
                     const int32_t* query_start_loc, int32_t num_seqs,
                     int32_t max_pages_per_seq, int64_t num_pages, int32_t num_kv_heads,
                     int32_t head_dim, int32_t page_size) {
  int rc = check_common(seq_lens, query_start_loc, num_seqs, max_pages_per_seq, num_kv_heads,
                        num_kv_heads, head_dim, page_size);
  if (rc) return rc;
  /* Check every destination page before writing anything. */
  for (int32_t r = 0; r < num_seqs; ++r) {
    int64_t L = query_start_loc[r + 1] - query_start_loc[r];
    int64_t S = seq_lens[r];
    for (int64_t i = 0; i < L; ++i) {
      int64_t pos = S - L + i;
      int64_t page = block_table[(int64_t)r * max_pages_per_seq + pos / page_size];
      if (page < 0 || page >= num_pages) return ORACLE_ERR_PAGE;
    }
  }
  for (int32_t r = 0; r < num_seqs; ++r) {
    int64_t L = query_start_loc[r + 1] - query_start_loc[r];
    int64_t S = seq_lens[r];
    for (int64_t i = 0; i < L; ++i) {
      int64_t tok = query_start_loc[r] + i;
      int64_t pos = S - L + i;
      int64_t page = block_table[(int64_t)r * max_pages_per_seq + pos / page_size];
      int64_t slot = pos % page_size;
      for (int32_t h = 0; h < num_kv_heads; ++h) {
        const uint16_t* ks = k_new + (tok * num_kv_heads + h) * head_dim;
        const uint16_t* vs = v_new + (tok * num_kv_heads + h) * head_dim;
        uint16_t* kd = k_cache + ((page * num_kv_heads + h) * page_size + slot) * head_dim;
        uint16_t* vd = v_cache + ((page * num_kv_heads + h) * page_size + slot) * head_dim;
        for (int32_t d = 0; d < head_dim; ++d) {
          kd[d] = ks[d];
          vd[d] = vs[d];
        }
      }
    }
  }
  return ORACLE_OK;
}

/* Step 5: value of an e4m3 code. */
double oracle_e4m3_to_double(uint8_t c) {
  int e = (c >> 3) & 15, m = c & 7;
  if (e == 15 && m == 7) return NAN;
  double v = e == 0 ? ldexp((double)m, -9) : ldexp((double)(8 + m), e - 10);
  return (c & 0x80) ? -v : v;
}

/* Step 5: nearest e4m3 code of a float, ties to even, saturating at 448.
 * The quantum of the binade [2^e, 2^(e+1)) is 2^(e-3) (subnormals: 2^-9). */
uint8_t oracle_float_to_e4m3(float x) {
  if (isnan(x)) return 0x7F;
  uint8_t sign = signbit(x) ? 0x80 : 0;
  double a = fabs((double)x);
  if (a >= 448.0) return sign | 0x7E;
  if (a == 0.0) return sign;
  int ex;
  frexp(a, &ex); /* a = f 2^ex, 0.5 <= f < 1 */
  int e = ex - 1;
  if (e < -6) e = -6;
  double q = ldexp(1.0, e - 3);
  double r = rint(a / q) * q; /* a / q is exact: q is a power of two */
  if (r == 0.0) return sign;
  if (r >= 448.0) return sign | 0x7E;
  if (r < ldexp(1.0, -6)) return sign | (uint8_t)(r / ldexp(1.0, -9)); /* subnormal */
  frexp(r, &ex);
  int E = ex - 1;
  int m = (int)(r / ldexp(1.0, E - 3)) - 8;
  return sign | (uint8_t)(((E + 7) << 3) | m);
}

/* Step 5 for one row of n bf16 values: codes and the scale. */
static void quantize_row(const uint16_t* x, int32_t n, uint8_t* codes, float* scale) {
  float a = 0.f;
  for (int32_t i = 0; i < n; ++i) {
    float v = (float)fabs(bf16_to_double(x[i]));
    if (v > a) a = v;
  }
  if (a == 0.f) {
    for (int32_t i = 0; i < n; ++i) codes[i] = 0;
    *scale = 0.f;
    return;
  }
  volatile float inv = 448.0f / a; /* float arithmetic, as defined */
  *scale = a / 448.0f;
  for (int32_t i = 0; i < n; ++i) {
    volatile float y = (float)bf16_to_double(x[i]) * inv;
    codes[i] = oracle_float_to_e4m3(y);
  }
}

/* Step 1 with step 5: scatter the quantized new rows into fp8 pools
 * k8/v8 [num_pages, H_kv, page, D] and scales [num_pages, H_kv, page]. */
int oracle_kv_append_fp8(const uint16_t* k_new, const uint16_t* v_new, uint8_t* k8, uint8_t* v8,
                         float* k_scale, float* v_scale, const int32_t* block_table,
                         const int32_t* seq_lens, const int32_t* query_start_loc, int32_t num_seqs,
                         int32_t max_pages_per_seq, int64_t num_pages, int32_t num_kv_heads,
                         int32_t head_dim, int32_t page_size) {
  int rc = check_common(seq_lens, query_start_loc, num_seqs, max_pages_per_seq, num_kv_heads,
                        num_kv_heads, head_dim, page_size);
  if (rc) return rc;
  for (int32_t r = 0; r < num_seqs; ++r) {
    int64_t L = query_start_loc[r + 1] - query_start_loc[r];
    int64_t S = seq_lens[r];
    for (int64_t i = 0; i < L; ++i) {
      int64_t page = block_table[(int64_t)r * max_pages_per_seq + (S - L + i) / page_size];
      if (page < 0 || page >= num_pages) return ORACLE_ERR_PAGE;
    }
  }
  for (int32_t r = 0; r < num_seqs; ++r) {
    int64_t L = query_start_loc[r + 1] - query_start_loc[r];
    int64_t S = seq_lens[r];
    for (int64_t i = 0; i < L; ++i) {
      int64_t tok = query_start_loc[r] + i;
      int64_t pos = S - L + i;
      int64_t page = block_table[(int64_t)r * max_pages_per_seq + pos / page_size];
      for (int32_t h = 0; h < num_kv_heads; ++h) {
        int64_t row = (page * num_kv_heads + h) * page_size + pos % page_size;
        quantize_row(k_new + (tok * num_kv_heads + h) * head_dim, head_dim, k8 + row * head_dim, k_scale + row);
        quantize_row(v_new + (tok * num_kv_heads + h) * head_dim, head_dim, v8 + row * head_dim, v_scale + row);
      }
    }
  }
  return ORACLE_OK;
}

/* Visible key range [lo, p] of a query at position p (step 2's mask). */
static int64_t first_visible(int64_t p, int32_t window) {
  if (window <= 0) return 0;
  int64_t lo = p - window + 1;
  return lo < 0 ? 0 : lo;
}

/* Where K and V come from: bf16 pools (step 2), or fp8 pools with their
 * per-row scales (step 5). Rows are (page * H_kv + kv head) * page + slot. */
typedef struct {
  const uint16_t *k16, *v16;
  const uint8_t *k8, *v8;
  const float *ks, *vs;
} kv_src;

static double kv_value(const kv_src* src, int is_v, int64_t row, int32_t d, int32_t head_dim) {
  if (src->k16) return bf16_to_double((is_v ? src->v16 : src->k16)[row * head_dim + d]);
  return oracle_e4m3_to_double((is_v ? src->v8 : src->k8)[row * head_dim + d]) *
         (double)(is_v ? src->vs : src->ks)[row];
}

/* Step 2 for one query vector: gathers its visible keys straight from the
 * pages and writes out[0..D) (bf16 bits) and *lse. */
static int attend_one(const uint16_t* qv, const kv_src* src,
                      const int32_t* bt_row, int64_t p, int32_t kvh, int32_t window,
                      double scale, double sink, int64_t num_pages, int32_t num_kv_heads,
                      int32_t head_dim, int32_t page_size, double* s, double* acc, uint16_t* out,
                      float* lse) {
  int64_t lo = first_visible(p, window);
  int64_t n = p - lo + 1;
  if (n <= 0) {
    for (int32_t d = 0; d < head_dim; ++d) out[d] = 0;
    *lse = (float)sink; /* ln exp(sigma); -inf without a sink */
    return ORACLE_OK;
  }
  /* scores */
  double m = -INFINITY;
  for (int64_t j = lo; j <= p; ++j) {
    int64_t page = bt_row[j / page_size];
    if (page < 0 || page >= num_pages) return ORACLE_ERR_PAGE;
    const int64_t kr = (page * num_kv_heads + kvh) * page_size + j % page_size;
    double dot = 0.0;
    for (int32_t d = 0; d < head_dim; ++d) dot += bf16_to_double(qv[d]) * kv_value(src, 0, kr, d, head_dim);
    s[j - lo] = scale * dot;
    if (s[j - lo] > m) m = s[j - lo];
  }
  /* normaliser (step 3: the sink joins the max and the sum) */
  if (sink > m) m = sink;
  double l = 0.0;
  for (int64_t j = 0; j < n; ++j) l += exp(s[j] - m);
  if (sink > -INFINITY) l += exp(sink - m);
  /* weighted sum of values */
  for (int32_t d = 0; d < head_dim; ++d) acc[d] = 0.0;
  for (int64_t j = lo; j <= p; ++j) {
    int64_t page = bt_row[j / page_size];
    const int64_t vr = (page * num_kv_heads + kvh) * page_size + j % page_size;
    double w = exp(s[j - lo] - m) / l;
    for (int32_t d = 0; d < head_dim; ++d) acc[d] += w * kv_value(src, 1, vr, d, head_dim);
  }
  for (int32_t d = 0; d < head_dim; ++d) out[d] = oracle_double_to_bf16(acc[d]);
  *lse = (float)(m + log(l));
  return ORACLE_OK;
}

static int row_of_token(const int32_t* qsl, int32_t num_seqs, int64_t t) {
  for (int32_t r = 0; r < num_seqs; ++r)
    if (t >= qsl[r] && t < qsl[r + 1]) return r;
  return -1;
}

/* Full attention: every query token of every row, every q head. */
static int paged_attention_impl(const uint16_t* q, const kv_src* src,
                                const int32_t* block_table, const int32_t* seq_lens,
                                const int32_t* query_start_loc, int32_t num_seqs,
                                int32_t max_pages_per_seq, int64_t num_pages, int32_t num_q_heads,
                                int32_t num_kv_heads, int32_t head_dim, int32_t page_size,
                                int32_t sliding_window, double softmax_scale, uint16_t* out,
                                float* lse, int32_t num_threads, const float* sinks) {
  int rc = check_common(seq_lens, query_start_loc, num_seqs, max_pages_per_seq, num_q_heads,
                        num_kv_heads, head_dim, page_size);
  if (rc) return rc;
  int64_t max_s = 1;
  for (int32_t r = 0; r < num_seqs; ++r)
    if (seq_lens[r] > max_s) max_s = seq_lens[r];
  const int32_t group = num_q_heads / num_kv_heads;
  const int64_t total_q = num_seqs > 0 ? query_start_loc[num_seqs] : 0;
  int err = ORACLE_OK;
#ifdef _OPENMP
  if (num_threads > 0) omp_set_num_threads(num_threads);
#else
  (void)num_threads;
#endif
#pragma omp parallel
  {
    double* s = (double*)malloc(sizeof(double) * (size_t)max_s);
    double* acc = (double*)malloc(sizeof(double) * (size_t)head_dim);
    if (!s || !acc) {
#pragma omp atomic write
      err = ORACLE_ERR_NOMEM;
    }
#pragma omp for schedule(dynamic, 1) collapse(2)
    for (int64_t t = 0; t < total_q; ++t) {
      for (int32_t h = 0; h < num_q_heads; ++h) {
        if (!s || !acc) continue;
        int32_t r = row_of_token(query_start_loc, num_seqs, t);
        int64_t S = seq_lens[r];
        int64_t L = query_start_loc[r + 1] - query_start_loc[r];
        int64_t p = S - L + (t - query_start_loc[r]);
        int e = attend_one(q + (t * num_q_heads + h) * head_dim, src,
                           block_table + (int64_t)r * max_pages_per_seq, p, h / group,
                           sliding_window, softmax_scale, sinks ? (double)sinks[h] : -INFINITY,
                           num_pages, num_kv_heads, head_dim, page_size, s, acc,
                           out + (t * num_q_heads + h) * head_dim, lse + t * num_q_heads + h);
        if (e) {
#pragma omp atomic write
          err = e;
        }
      }
    }
    free(s);
    free(acc);
  }
  return err;
}

/* The same at listed (token, q head) pairs. */
static int paged_attention_sampled_impl(const uint16_t* q, const kv_src* src,
                                   const int32_t* block_table,
                                   const int32_t* seq_lens, const int32_t* query_start_loc,
                                   int32_t num_seqs, int32_t max_pages_per_seq, int64_t num_pages,
                                   int32_t num_q_heads, int32_t num_kv_heads, int32_t head_dim,
                                   int32_t page_size, int32_t sliding_window,
                                   double softmax_scale, const int64_t* sample_token,
                                   const int32_t* sample_head, int64_t n_samples,
                                   uint16_t* out_samples, float* lse_samples,
                                   int32_t num_threads, const float* sinks) {
  int rc = check_common(seq_lens, query_start_loc, num_seqs, max_pages_per_seq, num_q_heads,
                        num_kv_heads, head_dim, page_size);
  if (rc) return rc;
  const int64_t total_q = num_seqs > 0 ? query_start_loc[num_seqs] : 0;
  for (int64_t i = 0; i < n_samples; ++i)
    if (sample_token[i] < 0 || sample_token[i] >= total_q || sample_head[i] < 0 ||
        sample_head[i] >= num_q_heads)
      return ORACLE_ERR_SHAPE;
  int64_t max_s = 1;
  for (int32_t r = 0; r < num_seqs; ++r)
    if (seq_lens[r] > max_s) max_s = seq_lens[r];
  const int32_t group = num_q_heads / num_kv_heads;
  int err = ORACLE_OK;
#ifdef _OPENMP
  if (num_threads > 0) omp_set_num_threads(num_threads);
#else
  (void)num_threads;
#endif
#pragma omp parallel
  {
    double* s = (double*)malloc(sizeof(double) * (size_t)max_s);
    double* acc = (double*)malloc(sizeof(double) * (size_t)head_dim);
    if (!s || !acc) {
#pragma omp atomic write
      err = ORACLE_ERR_NOMEM;
    }
#pragma omp for schedule(dynamic, 1)
    for (int64_t i = 0; i < n_samples; ++i) {
      if (!s || !acc) continue;
      int64_t t = sample_token[i];
      int32_t h = sample_head[i];
      int32_t r = row_of_token(query_start_loc, num_seqs, t);
      int64_t S = seq_lens[r];
      int64_t L = query_start_loc[r + 1] - query_start_loc[r];
      int64_t p = S - L + (t - query_start_loc[r]);
      int e = attend_one(q + (t * num_q_heads + h) * head_dim, src,
                         block_table + (int64_t)r * max_pages_per_seq, p, h / group,
                         sliding_window, softmax_scale, sinks ? (double)sinks[h] : -INFINITY,
                         num_pages, num_kv_heads, head_dim, page_size, s, acc,
                         out_samples + i * head_dim, lse_samples + i);
      if (e) {
#pragma omp atomic write
        err = e;
      }
    }
    free(s);
    free(acc);
  }
  return err;
}

/* Step 4 on x [n, heads, D] (bf16 bits, rotated in place): row t sits at
 * position positions[t]; cos_sin is [max_position, D] float. */
int oracle_rope(uint16_t* x, int64_t n, int32_t heads, int32_t head_dim, const int64_t* positions,
                const float* cos_sin, int64_t max_position) {
  if (n < 0 || heads <= 0 || head_dim <= 0 || head_dim % 2) return ORACLE_ERR_SHAPE;
  for (int64_t t = 0; t < n; ++t)
    if (positions[t] < 0 || positions[t] >= max_position) return ORACLE_ERR_LENGTH;
  const int32_t half = head_dim / 2;
  for (int64_t t = 0; t < n; ++t) {
    const float* cs = cos_sin + positions[t] * head_dim;
    for (int32_t h = 0; h < heads; ++h) {
      uint16_t* v = x + (t * heads + h) * head_dim;
      for (int32_t i = 0; i < half; ++i) {
        double a = bf16_to_double(v[i]), b = bf16_to_double(v[i + half]);
        double c = (double)cs[i], s = (double)cs[half + i];
        v[i] = oracle_double_to_bf16(a * c - b * s);
        v[i + half] = oracle_double_to_bf16(b * c + a * s);
      }
    }
  }
  return ORACLE_OK;
}

/* Full attention (steps 2-3) over bf16 pools. num_threads <= 0 uses the
 * OpenMP default. */
int oracle_paged_attention(const uint16_t* q, const uint16_t* k_cache, const uint16_t* v_cache,
                           const int32_t* block_table, const int32_t* seq_lens,
                           const int32_t* query_start_loc, int32_t num_seqs,
                           int32_t max_pages_per_seq, int64_t num_pages, int32_t num_q_heads,
                           int32_t num_kv_heads, int32_t head_dim, int32_t page_size,
                           int32_t sliding_window, double softmax_scale, uint16_t* out,
                           float* lse, int32_t num_threads, const float* sinks) {
  kv_src src = {k_cache, v_cache, NULL, NULL, NULL, NULL};
  return paged_attention_impl(q, &src, block_table, seq_lens, query_start_loc, num_seqs, max_pages_per_seq,
                              num_pages, num_q_heads, num_kv_heads, head_dim, page_size, sliding_window,
                              softmax_scale, out, lse, num_threads, sinks);
}

/* The same over fp8 pools with per-row scales (step 5). */
int oracle_paged_attention_fp8(const uint16_t* q, const uint8_t* k8, const uint8_t* v8, const float* k_scale,
                               const float* v_scale, const int32_t* block_table, const int32_t* seq_lens,
                               const int32_t* query_start_loc, int32_t num_seqs, int32_t max_pages_per_seq,
                               int64_t num_pages, int32_t num_q_heads, int32_t num_kv_heads, int32_t head_dim,
                               int32_t page_size, int32_t sliding_window, double softmax_scale, uint16_t* out,
                               float* lse, int32_t num_threads, const float* sinks) {
  kv_src src = {NULL, NULL, k8, v8, k_scale, v_scale};
  return paged_attention_impl(q, &src, block_table, seq_lens, query_start_loc, num_seqs, max_pages_per_seq,
                              num_pages, num_q_heads, num_kv_heads, head_dim, page_size, sliding_window,
                              softmax_scale, out, lse, num_threads, sinks);
}

/* The definition evaluated only at listed (token, q head) pairs, for spot
 * checks of workloads too large to run in full. out_samples is
 * [n_samples, D] bf16 bits, lse_samples [n_samples]. */
int oracle_paged_attention_sampled(const uint16_t* q, const uint16_t* k_cache,
                                   const uint16_t* v_cache, const int32_t* block_table,
                                   const int32_t* seq_lens, const int32_t* query_start_loc,
                                   int32_t num_seqs, int32_t max_pages_per_seq, int64_t num_pages,
                                   int32_t num_q_heads, int32_t num_kv_heads, int32_t head_dim,
                                   int32_t page_size, int32_t sliding_window,
                                   double softmax_scale, const int64_t* sample_token,
                                   const int32_t* sample_head, int64_t n_samples,
                                   uint16_t* out_samples, float* lse_samples,
                                   int32_t num_threads, const float* sinks) {
  kv_src src = {k_cache, v_cache, NULL, NULL, NULL, NULL};
  return paged_attention_sampled_impl(q, &src, block_table, seq_lens, query_start_loc, num_seqs,
                                      max_pages_per_seq, num_pages, num_q_heads, num_kv_heads, head_dim,
                                      page_size, sliding_window, softmax_scale, sample_token, sample_head,
                                      n_samples, out_samples, lse_samples, num_threads, sinks);
}

int oracle_paged_attention_sampled_fp8(const uint16_t* q, const uint8_t* k8, const uint8_t* v8,
                                       const float* k_scale, const float* v_scale, const int32_t* block_table,
                                       const int32_t* seq_lens, const int32_t* query_start_loc, int32_t num_seqs,
                                       int32_t max_pages_per_seq, int64_t num_pages, int32_t num_q_heads,
                                       int32_t num_kv_heads, int32_t head_dim, int32_t page_size,
                                       int32_t sliding_window, double softmax_scale, const int64_t* sample_token,
                                       const int32_t* sample_head, int64_t n_samples, uint16_t* out_samples,
                                       float* lse_samples, int32_t num_threads, const float* sinks) {
  kv_src src = {NULL, NULL, k8, v8, k_scale, v_scale};
  return paged_attention_sampled_impl(q, &src, block_table, seq_lens, query_start_loc, num_seqs,
                                      max_pages_per_seq, num_pages, num_q_heads, num_kv_heads, head_dim,
                                      page_size, sliding_window, softmax_scale, sample_token, sample_head,
                                      n_samples, out_samples, lse_samples, num_threads, sinks);
}

int oracle_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}
