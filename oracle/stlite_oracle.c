/*
 * ST-Lite reference oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, single-threaded CPU restatement of the ST-Lite per-layer
 * KV-cache compression procedure (Algorithm 1 of "ST-Lite: Training-Free KV
 * Cache Compression with Spatio-Trajectory Guidance for Long-Horizon GUI
 * Agents", arXiv 2603.00188).  Every quantity is computed in IEEE double from
 * inputs that the caller has already converted exactly (bf16/fp32 -> double).
 * There is no blocking, fusion or reordering beyond what the definitions state.
 *
 * Only the test suite, the package smoke check and the benchmark's CPU
 * baseline leg may load this code.  It shares no code, header or constant with
 * the CUDA library; neither side includes or links the other.
 *
 * Layouts (all row-major, C order):
 *   q  [w][Hq][d]   window queries; query head g belongs to KV head g / G,
 *                   G = Hq / Hkv (grouped-query attention).
 *   k  [n][Hkv][d]  cached keys of one layer.
 *   Frame f owns the contiguous visual span [off[f], off[f] + gh[f]*gw[f]),
 *   laid out row-major on a gh[f] x gw[f] patch grid (u = row, v = column).
 *   The last frame is the current frame; every token outside a frame is text.
 *
 * Readings of points the paper leaves open (each restated where it is used):
 *   R1  GQA: A_base of a KV head is the mean over its G query heads of the
 *       single-head window score of Eq. (2).
 *   R2  Cosine: a.b / (max(|a|,1e-8) * max(|b|,1e-8)); a zero vector has
 *       cosine 0 with everything.
 *   R3  CSS neighbours: only the in-grid cells of the 3x3 Moore neighbourhood
 *       of the same frame; a cell with no neighbour (1x1 grid) has Phi = 0.
 *   R4  Budget: B = floor(beta * L + 1e-9), at least 1, unless overridden.
 *   R5  Top-B ties: equal scores are ranked by ascending token index.
 *   R6  Per-KV-head selection: each KV head keeps its own B tokens.
 *   R7  Undefined entries (Phi of a text token, rho of a token outside the
 *       historical pool) are reported as NaN.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ---------------------------------------------------------------- helpers */

static double dot(const double* a, const double* b, int32_t d) {
  double s = 0.0;
  for (int32_t t = 0; t < d; ++t) s += a[t] * b[t];
  return s;
}

static double norm_clamped(const double* a, int32_t d) {
  double n = sqrt(dot(a, a, d));
  return n > 1e-8 ? n : 1e-8;
}

/* Cosine similarity used by both CSS (Eq. 4) and TSG (Eq. 6), reading R2. */
static double cosine(const double* a, const double* b, int32_t d) {
  return dot(a, b, d) / (norm_clamped(a, d) * norm_clamped(b, d));
}

static const double* key_row(const double* k, int32_t hkv, int32_t d, int32_t j, int32_t h) {
  return k + ((size_t)j * hkv + h) * d;
}

/* Frame membership: returns the frame holding token j, or -1 for text. */
static int32_t frame_of(int32_t j, int32_t n_frames, const int32_t* off, const int32_t* gh,
                        const int32_t* gw) {
  for (int32_t f = 0; f < n_frames; ++f)
    if (j >= off[f] && j < off[f] + gh[f] * gw[f]) return f;
  return -1;
}

/* --------------------------------------------------------------- budget */

/* Flat per-layer budget, Sec. 2.1 and Algorithm 1 (initialisation):
 * B = floor(beta * L); reading R4 adds a 1e-9 guard against beta*L landing
 * just below an integer and keeps B >= 1.  k_override > 0 replaces it. */
int32_t orc_budget(int32_t n, double beta, int32_t k_override) {
  if (k_override > 0) return k_override < n ? k_override : n;
  int64_t b = (int64_t)floor(beta * (double)n + 1e-9);
  if (b < 1) b = 1;
  if (b > n) b = n;
  return (int32_t)b;
}

/* ------------------------------------------------- window score (Eq. 2) */

/* A_base for KV head h (Sec. 2.1, Eq. 2, SnapKV-style voting):
 *   A[j] = (1/G) * sum_{g in group h} sum_{r < w} softmax_j(q_{r,g} . k_{j,h} / sqrt(d)).
 * Each softmax row is materialised in full over all n cached keys (no mask,
 * nothing force-kept). */
void orc_abase(const double* q, const double* k, int32_t n, int32_t w, int32_t hq,
               int32_t hkv, int32_t d, int32_t h, double* a_out) {
  int32_t G = hq / hkv;
  double inv_sqrt_d = 1.0 / sqrt((double)d);
  double* logit = (double*)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
  for (int32_t j = 0; j < n; ++j) a_out[j] = 0.0;
  for (int32_t g = h * G; g < (h + 1) * G; ++g) {
    for (int32_t r = 0; r < w; ++r) {
      const double* qrow = q + ((size_t)r * hq + g) * d;
      double mx = -INFINITY;
      for (int32_t j = 0; j < n; ++j) {
        logit[j] = dot(qrow, key_row(k, hkv, d, j, h), d) * inv_sqrt_d;
        if (logit[j] > mx) mx = logit[j];
      }
      double z = 0.0;
      for (int32_t j = 0; j < n; ++j) z += exp(logit[j] - mx);
      for (int32_t j = 0; j < n; ++j) a_out[j] += exp(logit[j] - mx) / z / (double)G;
    }
  }
  free(logit);
}

/* The inner sum of Eq. 2 for the single query head g: partial[j] =
 * sum_{r < w} softmax_j(q_{r,g} . k_{j,h} / sqrt(d)), h = g / G (not yet
 * divided by G).  A_base of KV head h is the mean of these partials over
 * the G query heads of its group (reading R1); the test drivers run the
 * query heads on separate threads and add the partials afterwards. */
void orc_abase_qhead(const double* q, const double* k, int32_t n, int32_t w, int32_t hq,
                     int32_t hkv, int32_t d, int32_t g, double* partial) {
  int32_t G = hq / hkv, h = g / G;
  double inv_sqrt_d = 1.0 / sqrt((double)d);
  double* logit = (double*)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
  for (int32_t j = 0; j < n; ++j) partial[j] = 0.0;
  for (int32_t r = 0; r < w; ++r) {
    const double* qrow = q + ((size_t)r * hq + g) * d;
    double mx = -INFINITY;
    for (int32_t j = 0; j < n; ++j) {
      logit[j] = dot(qrow, key_row(k, hkv, d, j, h), d) * inv_sqrt_d;
      if (logit[j] > mx) mx = logit[j];
    }
    double z = 0.0;
    for (int32_t j = 0; j < n; ++j) z += exp(logit[j] - mx);
    for (int32_t j = 0; j < n; ++j) partial[j] += exp(logit[j] - mx) / z;
  }
  free(logit);
}

/* Prompt-wide base scores (appendix "Sensitivity to the Base Attention
 * Scoring Function": the Mean Attention base and the full-attention
 * "snapshot" base), partial sum of the single query head g.  The last n_q
 * cached positions are the prompt's query rows: row r sits at position
 * p_r = n - n_q + r and, as in the model's causal prefill, attends to the
 * keys j <= p_r only (reading R18):
 *   partial[j] = sum_{r : p_r >= j} softmax_{j' <= p_r}(q_{r,g} . k_{j',h} / sqrt(d))_j,
 * h = g / G.  The full-attention base of KV head h is the mean of these
 * partials over its G query heads; the Mean Attention base divides that by
 * the number of prompt rows that attend to j (reading R19). */
void orc_prompt_qhead(const double* q, const double* k, int32_t n, int32_t n_q, int32_t hq,
                      int32_t hkv, int32_t d, int32_t g, double* partial) {
  int32_t G = hq / hkv, h = g / G;
  double inv_sqrt_d = 1.0 / sqrt((double)d);
  double* logit = (double*)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
  for (int32_t j = 0; j < n; ++j) partial[j] = 0.0;
  for (int32_t r = 0; r < n_q; ++r) {
    const int32_t pos = n - n_q + r;  /* keys 0..pos are visible */
    const double* qrow = q + ((size_t)r * hq + g) * d;
    double mx = -INFINITY;
    for (int32_t j = 0; j <= pos; ++j) {
      logit[j] = dot(qrow, key_row(k, hkv, d, j, h), d) * inv_sqrt_d;
      if (logit[j] > mx) mx = logit[j];
    }
    double z = 0.0;
    for (int32_t j = 0; j <= pos; ++j) z += exp(logit[j] - mx);
    for (int32_t j = 0; j <= pos; ++j) partial[j] += exp(logit[j] - mx) / z;
  }
  free(logit);
}

/* --------------------------------------------- CSS saliency (Eqs. 4-5) */

/* Phi for one visual token at (u, v) of frame f, KV head h (Eqs. 4-5):
 *   H = (1/|N|) sum_{(p,q) in N(u,v)} cos(k_{u,v}, k_{p,q}),  Phi = 1 - H,
 * with N(u,v) the in-grid cells of the (2 radius + 1)^2 neighbourhood other
 * than (u, v) itself: radius 1 is the 3x3 Moore neighbourhood of the method
 * (reading R3), radius 2-4 the 5x5 to 9x9 kernels of the neighbourhood-size
 * ablation. */
double orc_css_phi_token(const double* k, int32_t hkv, int32_t d, int32_t h, int32_t off,
                         int32_t gh, int32_t gw, int32_t u, int32_t v, int32_t radius) {
  const double* c = key_row(k, hkv, d, off + u * gw + v, h);
  double sum = 0.0;
  int32_t cnt = 0;
  for (int32_t du = -radius; du <= radius; ++du) {
    for (int32_t dv = -radius; dv <= radius; ++dv) {
      if (du == 0 && dv == 0) continue;
      int32_t pu = u + du, pv = v + dv;
      if (pu < 0 || pu >= gh || pv < 0 || pv >= gw) continue;
      sum += cosine(c, key_row(k, hkv, d, off + pu * gw + pv, h), d);
      ++cnt;
    }
  }
  if (cnt == 0) return 0.0;
  return 1.0 - sum / (double)cnt;
}

/* Phi over all tokens of KV head h; text tokens get NaN (reading R7). */
void orc_css_phi(const double* k, int32_t n, int32_t hkv, int32_t d, int32_t h,
                 int32_t n_frames, const int32_t* off, const int32_t* gh, const int32_t* gw,
                 int32_t radius, double* phi_out) {
  for (int32_t j = 0; j < n; ++j) phi_out[j] = NAN;
  for (int32_t f = 0; f < n_frames; ++f)
    for (int32_t u = 0; u < gh[f]; ++u)
      for (int32_t v = 0; v < gw[f]; ++v)
        phi_out[off[f] + u * gw[f] + v] =
            orc_css_phi_token(k, hkv, d, h, off[f], gh[f], gw[f], u, v, radius);
}

/* ----------------------------------------------- TSG redundancy (Eq. 6) */

/* rho_i = max over current-frame visual keys k_j of cos(k_i, k_j) (Sec. 3.2). */
/* TSG similarity of two keys.  metric 0: cosine (Eq. 6, the method);
 * 1: dot product; 2: negative squared L2 distance -|a - b|^2 (the two
 * alternatives of the similarity-metric ablation). */
static double tsg_similarity(const double* a, const double* b, int32_t d, int32_t metric) {
  if (metric == 1) return dot(a, b, d);
  if (metric == 2) {
    double s = 0.0;
    for (int32_t e = 0; e < d; ++e) s += (a[e] - b[e]) * (a[e] - b[e]);
    return -s;
  }
  return cosine(a, b, d);
}

double orc_tsg_rho_token(const double* k, int32_t hkv, int32_t d, int32_t h, int32_t i,
                         int32_t cur_off, int32_t cur_len, int32_t metric) {
  double best = -INFINITY;
  const double* ki = key_row(k, hkv, d, i, h);
  for (int32_t j = cur_off; j < cur_off + cur_len; ++j) {
    double c = tsg_similarity(ki, key_row(k, hkv, d, j, h), d, metric);
    if (c > best) best = c;
  }
  return best;
}

/* rho of the listed tokens (each a member of the historical pool) against
 * the current frame [cur_off, cur_off + cur_len): the per-token step of
 * Algorithm 1's ComputeScores, for test drivers that spread the pool over
 * threads. */
void orc_tsg_rho_tokens(const double* k, int32_t hkv, int32_t d, int32_t h, const int32_t* tok,
                        int32_t count, int32_t cur_off, int32_t cur_len, int32_t metric, double* out) {
  for (int32_t t = 0; t < count; ++t)
    out[t] = orc_tsg_rho_token(k, hkv, d, h, tok[t], cur_off, cur_len, metric);
}

/* rho for every token of the historical pool T_pool (visual tokens of frames
 * 0..F-2, Algorithm 1 ComputeScores); NaN for every other token (R7). */
void orc_tsg_rho(const double* k, int32_t n, int32_t hkv, int32_t d, int32_t h,
                 int32_t n_frames, const int32_t* off, const int32_t* gh, const int32_t* gw,
                 int32_t metric, double* rho_out) {
  for (int32_t j = 0; j < n; ++j) rho_out[j] = NAN;
  if (n_frames < 2) return;
  int32_t cf = n_frames - 1;
  int32_t cur_off = off[cf], cur_len = gh[cf] * gw[cf];
  for (int32_t f = 0; f < cf; ++f)
    for (int32_t i = off[f]; i < off[f] + gh[f] * gw[f]; ++i)
      rho_out[i] = orc_tsg_rho_token(k, hkv, d, h, i, cur_off, cur_len, metric);
}

/* ---------------------------------------- TSG threshold and gate (7-8) */

static int cmp_double_asc(const void* a, const void* b) {
  double x = *(const double*)a, y = *(const double*)b;
  return (x > y) - (x < y);
}

/* Threshold (Eq. 7): sort the pool's rho ascending and take the
 * min(B, |T_pool|)-th smallest (1-indexed).  Gate (Eq. 8): M_i = [rho_i <= tau]
 * for historical visual tokens; the current frame is exempt (M = 1, Sec. 3.3);
 * text tokens carry M = 1 (they are never gated).  With an empty pool or TSG
 * disabled every M is 1 and tau is reported as NaN.  Returns |T_pool|. */
/* tau and the gate (Eqs. 7-8).  fixed_gate != 0 replaces the adaptive tau by
 * the constant fixed_tau (the fixed-threshold control of the necessity
 * study: every pool token with similarity above it is gated). */
int32_t orc_tsg_gate(const double* rho, int32_t n, int32_t n_frames, const int32_t* off,
                     const int32_t* gh, const int32_t* gw, int32_t budget, int32_t tsg_enable,
                     int32_t fixed_gate, double fixed_tau, double* tau_out, uint8_t* gate_out) {
  for (int32_t j = 0; j < n; ++j) gate_out[j] = 1;
  *tau_out = NAN;
  int32_t pool = 0;
  for (int32_t f = 0; f + 1 < n_frames; ++f) pool += gh[f] * gw[f];
  if (!tsg_enable || pool == 0) return pool;
  if (fixed_gate) {
    *tau_out = fixed_tau;
    for (int32_t f = 0; f + 1 < n_frames; ++f)
      for (int32_t i = off[f]; i < off[f] + gh[f] * gw[f]; ++i) gate_out[i] = rho[i] <= fixed_tau;
    return pool;
  }
  double* sorted = (double*)malloc(sizeof(double) * (size_t)pool);
  int32_t t = 0;
  for (int32_t f = 0; f + 1 < n_frames; ++f)
    for (int32_t i = off[f]; i < off[f] + gh[f] * gw[f]; ++i) sorted[t++] = rho[i];
  qsort(sorted, (size_t)pool, sizeof(double), cmp_double_asc);
  int32_t m = budget < pool ? budget : pool;
  double tau = sorted[m - 1];
  free(sorted);
  *tau_out = tau;
  for (int32_t f = 0; f + 1 < n_frames; ++f)
    for (int32_t i = off[f]; i < off[f] + gh[f] * gw[f]; ++i) gate_out[i] = rho[i] <= tau;
  return pool;
}

/* ------------------------------------------- integrated score (Eq. 9) */

/* S = A_base for text; S = M * (A_base + alpha * Phi) for visual tokens.
 * css_enable = 0 means alpha = 0 (Phi does not enter). */
void orc_combine(const double* a, const double* phi, const uint8_t* gate, int32_t n,
                 int32_t n_frames, const int32_t* off, const int32_t* gh, const int32_t* gw,
                 double alpha, int32_t css_enable, double* s_out) {
  double al = css_enable ? alpha : 0.0;
  for (int32_t j = 0; j < n; ++j) {
    if (frame_of(j, n_frames, off, gh, gw) < 0) {
      s_out[j] = a[j];
    } else {
      s_out[j] = (double)gate[j] * (a[j] + al * phi[j]);
    }
  }
}

/* ------------------------------------------------------- top-B (Sec 3.3) */

typedef struct {
  double s;
  int32_t i;
} scored_token;

static int cmp_rank(const void* a, const void* b) {
  const scored_token* x = (const scored_token*)a;
  const scored_token* y = (const scored_token*)b;
  if (x->s > y->s) return -1;
  if (x->s < y->s) return 1;
  return (x->i > y->i) - (x->i < y->i); /* reading R5: lower index first among equal S */
}
static int cmp_int_asc(const void* a, const void* b) {
  int32_t x = *(const int32_t*)a, y = *(const int32_t*)b;
  return (x > y) - (x < y);
}

/* I_keep = Top_B(S): rank every token by (S descending, index ascending),
 * keep the first B and return them in ascending index order. */
void orc_topk(const double* s, int32_t n, int32_t budget, int32_t* idx_out) {
  scored_token* order = (scored_token*)malloc(sizeof(scored_token) * (size_t)(n > 0 ? n : 1));
  for (int32_t j = 0; j < n; ++j) {
    order[j].s = s[j];
    order[j].i = j;
  }
  qsort(order, (size_t)n, sizeof(scored_token), cmp_rank);
  int32_t b = budget < n ? budget : n;
  for (int32_t r = 0; r < b; ++r) idx_out[r] = order[r].i;
  qsort(idx_out, (size_t)b, sizeof(int32_t), cmp_int_asc);
  free(order);
}

/* ------------------------------------------------------------- gather */

/* K'[r, h, :] = K[idx[r], h, :] and the same for V, copied byte for byte
 * (Algorithm 1, return statement).  elem_bytes is 2 (bf16) or 4 (fp32). */
void orc_gather(const uint8_t* k, const uint8_t* v, int32_t hkv, int32_t d, int32_t elem_bytes,
                int32_t h, const int32_t* idx, int32_t budget, uint8_t* k_out, uint8_t* v_out) {
  size_t row = (size_t)d * (size_t)elem_bytes;
  for (int32_t r = 0; r < budget; ++r) {
    size_t src = ((size_t)idx[r] * hkv + h) * row;
    size_t dst = ((size_t)r * hkv + h) * row;
    memcpy(k_out + dst, k + src, row);
    memcpy(v_out + dst, v + src, row);
  }
}

/* ------------------------------------------------ Algorithm 1, one head */

/* The whole procedure for KV head h.  Scratch outputs (a, phi, rho, gate, s;
 * each [n]) and tau are returned for inspection; idx_out receives the B kept
 * token indices in ascending order. */
void orc_compress_head(const double* q, const double* k, int32_t n, int32_t w, int32_t hq,
                       int32_t hkv, int32_t d, int32_t h, int32_t n_frames, const int32_t* off,
                       const int32_t* gh, const int32_t* gw, int32_t budget, double alpha,
                       int32_t tsg_enable, int32_t css_enable, double* a, double* phi,
                       double* rho, uint8_t* gate, double* s, double* tau, int32_t* idx_out) {
  orc_abase(q, k, n, w, hq, hkv, d, h, a);
  orc_css_phi(k, n, hkv, d, h, n_frames, off, gh, gw, 1, phi);
  if (tsg_enable)
    orc_tsg_rho(k, n, hkv, d, h, n_frames, off, gh, gw, 0, rho);
  else
    for (int32_t j = 0; j < n; ++j) rho[j] = NAN;
  orc_tsg_gate(rho, n, n_frames, off, gh, gw, budget, tsg_enable, 0, 0.0, tau, gate);
  orc_combine(a, phi, gate, n, n_frames, off, gh, gw, alpha, css_enable, s);
  orc_topk(s, n, budget, idx_out);
}

/* ------------------------------------ consumer: decode over the cache */

/* Scaled dot-product attention of one query row over a KV cache, the
 * operation a decoder runs at every generated token (the consumer of the
 * compressed cache: the efficiency study's decode latency compares the full
 * and the compressed cache).  For query head g of window row r:
 *   out = sum_j softmax_j(q_{r,g} . k_{j,h} / sqrt(d)) v_{j,h},  h = g / G,
 * over all n cached tokens, with the softmax materialised in full. */
void orc_decode_row(const double* q, const double* k, const double* v, int32_t n, int32_t hq,
                    int32_t hkv, int32_t d, int32_t r, int32_t g, double* out) {
  const int32_t G = hq / hkv, h = g / G;
  const double* qrow = q + ((size_t)r * hq + g) * d;
  double* logit = (double*)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
  double mx = -INFINITY;
  for (int32_t j = 0; j < n; ++j) {
    logit[j] = dot(qrow, key_row(k, hkv, d, j, h), d) / sqrt((double)d);
    if (logit[j] > mx) mx = logit[j];
  }
  double z = 0.0;
  for (int32_t j = 0; j < n; ++j) z += exp(logit[j] - mx);
  for (int32_t e = 0; e < d; ++e) out[e] = 0.0;
  for (int32_t j = 0; j < n; ++j) {
    const double p = exp(logit[j] - mx) / z;
    const double* vrow = key_row(v, hkv, d, j, h);
    for (int32_t e = 0; e < d; ++e) out[e] += p * vrow[e];
  }
  free(logit);
}
