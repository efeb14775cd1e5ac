/*
 * kvr_oracle.c -- plain, slow CPU oracle for budgeted KV-cache repair.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product library links, loads or
 * calls this file; only the test suite, the smoke check and the benchmark's
 * CPU-baseline leg do.  It shares no code, header or table with the CUDA path.
 *
 * What it computes (paper: "Contiguity, Not Importance: Budgeted Repair of
 * Stale KV Caches After Document Edits", Sec. 3):
 *   - the repair operator R(K(C), C', P) of Sec. 3 "The repair interface":
 *     positions P are recomputed from the edited context C' one layer at a time,
 *     every other cache entry is left as it is;
 *   - full prefill K(C') as the special case P = {0..n-1} on an empty cache
 *     (the endpoint identity, Eq. 1);
 *   - the two selector forwards of Table 1 that need a model pass
 *     (stale-query Attention and CacheBlend-style KV deviation);
 *   - the fresh-query logits of Sec. 3 (a query computed anew, kept out of
 *     the cache).
 * The model is a textbook Llama-style decoder (RMSNorm, rotate-half RoPE at
 * the original position ids, grouped-query causal attention, SwiGLU MLP),
 * which is what the paper's three model families are.
 *
 * Arithmetic: IEEE double everywhere.  Weights arrive as fp32 or as bf16 bit
 * patterns and are widened exactly.  Cache entries are stored in the cache's
 * dtype (fp32 or bf16, round-to-nearest-even) because the cache is a stored
 * data structure of that dtype; everything else stays in double -- except, on
 * the bf16 path (orc_config.operands), the operands of the matrix products,
 * which that path holds in bf16: they are rounded where they enter a product
 * and every sum stays in double.  Build with
 * -ffp-contract=off so that a*b+c is never fused: each output element is one
 * sequential sum in a fixed order, independent of which other rows are in the
 * batch and of the thread count.  That is what makes the bit-exact invariants
 * (endpoint identity, no-op edit, token-major == layer-major) hold here.
 *
 * Loops are written in the order the definitions read.  OpenMP only spreads
 * independent output elements (rows, features, heads) over threads.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

typedef struct {
  int32_t vocab, d_model, n_layers, n_heads, n_kv_heads, head_dim, ffn;
  int32_t qkv_bias; /* 1: the q/k/v projections carry a bias (Qwen-style) */
  int32_t wdtype;   /* storage of every weight: 0 = fp32, 1 = bf16 bit patterns */
  int32_t cdtype;   /* storage of cache entries: 0 = fp32, 1 = bf16 */
  /* Operands of the matrix products (the bf16 path of Sec. 4 takes them in
   * bf16 and accumulates wider): 0 = kept in double; bit 0 = the rows that
   * enter a weight product (normalised rows into the QKV and gate/up
   * projections and the lm_head, the attention output into O, the SwiGLU
   * activation into down) are rounded to bf16; bit 1 = so are the two
   * attention products' operands: the post-RoPE query, and the weights of V,
   * 2^(x_j - E) with x_j = log2(e) s_j the scores in base 2 and E an integer
   * at or above their maximum (any integer gives the same bf16 mantissas;
   * O = sum_j bf16(2^(x_j - E)) v_j / sum_j 2^(x_j - E)).  Accumulation and
   * everything else stay in double -- unless bit 2 is set: then every weight
   * product's result and the residual stream are rounded to fp32 as well (the
   * bf16 path with fp32 sums; a null control, which measures how far a last-
   * bit change of the sums carries through the layers). */
  int32_t operands;
  double rope_theta, rms_eps;
} orc_config;

/* All matrices are row-major [out_features][in_features]; vectors are [n]. */
typedef struct {
  const void *embed;      /* [vocab][d_model] */
  const void *final_norm; /* [d_model] */
  const void *lm_head;    /* [vocab][d_model] */
  const void *const *attn_norm, *const *wq, *const *wk, *const *wv, *const *wo;
  const void *const *bq, *const *bk, *const *bv; /* NULL entries when qkv_bias == 0 */
  const void *const *mlp_norm, *const *wg, *const *wu, *const *wd;
} orc_weights;

enum { ORC_OK = 0, ORC_EINVAL = 1, ORC_ENOMEM = 2 };

static const double LOG2E = 1.44269504088896340736; /* log2(e) */

/* ---------------------------------------------------------------- helpers */

static double wval(const void *p, size_t i, int bf16) {
  if (bf16) {
    uint32_t bits = (uint32_t)((const uint16_t *)p)[i] << 16;
    float f;
    memcpy(&f, &bits, 4);
    return (double)f;
  }
  return (double)((const float *)p)[i];
}

/* Round a double to the cache dtype: first to fp32 (round to nearest even),
 * then, for bf16, to the nearest bf16 (ties to even).  Returned as the fp32
 * value that holds it exactly. */
static float to_cache(double x, int cdtype) {
  float f = (float)x;
  if (cdtype == 1) {
    uint32_t u;
    memcpy(&u, &f, 4);
    u = (u + 0x7FFFu + ((u >> 16) & 1u)) & 0xFFFF0000u;
    memcpy(&f, &u, 4);
  }
  return f;
}

/* An operand of a matrix product as the bf16 path holds it: rounded to bf16
 * (through fp32, as to_cache) when `on`, else unchanged. */
static double operand(double x, int on) { return on ? (double)to_cache(x, 1) : x; }

static void round_operands(double *x, size_t n, int on) {
  if (on)
    for (size_t i = 0; i < n; ++i) x[i] = operand(x[i], 1);
}

/* RMSNorm: y_i = x_i / sqrt(mean(x^2) + eps) * g_i. */
static void rmsnorm(const double *x, const void *g, int gbf16, int d, double eps, double *y) {
  double ss = 0.0;
  for (int i = 0; i < d; ++i) ss += x[i] * x[i];
  double r = 1.0 / sqrt(ss / (double)d + eps);
  for (int i = 0; i < d; ++i) y[i] = x[i] * r * wval(g, (size_t)i, gbf16);
}

/* Set by the entry points from orc_config.operands bit 2: round the results
 * of the weight products and the residual stream to fp32. */
static int g_f32_sums = 0;

static double sum_round(double x) { return g_f32_sums ? (double)(float)x : x; }

/* y[r][o] = sum_k W[o][k] * x[r][k] (+ b[o]) for m rows. */
static void linear_rows(const double *x, int m, int in, const void *W, const void *b, int bf16,
                        int out, double *y) {
#pragma omp parallel for schedule(static)
  for (int o = 0; o < out; ++o) {
    for (int r = 0; r < m; ++r) {
      const double *xr = x + (size_t)r * in;
      double acc = 0.0;
      for (int k = 0; k < in; ++k) acc += wval(W, (size_t)o * in + k, bf16) * xr[k];
      if (b) acc += wval(b, (size_t)o, bf16);
      y[(size_t)r * out + o] = sum_round(acc);
    }
  }
}

/* Rotate-half rotary embedding of one head vector at position pos:
 * pair (i, i + dh/2) is rotated by angle pos * theta^(-2i/dh). */
static void rope(double *x, int dh, int64_t pos, double theta) {
  int half = dh / 2;
  for (int i = 0; i < half; ++i) {
    double inv_freq = pow(theta, -2.0 * (double)i / (double)dh);
    double ang = (double)pos * inv_freq;
    double c = cos(ang), s = sin(ang);
    double x1 = x[i], x2 = x[i + half];
    x[i] = x1 * c - x2 * s;
    x[i + half] = x2 * c + x1 * s;
  }
}

static double silu(double x) { return x / (1.0 + exp(-x)); }

static size_t cache_index(const orc_config *c, int cap, int l, int64_t pos, int g) {
  return (((size_t)l * cap + (size_t)pos) * c->n_kv_heads + g) * c->head_dim;
}

/* ------------------------------------------------------------ layer stages */

/* Stage 1 of layer l for m rows: a = RMSNorm(h); q, k, v = a W (+ b);
 * RoPE on q and k at each row's original position. */
static void stage_qkv(const orc_config *c, const orc_weights *w, int l, const double *h, int m,
                      const int64_t *pos, double *q, double *k, double *v, double *scratch) {
  int d = c->d_model, dh = c->head_dim, H = c->n_heads, G = c->n_kv_heads, bf = c->wdtype;
  for (int r = 0; r < m; ++r)
    rmsnorm(h + (size_t)r * d, w->attn_norm[l], bf, d, c->rms_eps, scratch + (size_t)r * d);
  round_operands(scratch, (size_t)m * d, c->operands & 1);
  linear_rows(scratch, m, d, w->wq[l], c->qkv_bias ? w->bq[l] : NULL, bf, H * dh, q);
  linear_rows(scratch, m, d, w->wk[l], c->qkv_bias ? w->bk[l] : NULL, bf, G * dh, k);
  linear_rows(scratch, m, d, w->wv[l], c->qkv_bias ? w->bv[l] : NULL, bf, G * dh, v);
  for (int r = 0; r < m; ++r) {
    for (int hh = 0; hh < H; ++hh) rope(q + ((size_t)r * H + hh) * dh, dh, pos[r], c->rope_theta);
    for (int g = 0; g < G; ++g) rope(k + ((size_t)r * G + g) * dh, dh, pos[r], c->rope_theta);
  }
}

/* Write the rows' fresh k, v into the cache of layer l at their positions. */
static void stage_write_kv(const orc_config *c, int l, float *kc, float *vc, int cap, const double *k,
                           const double *v, int m, const int64_t *pos) {
  int G = c->n_kv_heads, dh = c->head_dim;
  for (int r = 0; r < m; ++r)
    for (int g = 0; g < G; ++g)
      for (int i = 0; i < dh; ++i) {
        size_t ci = cache_index(c, cap, l, pos[r], g) + i;
        size_t si = ((size_t)r * G + g) * dh + i;
        kc[ci] = to_cache(k[si], c->cdtype);
        vc[ci] = to_cache(v[si], c->cdtype);
      }
}

/* Causal grouped-query attention of one row at position p over the cache of
 * layer l: head hh reads kv head hh / (H / G); keys j = 0..p. */
static void attend_row(const orc_config *c, int l, const float *kc, const float *vc, int cap,
                       const double *q, int64_t p, double *o, double *sbuf) {
  int H = c->n_heads, G = c->n_kv_heads, dh = c->head_dim, grp = H / G;
  const int rnd = c->operands & 2;
  double scale = 1.0 / sqrt((double)dh);
  for (int hh = 0; hh < H; ++hh) {
    int g = hh / grp;
    const double *qh = q + (size_t)hh * dh;
    double mx = -INFINITY;
    for (int64_t j = 0; j <= p; ++j) {
      const float *kj = kc + cache_index(c, cap, l, j, g);
      double s = 0.0;
      for (int i = 0; i < dh; ++i) s += operand(qh[i], rnd) * (double)kj[i];
      sbuf[j] = s * scale;
      if (sbuf[j] > mx) mx = sbuf[j];
    }
    double z = 0.0;
    if (rnd) {
      /* base-2 scores against the integer E = ceil(max): the weights of V
       * are rounded, their sum is not */
      const double E = ceil(mx * LOG2E);
      for (int64_t j = 0; j <= p; ++j) {
        sbuf[j] = exp2(sbuf[j] * LOG2E - E);
        z += sbuf[j];
        sbuf[j] = operand(sbuf[j], 1);
      }
    } else {
      for (int64_t j = 0; j <= p; ++j) {
        sbuf[j] = exp(sbuf[j] - mx);
        z += sbuf[j];
      }
    }
    double *oh = o + (size_t)hh * dh;
    for (int i = 0; i < dh; ++i) {
      double acc = 0.0;
      for (int64_t j = 0; j <= p; ++j) acc += sbuf[j] * (double)vc[cache_index(c, cap, l, j, g) + i];
      oh[i] = acc / z;
    }
  }
}

/* Stage 2 of layer l: attention for all m rows, then h += o Wo, then
 * h += Wd (silu(Wg b) * (Wu b)) with b = RMSNorm(h). */
static int stage_attn_mlp(const orc_config *c, const orc_weights *w, int l, const float *kc,
                          const float *vc, int cap, double *h, int m, const int64_t *pos,
                          const double *q) {
  int d = c->d_model, H = c->n_heads, dh = c->head_dim, F = c->ffn, bf = c->wdtype;
  int64_t pmax = 0;
  for (int r = 0; r < m; ++r)
    if (pos[r] > pmax) pmax = pos[r];
  double *o = malloc(sizeof(double) * (size_t)m * H * dh);
  double *t = malloc(sizeof(double) * (size_t)m * d);
  if (!o || !t) {
    free(o);
    free(t);
    return ORC_ENOMEM;
  }
  int fail = 0;
#pragma omp parallel
  {
    double *sbuf = malloc(sizeof(double) * (size_t)(pmax + 1));
    if (!sbuf) {
#pragma omp atomic write
      fail = 1;
    } else {
#pragma omp for schedule(dynamic, 1)
      for (int r = 0; r < m; ++r)
        attend_row(c, l, kc, vc, cap, q + (size_t)r * H * dh, pos[r], o + (size_t)r * H * dh, sbuf);
    }
    free(sbuf);
  }
  if (fail) {
    free(o);
    free(t);
    return ORC_ENOMEM;
  }
  /* h += o Wo */
  round_operands(o, (size_t)m * H * dh, c->operands & 1);
  linear_rows(o, m, H * dh, w->wo[l], NULL, bf, d, t);
  for (size_t i = 0; i < (size_t)m * d; ++i) h[i] = sum_round(h[i] + t[i]);
  /* h += Wd (silu(Wg b) * (Wu b)) */
  double *bb = malloc(sizeof(double) * (size_t)m * d);
  double *gg = malloc(sizeof(double) * (size_t)m * F);
  double *uu = malloc(sizeof(double) * (size_t)m * F);
  if (!bb || !gg || !uu) {
    free(bb);
    free(gg);
    free(uu);
    free(o);
    free(t);
    return ORC_ENOMEM;
  }
  for (int r = 0; r < m; ++r)
    rmsnorm(h + (size_t)r * d, w->mlp_norm[l], bf, d, c->rms_eps, bb + (size_t)r * d);
  round_operands(bb, (size_t)m * d, c->operands & 1);
  linear_rows(bb, m, d, w->wg[l], NULL, bf, F, gg);
  linear_rows(bb, m, d, w->wu[l], NULL, bf, F, uu);
  for (size_t i = 0; i < (size_t)m * F; ++i) gg[i] = silu(gg[i]) * uu[i];
  round_operands(gg, (size_t)m * F, c->operands & 1);
  linear_rows(gg, m, F, w->wd[l], NULL, bf, d, t);
  for (size_t i = 0; i < (size_t)m * d; ++i) h[i] = sum_round(h[i] + t[i]);
  free(bb);
  free(gg);
  free(uu);
  free(o);
  free(t);
  return ORC_OK;
}

static void embed_rows(const orc_config *c, const orc_weights *w, const int32_t *tokens,
                       const int64_t *pos, int m, double *h) {
  int d = c->d_model;
  for (int r = 0; r < m; ++r) {
    size_t base = (size_t)tokens[pos[r]] * d;
    for (int i = 0; i < d; ++i) h[(size_t)r * d + i] = wval(w->embed, base + i, c->wdtype);
  }
}

static int check_rows(const orc_config *c, int cap, const int32_t *tokens, const int64_t *pos, int m) {
  for (int r = 0; r < m; ++r) {
    if (pos[r] < 0 || pos[r] >= cap) return ORC_EINVAL;
    if (r > 0 && pos[r] <= pos[r - 1]) return ORC_EINVAL;
    if (tokens[pos[r]] < 0 || tokens[pos[r]] >= c->vocab) return ORC_EINVAL;
  }
  if (c->n_heads % c->n_kv_heads != 0 || c->head_dim % 2 != 0) return ORC_EINVAL;
  return ORC_OK;
}

/* ------------------------------------------------------------- entry points */

int orc_set_threads(int n) {
#ifdef _OPENMP
  if (n > 0) omp_set_num_threads(n);
  return omp_get_max_threads();
#else
  (void)n;
  return 1;
#endif
}

/* The repair operator R of Sec. 3, layer-major: the rows at positions pos[0..m)
 * (strictly increasing) are recomputed from tokens (the edited context C')
 * through every layer.  At each layer all m rows' fresh k, v are written into
 * the cache before any of them attends, which is what Eq. 1 needs (with P
 * the full range the result must be the prefill of C').  Cache layout:
 * kc, vc = [n_layers][cap][n_kv_heads][head_dim].  If h_out is not NULL it
 * receives the rows' final residual stream [m][d_model]. */
int orc_recompute(const orc_config *c, const orc_weights *w, float *kc, float *vc, int cap,
                  const int32_t *tokens, const int64_t *pos, int m, double *h_out) {
  g_f32_sums = (c->operands & 4) != 0;
  if (m <= 0) return ORC_OK;
  int rc = check_rows(c, cap, tokens, pos, m);
  if (rc) return rc;
  int d = c->d_model, H = c->n_heads, G = c->n_kv_heads, dh = c->head_dim;
  double *h = malloc(sizeof(double) * (size_t)m * d);
  double *q = malloc(sizeof(double) * (size_t)m * H * dh);
  double *k = malloc(sizeof(double) * (size_t)m * G * dh);
  double *v = malloc(sizeof(double) * (size_t)m * G * dh);
  double *s = malloc(sizeof(double) * (size_t)m * d);
  if (!h || !q || !k || !v || !s) {
    rc = ORC_ENOMEM;
    goto done;
  }
  embed_rows(c, w, tokens, pos, m, h);
  for (int l = 0; l < c->n_layers && !rc; ++l) {
    stage_qkv(c, w, l, h, m, pos, q, k, v, s);
    stage_write_kv(c, l, kc, vc, cap, k, v, m, pos);
    rc = stage_attn_mlp(c, w, l, kc, vc, cap, h, m, pos, q);
  }
  if (!rc && h_out) memcpy(h_out, h, sizeof(double) * (size_t)m * d);
done:
  free(h);
  free(q);
  free(k);
  free(v);
  free(s);
  return rc;
}

/* Brute-force token-major recompute: one position at a time, in ascending
 * order, through all layers (decode order).  Valid because of causality:
 * position p only reads cache entries j <= p, and every j < p in the set has
 * already been refreshed in every layer. */
int orc_recompute_token_major(const orc_config *c, const orc_weights *w, float *kc, float *vc,
                              int cap, const int32_t *tokens, const int64_t *pos, int m,
                              double *h_out) {
  int rc = check_rows(c, cap, tokens, pos, m);
  for (int r = 0; r < m && !rc; ++r)
    rc = orc_recompute(c, w, kc, vc, cap, tokens, pos + r, 1,
                       h_out ? h_out + (size_t)r * c->d_model : NULL);
  return rc;
}

/* Stale-query Attention selector score (Table 1: positions ranked by the
 * attention a query pays them in the stale cache), with the edit-span rows as
 * the queries.
 * The span rows [s_start, s_end) are run through every layer exactly as in
 * repair (their fresh k, v are written into kc/vc, which the caller passes
 * as a copy).  At layer l, for each span row and query head, logits to the
 * stale keys of the pool D = [s_end, n) are softmaxed over D alone, and
 * score[j] accumulates the probability, summed over rows, heads and layers.
 * score has n entries; entries outside D are set to 0. */
int orc_score_attention(const orc_config *c, const orc_weights *w, float *kc, float *vc, int cap,
                        int n, const int32_t *tokens, int s_start, int s_end, double *score) {
  g_f32_sums = (c->operands & 4) != 0;
  int m = s_end - s_start;
  if (m <= 0 || s_start < 0 || s_end > n || n > cap) return ORC_EINVAL;
  int d = c->d_model, H = c->n_heads, G = c->n_kv_heads, dh = c->head_dim, grp = H / G;
  int64_t *pos = malloc(sizeof(int64_t) * (size_t)m);
  double *h = malloc(sizeof(double) * (size_t)m * d);
  double *q = malloc(sizeof(double) * (size_t)m * H * dh);
  double *k = malloc(sizeof(double) * (size_t)m * G * dh);
  double *v = malloc(sizeof(double) * (size_t)m * G * dh);
  double *s = malloc(sizeof(double) * (size_t)m * d);
  double *lg = malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
  int rc = ORC_OK;
  if (!pos || !h || !q || !k || !v || !s || !lg) {
    rc = ORC_ENOMEM;
    goto done;
  }
  for (int r = 0; r < m; ++r) pos[r] = s_start + r;
  rc = check_rows(c, cap, tokens, pos, m);
  if (rc) goto done;
  for (int j = 0; j < n; ++j) score[j] = 0.0;
  double scale = 1.0 / sqrt((double)dh);
  embed_rows(c, w, tokens, pos, m, h);
  for (int l = 0; l < c->n_layers && !rc; ++l) {
    stage_qkv(c, w, l, h, m, pos, q, k, v, s);
    stage_write_kv(c, l, kc, vc, cap, k, v, m, pos);
    for (int r = 0; r < m; ++r)
      for (int hh = 0; hh < H; ++hh) {
        int g = hh / grp;
        const double *qh = q + ((size_t)r * H + hh) * dh;
        double mx = -INFINITY, z = 0.0;
#pragma omp parallel for schedule(static)
        for (int j = s_end; j < n; ++j) {
          const float *kj = kc + cache_index(c, cap, l, j, g);
          double a = 0.0;
          for (int i = 0; i < dh; ++i) a += qh[i] * (double)kj[i];
          lg[j] = a * scale;
        }
        for (int j = s_end; j < n; ++j)
          if (lg[j] > mx) mx = lg[j];
        for (int j = s_end; j < n; ++j) {
          lg[j] = exp(lg[j] - mx);
          z += lg[j];
        }
        for (int j = s_end; j < n; ++j) score[j] += lg[j] / z;
      }
    rc = stage_attn_mlp(c, w, l, kc, vc, cap, h, m, pos, q);
  }
done:
  free(pos);
  free(h);
  free(q);
  free(k);
  free(v);
  free(s);
  free(lg);
  return rc;
}

/* CacheBlend-style KV-deviation score (Table 1, "top-K by key/value
 * deviation" at the second layer, index 1).  On the caller's copy of the
 * cache: refresh the span's layer-0 k, v; recompute layer 0 for every pool
 * row j in D = [s_end, n); project the result to layer 1's k (with RoPE at j)
 * and v, rounded to the cache dtype as a repaired entry would be stored; and
 * score[j] = ||k1_fresh - k1_stale||_2 + ||v1_fresh - v1_stale||_2, each norm
 * over all kv heads and dims.  Entries outside D are 0.  Needs >= 2 layers. */
int orc_score_cacheblend(const orc_config *c, const orc_weights *w, float *kc, float *vc, int cap,
                         int n, const int32_t *tokens, int s_start, int s_end, double *score) {
  g_f32_sums = (c->operands & 4) != 0;
  int ms = s_end - s_start, md = n - s_end;
  if (ms <= 0 || s_start < 0 || s_end > n || n > cap || c->n_layers < 2) return ORC_EINVAL;
  int d = c->d_model, H = c->n_heads, G = c->n_kv_heads, dh = c->head_dim;
  int mm = ms > md ? ms : md;
  if (mm <= 0) mm = 1;
  int64_t *pos = malloc(sizeof(int64_t) * (size_t)mm);
  double *h = malloc(sizeof(double) * (size_t)mm * d);
  double *q = malloc(sizeof(double) * (size_t)mm * H * dh);
  double *k = malloc(sizeof(double) * (size_t)mm * G * dh);
  double *v = malloc(sizeof(double) * (size_t)mm * G * dh);
  double *s = malloc(sizeof(double) * (size_t)mm * d);
  int rc = ORC_OK;
  if (!pos || !h || !q || !k || !v || !s) {
    rc = ORC_ENOMEM;
    goto done;
  }
  for (int j = 0; j < n; ++j) score[j] = 0.0;
  /* refresh the span's layer-0 k, v */
  for (int r = 0; r < ms; ++r) pos[r] = s_start + r;
  rc = check_rows(c, cap, tokens, pos, ms);
  if (rc) goto done;
  embed_rows(c, w, tokens, pos, ms, h);
  stage_qkv(c, w, 0, h, ms, pos, q, k, v, s);
  stage_write_kv(c, 0, kc, vc, cap, k, v, ms, pos);
  if (md <= 0) goto done;
  /* layer 0 for every pool row */
  for (int r = 0; r < md; ++r) pos[r] = s_end + r;
  rc = check_rows(c, cap, tokens, pos, md);
  if (rc) goto done;
  embed_rows(c, w, tokens, pos, md, h);
  stage_qkv(c, w, 0, h, md, pos, q, k, v, s);
  stage_write_kv(c, 0, kc, vc, cap, k, v, md, pos);
  rc = stage_attn_mlp(c, w, 0, kc, vc, cap, h, md, pos, q);
  if (rc) goto done;
  /* layer-1 k (post-RoPE) and v of the fresh rows against the stale cache */
  stage_qkv(c, w, 1, h, md, pos, q, k, v, s);
  for (int r = 0; r < md; ++r) {
    double dk = 0.0, dv = 0.0;
    for (int g = 0; g < G; ++g)
      for (int i = 0; i < dh; ++i) {
        size_t ci = cache_index(c, cap, 1, pos[r], g) + i;
        size_t si = ((size_t)r * G + g) * dh + i;
        double ek = (double)to_cache(k[si], c->cdtype) - (double)kc[ci];
        double ev = (double)to_cache(v[si], c->cdtype) - (double)vc[ci];
        dk += ek * ek;
        dv += ev * ev;
      }
    score[pos[r]] = sqrt(dk) + sqrt(dv);
  }
done:
  free(pos);
  free(h);
  free(q);
  free(k);
  free(v);
  free(s);
  return rc;
}

/* Logits of every row of a fresh query: rows n..n+m-1 of `tokens` attend
 * to the caller's copy of the cache (cap >= n+m); logits [m][vocab] =
 * lm_head RMSNorm(h_row).  Used for teacher-forced answer scoring (Eq. 2). */
int orc_logits_all(const orc_config *c, const orc_weights *w, float *kc, float *vc, int cap,
                   int n, const int32_t *tokens, int m, double *logits) {
  g_f32_sums = (c->operands & 4) != 0;
  if (m <= 0 || n < 0 || n + m > cap) return ORC_EINVAL;
  int d = c->d_model;
  int64_t *pos = malloc(sizeof(int64_t) * (size_t)m);
  double *h = malloc(sizeof(double) * (size_t)m * d);
  double *a = malloc(sizeof(double) * (size_t)m * d);
  int rc = ORC_OK;
  if (!pos || !h || !a) {
    rc = ORC_ENOMEM;
    goto done;
  }
  for (int r = 0; r < m; ++r) pos[r] = n + r;
  rc = orc_recompute(c, w, kc, vc, cap, tokens, pos, m, h);
  if (rc) goto done;
  for (int r = 0; r < m; ++r)
    rmsnorm(h + (size_t)r * d, w->final_norm, c->wdtype, d, c->rms_eps, a + (size_t)r * d);
  round_operands(a, (size_t)m * d, c->operands & 1);
  linear_rows(a, m, d, w->lm_head, NULL, c->wdtype, c->vocab, logits);
done:
  free(pos);
  free(h);
  free(a);
  return rc;
}

/* Fresh-query logits (Sec. 3: the query that scores a cache state is
 * computed anew each time and kept out of the cache).  The m query tokens sit at positions n..n+m-1;
 * their k, v go into the caller's copy of the cache (cap >= n+m) and never
 * into the document's entries.  logits[vocab] = lm_head RMSNorm(h_last). */
int orc_logits(const orc_config *c, const orc_weights *w, float *kc, float *vc, int cap, int n,
               const int32_t *tokens /* [n+m], query at n.. */, int m, double *logits) {
  g_f32_sums = (c->operands & 4) != 0;
  if (m <= 0 || n < 0 || n + m > cap) return ORC_EINVAL;
  int d = c->d_model;
  int64_t *pos = malloc(sizeof(int64_t) * (size_t)m);
  double *h = malloc(sizeof(double) * (size_t)m * d);
  double *a = malloc(sizeof(double) * (size_t)d);
  int rc = ORC_OK;
  if (!pos || !h || !a) {
    rc = ORC_ENOMEM;
    goto done;
  }
  for (int r = 0; r < m; ++r) pos[r] = n + r;
  rc = orc_recompute(c, w, kc, vc, cap, tokens, pos, m, h);
  if (rc) goto done;
  rmsnorm(h + (size_t)(m - 1) * d, w->final_norm, c->wdtype, d, c->rms_eps, a);
  round_operands(a, (size_t)d, c->operands & 1);
  linear_rows(a, 1, d, w->lm_head, NULL, c->wdtype, c->vocab, logits);
done:
  free(pos);
  free(h);
  free(a);
  return rc;
}
