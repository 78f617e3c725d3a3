/*
 * pced_oracle.c -- CPU oracle of one PCED decode step.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the
 * benchmark's CPU-baseline leg use this file; the CUDA decoding library
 * shares no code with it.
 *
 * Everything is computed in fp64 straight from the definitions, with no
 * blocking, online softmax, splitting or fusion:
 *   - decode attention: full score vector, max-subtracted softmax, weighted
 *     sum of values (each expert attends over its own cache, Sec. 3
 *     "Parallel Context-of-Experts");
 *   - unembedding + log-softmax: full logit row, log-sum-exp;
 *   - retrieval-aware contrastive score (Eq. 2) and the max over experts and
 *     vocabulary (Eq. 3), by brute-force scan of every (expert, token);
 *   - the chosen token feeds every expert at the next step (shared history,
 *     Sec. 3 after Eq. 3).
 * Threads only split independent outputs (sequence/head pairs, vocabulary
 * rows); each output is computed by one thread in a fixed order, so results
 * do not depend on the thread count.
 */
#include "pced_oracle.h"

#include <math.h>
#include <pthread.h>
#include <stdlib.h>
#include <string.h>

/* ---------------------------------------------------------------- helpers */

double oracle_bf16_value(uint16_t bits) {
  union { uint32_t u; float f; } c;
  c.u = (uint32_t)bits << 16;
  return (double)c.f;
}

uint16_t oracle_round_bf16(double x) {
  /* bf16 keeps 8 significant bits.  frexp gives x = m * 2^e, 0.5 <= |m| < 1;
   * m * 2^8 rounded to an integer (ties to even, the default rounding mode)
   * is the 8-bit significand of the nearest bf16. */
  if (x == 0.0) return signbit(x) ? 0x8000u : 0u;
  int e;
  double m = frexp(x, &e);
  double r = ldexp(nearbyint(ldexp(m, 8)), e - 8);
  union { uint32_t u; float f; } c;
  c.f = (float)r; /* exact: r has at most 8 significant bits */
  return (uint16_t)(c.u >> 16);
}

void oracle_rmsnorm(const double* x, int32_t n, double eps, double* y) {
  double ss = 0.0;
  for (int32_t i = 0; i < n; ++i) ss += x[i] * x[i];
  double inv = 1.0 / sqrt(ss / (double)n + eps);
  for (int32_t i = 0; i < n; ++i) y[i] = x[i] * inv;
}

typedef void (*item_fn)(void* ctx, int64_t item);
typedef struct {
  item_fn fn;
  void* ctx;
  int64_t n;
  int32_t nthreads, tid;
} pf_job;

static void* pf_worker(void* p) {
  pf_job* j = (pf_job*)p;
  for (int64_t i = j->tid; i < j->n; i += j->nthreads) j->fn(j->ctx, i);
  return NULL;
}

static void parallel_for(int64_t n, item_fn fn, void* ctx, int32_t nthreads) {
  if (nthreads < 1) nthreads = 1;
  if (nthreads > 256) nthreads = 256;
  if ((int64_t)nthreads > n) nthreads = (int32_t)(n > 0 ? n : 1);
  if (nthreads == 1) {
    for (int64_t i = 0; i < n; ++i) fn(ctx, i);
    return;
  }
  pthread_t th[256];
  pf_job jobs[256];
  for (int32_t t = 0; t < nthreads; ++t) {
    pf_job j = {fn, ctx, n, nthreads, t};
    jobs[t] = j;
    pthread_create(&th[t], NULL, pf_worker, &jobs[t]);
  }
  for (int32_t t = 0; t < nthreads; ++t) pthread_join(th[t], NULL);
}

/* -------------------------------------------------------- decode attention */

typedef struct {
  const uint16_t *q, *kc, *vc;
  const int64_t* kv_off;
  const int32_t *cap, *len;
  int32_t Hq, Hkv, D;
  double scale;
  double* out;
} attn_ctx;

/* one (sequence, query head): o = sum_j softmax_j(scale * q.k_j) v_j */
static void attn_item(void* p, int64_t item) {
  attn_ctx* c = (attn_ctx*)p;
  int32_t s = (int32_t)(item / c->Hq), hq = (int32_t)(item % c->Hq);
  int32_t G = c->Hq / c->Hkv, h = hq / G, D = c->D, n = c->len[s];
  const uint16_t* q = c->q + ((int64_t)s * c->Hq + hq) * D;
  const uint16_t* K = c->kc + c->kv_off[s] + (int64_t)h * c->cap[s] * D;
  const uint16_t* Vv = c->vc + c->kv_off[s] + (int64_t)h * c->cap[s] * D;
  double* o = c->out + ((int64_t)s * c->Hq + hq) * D;
  double* sc = (double*)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
  double mx = -INFINITY;
  for (int32_t j = 0; j < n; ++j) {
    double dot = 0.0;
    for (int32_t i = 0; i < D; ++i) dot += oracle_bf16_value(q[i]) * oracle_bf16_value(K[(int64_t)j * D + i]);
    sc[j] = c->scale * dot;
    if (sc[j] > mx) mx = sc[j];
  }
  double sum = 0.0;
  for (int32_t j = 0; j < n; ++j) {
    sc[j] = exp(sc[j] - mx);
    sum += sc[j];
  }
  for (int32_t i = 0; i < D; ++i) o[i] = 0.0;
  for (int32_t j = 0; j < n; ++j) {
    double p = sc[j] / sum;
    for (int32_t i = 0; i < D; ++i) o[i] += p * oracle_bf16_value(Vv[(int64_t)j * D + i]);
  }
  free(sc);
}

int32_t oracle_attention(const uint16_t* q, const uint16_t* kc, const uint16_t* vc, const int64_t* kv_off,
                         const int32_t* cap, const int32_t* len, int32_t S, int32_t Hq, int32_t Hkv, int32_t D,
                         double scale, double* out, int32_t nthreads) {
  if (!q || !kc || !vc || !kv_off || !cap || !len || !out || S < 0 || Hq < 1 || Hkv < 1 || D < 1 ||
      Hq % Hkv != 0)
    return -1;
  for (int32_t s = 0; s < S; ++s)
    if (len[s] < 1 || len[s] > cap[s]) return -1;
  attn_ctx c = {q, kc, vc, kv_off, cap, len, Hq, Hkv, D, scale, out};
  parallel_for((int64_t)S * Hq, attn_item, &c, nthreads);
  return 0;
}

/* ------------------------------------------------- unembedding + log-softmax */

typedef struct {
  const uint16_t *h, *w;
  int32_t S, d, V;
  double* lp;
} logit_ctx;

/* one vocabulary row v: z[s][v] = sum_i h[s][i] W[v][i] for all s */
static void logit_item(void* p, int64_t v) {
  logit_ctx* c = (logit_ctx*)p;
  const uint16_t* wr = c->w + v * c->d;
  for (int32_t s = 0; s < c->S; ++s) {
    const uint16_t* hr = c->h + (int64_t)s * c->d;
    double z = 0.0;
    for (int32_t i = 0; i < c->d; ++i) z += oracle_bf16_value(hr[i]) * oracle_bf16_value(wr[i]);
    c->lp[(int64_t)s * c->V + v] = z;
  }
}

int32_t oracle_lm_head_logprobs(const uint16_t* h, const uint16_t* w, int32_t S, int32_t d, int32_t V, double* lp,
                                double* lse, int32_t nthreads) {
  if (!h || !w || !lp || !lse || S < 0 || d < 1 || V < 1) return -1;
  logit_ctx c = {h, w, S, d, V, lp};
  parallel_for(V, logit_item, &c, nthreads);
  for (int32_t s = 0; s < S; ++s) {
    double* z = lp + (int64_t)s * V;
    double mx = -INFINITY, sum = 0.0;
    for (int32_t v = 0; v < V; ++v)
      if (z[v] > mx) mx = z[v];
    for (int32_t v = 0; v < V; ++v) sum += exp(z[v] - mx);
    lse[s] = mx + log(sum);
    for (int32_t v = 0; v < V; ++v) z[v] -= lse[s];
  }
  return 0;
}

/* ------------------------------------------ Eq. 2 + Eq. 3 (brute-force scan) */

static double clip_relevance(float r) {
  const double eps = 1e-8;
  double x = (double)r;
  if (x < eps) x = eps;
  if (x > 1.0 - eps) x = 1.0 - eps;
  return x;
}

int32_t oracle_contrastive_select(const double* lp, const float* beta, const float* r, double gamma, int32_t B,
                                  int32_t N, int32_t V, int32_t* token, int32_t* expert, double* score,
                                  double* token_gap, double* expert_gap) {
  if (!lp || !beta || !r || !token || !expert || !score || B < 1 || N < 1 || V < 1) return -1;
  for (int32_t b = 0; b < B; ++b) {
    const double* lp0 = lp + (int64_t)b * (N + 1) * V; /* amateur row */
    double best = -INFINITY;
    int32_t bv = -1, bk = -1;
    /* scan tokens in increasing id and experts in increasing index; a later
     * candidate replaces the incumbent only when strictly larger, which gives
     * the lowest-token-then-lowest-expert tie rule */
    for (int32_t v = 0; v < V; ++v) {
      for (int32_t k = 1; k <= N; ++k) {
        double bt = (double)beta[(int64_t)b * N + (k - 1)];
        double prior = gamma * log(clip_relevance(r[(int64_t)b * N + (k - 1)]));
        double lpk = lp[((int64_t)b * (N + 1) + k) * V + v];
        double shat = (1.0 + bt) * lpk - bt * lp0[v] + prior;
        if (shat > best) {
          best = shat;
          bv = v;
          bk = k;
        }
      }
    }
    token[b] = bv;
    expert[b] = bk;
    score[b] = best;
    if (token_gap || expert_gap) {
      double runner_tok = -INFINITY, runner_exp = -INFINITY;
      for (int32_t v = 0; v < V; ++v) {
        for (int32_t k = 1; k <= N; ++k) {
          double bt = (double)beta[(int64_t)b * N + (k - 1)];
          double prior = gamma * log(clip_relevance(r[(int64_t)b * N + (k - 1)]));
          double shat = (1.0 + bt) * lp[((int64_t)b * (N + 1) + k) * V + v] - bt * lp0[v] + prior;
          if (v != bv && shat > runner_tok) runner_tok = shat;
          if (v == bv && k != bk && shat > runner_exp) runner_exp = shat;
        }
      }
      if (token_gap) token_gap[b] = best - runner_tok;
      if (expert_gap) expert_gap[b] = best - runner_exp;
    }
  }
  return 0;
}

/* ------------------------------------- dynamic contrast strength (AdaCAD) */

int32_t oracle_aggregate_select(const double* lp, const float* beta, const float* r, int32_t B, int32_t N, int32_t V,
                                int32_t rule, int32_t* token, int32_t* expert, double* score, double* token_gap,
                                double* expert_gap) {
  if (!lp || !beta || !r || !token || !expert || !score || B < 1 || N < 1 || V < 1 || (rule != 1 && rule != 2))
    return -1;
  double* c = (double*)malloc(sizeof(double) * (size_t)N * V); /* c_k(v) - LSE_k = log p_k(v) */
  double* agg = (double*)malloc(sizeof(double) * (size_t)V);
  double* w = (double*)malloc(sizeof(double) * (size_t)N);
  if (!c || !agg || !w) {
    free(c); free(agg); free(w);
    return -1;
  }
  for (int32_t b = 0; b < B; ++b) {
    const double* lp0 = lp + (int64_t)b * (N + 1) * V;
    double wsum = 0.0;
    for (int32_t k = 0; k < N; ++k) {
      w[k] = clip_relevance(r[(int64_t)b * N + k]);
      wsum += w[k];
    }
    for (int32_t k = 0; k < N; ++k) w[k] /= wsum;
    for (int32_t k = 0; k < N; ++k) {
      const double bt = (double)beta[(int64_t)b * N + k];
      const double* lpk = lp + ((int64_t)b * (N + 1) + k + 1) * V;
      double* ck = c + (int64_t)k * V;
      double m = -INFINITY;
      for (int32_t v = 0; v < V; ++v) {
        ck[v] = (1.0 + bt) * lpk[v] - bt * lp0[v];
        if (ck[v] > m) m = ck[v];
      }
      double se = 0.0;
      for (int32_t v = 0; v < V; ++v) se += exp(ck[v] - m);
      const double lse = m + log(se);
      for (int32_t v = 0; v < V; ++v) ck[v] -= lse;
    }
    for (int32_t v = 0; v < V; ++v) {
      double a = 0.0;
      if (rule == 1) {
        for (int32_t k = 0; k < N; ++k) a += w[k] * exp(c[(int64_t)k * V + v]);
        a = log(a);
      } else {
        for (int32_t k = 0; k < N; ++k) a += w[k] * c[(int64_t)k * V + v];
      }
      agg[v] = a;
    }
    int32_t bv = 0;
    for (int32_t v = 1; v < V; ++v)
      if (agg[v] > agg[bv]) bv = v;
    double runner = -INFINITY;
    for (int32_t v = 0; v < V; ++v)
      if (v != bv && agg[v] > runner) runner = agg[v];
    int32_t bk = 0;
    for (int32_t k = 1; k < N; ++k)
      if (w[k] * exp(c[(int64_t)k * V + bv]) > w[bk] * exp(c[(int64_t)bk * V + bv])) bk = k;
    token[b] = bv;
    expert[b] = bk + 1;
    score[b] = agg[bv];
    if (token_gap) token_gap[b] = agg[bv] - runner;
    if (expert_gap) {
      /* the attribution's margin in log units: log(w p) of the chosen
       * expert at the token against the best other expert's */
      double other = -INFINITY;
      for (int32_t k = 0; k < N; ++k) {
        const double lk = log(w[k]) + c[(int64_t)k * V + bv];
        if (k != bk && lk > other) other = lk;
      }
      expert_gap[b] = log(w[bk]) + c[(int64_t)bk * V + bv] - other;
    }
  }
  free(c); free(agg); free(w);
  return 0;
}

int32_t oracle_adacad_beta(const double* lp, int32_t B, int32_t N, int32_t V, double* beta) {
  if (!lp || !beta || B < 1 || N < 1 || V < 1) return -1;
  for (int32_t b = 0; b < B; ++b) {
    const double* lp0 = lp + (int64_t)b * (N + 1) * V; /* amateur row */
    for (int32_t k = 1; k <= N; ++k) {
      const double* lpk = lp + ((int64_t)b * (N + 1) + k) * V;
      /* Jensen-Shannon divergence in bits: the mean of the two
       * Kullback-Leibler divergences to the midpoint distribution */
      double kl_k = 0.0, kl_0 = 0.0;
      for (int32_t v = 0; v < V; ++v) {
        double pk = exp(lpk[v]), p0 = exp(lp0[v]);
        double m = 0.5 * (pk + p0);
        if (pk > 0.0) kl_k += pk * log2(pk / m);
        if (p0 > 0.0) kl_0 += p0 * log2(p0 / m);
      }
      beta[(int64_t)b * N + (k - 1)] = 0.5 * (kl_k + kl_0);
    }
  }
  return 0;
}

/* ------------------------------------------------------------- full step */

int32_t oracle_decode_step(const oracle_dims* dm, uint16_t* kc, uint16_t* vc, int64_t layer_elems,
                           const int64_t* kv_off, const int32_t* cap, int32_t* len, const uint16_t* emb_rows,
                           const uint16_t* w, const float* beta, const float* r, int32_t* token, int32_t* expert,
                           double* score, double* token_gap, double* expert_gap, uint16_t* h_out, double* lse_out,
                           int32_t nthreads) {
  return oracle_decode_step_ex(dm, kc, vc, layer_elems, kv_off, cap, len, emb_rows, w, beta, r, token, expert,
                               score, token_gap, expert_gap, h_out, lse_out, NULL, nthreads);
}

static double clip_unit(double x, double eps) {
  if (x < 0.0) return 0.0;
  if (x > 1.0 - eps) return 1.0 - eps;
  return x;
}

int32_t oracle_relevance(const double* s, int32_t mode, const double* z, int32_t n, double eps, double* r) {
  if (!s || !r || n < 0 || eps < 0.0 || (mode != 0 && mode != 1)) return -1;
  const double pi = 3.14159265358979323846;
  for (int32_t k = 0; k < n; ++k) {
    const double rr = mode == 0 ? clip_unit((s[k] + 1.0) / 2.0, eps)
                                : clip_unit(2.0 / pi * atan(s[k] > 0.0 ? s[k] : 0.0), eps);
    if (!z) {
      r[k] = rr;
      continue;
    }
    const double rz = clip_unit(1.0 / (1.0 + exp(-z[k])), eps);
    r[k] = 2.0 * rr * rz / (rr + rz + eps);
  }
  return 0;
}

void oracle_rope(const double* x, int32_t D, int64_t pos, double theta, double* y) {
  const int32_t half = D / 2;
  for (int32_t f = 0; f < half; ++f) {
    const float inv_freq = (float)pow(theta, -2.0 * (double)f / (double)D);
    const float angle = (float)pos * inv_freq; /* fp32 product, as the models compute it */
    const double c = cos((double)angle), sn = sin((double)angle);
    const double a = x[f], b = x[f + half];
    y[f] = a * c - b * sn;
    y[f + half] = b * c + a * sn;
  }
}

int32_t oracle_decode_step_ex(const oracle_dims* dm, uint16_t* kc, uint16_t* vc, int64_t layer_elems,
                              const int64_t* kv_off, const int32_t* cap, int32_t* len, const uint16_t* emb_rows,
                              const uint16_t* w, const float* beta, const float* r, int32_t* token, int32_t* expert,
                              double* score, double* token_gap, double* expert_gap, uint16_t* h_out,
                              double* lse_out, float* beta_dyn, int32_t nthreads) {
  if (!dm || !kc || !vc || !kv_off || !cap || !len || !emb_rows || !w || !beta || !r || !token || !expert ||
      !score)
    return -1;
  const int32_t B = dm->B, N = dm->N, L = dm->L, Hq = dm->Hq, Hkv = dm->Hkv, D = dm->D, V = dm->V;
  if (B < 1 || N < 1 || L < 1 || Hkv < 1 || Hq % Hkv != 0 || 2 * Hkv > Hq || D < 1 || V < 1) return -1;
  if (dm->rope_theta < 0.0 || (dm->rope_theta > 0.0 && D % 2 != 0)) return -1;
  if (dm->score_mode < 0 || dm->score_mode > 1 || dm->aggregation < 0 || dm->aggregation > 2) return -1;
  const int32_t S = B * (N + 1), d = Hq * D;
  for (int32_t s = 0; s < S; ++s)
    if (len[s] < 0 || len[s] >= cap[s]) return -2;

  double* x = (double*)malloc(sizeof(double) * (size_t)S * d);  /* residual stream */
  double* xn = (double*)malloc(sizeof(double) * (size_t)d);
  double* xq = (double*)malloc(sizeof(double) * (size_t)d); /* rotated query heads */
  uint16_t* u = (uint16_t*)malloc(sizeof(uint16_t) * (size_t)S * d); /* bf16 layer input */
  double* o = (double*)malloc(sizeof(double) * (size_t)S * d);
  double* lp = (double*)malloc(sizeof(double) * (size_t)S * V);
  double* lse = (double*)malloc(sizeof(double) * (size_t)S);
  if (!x || !xn || !xq || !u || !o || !lp || !lse) {
    free(x); free(xn); free(xq); free(u); free(o); free(lp); free(lse);
    return -1;
  }

  /* shared history: every expert of query b consumes the same previous token */
  for (int32_t s = 0; s < S; ++s) {
    int32_t b = s / (N + 1);
    for (int32_t i = 0; i < d; ++i) x[(int64_t)s * d + i] = oracle_bf16_value(emb_rows[(int64_t)b * d + i]);
    len[s] += 1; /* the new token joins every expert's cache */
  }

  for (int32_t l = 0; l < L; ++l) {
    uint16_t* K = kc + (int64_t)l * layer_elems;
    uint16_t* Vc = vc + (int64_t)l * layer_elems;
    for (int32_t s = 0; s < S; ++s) {
      oracle_rmsnorm(x + (int64_t)s * d, d, dm->rms_eps, xn);
      const int64_t pos = len[s] - 1; /* the new token's position */
      for (int32_t hq = 0; hq < Hq; ++hq) {
        if (dm->rope_theta > 0.0)
          oracle_rope(xn + (int64_t)hq * D, D, pos, dm->rope_theta, xq + (int64_t)hq * D);
        else
          memcpy(xq + (int64_t)hq * D, xn + (int64_t)hq * D, sizeof(double) * (size_t)D);
      }
      for (int32_t i = 0; i < d; ++i) u[(int64_t)s * d + i] = oracle_round_bf16(xq[i]);
      for (int32_t h = 0; h < Hkv; ++h) {
        uint16_t* kr = K + kv_off[s] + ((int64_t)h * cap[s] + pos) * D;
        uint16_t* vr = Vc + kv_off[s] + ((int64_t)h * cap[s] + pos) * D;
        memcpy(kr, u + (int64_t)s * d + (int64_t)h * D, sizeof(uint16_t) * (size_t)D);
        for (int32_t i = 0; i < D; ++i) vr[i] = oracle_round_bf16(xn[(int64_t)(Hkv + h) * D + i]);
      }
    }
    oracle_attention(u, K, Vc, kv_off, cap, len, S, Hq, Hkv, D, dm->attn_scale, o, nthreads);
    for (int64_t i = 0; i < (int64_t)S * d; ++i) x[i] += o[i];
  }

  for (int32_t s = 0; s < S; ++s) {
    oracle_rmsnorm(x + (int64_t)s * d, d, dm->rms_eps, xn);
    for (int32_t i = 0; i < d; ++i) u[(int64_t)s * d + i] = oracle_round_bf16(xn[i]);
  }
  if (h_out) memcpy(h_out, u, sizeof(uint16_t) * (size_t)S * d);

  oracle_lm_head_logprobs(u, w, S, d, V, lp, lse, nthreads);
  if (lse_out) memcpy(lse_out, lse, sizeof(double) * (size_t)S);
  int32_t rc = 0;
  if (beta_dyn) {
    /* first generated token of a dynamic-beta run: beta from this step's
     * distributions, rounded to the fp32 the selection takes */
    double* bd = (double*)malloc(sizeof(double) * (size_t)B * N);
    if (!bd) {
      rc = -1;
    } else {
      oracle_adacad_beta(lp, B, N, V, bd);
      for (int64_t i = 0; i < (int64_t)B * N; ++i) beta_dyn[i] = (float)bd[i];
      free(bd);
      beta = beta_dyn;
    }
  }
  if (rc == 0 && dm->aggregation != 0) {
    rc = oracle_aggregate_select(lp, beta, r, B, N, V, dm->aggregation, token, expert, score, token_gap, expert_gap);
  } else if (rc == 0) {
    if (dm->score_mode == 1) /* raw logits: z = lp + lse */
      for (int32_t s = 0; s < S; ++s)
        for (int32_t v = 0; v < V; ++v) lp[(int64_t)s * V + v] += lse[s];
    oracle_contrastive_select(lp, beta, r, dm->gamma, B, N, V, token, expert, score, token_gap, expert_gap);
  }

  free(x); free(xn); free(xq); free(u); free(o); free(lp); free(lse);
  return rc;
}
