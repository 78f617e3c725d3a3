/*
 * pced_oracle.h -- CPU oracle of one Parallel Context-of-Experts Decoding
 * (PCED) step.  TEST INFRASTRUCTURE ONLY: the tests, the smoke check and the
 * benchmark's CPU-baseline leg call it; the decoding library never does.
 *
 * Plain fp64 statement of what the decode step computes (paper Sec. 3,
 * "Parallel Context-of-Experts" and "Retrieval-aware contrastive decoding",
 * Eq. 2 and Eq. 3), written for checkability rather than speed.  bf16
 * tensors are passed as raw uint16 bit patterns.
 */
#ifndef PCED_ORACLE_H
#define PCED_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* exact value of a bf16 bit pattern */
double oracle_bf16_value(uint16_t bits);
/* nearest bf16 to x, ties to even (x finite, |x| < 3e38) */
uint16_t oracle_round_bf16(double x);
/* y = x / sqrt(mean(x^2) + eps) */
void oracle_rmsnorm(const double* x, int32_t n, double eps, double* y);

/* One layer of decode attention for S sequences.
 * q: bf16 [S][Hq][D].  kc/vc: one layer's cache region; the slab of
 * (sequence s, kv-head h) starts at element kv_off[s] + h*cap[s]*D and its
 * first len[s] rows of D elements are the keys/values attended to.
 * Query head hq reads kv-head hq / (Hq/Hkv) (grouped-query attention).
 * out: fp64 [S][Hq][D] = softmax(scale * q K^T) V.  Returns 0, or -1 on bad
 * arguments. */
int32_t oracle_attention(const uint16_t* q, const uint16_t* kc, const uint16_t* vc, const int64_t* kv_off,
                         const int32_t* cap, const int32_t* len, int32_t S, int32_t Hq, int32_t Hkv, int32_t D,
                         double scale, double* out, int32_t nthreads);

/* Unembedding + log-softmax: z[s][v] = sum_i h[s][i] * W[v][i];
 * lse[s] = log sum_v exp(z[s][v]); lp[s][v] = z[s][v] - lse[s].
 * h: bf16 [S][d], W: bf16 [V][d]; lp: fp64 [S][V]; lse: fp64 [S]. */
int32_t oracle_lm_head_logprobs(const uint16_t* h, const uint16_t* w, int32_t S, int32_t d, int32_t V, double* lp,
                                double* lse, int32_t nthreads);

/* Eq. 2 + Eq. 3 on log-probabilities lp [S][V] (row b*(N+1) is query b's
 * amateur, rows b*(N+1)+k, k = 1..N, its contextual experts).
 *   shat_k(v) = (1 + beta[b][k-1]) lp_k(v) - beta[b][k-1] lp_0(v) + gamma log r~[b][k-1],
 *   r~ = min(max(r, 1e-8), 1 - 1e-8),
 *   token[b] = argmax_v max_k shat_k(v), expert[b] = the maximising k (1-based).
 * Exact ties: highest score, then lowest token id, then lowest expert.
 * token_gap[b] = score - max_{v != token} max_k shat_k(v);
 * expert_gap[b] = score - max_{k != expert} shat_k(token)  (+inf when N = 1). */
int32_t oracle_contrastive_select(const double* lp, const float* beta, const float* r, double gamma, int32_t B,
                                  int32_t N, int32_t V, int32_t* token, int32_t* expert, double* score,
                                  double* token_gap, double* expert_gap);

/* Aggregation variants of the experts (App. "Ablation of Expert Aggregation
 * Rule": Mixture-of-Experts, a weighted sum, and Product-of-Experts, a
 * weighted product, in probability space, weights derived from retrieval
 * scores).  Reading (the paper gives no formula): per contextual expert the
 * contrastive scores c_k(v) = (1 + beta_k) lp_k(v) - beta_k lp_0(v) of Eq. 2
 * without the prior, p_k = softmax_v(c_k), weights w_k = r~_k / sum_j r~_j
 * with r~ clipped as in Eq. 2;
 *   rule 1 (MoE): agg(v) = log sum_k w_k p_k(v)
 *   rule 2 (PoE): agg(v) = sum_k w_k log p_k(v)
 * token = argmax_v agg (lowest id on exact ties), score = agg(token),
 * expert = argmax_k w_k p_k(token) (1-based, lowest k on ties),
 * token_gap = agg(token) - max_{v != token} agg(v) (+inf when V = 1),
 * expert_gap = log(w p)_expert(token) - max_{k != expert} log(w_k p_k(token))
 * (+inf when N = 1; the near-tie margin of the attribution, in log units).
 * lp [S][V] as in oracle_contrastive_select; gamma does not enter.
 * Parity unpinned against the paper (it names the rules, not the weighting);
 * the tests pin this reading by closed forms. */
int32_t oracle_aggregate_select(const double* lp, const float* beta, const float* r, int32_t B, int32_t N, int32_t V,
                                int32_t rule, int32_t* token, int32_t* expert, double* score, double* token_gap,
                                double* expert_gap);

/* Dynamic contrast strength (Sec. 3 after Eq. 2: beta_0 is computed as in
 * AdaCAD for the first generated token and kept fixed thereafter).  Reading
 * used here: one beta per contextual expert, the Jensen-Shannon divergence in
 * bits between the expert's next-token distribution and the amateur's,
 *   beta[b][k-1] = 1/2 sum_v [ p_k(v) log2(p_k(v)/m(v)) + p_0(v) log2(p_0(v)/m(v)) ],
 *   m = (p_k + p_0)/2,  p = exp(lp),  terms with p = 0 contribute 0,
 * so 0 <= beta <= 1.  lp [S][V] as in oracle_contrastive_select.
 * Parity unpinned against the paper (it names AdaCAD, not the formula); the
 * tests pin the divergence itself. */
int32_t oracle_adacad_beta(const double* lp, int32_t B, int32_t N, int32_t V, double* beta);

/* Rotary position embedding of one head (the decoder LLM's positional
 * encoding; the paper runs Llama / Qwen models, which use it), rotate-half
 * pairing: for f < D/2, with angle a_f = fp32(pos * fp32(theta^(-2f/D)))
 * (the fp32 angle of the models' reference implementations),
 *   y[f]       = x[f] cos a_f - x[f + D/2] sin a_f,
 *   y[f + D/2] = x[f + D/2] cos a_f + x[f] sin a_f,
 * cos and sin evaluated in double.  D even, pos >= 0, theta > 0. */
void oracle_rope(const double* x, int32_t D, int64_t pos, double theta, double* y);

/* Relevance scores r_k in [0, 1) from a retriever's and a reranker's raw
 * scores (Sec. 3 "Retrieval and relevance scoring", App. "Normalization of
 * Retrieval and Reranker Scores"):
 *   retrieval, mode 0 (dense / ColBERT): r_ret = clip((s + 1)/2, 0, 1 - eps)
 *   retrieval, mode 1 (sparse):          r_ret = clip((2/pi) atan(max(s, 0)), 0, 1 - eps)
 *   reranker logit z:                    r_rer = clip(1/(1 + exp(-z)), 0, 1 - eps)
 *   fusion (harmonic mean, appendix form with eps in the denominator):
 *                                        r = 2 r_ret r_rer / (r_ret + r_rer + eps)
 * With z == NULL the result is r_ret alone.  n scores; returns 0, or -1 on bad
 * arguments (mode not 0/1, n < 0, eps < 0). */
int32_t oracle_relevance(const double* s, int32_t mode, const double* z, int32_t n, double eps, double* r);

typedef struct oracle_dims {
  int32_t B, N, L, Hq, Hkv, D, V; /* S = B*(N+1), d = Hq*D, requires 2*Hkv <= Hq */
  double gamma;                   /* retrieval-prior weight of Eq. 2 */
  double rms_eps;                 /* RMSNorm epsilon */
  double attn_scale;              /* softmax scale, 1/sqrt(D) */
  double rope_theta;              /* rotary base; 0: no rotary embedding */
  int32_t score_mode;             /* s_k of Eq. 2: 0 log-probabilities, 1 raw logits */
  int32_t aggregation;            /* 0 max over experts (Eq. 3), 1 MoE, 2 PoE (oracle_aggregate_select) */
} oracle_dims;

/* One full decode step of the synthetic PCED model.
 *   x_0[s]    = emb_rows[b]            (embedding of query b's previous token)
 *   per layer l:  n = rmsnorm(x_l[s]);  q = bf16(R(n)) as [Hq][D];
 *                 K_l[s][h][len] = q[h], V_l[s][h][len] = bf16(n[Hkv + h])
 *                 (h < Hkv, appended at the old length = the token's position p;
 *                 the length grows by one per step)
 *                 x_{l+1}[s] = x_l[s] + attention(q, K_l, V_l)
 *                 R: oracle_rope at position p on every head when
 *                 rope_theta > 0, else the identity
 *   h[s]      = bf16(rmsnorm(x_L[s]))
 *   then the unembedding/log-softmax and Eq. 2 + Eq. 3 selection.
 * kc/vc span L layers of layer_elems elements (slab layout as in
 * oracle_attention); len[S] is updated in place; h_out (bf16 [S][d]) and
 * lse_out ([S]) may be NULL.  score_mode 1 feeds the raw logits z = lp + lse
 * to Eq. 2 instead of the log-probabilities (max rule; MoE / PoE do not
 * depend on it: a per-expert constant drops out of the softmax); with
 * aggregation 1 or 2 the token, expert and both gaps come from
 * oracle_aggregate_select.  Returns 0, -1 on bad arguments, -2 when a
 * cache is full. */
int32_t oracle_decode_step(const oracle_dims* dm, uint16_t* kc, uint16_t* vc, int64_t layer_elems,
                           const int64_t* kv_off, const int32_t* cap, int32_t* len, const uint16_t* emb_rows,
                           const uint16_t* w, const float* beta, const float* r, int32_t* token, int32_t* expert,
                           double* score, double* token_gap, double* expert_gap, uint16_t* h_out, double* lse_out,
                           int32_t nthreads);
/* The same step; when beta_dyn is not NULL the contrast strengths are not
 * taken from `beta` but computed from this step's log-probabilities with
 * oracle_adacad_beta, rounded to fp32, stored in beta_dyn [B][N] and used for
 * the selection (the first generated token of a dynamic-beta run). */
int32_t oracle_decode_step_ex(const oracle_dims* dm, uint16_t* kc, uint16_t* vc, int64_t layer_elems,
                              const int64_t* kv_off, const int32_t* cap, int32_t* len, const uint16_t* emb_rows,
                              const uint16_t* w, const float* beta, const float* r, int32_t* token, int32_t* expert,
                              double* score, double* token_gap, double* expert_gap, uint16_t* h_out,
                              double* lse_out, float* beta_dyn, int32_t nthreads);

#ifdef __cplusplus
}
#endif
#endif /* PCED_ORACLE_H */
