// aggregate.cuh -- MoE / PoE aggregation of the experts from materialised
// log-probabilities (the appendix's aggregation-rule ablation).
#pragma once
#include "common.cuh"

namespace pced {

struct AggArgs {
  // [S][V] log-probabilities, query-major, amateur first; or, with rec_stats
  // set (MoE / PoE only), the raw logits z: p_k and the aggregates do not
  // depend on the rows' log-sum-exps L (the constant (1+beta) L_k - beta L_0
  // cancels in the softmax of the contrastive scores)
  const float* lp;
  const float2* rec_stats;  // raw logits: the LM head's per-tile (max, sum exp) of every row, [S][nrec]
  int32_t nrec;
  float* lse_rows;      // raw logits: [S] log-sum-exps formed from rec_stats (what lse points to)
  const float* beta;    // [B][N]
  const float* r;       // [B][N] relevance scores
  const float* lse;     // [S] log-sum-exps of the rows (copied to lse_out)
  int32_t B, N, V, rule, nchunks;  // rule 0 Eq. 3 (max over experts), 1 MoE, 2 PoE
  float gamma;          // rule 0: weight of the retrieval prior
  int raw_logits;       // rule 0: s_k of Eq. 2 are the raw logits lp + lse
  float2* part;         // [B][N][nchunks] (max, sum exp) of c_k over each chunk
  int32_t* kdone;       // [B][N] chunks finished per expert (zero at launch; the last resets it)
  float* lse_k;         // [B][N] log-sum-exp of c_k (the softmax normaliser of p_k)
  float2* best;         // [B][nchunks] (aggregate, token) of each chunk
  float* best2;         // [B][nchunks] the chunk's best aggregate at another token
  int32_t* qdone;       // [B] chunks finished (zero at launch; the last resets it)
  int* tile_ctr;        // optional: the LM head's tile counter, reset for its next launch
  int32_t* token;       // optional [B]
  int32_t* expert;      // optional [B]
  float* score;         // optional [B]
  float* lse_out;       // optional [S]
  // step bookkeeping (optional), as in the max-rule selection
  int32_t* step;
  int32_t* history;
  int32_t* expert_trace;
  float* score_trace;
  float2* gap_trace;    // optional [B][max_steps]: (token gap, attribution margin)
  int64_t* key_out;     // rule 0, expert-partitioned step: packed choices [B], nothing appended
  int32_t expert_base;
  int32_t max_steps;
  int32_t* done_counter;
  int* status;
};

constexpr int AGG_CHUNK = 1024;  // vocabulary entries per CTA (about 125 CTAs per query at V = 128K)
constexpr int AGG_MAX_N = 512;   // experts per query (the LM head's row limit)
inline int32_t agg_chunks(int32_t V) { return (V + AGG_CHUNK - 1) / AGG_CHUNK; }
// (1) per (query, expert, chunk) statistics, (2) per (query, chunk) best and the pick
cudaError_t agg_partials_launch(const AggArgs& a, cudaStream_t stream);
cudaError_t agg_select_launch(const AggArgs& a, cudaStream_t stream);

}  // namespace pced
