// lm_head.cuh -- unembedding GEMM with fused log-softmax statistics and the
// contrastive per-tile maxima, plus the cross-tile reductions.
#pragma once
#include "common.cuh"

namespace pced {

constexpr int LM_EPI_THREADS = 256;  // eight epilogue warps: two per TMEM lane quarter, each half of the columns
constexpr int LM_THREADS = 64 + LM_EPI_THREADS;  // warp 0 TMA, warp 1 MMA + TMEM owner, warps 2-9 epilogue
constexpr int LM_TILE_V = 128;   // vocabulary rows per tile (UMMA M)
constexpr int LM_TILE_K = 64;    // hidden elements per stage (one 128-byte swizzle row)
constexpr int LM_MAX_S = 512;
constexpr int LM_MAX_N1 = 256;   // experts + amateur per query in the selection kernels
constexpr int LM_TRING = 16;     // claimed-tile ring between the TMA and MMA warps (> stages + 2 tiles in flight)

struct LmGeom {
  int32_t S, S_pad, nchunk, chunk_n, d, V, ntiles, nks, slabs, nst, stages, acc_bufs, grid;
  uint32_t tmem_cols;
  size_t smem;
};
// returns false when the shape is unsupported
bool lm_geometry(int32_t S, int32_t d, int32_t V, LmGeom* g);

struct LmArgs {
  int mode;  // 0: write logits[S][V]; 1: contrastive records (needs N, beta)
  int32_t S, N, V, ntiles, nks, slabs, nst, stages, acc_bufs, S_pad, nchunk, chunk_n;
  uint32_t tmem_cols;
  float* logits;      // mode 0
  float2* rec_stats;  // [S][ntiles] (max z, sum exp(z - max)) of each vocabulary tile
  float2* rec_arg;    // [S][ntiles] (max u, argmax v as int bits) for expert columns, mode 1
  float* rec_u2;      // [S][ntiles] the tile's second-largest u (another token), mode 1
  int* tile_ctr;      // tiles claimed so far (zero at launch)
  const float* beta;  // [B][N]
  int pdl;            // launched as a programmatic dependent of the kernel that writes H
  int* status;
};

cudaError_t lm_head_launch(const CUtensorMap& wmap, const CUtensorMap& hmap, const LmGeom& g, const LmArgs& a,
                           cudaStream_t stream);
// mode-0 finish: lse[s] from the tile records, logits -> log-probs in place
cudaError_t lm_lse_finalize_launch(float* logits, const float2* rec_stats, float* lse, int32_t S, int32_t V,
                                   int32_t nrec, cudaStream_t stream);

// Selection from mode-1 records (Eq. 2 + Eq. 3), one CTA per query.
struct SelectArgs {
  const float2* rec_stats;
  const float2* rec_arg;
  const float* rec_u2;
  int32_t B, N, nrec;  // records per row (the LM head's vocabulary tiles)
  int32_t V;
  int* tile_ctr;       // optional: the LM head's tile counter, reset here for its next launch
  const float* beta;
  const float* r;
  float gamma;
  int32_t* token;     // optional [B]
  int32_t* expert;    // optional [B]
  float* score;       // optional [B]
  float* lse_out;     // optional [S]
  // step bookkeeping (optional): history[b][t] etc. with t = *step, then *step += 1
  int32_t* step;
  int32_t* history;
  int32_t* expert_trace;
  float* score_trace;
  int32_t max_steps;
  int32_t* done_counter;
  // per-row results and per-query counters (zero at the first launch; the
  // last CTA of a query resets its counter)
  float* sel_L;       // [S] log-sum-exp of each row
  float* sel_u;       // [S] best u_k of each expert row
  int32_t* sel_tok;   // [S] its token
  float* sel_u2;      // [S] the row's best u_k at another token
  // near-tie margins of the choice (optional): gap_trace[b][t] = (token gap,
  // expert gap); the expert gap recomputes z_s(y) = h_s . W[y] for the
  // query's rows
  float2* gap_trace;
  int64_t* key_out;   // expert-partitioned step: packed choices [B], nothing appended
  int32_t expert_base;
  const __nv_bfloat16* hidden;     // [S][d]
  const __nv_bfloat16* w_unembed;  // [V][d]
  int32_t d;
  int32_t* qdone;     // [B] rows of the query finished
  int pdl;            // launched as a programmatic dependent of the LM head
  int raw_logits;     // s_k of Eq. 2 are the raw logits: c_k = gamma log r_k alone
  int* status;
};
cudaError_t select_from_records_launch(const SelectArgs& a, cudaStream_t stream);

}  // namespace pced
