// step.cu -- one greedy PCED decode step for all queries (paper Sec. 3: the
// N+1 experts run as one batch; Eq. 2 + Eq. 3 pick the token, which joins
// every expert's history).  Three launches on one stream, no host sync:
//   attention  one cooperative kernel: x_0 = E[y_{t-1}], then for every layer
//              u = bf16(rmsnorm(x)), append K/V row of u, x += attention(u);
//              h = bf16(rmsnorm(x_L)); seq_len += 1
//   lm head    tcgen05 GEMM with log-softmax statistics + contrastive tile maxima
//   select     Eq. 2 + Eq. 3 per query, history[b][t] = y, t += 1
// Every quantity that changes between steps (t, lengths, history) lives on
// the device, so one captured call replays as the next step.
#include <cmath>
#include <math.h>
#include <nvtx3/nvToolsExt.h>
#include <stdlib.h>

#include "adacad.cuh"
#include "aggregate.cuh"
#include "attention.cuh"
#include "lm_head.cuh"
#include "select_key.cuh"

namespace pced {

struct StepLayout {
  int* status;
  int32_t* done_counter;  // selection kernel: queries finished this step
  int32_t* att_done;      // attention: CTAs finished
  int32_t* att_epoch;     // attention: launches completed
  int32_t* lm_tile_ctr;   // LM head: vocabulary tiles claimed (reset by the selection)
  int32_t* sel_qdone;     // selection: rows finished per query
  float* sel_L;
  float* sel_u;
  int32_t* sel_tok;
  float* lp;              // [S][V] log-probabilities of a dynamic-beta first step
  void* ada;              // scratch of the beta kernel (counters zero between uses)
  float2* agg_part;       // MoE / PoE: per (query, expert, chunk) statistics
  float2* agg_best;       // MoE / PoE: per (query, chunk) best
  float* agg_best2;       // MoE / PoE: per (query, chunk) best at another token
  int32_t* agg_kdone;     // MoE / PoE: chunks finished per (query, expert)
  float* agg_lse;         // MoE / PoE: per (query, expert) log-sum-exp of the contrastive scores
  int32_t* agg_qdone;     // MoE / PoE: chunks finished per query
  uint64_t* part_ss;
  uint64_t* resid;
  uint64_t* rec_o;
  uint64_t* rec_ml;
  __nv_bfloat16* h;
  float2* lm_stats;
  float2* lm_arg;
  float* lm_u2;
  float* sel_u2;
  size_t bytes;
};

static StepLayout step_layout(const pced_dims* dm, void* ws) {
  const int32_t S = dm->B * (dm->N + 1), d = dm->Hq * dm->D, G = dm->Hq / dm->Hkv;
  const int64_t slots = att_step_slots(S, dm->Hkv);
  const int64_t ntiles = (dm->V + LM_TILE_V - 1) / LM_TILE_V;
  StepLayout L;
  pced_host::Carver c(ws);
  L.status = c.take<int>(64);
  L.done_counter = c.take<int32_t>(1);
  L.att_done = c.take<int32_t>(1);
  L.att_epoch = c.take<int32_t>(1);
  // the words the attention CTAs exchange start on 4 KB boundaries (an
  // offset that is not a multiple of 1 KB measured ~1 % slower)
  L.part_ss = c.take<uint64_t>((size_t)2 * S * dm->Hkv * ATT_CONSUMERS, 4096);
  L.resid = c.take<uint64_t>((size_t)2 * S * d, 4096);
  L.rec_o = c.take<uint64_t>((size_t)(slots * G * dm->D), 4096);
  L.rec_ml = c.take<uint64_t>((size_t)(slots * G * 2), 4096);
  L.h = c.take<__nv_bfloat16>((size_t)S * d);
  L.lm_stats = c.take<float2>((size_t)(S * ntiles));
  L.lm_arg = c.take<float2>((size_t)(S * ntiles));
  L.lm_u2 = c.take<float>((size_t)(S * ntiles));
  L.sel_u2 = c.take<float>((size_t)S);
  L.lm_tile_ctr = c.take<int32_t>(1);
  L.sel_qdone = c.take<int32_t>((size_t)dm->B);
  L.sel_L = c.take<float>((size_t)S);
  L.sel_u = c.take<float>((size_t)S);
  L.sel_tok = c.take<int32_t>((size_t)S);
  L.lp = c.take<float>((size_t)S * dm->V);
  L.ada = c.take<char>(adacad_scratch_bytes(dm->B, dm->N, dm->V));
  L.agg_part = c.take<float2>((size_t)dm->B * dm->N * agg_chunks(dm->V));
  L.agg_best = c.take<float2>((size_t)dm->B * agg_chunks(dm->V));
  L.agg_best2 = c.take<float>((size_t)dm->B * agg_chunks(dm->V));
  L.agg_kdone = c.take<int32_t>((size_t)dm->B * dm->N);
  L.agg_lse = c.take<float>((size_t)dm->B * dm->N);
  L.agg_qdone = c.take<int32_t>((size_t)dm->B);
  L.bytes = c.used() + 4 * (4096 - 256);  // room for the 4 KB alignment of four arrays
  return L;
}

// NVTX ranges on the host thread that enqueues a step, for timeline tools:
// one over the call and, inside it, one per launch named by its kind (the
// names of pced_step_launch_kind).  Without a tool attached they cost a
// branch each.
struct StepRanges {
  bool open = false;
  StepRanges() { nvtxRangePushA("pced_step"); }
  void next(const char* kind) {
    if (open) nvtxRangePop();
    nvtxRangePushA(kind);
    open = true;
  }
  ~StepRanges() {
    if (open) nvtxRangePop();
    nvtxRangePop();
  }
};

}  // namespace pced

using namespace pced;
using namespace pced_host;

extern "C" size_t pced_step_workspace_size(const pced_dims* dm) {
  if (!dm || dm->B < 1 || dm->N < 1 || dm->Hq < 1 || dm->Hkv < 1 || dm->D < 1 || dm->V < 1 || dm->Hq % dm->Hkv)
    return 0;
  return step_layout(dm, nullptr).bytes;
}

// The kernels one pced_step call with these arguments launches, in order
// (kinds may be NULL); returns their number.
static int32_t step_plan(const pced_step_args* p, const char** kinds) {
  int32_t n = 0;
  auto add = [&](const char* k) {
    if (kinds) kinds[n] = k;
    ++n;
  };
  const bool dyn = p->beta_from_step != 0, agg = p->aggregation != PCED_AGG_MAX;
  add("attention");
  if (dyn || agg) {
    add("lm_head");  // logits mode: the logits materialised
    if (dyn) {
      add("lse_finalize");  // normalised to log-probabilities for beta
      add("adacad_beta");
    }
  }
  if (agg) {
    add("agg_partials");
    add("agg_select");
  } else if (dyn) {
    add("agg_select");  // Eq. 3 on the log-probabilities written for beta
  } else {
    add("lm_head");  // fused log-softmax statistics and contrastive tile maxima
    add("select");
  }
  return n;
}

extern "C" int32_t pced_step_launch_count(const pced_step_args* p) { return p ? step_plan(p, nullptr) : 0; }

extern "C" const char* pced_step_launch_kind(const pced_step_args* p, int32_t i) {
  const char* kinds[8];
  if (!p || i < 0 || i >= step_plan(p, kinds)) return nullptr;
  return kinds[i];
}

// Host-side validation of a pced_step call; on success *g and *num_blocks
// hold the LM-head geometry and the paged pool's block count.
static pced_status step_check(const pced_step_args* p, LmGeom* g_out, int64_t* num_blocks_out) {
  if (!p) return fail(PCED_ERR_INVALID_ARG, "pced_step: null args");
  const pced_dims dm = p->dims;
  const bool paged = p->block_table != nullptr;
  if (!p->embed || !p->w_unembed || !p->k_cache || !p->v_cache || (!paged && !p->kv_offset) || !p->cap || !p->seq_len ||
      !p->step || !p->history || !p->beta || !p->r || !p->workspace || (p->beta_from_step && !p->beta_out))
    return fail(PCED_ERR_INVALID_ARG, "pced_step: null pointer");
  if (dm.B < 1 || dm.N < 1 || dm.L < 1 || dm.Hq < 1 || dm.Hkv < 1 || dm.D < 1 || dm.V < 1 || dm.Hq % dm.Hkv != 0 ||
      2 * dm.Hkv > dm.Hq || dm.L > ATT_MAX_LAYERS || p->max_steps < 1 || p->layer_elems < dm.D || p->total_cap < 1)
    return fail(PCED_ERR_INVALID_ARG, "pced_step: bad dimensions");
  if (!isfinite(p->gamma) || !(p->attn_scale > 0.f) || !(p->rms_eps >= 0.f))
    return fail(PCED_ERR_INVALID_ARG, "pced_step: bad gamma / scale / eps");
  if (p->bos_token < 0 || p->bos_token >= dm.V) return fail(PCED_ERR_INVALID_ARG, "pced_step: bos out of range");
  const int32_t S = dm.B * (dm.N + 1), d = dm.Hq * dm.D, G = dm.Hq / dm.Hkv;
  if (dm.D != 64 && dm.D != 128) return fail(PCED_ERR_UNSUPPORTED, "pced_step: D=%d (supported: 64, 128)", dm.D);
  if (G > ATT_MAX_G) return fail(PCED_ERR_UNSUPPORTED, "pced_step: Hq/Hkv > %d", ATT_MAX_G);
  if (S > ATT_MAX_S || S > LM_MAX_S) return fail(PCED_ERR_UNSUPPORTED, "pced_step: S=%d too large", S);
  if (dm.N + 1 > LM_MAX_N1) return fail(PCED_ERR_UNSUPPORTED, "pced_step: N too large");
  if (d > 8192) return fail(PCED_ERR_UNSUPPORTED, "pced_step: hidden size %d > 8192", d);
  if (p->layer_elems % dm.D != 0 || (int64_t)dm.L * (p->layer_elems / dm.D) >= ((int64_t)1 << 31))
    return fail(PCED_ERR_UNSUPPORTED, "pced_step: cache too large for 32-bit row coordinates");
  if (p->score_mode != PCED_SCORE_LOGPROB && p->score_mode != PCED_SCORE_LOGIT)
    return fail(PCED_ERR_INVALID_ARG, "pced_step: score_mode %d", p->score_mode);
  if (p->aggregation < PCED_AGG_MAX || p->aggregation > PCED_AGG_POE)
    return fail(PCED_ERR_INVALID_ARG, "pced_step: aggregation %d", p->aggregation);
  if (p->aggregation != PCED_AGG_MAX && dm.N > AGG_MAX_N)
    return fail(PCED_ERR_UNSUPPORTED, "pced_step: MoE / PoE take at most %d experts", AGG_MAX_N);
  if (p->key_out && (p->aggregation != PCED_AGG_MAX || dm.V > KEY_MAX_TOKENS || p->expert_base < 0 ||
                     p->expert_base + dm.N > KEY_MAX_EXPERTS))
    return fail(PCED_ERR_UNSUPPORTED, "pced_step: expert-partitioned step needs the max rule, V <= 2^20 and "
                                      "expert_base + N <= 4096");
  if (!(p->rope_theta >= 0.f) || !std::isfinite(p->rope_theta))
    return fail(PCED_ERR_INVALID_ARG, "pced_step: rope_theta must be finite and >= 0");
  int64_t num_blocks = 0;
  if (paged) {
    if (p->block_rows < ATT_BLOCK_N || p->block_rows % ATT_BLOCK_N != 0 || p->max_blocks < 1)
      return fail(PCED_ERR_INVALID_ARG, "pced_step: block_rows must be a positive multiple of %d", ATT_BLOCK_N);
    if ((int64_t)S * p->max_blocks >= ((int64_t)1 << 31))
      return fail(PCED_ERR_UNSUPPORTED, "pced_step: block table too large for 32-bit entry indices");
    const int64_t block_elems = (int64_t)dm.Hkv * p->block_rows * dm.D;
    if (p->layer_elems % block_elems != 0)
      return fail(PCED_ERR_INVALID_ARG, "pced_step: layer_elems is not a whole number of blocks");
    num_blocks = p->layer_elems / block_elems;
    if (num_blocks >= ((int64_t)1 << 31)) return fail(PCED_ERR_UNSUPPORTED, "pced_step: too many blocks");
  }
  LmGeom g;
  if (!lm_geometry(S, d, dm.V, &g)) return fail(PCED_ERR_UNSUPPORTED, "pced_step: LM-head shape unsupported");
  if ((((uintptr_t)p->k_cache) | ((uintptr_t)p->v_cache) | ((uintptr_t)p->w_unembed) | ((uintptr_t)p->embed)) & 15u)
    return fail(PCED_ERR_INVALID_ARG, "pced_step: tensors must be 16-byte aligned");
  if (((uintptr_t)p->workspace) & 255u || p->workspace_bytes < pced_step_workspace_size(&dm))
    return fail(PCED_ERR_WORKSPACE, "pced_step: workspace too small or misaligned");
  if (num_sms() <= 0) return fail(PCED_ERR_NO_DEVICE, "pced_step: no CUDA device");
  *g_out = g;
  *num_blocks_out = num_blocks;
  return PCED_OK;
}

extern "C" pced_status pced_step(const pced_step_args* p, void* stream) {
  LmGeom g;
  int64_t num_blocks = 0;
  const pced_status chk = step_check(p, &g, &num_blocks);
  if (chk != PCED_OK) return chk;
  const pced_dims dm = p->dims;
  const bool paged = p->block_table != nullptr;
  const int32_t S = dm.B * (dm.N + 1), d = dm.Hq * dm.D, G = dm.Hq / dm.Hkv;

  const StepLayout W = step_layout(&dm, p->workspace);
  CUtensorMap kmap, vmap, wmap, hmap;
  const uint64_t rows = (uint64_t)dm.L * (uint64_t)(p->layer_elems / dm.D);
  pced_status st = make_tmap_kv(&kmap, p->k_cache, rows, (uint32_t)dm.D, ATT_BLOCK_N);
  if (st == PCED_OK) st = make_tmap_kv(&vmap, p->v_cache, rows, (uint32_t)dm.D, ATT_BLOCK_N);
  if (st == PCED_OK) st = make_tmap_2d(&wmap, p->w_unembed, (uint64_t)dm.V, (uint64_t)d, LM_TILE_V, LM_TILE_K, true);
  if (st == PCED_OK) st = make_tmap_2d(&hmap, W.h, (uint64_t)S, (uint64_t)d, (uint32_t)g.chunk_n, LM_TILE_K, false);
  if (st != PCED_OK) return st;
  cudaStream_t s = (cudaStream_t)stream;
  const bool dyn = p->beta_from_step != 0;
  const bool agg = p->aggregation != PCED_AGG_MAX;
  const bool timed = p->stage_events && p->n_stage_events >= step_plan(p, nullptr) + 1;
  cudaStreamCaptureStatus cap_status = cudaStreamCaptureStatusNone;
  if (timed && cudaStreamIsCapturing(s, &cap_status) != cudaSuccess) return cuda_status(cudaGetLastError(), "capture query");
  int mark_i = 0;
  // inside a stream capture the events become external event-record nodes, so
  // they can still be timed after each replay
  auto mark = [&]() -> cudaError_t {
    if (!timed) return cudaSuccess;
    cudaEvent_t ev = (cudaEvent_t)p->stage_events[mark_i++];
    return cap_status == cudaStreamCaptureStatusActive ? cudaEventRecordWithFlags(ev, s, cudaEventRecordExternal)
                                                       : cudaEventRecord(ev, s);
  };
  StepRanges ranges;
  cudaError_t e = mark();
  if (e != cudaSuccess) return cuda_status(e, "stage event");

  StepAttArgs at = {};
  at.S = S;
  at.Hq = dm.Hq;
  at.Hkv = dm.Hkv;
  at.G = G;
  at.L = dm.L;
  at.n1 = dm.N + 1;
  at.V = dm.V;
  at.bos = p->bos_token;
  at.max_steps = p->max_steps;
  at.rows_per_layer = p->layer_elems / dm.D;
  at.layer_elems = p->layer_elems;
  at.scale_log2 = p->attn_scale * 1.4426950408889634f;
  at.rms_eps = p->rms_eps;
  at.seg_cost = att_step_seg_cost(dm.D);
  at.pf_tiles = att_step_pf_tiles();
  at.groups = att_step_groups();
  at.seg_lead = att_step_seg_lead(at.seg_cost);
  if (paged) {
    // whole tiles: with every extent, lead and CTA share a multiple of the
    // tile size, each piece starts on a tile (and so block) boundary
    at.seg_cost = (at.seg_cost + ATT_BLOCK_N - 1) & ~(ATT_BLOCK_N - 1);
    at.seg_lead = (at.seg_lead + ATT_BLOCK_N - 1) & ~(ATT_BLOCK_N - 1);
    if (at.seg_lead > at.seg_cost) at.seg_lead = at.seg_cost;
  }
  at.kv_offset = p->kv_offset;
  at.cap = p->cap;
  at.block_table = p->block_table;
  at.block_rows = paged ? p->block_rows : 0;
  at.max_blocks = paged ? p->max_blocks : 0;
  at.num_blocks = (int32_t)num_blocks;
  at.rope_theta = p->rope_theta;
  at.block_shift = -1;
  if (paged && (p->block_rows & (p->block_rows - 1)) == 0)
    for (at.block_shift = 0; (1 << at.block_shift) < p->block_rows; ++at.block_shift) {
    }
  at.seq_len = p->seq_len;
  at.step = p->step;
  at.history = p->history;
  at.embed = (const __nv_bfloat16*)p->embed;
  at.k_cache = (__nv_bfloat16*)p->k_cache;
  at.v_cache = (__nv_bfloat16*)p->v_cache;
  at.resid = W.resid;
  at.part_ss = W.part_ss;
  at.rec_o = W.rec_o;
  at.rec_ml = W.rec_ml;
  at.epoch = W.att_epoch;
  at.done_cnt = W.att_done;
  at.hidden = W.h;
  at.hidden_copy = (__nv_bfloat16*)p->hidden_out;
  at.status = W.status;
  at.wait_ns = p->wait_limit_ns ? p->wait_limit_ns : kWaitLimitNs;
  ranges.next("attention");
  e = att_step_launch(dm.D, kmap, vmap, at, att_grid(p->total_cap * dm.Hkv), s);
  if (e == cudaSuccess) e = mark();
  if (e != cudaSuccess) return cuda_status(e, "attention launch");

  // dynamic contrast strength or MoE / PoE: materialise this step's
  // log-probabilities; beta from their divergences, then either the usual
  // fused LM head with that beta or the aggregation kernels
  const float* beta = p->beta;
  if (dyn || agg) {
    LmArgs lz = {};
    lz.mode = 0;
    lz.S = S;
    lz.N = 0;
    lz.V = dm.V;
    lz.ntiles = g.ntiles;
    lz.nks = g.nks;
    lz.slabs = g.slabs;
    lz.nst = g.nst;
    lz.stages = g.stages;
    lz.acc_bufs = g.acc_bufs;
    lz.S_pad = g.S_pad;
    lz.nchunk = g.nchunk;
    lz.chunk_n = g.chunk_n;
    lz.tmem_cols = g.tmem_cols;
    lz.logits = W.lp;
    lz.rec_stats = W.lm_stats;
    lz.tile_ctr = W.lm_tile_ctr;
    lz.status = W.status;
    lz.pdl = timed ? 0 : 1;  // streams weights while the attention kernel finishes
    ranges.next("lm_head");
    e = lm_head_launch(wmap, hmap, g, lz, s);
    if (e == cudaSuccess) e = mark();
    // MoE / PoE alone need no log-probabilities (the aggregation kernels
    // read the raw logits and form the rows' log-sum-exps themselves); beta
    // needs the normalised rows
    if (e == cudaSuccess && dyn) {
      ranges.next("lse_finalize");
      e = lm_lse_finalize_launch(W.lp, W.lm_stats, W.sel_L, S, dm.V, g.ntiles, s);
      if (e == cudaSuccess) e = mark();
    }
    // the JSD kernel also re-arms the LM head's tile counter for the fused pass
    if (e == cudaSuccess && dyn) {
      ranges.next("adacad_beta");
      e = adacad_beta_launch(W.lp, dm.B, dm.N, dm.V, p->beta_out, W.ada, W.lm_tile_ctr, s);
      if (e == cudaSuccess) e = mark();
    }
    if (e != cudaSuccess) return cuda_status(e, "log-probability launches");
    if (dyn) beta = p->beta_out;
  }
  if (agg || dyn) {
    // MoE / PoE, or Eq. 3 on the log-probabilities the first step of a
    // dynamic-beta decode has written anyway (no second LM-head pass)
    AggArgs ag = {};
    ag.lp = W.lp;
    if (!dyn) {  // raw logits (MoE / PoE without a dynamic beta)
      ag.rec_stats = W.lm_stats;
      ag.nrec = g.ntiles;
      ag.lse_rows = W.sel_L;
    }
    ag.beta = beta;
    ag.r = p->r;
    ag.lse = W.sel_L;
    ag.B = dm.B;
    ag.N = dm.N;
    ag.V = dm.V;
    ag.rule = p->aggregation;
    ag.gamma = p->gamma;
    ag.raw_logits = p->score_mode == PCED_SCORE_LOGIT;
    ag.nchunks = agg_chunks(dm.V);
    ag.part = W.agg_part;
    ag.best = W.agg_best;
    ag.best2 = W.agg_best2;
    ag.kdone = W.agg_kdone;
    ag.lse_k = W.agg_lse;
    ag.gap_trace = p->key_out ? nullptr : reinterpret_cast<float2*>(p->gap_trace);
    ag.key_out = p->key_out;
    ag.expert_base = p->expert_base;
    ag.qdone = W.agg_qdone;
    ag.tile_ctr = W.lm_tile_ctr;
    ag.lse_out = p->lse_out;
    ag.step = p->step;
    ag.history = p->history;
    ag.expert_trace = p->expert_trace;
    ag.score_trace = p->score_trace;
    ag.max_steps = p->max_steps;
    ag.done_counter = W.done_counter;
    ag.token = p->token_out;
    ag.expert = p->expert_out;
    ag.score = p->score_out;
    ag.status = W.status;
    if (agg) {
      ranges.next("agg_partials");
      e = agg_partials_launch(ag, s);
      if (e == cudaSuccess) e = mark();
    }
    if (e == cudaSuccess) ranges.next("agg_select");
    if (e == cudaSuccess) e = agg_select_launch(ag, s);
    if (e == cudaSuccess) e = mark();
    if (e != cudaSuccess) return cuda_status(e, "aggregation launches");
    return PCED_OK;
  }

  LmArgs la = {};
  la.mode = 1;
  la.S = S;
  la.N = dm.N;
  la.V = dm.V;
  la.ntiles = g.ntiles;
  la.nks = g.nks;
  la.slabs = g.slabs;
  la.nst = g.nst;
  la.stages = g.stages;
  la.acc_bufs = g.acc_bufs;
  la.S_pad = g.S_pad;
  la.nchunk = g.nchunk;
  la.chunk_n = g.chunk_n;
  la.tmem_cols = g.tmem_cols;
  la.rec_stats = W.lm_stats;
  la.rec_arg = W.lm_arg;
  la.rec_u2 = W.lm_u2;
  la.tile_ctr = W.lm_tile_ctr;
  la.beta = beta;
  la.status = W.status;
  la.pdl = (timed || dyn) ? 0 : 1;  // stage events between the launches would break the overlap
  ranges.next("lm_head");
  e = lm_head_launch(wmap, hmap, g, la, s);
  if (e == cudaSuccess) e = mark();
  if (e != cudaSuccess) return cuda_status(e, "lm head launch");

  SelectArgs sa = {};
  sa.rec_stats = W.lm_stats;
  sa.rec_arg = W.lm_arg;
  sa.rec_u2 = W.lm_u2;
  sa.V = dm.V;
  sa.sel_u2 = W.sel_u2;
  sa.gap_trace = reinterpret_cast<float2*>(p->gap_trace);
  sa.key_out = p->key_out;
  sa.expert_base = p->expert_base;
  sa.hidden = W.h;
  sa.w_unembed = (const __nv_bfloat16*)p->w_unembed;
  sa.d = d;
  sa.B = dm.B;
  sa.N = dm.N;
  sa.nrec = g.ntiles;
  sa.tile_ctr = W.lm_tile_ctr;
  sa.sel_L = W.sel_L;
  sa.sel_u = W.sel_u;
  sa.sel_tok = W.sel_tok;
  sa.qdone = W.sel_qdone;
  sa.beta = beta;
  sa.r = p->r;
  sa.gamma = p->gamma;
  sa.lse_out = p->lse_out;
  sa.step = p->step;
  sa.history = p->history;
  sa.expert_trace = p->expert_trace;
  sa.score_trace = p->score_trace;
  sa.max_steps = p->max_steps;
  sa.done_counter = W.done_counter;
  sa.token = p->token_out;
  sa.expert = p->expert_out;
  sa.score = p->score_out;
  sa.status = W.status;
  sa.pdl = (timed || dyn) ? 0 : 1;
  sa.raw_logits = p->score_mode == PCED_SCORE_LOGIT;
  ranges.next("select");
  e = select_from_records_launch(sa, s);
  if (e == cudaSuccess) e = mark();
  if (e != cudaSuccess) return cuda_status(e, "select launch");
  return PCED_OK;
}

// A "host" buffer that is device memory would make the copy device to
// device; refuse it where the runtime can say (not inside a stream capture,
// where a pointer query is not a capturable call).
static bool is_device_memory(const void* ptr) {
  cudaPointerAttributes at = {};
  if (cudaPointerGetAttributes(&at, ptr) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeDevice;
}

extern "C" pced_status pced_step_host_io(const pced_step_args* p, const float* beta_host, const float* r_host,
                                         int32_t* token_host, int32_t* expert_host, float* score_host,
                                         void* stream) {
  if (!p) return fail(PCED_ERR_INVALID_ARG, "pced_step_host_io: null args");
  if (p->key_out) return fail(PCED_ERR_INVALID_ARG, "pced_step_host_io: not for an expert-partitioned step");
  if ((token_host && !p->token_out) || (expert_host && !p->expert_out) || (score_host && !p->score_out))
    return fail(PCED_ERR_INVALID_ARG, "pced_step_host_io: a host output needs its device output in args");
  LmGeom g;
  int64_t num_blocks = 0;
  const pced_status chk = step_check(p, &g, &num_blocks);
  if (chk != PCED_OK) return chk;
  cudaStream_t s = (cudaStream_t)stream;
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(s, &cap) != cudaSuccess) return cuda_status(cudaGetLastError(), "capture query");
  if (cap == cudaStreamCaptureStatusNone) {
    const void* host[5] = {beta_host, r_host, token_host, expert_host, score_host};
    for (const void* h : host)
      if (h && is_device_memory(h))
        return fail(PCED_ERR_INVALID_ARG, "pced_step_host_io: a host buffer is device memory");
  }
  const size_t BN = (size_t)p->dims.B * p->dims.N, B = (size_t)p->dims.B;
  // Each copy costs a few microseconds of copy-engine latency on the step's
  // critical path, far more than its bytes: buffers that lie side by side on
  // both sides (r after beta; expert after token, score after expert) move
  // in one copy.
  auto adjacent = [](const void* a, const void* b, size_t bytes) {
    return (const char*)b == (const char*)a + bytes;
  };
  const bool one_in = beta_host && r_host && adjacent(beta_host, r_host, BN * 4) && adjacent(p->beta, p->r, BN * 4);
  const bool one_out = token_host && expert_host && score_host && adjacent(token_host, expert_host, B * 4) &&
                       adjacent(expert_host, score_host, B * 4) && adjacent(p->token_out, p->expert_out, B * 4) &&
                       adjacent(p->expert_out, p->score_out, B * 4);
  cudaError_t e = cudaSuccess;
  if (one_in) {
    e = cudaMemcpyAsync((void*)p->beta, beta_host, 2 * BN * sizeof(float), cudaMemcpyHostToDevice, s);
  } else {
    if (beta_host) e = cudaMemcpyAsync((void*)p->beta, beta_host, BN * sizeof(float), cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess && r_host)
      e = cudaMemcpyAsync((void*)p->r, r_host, BN * sizeof(float), cudaMemcpyHostToDevice, s);
  }
  if (e != cudaSuccess) return cuda_status(e, "pced_step_host_io: upload");
  const pced_status st = pced_step(p, stream);
  if (st != PCED_OK) return st;
  if (one_out) {
    e = cudaMemcpyAsync(token_host, p->token_out, 3 * B * 4, cudaMemcpyDeviceToHost, s);
  } else {
    if (token_host) e = cudaMemcpyAsync(token_host, p->token_out, B * sizeof(int32_t), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess && expert_host)
      e = cudaMemcpyAsync(expert_host, p->expert_out, B * sizeof(int32_t), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess && score_host)
      e = cudaMemcpyAsync(score_host, p->score_out, B * sizeof(float), cudaMemcpyDeviceToHost, s);
  }
  if (e != cudaSuccess) return cuda_status(e, "pced_step_host_io: read-back");
  return PCED_OK;
}
