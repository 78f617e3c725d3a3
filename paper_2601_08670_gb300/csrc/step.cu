// step.cu -- one greedy PCED decode step for all queries (paper Sec. 3: the
// N+1 experts run as one batch; Eq. 2 + Eq. 3 pick the token, which joins
// every expert's history).  Launch sequence on one stream, no host sync:
//   embed      x_0 = E[y_{t-1}], u = bf16(rmsnorm(x_0)), append layer-0 K/V, seq_len += 1
//   L times    split-KV attention, then combine: x += o, u = bf16(rmsnorm(x)),
//              append the next layer's K/V (or write h after the last layer)
//   lm head    tcgen05 GEMM with log-softmax statistics + contrastive tile maxima
//   select     Eq. 2 + Eq. 3 per query, history[b][t] = y, t += 1
// Every quantity that changes between steps (t, lengths, history) lives on
// the device, so one captured call replays as the next step.
#include <math.h>

#include "attention.cuh"
#include "lm_head.cuh"

namespace pced {

constexpr int EMB_THREADS = 256;
constexpr int EMB_MAX_PER_THREAD = 32;  // d <= 8192

struct EmbedArgs {
  const __nv_bfloat16* embed;
  int32_t S, n1, d, Hkv, D, V, max_steps, bos;
  const int32_t* step;
  const int32_t* history;
  int32_t* seq_len;
  const int32_t* cap;
  const int64_t* kv_offset;
  __nv_bfloat16* k_cache;
  __nv_bfloat16* v_cache;
  float* resid;
  __nv_bfloat16* q;
  float rms_eps;
  int* status;
};

__global__ void __launch_bounds__(EMB_THREADS) step_embed_kernel(EmbedArgs a) {
  const int s = blockIdx.x, tid = threadIdx.x, b = s / a.n1, d = a.d;
  __shared__ int sh_tok, sh_pos;
  __shared__ float red[EMB_THREADS / 32];
  if (tid == 0) {
    const int t = *a.step;
    int tok = a.bos;
    if (t > 0 && t <= a.max_steps) tok = a.history[(int64_t)b * a.max_steps + t - 1];
    if (t >= a.max_steps) dev_flag(a.status, PCED_DEV_STEP_LIMIT);
    if (tok < 0 || tok >= a.V) {
      dev_flag(a.status, PCED_DEV_BAD_TOKEN);
      tok = 0;
    }
    const int L = a.seq_len[s], c = a.cap[s];
    int pos = -1;
    if (L < 0 || L >= c) {
      dev_flag(a.status, PCED_DEV_CACHE_FULL);
    } else {
      a.seq_len[s] = L + 1;
      pos = L;
    }
    sh_tok = tok;
    sh_pos = pos;
  }
  __syncthreads();
  const __nv_bfloat16* e = a.embed + (int64_t)sh_tok * d;
  float xv[EMB_MAX_PER_THREAD];
  float ss = 0.f;
#pragma unroll
  for (int j = 0; j < EMB_MAX_PER_THREAD; ++j) {
    const int i = tid + j * EMB_THREADS;
    xv[j] = 0.f;
    if (i < d) {
      xv[j] = __bfloat162float(e[i]);
      a.resid[(int64_t)s * d + i] = xv[j];
      ss += xv[j] * xv[j];
    }
  }
  ss = warp_sum(ss);
  if ((tid & 31) == 0) red[tid >> 5] = ss;
  __syncthreads();
  if (tid < 32) {
    float v = tid < EMB_THREADS / 32 ? red[tid] : 0.f;
    v = warp_sum(v);
    if (tid == 0) red[0] = v;
  }
  __syncthreads();
  const float inv = 1.0f / sqrtf(red[0] / (float)d + a.rms_eps);
  const int pos = sh_pos, capv = a.cap[s];
#pragma unroll
  for (int j = 0; j < EMB_MAX_PER_THREAD; ++j) {
    const int i = tid + j * EMB_THREADS;
    if (i >= d) continue;
    const __nv_bfloat16 u = __float2bfloat16_rn(xv[j] * inv);
    a.q[(int64_t)s * d + i] = u;
    if (pos >= 0 && i < 2 * a.Hkv * a.D) {
      const int hh = i / a.D, dd = i - hh * a.D;
      const bool isv = hh >= a.Hkv;
      const int hk = isv ? hh - a.Hkv : hh;
      const int64_t el = a.kv_offset[s] + ((int64_t)hk * capv + pos) * a.D + dd;
      (isv ? a.v_cache : a.k_cache)[el] = u;
    }
  }
}

struct StepLayout {
  int* status;
  float* resid;
  __nv_bfloat16* q;
  __nv_bfloat16* h;
  float* rec_o;
  float2* rec_ml;
  int64_t* plan_pre;
  int64_t* plan_per;
  float2* lm_stats;
  float2* lm_arg;
  int32_t* done_counter;
  float* part_ss;
  int32_t* seq_counters;
  size_t bytes;
};

static StepLayout step_layout(const pced_dims* dm, void* ws) {
  const int32_t S = dm->B * (dm->N + 1), d = dm->Hq * dm->D, G = dm->Hq / dm->Hkv;
  const int64_t slots = ATT_MAX_CTAS + (int64_t)S * dm->Hkv;
  const int64_t ntiles = (dm->V + LM_TILE_V - 1) / LM_TILE_V;
  StepLayout L;
  pced_host::Carver c(ws);
  L.status = c.take<int>(64);
  L.done_counter = c.take<int32_t>(1);
  L.seq_counters = c.take<int32_t>((size_t)S);
  L.part_ss = c.take<float>((size_t)S * dm->Hkv);
  L.resid = c.take<float>((size_t)S * d);
  L.q = c.take<__nv_bfloat16>((size_t)S * d);
  L.h = c.take<__nv_bfloat16>((size_t)S * d);
  L.rec_o = c.take<float>((size_t)(slots * G * dm->D));
  L.rec_ml = c.take<float2>((size_t)(slots * G));
  L.plan_pre = c.take<int64_t>((size_t)S + 1);
  L.plan_per = c.take<int64_t>(1);
  L.lm_stats = c.take<float2>((size_t)(S * ntiles));
  L.lm_arg = c.take<float2>((size_t)(S * ntiles));
  L.bytes = c.used();
  return L;
}

}  // namespace pced

using namespace pced;
using namespace pced_host;

extern "C" size_t pced_step_workspace_size(const pced_dims* dm) {
  if (!dm || dm->B < 1 || dm->N < 1 || dm->Hq < 1 || dm->Hkv < 1 || dm->D < 1 || dm->V < 1 || dm->Hq % dm->Hkv)
    return 0;
  return step_layout(dm, nullptr).bytes;
}

extern "C" int32_t pced_step_launch_count(const pced_dims* dm) { return dm ? 1 + 2 * dm->L + 2 : 0; }

extern "C" const char* pced_step_launch_kind(const pced_dims* dm, int32_t i) {
  if (!dm || i < 0 || i >= pced_step_launch_count(dm)) return nullptr;
  if (i == 0) return "embed";
  if (i <= 2 * dm->L) return (i % 2 == 1) ? "attn_split" : "attn_combine";
  return i == 2 * dm->L + 1 ? "lm_head" : "select";
}

extern "C" pced_status pced_step(const pced_step_args* p, void* stream) {
  if (!p) return fail(PCED_ERR_INVALID_ARG, "pced_step: null args");
  const pced_dims dm = p->dims;
  if (!p->embed || !p->w_unembed || !p->k_cache || !p->v_cache || !p->kv_offset || !p->cap || !p->seq_len ||
      !p->step || !p->history || !p->beta || !p->r || !p->workspace)
    return fail(PCED_ERR_INVALID_ARG, "pced_step: null pointer");
  if (dm.B < 1 || dm.N < 1 || dm.L < 1 || dm.Hq < 1 || dm.Hkv < 1 || dm.D < 1 || dm.V < 1 || dm.Hq % dm.Hkv != 0 ||
      2 * dm.Hkv > dm.Hq || p->max_steps < 1 || p->layer_elems < dm.D || p->total_cap < 1)
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
  LmGeom g;
  if (!lm_geometry(S, d, dm.V, &g)) return fail(PCED_ERR_UNSUPPORTED, "pced_step: LM-head shape unsupported");
  if ((((uintptr_t)p->k_cache) | ((uintptr_t)p->v_cache) | ((uintptr_t)p->w_unembed) | ((uintptr_t)p->embed)) & 15u)
    return fail(PCED_ERR_INVALID_ARG, "pced_step: tensors must be 16-byte aligned");
  if (((uintptr_t)p->workspace) & 255u || p->workspace_bytes < pced_step_workspace_size(&dm))
    return fail(PCED_ERR_WORKSPACE, "pced_step: workspace too small or misaligned");
  if (num_sms() <= 0) return fail(PCED_ERR_NO_DEVICE, "pced_step: no CUDA device");

  const StepLayout W = step_layout(&dm, p->workspace);
  CUtensorMap kmap, vmap, wmap, hmap;
  const uint64_t rows = (uint64_t)dm.L * (uint64_t)(p->layer_elems / dm.D);
  pced_status st = make_tmap_2d(&kmap, p->k_cache, rows, (uint64_t)dm.D, ATT_BLOCK_N, 64, true);
  if (st == PCED_OK) st = make_tmap_2d(&vmap, p->v_cache, rows, (uint64_t)dm.D, ATT_BLOCK_N, 64, true);
  if (st == PCED_OK) st = make_tmap_2d(&wmap, p->w_unembed, (uint64_t)dm.V, (uint64_t)d, LM_TILE_V, LM_TILE_K, true);
  if (st == PCED_OK) st = make_tmap_2d(&hmap, W.h, (uint64_t)S, (uint64_t)d, (uint32_t)g.chunk_n, LM_TILE_K, false);
  if (st != PCED_OK) return st;
  cudaStream_t s = (cudaStream_t)stream;
  const bool timed = p->stage_events && p->n_stage_events >= pced_step_launch_count(&dm) + 1;
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
  cudaError_t e = mark();
  if (e != cudaSuccess) return cuda_status(e, "stage event");

  EmbedArgs ea;
  ea.embed = (const __nv_bfloat16*)p->embed;
  ea.S = S;
  ea.n1 = dm.N + 1;
  ea.d = d;
  ea.Hkv = dm.Hkv;
  ea.D = dm.D;
  ea.V = dm.V;
  ea.max_steps = p->max_steps;
  ea.bos = p->bos_token;
  ea.step = p->step;
  ea.history = p->history;
  ea.seq_len = p->seq_len;
  ea.cap = p->cap;
  ea.kv_offset = p->kv_offset;
  ea.k_cache = (__nv_bfloat16*)p->k_cache;
  ea.v_cache = (__nv_bfloat16*)p->v_cache;
  ea.resid = W.resid;
  ea.q = W.q;
  ea.rms_eps = p->rms_eps;
  ea.status = W.status;
  step_embed_kernel<<<S, EMB_THREADS, 0, s>>>(ea);
  e = cudaGetLastError();
  if (e == cudaSuccess) e = mark();
  if (e != cudaSuccess) return cuda_status(e, "embed launch");

  const int ctas = att_grid(p->total_cap * dm.Hkv);
  for (int l = 0; l < dm.L; ++l) {
    AttArgs a;
    a.q = W.q;
    a.kv_offset = p->kv_offset;
    a.cap = p->cap;
    a.seq_len = p->seq_len;
    a.S = S;
    a.Hq = dm.Hq;
    a.Hkv = dm.Hkv;
    a.G = G;
    a.row_base = (int64_t)l * (p->layer_elems / dm.D);
    a.scale_log2 = p->attn_scale * 1.4426950408889634f;
    a.rec_o = W.rec_o;
    a.rec_ml = W.rec_ml;
    a.plan_pre = W.plan_pre;
    a.plan_per = W.plan_per;
    a.status = W.status;
    e = att_split_launch(dm.D, kmap, vmap, a, ctas, s);
    if (e == cudaSuccess) e = mark();
    if (e != cudaSuccess) return cuda_status(e, "attention split launch");
    CombineArgs c = {};
    c.mode = 1;
    c.S = S;
    c.Hq = dm.Hq;
    c.Hkv = dm.Hkv;
    c.G = G;
    c.D = dm.D;
    c.rec_o = W.rec_o;
    c.rec_ml = W.rec_ml;
    c.plan_pre = W.plan_pre;
    c.plan_per = W.plan_per;
    c.seq_len = p->seq_len;
    c.resid = W.resid;
    c.part_ss = W.part_ss;
    c.counters = W.seq_counters;
    c.rms_eps = p->rms_eps;
    c.k_cache = (__nv_bfloat16*)p->k_cache;
    c.v_cache = (__nv_bfloat16*)p->v_cache;
    c.kv_offset = p->kv_offset;
    c.cap = p->cap;
    c.status = W.status;
    if (l + 1 < dm.L) {
      c.append = 1;
      c.q_next = W.q;
      c.next_layer_elem_base = (int64_t)(l + 1) * p->layer_elems;
    } else {
      c.append = 0;
      c.hidden = W.h;
      c.hidden_copy = (__nv_bfloat16*)p->hidden_out;
    }
    e = att_combine_launch(c, s);
    if (e == cudaSuccess) e = mark();
    if (e != cudaSuccess) return cuda_status(e, "attention combine launch");
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
  la.nbeta = dm.B * dm.N;
  la.stages = g.stages;
  la.acc_bufs = g.acc_bufs;
  la.S_pad = g.S_pad;
  la.nchunk = g.nchunk;
  la.chunk_n = g.chunk_n;
  la.tmem_cols = g.tmem_cols;
  la.rec_stats = W.lm_stats;
  la.rec_arg = W.lm_arg;
  la.beta = p->beta;
  la.status = W.status;
  e = lm_head_launch(wmap, hmap, g, la, s);
  if (e == cudaSuccess) e = mark();
  if (e != cudaSuccess) return cuda_status(e, "lm head launch");

  SelectArgs sa = {};
  sa.rec_stats = W.lm_stats;
  sa.rec_arg = W.lm_arg;
  sa.B = dm.B;
  sa.N = dm.N;
  sa.nrec = g.grid;
  sa.beta = p->beta;
  sa.r = p->r;
  sa.gamma = p->gamma;
  sa.lse_out = p->lse_out;
  sa.step = p->step;
  sa.history = p->history;
  sa.expert_trace = p->expert_trace;
  sa.score_trace = p->score_trace;
  sa.max_steps = p->max_steps;
  sa.done_counter = W.done_counter;
  sa.status = W.status;
  e = select_from_records_launch(sa, s);
  if (e == cudaSuccess) e = mark();
  if (e != cudaSuccess) return cuda_status(e, "select launch");
  return PCED_OK;
}
