/*
 * pced.h -- C ABI of the GB300 (sm_103a) implementation of one decode step of
 * Parallel Context-of-Experts Decoding (PCED, arXiv 2601.08670).
 *
 * The paper (Sec. 3, "Parallel Context-of-Experts") runs N+1 streams in one
 * batched pass: an amateur with no document (model prior) and N contextual
 * experts, each attending over its own independently encoded KV cache.  Each
 * step turns every expert's hidden state into log-probabilities s_k, scores
 *   shat_k = (1 + beta) s_k - beta s_0 + gamma log r_k          (Eq. 2)
 * and picks  y_t = argmax_v max_{k in 1..N} shat_k(v)            (Eq. 3),
 * then appends y_t to the shared history of all experts.
 *
 * Conventions shared by every entry point
 *   - All tensor pointers are DEVICE pointers owned by the caller (the one
 *     exception: the *_host buffers of pced_step_host_io, in host memory);
 *     the library allocates nothing and never synchronises.  `stream` is a
 *     cudaStream_t (NULL = legacy default stream).
 *   - bf16 tensors are raw bf16 arrays (2 bytes per element).
 *   - Sequences are query-major: sequence s = b*(N+1) + j belongs to query b;
 *     j = 0 is the amateur, j = 1..N are the contextual experts.
 *   - KV-cache slabs: for layer l, sequence s and kv-head h the keys (values)
 *     are cap[s] rows of D elements starting at element
 *         l*layer_elems + kv_offset[s] + h*cap[s]*D
 *     of k_cache (v_cache); rows [0, seq_len[s]) are live.
 *   - Every call validates its host-visible arguments before launching and
 *     returns a pced_status; nothing is launched on failure.  Conditions only
 *     visible on the device (a length above its capacity, a token outside the
 *     vocabulary, a full cache, a bounded wait that ran out) set bits of the
 *     32-bit device status word at byte 0 of the caller's workspace; the
 *     library only ORs bits into it, so the caller zeroes it once and reads it
 *     when convenient.
 *   - Workspaces must be 256-byte aligned and at least as large as the
 *     matching *_workspace_size() result.
 */
#ifndef PCED_H
#define PCED_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum pced_status {
  PCED_OK = 0,
  PCED_ERR_INVALID_ARG = 1, /* null pointer, inconsistent or out-of-range size */
  PCED_ERR_WORKSPACE = 2,   /* workspace too small or misaligned */
  PCED_ERR_UNSUPPORTED = 3, /* shape the kernels do not implement (see each call) */
  PCED_ERR_CUDA = 4,        /* a CUDA runtime/driver call failed */
  PCED_ERR_NO_DEVICE = 5    /* no usable sm_103 device */
} pced_status;

/* device status word bits (byte 0 of the workspace) */
#define PCED_DEV_BAD_LENGTH 0x1u  /* seq_len outside [1, cap] */
#define PCED_DEV_CACHE_FULL 0x2u  /* pced_step found no room for the new token */
#define PCED_DEV_TIMEOUT 0x4u     /* a bounded in-kernel wait expired */
#define PCED_DEV_BAD_TOKEN 0x8u   /* history token outside [0, V) */
#define PCED_DEV_STEP_LIMIT 0x10u /* step counter reached max_steps */
#define PCED_DEV_BAD_BLOCK 0x20u  /* paged caches: a needed block-table entry is missing or outside the pool */
#define PCED_DEV_BOUNDS 0x40u     /* bounds-checked build only: an index outside its buffer (the access was skipped) */

/* Static description of a status code (host). */
const char* pced_status_string(int32_t status);
/* Detail of the last failing call on this host thread (host, static storage). */
const char* pced_last_error(void);

typedef struct pced_dims {
  int32_t B;   /* independent queries */
  int32_t N;   /* contextual experts per query; the amateur is extra, S = B*(N+1) */
  int32_t L;   /* layers */
  int32_t Hq;  /* query heads */
  int32_t Hkv; /* kv heads (grouped-query attention, Hq % Hkv == 0) */
  int32_t D;   /* head dim; hidden size d = Hq*D */
  int32_t V;   /* vocabulary size */
} pced_dims;

/* ------------------------------------------------------------------------
 * pced_decode_attention -- one layer of decode attention for all S
 * sequences, each over its own cache (Sec. 3: each expert keeps its own KV
 * cache and attends only to it; grouped-query heads).
 *   q        bf16 [S][Hq][D]   query of the token being decoded
 *   k_cache, v_cache           bf16 cache region of THIS layer: slab (s, h)
 *                              at kv_offset[s] + h*cap[s]*D, cache_elems
 *                              elements in total
 *   kv_offset int64 [S], cap int32 [S], seq_len int32 [S] (device; the token
 *                              being decoded is already appended, so it is
 *                              row seq_len[s]-1 and attends to itself)
 *   total_cap                  host upper bound of sum(seq_len) (e.g. sum(cap));
 *                              sizes the grid only
 *   scale                      softmax scale, usually 1/sqrt(D)
 *   out      fp32 [S][Hq][D]   o = softmax(scale q K^T) V
 * Query head hq reads kv-head hq / (Hq/Hkv).  Supports D in {64, 128},
 * Hq/Hkv <= 8, cache_elems/D < 2^31, 16-byte aligned caches.
 * ------------------------------------------------------------------------ */
size_t pced_decode_attention_workspace_size(int32_t S, int32_t Hq, int32_t Hkv, int32_t D);
pced_status pced_decode_attention(const void* q, const void* k_cache, const void* v_cache, int64_t cache_elems,
                                  const int64_t* kv_offset, const int32_t* cap, const int32_t* seq_len, int32_t S,
                                  int32_t Hq, int32_t Hkv, int32_t D, int64_t total_cap, float scale, float* out,
                                  void* workspace, size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------
 * pced_decode_attention_noalloc -- pced_decode_attention for callers that
 * cannot allocate device memory when they need it (the paper has no
 * counterpart; this is a deployment convenience).  Examples: code that runs
 * while the caller's allocator is locked or shutting down, host callbacks
 * that must not enter the CUDA allocator, or an embedding runtime whose
 * memory pool is capped and owned by someone else.  The caller passes only
 * inputs and outputs; the split-KV partial records live in one fixed device
 * array inside this library, PCED_NOALLOC_SCRATCH_BYTES large, which every
 * GPU that loads the library reserves until the process exits.
 *   Arguments q ... out are those of pced_decode_attention.
 *   status   optional device int32 word the kernels OR PCED_DEV_* bits into
 *            (the caller zeroes it); NULL discards device-side conditions.
 * Sizes: the call needs about (SMs + S*Hkv) * (4*G*D + 8*G) + 8*S bytes of
 * scratch (G = Hq/Hkv, SMs = multiprocessors of the device); above
 * PCED_NOALLOC_SCRATCH_BYTES it returns PCED_ERR_UNSUPPORTED with the needed
 * size in pced_last_error() and launches nothing.  On a 152-SM device with
 * G = 4 and D = 128 that allows S*Hkv up to about 7900.
 * The call allocates no memory.  Its first call on a device (with that device
 * current) looks up the array's device address once, so make that first call
 * before any stream capture on the device.  Every call shares the one array
 * and overwrites it: calls that can overlap on the GPU (different streams, or
 * different host threads) race and give wrong results; serialise them.
 * Nothing in the array needs to start at zero.
 * ------------------------------------------------------------------------ */
#define PCED_NOALLOC_SCRATCH_BYTES (16u << 20)
pced_status pced_decode_attention_noalloc(const void* q, const void* k_cache, const void* v_cache,
                                          int64_t cache_elems, const int64_t* kv_offset, const int32_t* cap,
                                          const int32_t* seq_len, int32_t S, int32_t Hq, int32_t Hkv, int32_t D,
                                          int64_t total_cap, float scale, float* out, int32_t* status, void* stream);

/* ------------------------------------------------------------------------
 * pced_lm_head_logprobs -- per-expert log-probabilities s_k over the
 * vocabulary (Sec. 3: "per-expert logits s_k in R^|V|"; read as
 * log-softmax outputs, the scale Eq. 2 mixes).
 *   hidden    bf16 [S][d]   final normalised hidden states
 *   w_unembed bf16 [V][d]   unembedding matrix (row v = token v)
 *   logprobs  fp32 [S][V]   z - lse with z = hidden W^T
 *   lse       fp32 [S]      log sum_v exp(z[s][v])
 * Supports 1 <= S <= 512, d % 64 == 0, d <= 16384, 16-byte aligned rows.
 * ------------------------------------------------------------------------ */
size_t pced_lm_head_workspace_size(int32_t S, int32_t V);
pced_status pced_lm_head_logprobs(const void* hidden, const void* w_unembed, int32_t S, int32_t d, int32_t V,
                                  float* logprobs, float* lse, void* workspace, size_t workspace_bytes,
                                  void* stream);

/* ------------------------------------------------------------------------
 * pced_contrastive_select -- Eq. 2 and Eq. 3 on materialised log-probs.
 *   logprobs fp32 [S][V], S = B*(N+1), query-major, amateur first
 *   beta     fp32 [B][N]  contrastive strength of each expert (a broadcast beta_0)
 *   r        fp32 [B][N]  relevance scores, clipped on the device to [1e-8, 1]
 *   gamma                 weight of the retrieval prior
 *   token    int32 [B]    argmax_v max_k shat_k(v)
 *   expert   int32 [B]    maximising expert, 1-based
 *   score    fp32 [B]     the maximal shat
 * Exact ties go to the lowest token id, then the lowest expert index.
 * ------------------------------------------------------------------------ */
size_t pced_contrastive_select_workspace_size(int32_t B, int32_t N, int32_t V);
pced_status pced_contrastive_select(const float* logprobs, const float* beta, const float* r, float gamma, int32_t B,
                                    int32_t N, int32_t V, int32_t* token, int32_t* expert, float* score,
                                    void* workspace, size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------
 * pced_adacad_beta -- dynamic contrast strength for the first generated
 * token (Sec. 3 after Eq. 2: beta_0 is computed as in AdaCAD for the first
 * generated token and kept fixed thereafter).  Reading: one beta per
 * contextual expert, the Jensen-Shannon divergence in bits between the
 * expert's distribution p_k = exp(lp_k) and the amateur's p_0 = exp(lp_0),
 *   beta[b][k-1] = 1/2 sum_v [p_k log2(p_k/m) + p_0 log2(p_0/m)],  m = (p_k + p_0)/2,
 * so 0 <= beta <= 1.
 *   logprobs fp32 [B*(N+1)][V]  query-major, amateur first (device)
 *   beta     fp32 [B][N]        output (device)
 * Deterministic (fixed summation order).
 * ------------------------------------------------------------------------ */
size_t pced_adacad_beta_workspace_size(int32_t B, int32_t N, int32_t V);
pced_status pced_adacad_beta(const float* logprobs, int32_t B, int32_t N, int32_t V, float* beta, void* workspace,
                             size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------
 * pced_relevance -- relevance scores r in [0, 1) for the retrieval prior of
 * Eq. 2 (Sec. 3 "Retrieval and relevance scoring": map retriever and
 * reranker scores to [0, 1) and fuse them by the harmonic mean; App.
 * "Normalization of Retrieval and Reranker Scores" gives the maps):
 *   ret_mode PCED_RET_DENSE (dense / ColBERT similarity in [-1, 1]):
 *       r_ret = clip((s + 1)/2, 0, 1 - eps)
 *   ret_mode PCED_RET_SPARSE (sparse lexical score, >= 0, unbounded):
 *       r_ret = clip((2/pi) atan(max(s, 0)), 0, 1 - eps)
 *   reranker logit z:  r_rer = clip(1/(1 + exp(-z)), 0, 1 - eps)
 *   r = 2 r_ret r_rer / (r_ret + r_rer + eps)   (the appendix's form, eps in the denominator)
 *   ret_scores fp32 [n] (device), rer_logits fp32 [n] (device) or NULL
 *   (then r = r_ret), r fp32 [n] output (device).  The paper uses eps = 1e-8.
 * Evaluated in fp64, rounded to fp32 once.  n = 0 does nothing.  Errors:
 * PCED_ERR_INVALID_ARG for n < 0, another mode, eps outside [0, 0.5), a
 * null or misaligned pointer.
 * ------------------------------------------------------------------------ */
#define PCED_RET_DENSE 0
#define PCED_RET_SPARSE 1
pced_status pced_relevance(const float* ret_scores, int32_t ret_mode, const float* rer_logits, int32_t n, double eps,
                           float* r, void* stream);

/* ------------------------------------------------------------------------
 * pced_step -- one full greedy decode step of all B queries (Sec. 3,
 * Eq. 2, Eq. 3 and the shared-history append) on the weight-free layer
 * chain used for synthetic workloads:
 *   x_0     = embed[y_{t-1}]           (y_{-1} = bos_token; shared by all experts of a query)
 *   layer l: u = bf16(rmsnorm(x_l));  append K row u[0:Hkv) and V row u[Hkv:2Hkv) (as heads)
 *            at position seq_len (then seq_len+1 rows are live)
 *            x_{l+1} = x_l + attention(u as [Hq][D], own cache of layer l)   (fp32)
 *   h       = bf16(rmsnorm(x_L))
 *   token   = Eq. 3 over Eq. 2 of log_softmax(h W^T); appended to history[b][t]
 * The step index t, lengths and history live on the device, so a captured
 * CUDA graph of one call can be replayed step after step.  Each call adds
 * one to *step and to every seq_len[s].  Requires 2*Hkv <= Hq plus the limits
 * of the three calls above.  The workspace must be zero-filled before the
 * first call: besides the status word it holds counters the kernels leave
 * at zero when they finish.
 * ------------------------------------------------------------------------ */
typedef struct pced_step_args {
  pced_dims dims;
  const void* embed;        /* bf16 [V][d] token embedding */
  const void* w_unembed;    /* bf16 [V][d] */
  void* k_cache;            /* bf16, L regions of layer_elems elements */
  void* v_cache;
  int64_t layer_elems;
  const int64_t* kv_offset; /* [S] */
  const int32_t* cap;       /* [S] rows per slab */
  int64_t total_cap;        /* host: sum of cap */
  int32_t* seq_len;         /* [S] live rows; +1 per step */
  int32_t* step;            /* [1] step counter t; +1 per step while t < max_steps (at the
                               limit nothing is appended and PCED_DEV_STEP_LIMIT is set) */
  int32_t* history;         /* [B][max_steps] chosen tokens */
  int32_t* expert_trace;    /* [B][max_steps] winning expert (1-based), may be NULL */
  float* score_trace;       /* [B][max_steps] winning score, may be NULL */
  /* [B][max_steps][2] near-tie margins of each choice (Eq. 3), may be NULL:
   * the token gap, score minus the best score at any other token over all
   * experts, and the expert gap, score minus the best other expert's score
   * at the chosen token (+inf with one expert).  MoE / PoE report the
   * aggregate's token gap and the attribution's margin in log(w p).  A
   * choice within a small gap is a near tie: its token or expert could flip
   * under a change of summation order. */
  float* gap_trace;
  int32_t max_steps;
  const float* beta;        /* [B][N] */
  const float* r;           /* [B][N] relevance scores */
  float gamma;
  float attn_scale;         /* usually 1/sqrt(D) */
  float rms_eps;            /* usually 1e-6 */
  int32_t bos_token;
  void* hidden_out;         /* optional bf16 [S][d]: h of this step */
  float* lse_out;           /* optional fp32 [S]: log-sum-exp of each row of h W^T */
  void* workspace;
  size_t workspace_bytes;
  /* Optional timing hooks: an array of pced_step_launch_count(args) + 1
   * cudaEvent_t handles (cast to void*).  Event 0 is recorded on `stream`
   * before the first launch and event i+1 right after launch i, so the time
   * between consecutive events is the device time of that launch (the
   * events keep consecutive launches from overlapping).  NULL (or fewer
   * events) disables recording. */
  void* const* stage_events;
  int32_t n_stage_events;
  /* Dynamic contrast strength: when beta_from_step is nonzero this call
   * computes beta from this step's distributions (as pced_adacad_beta), writes
   * it to beta_out (device fp32 [B][N], may be the array `beta` points to)
   * and uses it for this step's selection; the caller passes it as `beta` to
   * the later steps.  Meant for the first step of a decode; such a call
   * materialises the log-probabilities (S x V fp32 in the workspace) in a
   * logits pass of the LM head and selects from them (Eq. 3 on materialised
   * log-probabilities). */
  int32_t beta_from_step;
  float* beta_out;
  /* Paged caches (PagedAttention-style, as the paper serves): when
   * block_table is not NULL, k_cache / v_cache hold per layer a pool of
   * layer_elems / (Hkv*block_rows*D) blocks of [Hkv][block_rows][D]; row pos
   * of (sequence s, kv-head h) is row pos % block_rows of block
   * block_table[s*max_blocks + pos / block_rows].  kv_offset is then unused
   * (may be NULL); cap[s] still bounds the length and must not exceed
   * max_blocks*block_rows.  block_rows: a multiple of 64 (else
   * PCED_ERR_INVALID_ARG); S*max_blocks must stay below 2^31 (else
   * PCED_ERR_UNSUPPORTED).  A table entry outside [0, number of blocks) sets
   * PCED_DEV_BAD_BLOCK: its keys read as zeros and the appended row is not
   * stored.  The table is read, never written. */
  const int32_t* block_table;
  int32_t block_rows;
  int32_t max_blocks;
  /* Rotary position embedding (the paper's decoders, Llama-3.1 / Mistral /
   * Qwen3, are rotary models): when rope_theta > 0 the queries and the
   * appended key row of every layer are rotated by the new token's position
   * p = seq_len[s] before the step (its row in the cache), rotate-half
   * pairing (f, f + D/2) with angle fp32(p * fp32(rope_theta^(-2f/D))); the
   * value row is not rotated and the cached rows are taken as stored (already
   * rotated).  0: no rotation.  Negative or non-finite: PCED_ERR_INVALID_ARG. */
  float rope_theta;
  /* s_k of Eq. 2 (Sec. 3 "per-expert logits"): PCED_SCORE_LOGPROB (0, the
   * default reading: log-softmax) or PCED_SCORE_LOGIT (1: raw logits, so the
   * per-expert constant is gamma log r alone).  Used by the max rule. */
  int32_t score_mode;
  /* How experts are combined (appendix "Ablation of Expert Aggregation
   * Rule"): PCED_AGG_MAX (0, Eq. 3), PCED_AGG_MOE (1) or PCED_AGG_POE (2).
   * MoE / PoE read: p_k = softmax_v((1 + beta_k) lp_k - beta_k lp_0), weights
   * w_k = r_k / sum_j r_j (r clipped to [1e-8, 1]); MoE picks
   * argmax_v log sum_k w_k p_k(v), PoE argmax_v sum_k w_k log p_k(v); the
   * expert reported is argmax_k w_k p_k(token), the score the aggregate;
   * gamma and score_mode do not enter (a per-expert constant drops out of the
   * softmax).  These rules materialise the logits (S x V fp32 in the
   * workspace) and take four launches (see pced_step_launch_kind). */
  int32_t aggregation;
  /* How long (ns) a warp of the attention kernel waits for another warp or
   * CTA (a layer's input, a partial record, a pipeline stage) before it sets
   * PCED_DEV_TIMEOUT and unwinds; the kernel then returns without its
   * results.  0: 2 s.  A CTA still waits for its own tile copies in flight
   * (up to 2 s) before it exits. */
  uint64_t wait_limit_ns;
  /* Expert-partitioned step (the experts of a query spread over several
   * GPUs; each holds the amateur, W_U and its own experts): when key_out is
   * not NULL the call computes the best choice of its experts per query as a
   * packed key (pced_select_key, with expert index expert_base + k for its
   * k-th expert) into key_out [B] (device int64) and appends nothing: t,
   * history and the traces stay as they were (gap_trace is not written).
   * After a max-reduction of the keys over the GPUs, pced_step_commit
   * appends the common token on each.  Requires the max rule of Eq. 3
   * (aggregation PCED_AGG_MAX), V <= 2^20 and expert_base + N <= 4096 (else
   * PCED_ERR_UNSUPPORTED).  The cache appends of this step are made either
   * way (every GPU appends the same input token). */
  int32_t expert_base;
  int64_t* key_out;
  /* Optional per-call outputs at fixed device addresses (each may be NULL):
   * this call's chosen token, its expert (1-based) and its score per query
   * ([B] each), the values history / expert_trace / score_trace receive at t.
   * The traces move with t; these do not, so a captured CUDA graph of the call
   * (or of pced_step_host_io) finds each step's choice at the same address.
   * An expert-partitioned call (key_out) does not write them. */
  int32_t* token_out;
  int32_t* expert_out;
  float* score_out;
} pced_step_args;

#define PCED_SCORE_LOGPROB 0
#define PCED_SCORE_LOGIT 1
#define PCED_AGG_MAX 0
#define PCED_AGG_MOE 1
#define PCED_AGG_POE 2

/* ------------------------------------------------------------------------
 * The choice of Eq. 3 as one int64 whose signed order is Eq. 3's order: the
 * higher score first, then the lower token id, then the lower expert index
 * (host; the device packs the same bits).  token in [0, 2^20), expert
 * (1-based, global) in [1, 4096].  The maximum of the keys of disjoint sets
 * of a query's experts is the key of the choice over their union (Eq. 3
 * couples experts only through this max), so an all-reduce-max of int64
 * (NCCL, gloo, torch.maximum) is the only exchange an expert-partitioned
 * step needs.  Unpack returns the fp32 score exactly; NULL outputs are skipped.
 * ------------------------------------------------------------------------ */
int64_t pced_select_key(float score, int32_t token, int32_t expert);
void pced_select_key_unpack(int64_t key, float* score, int32_t* token, int32_t* expert);

/* Append the reduced choices of an expert-partitioned step: for each query
 * b, history[b][t] = token, expert_trace / score_trace (may be NULL) from
 * keys[b] (device int64 [B]), then t += 1 (step, device int32).  A t outside
 * [0, max_steps) writes nothing and sets PCED_DEV_STEP_LIMIT in *status
 * (device, may be NULL).  One launch on `stream`. */
pced_status pced_step_commit(const int64_t* keys, int32_t B, int32_t* step, int32_t* history, int32_t* expert_trace,
                             float* score_trace, int32_t max_steps, int* status, void* stream);

size_t pced_step_workspace_size(const pced_dims* dims);
pced_status pced_step(const pced_step_args* args, void* stream);

/* One decode step with its per-step inputs and outputs in host memory, as a
 * serving loop runs it (Sec. 3: every step scores the experts with their
 * retrieval-derived weights r_k and contrast strengths beta_k of Eq. 2, and
 * the chosen token leaves the GPU to be emitted).  In stream order:
 *   1. beta_host, r_host (host fp32 [B][N] each; NULL: leave the device
 *      values) are copied into the device arrays args->beta and args->r
 *      point to (this call writes them);
 *   2. pced_step(args, stream);
 *   3. the step's choice is copied from args->token_out / expert_out /
 *      score_out into token_host / expert_host / score_host (host [B] each;
 *      NULL: not copied).
 * The call returns without waiting: the host outputs hold the step's values
 * once the stream has passed the call (synchronise it or an event recorded
 * after it).  Host buffers should be page-locked (cudaHostAlloc or
 * cudaHostRegister): the copies are then asynchronous, and a stream capture
 * of the call records them as graph nodes, so one graph replay is one step
 * with its uploads and read-backs; pageable buffers are staged by the CUDA
 * runtime and may block the calling thread.  Each copy adds a few
 * microseconds of latency to the step: buffers that lie side by side on both
 * sides (r right after beta; expert right after token, score right after
 * expert) move in one copy each way.  Errors (nothing is enqueued):
 * PCED_ERR_INVALID_ARG for a host output without its device output in args,
 * for an expert-partitioned call (key_out set) and, outside a stream capture,
 * for a "host" pointer that is device memory; any error pced_step reports
 * for args.  With beta_from_step the step overwrites beta_out after the
 * upload (upload nothing then, or a starting beta that is ignored). */
pced_status pced_step_host_io(const pced_step_args* args, const float* beta_host, const float* r_host,
                              int32_t* token_host, int32_t* expert_host, float* score_host, void* stream);

/* Number of kernel launches one pced_step call with these arguments makes:
 * 3 for the max rule with a fixed beta (attention, LM head, selection); a
 * first step with beta_from_step runs attention, a logits pass, its
 * log-sum-exp finalise, the beta kernel and a selection from the
 * log-probabilities (5); MoE / PoE run attention, the logits pass and two
 * aggregation kernels, which read the raw logits (4; with beta_from_step
 * also the finalise and the beta kernel, 6).  Only the
 * fields dims, beta_from_step and aggregation are read; NULL gives 0. */
int32_t pced_step_launch_count(const pced_step_args* args);
/* Kind of launch i (0-based) of such a call: "attention", "lm_head",
 * "lse_finalize", "adacad_beta", "agg_partials", "agg_select" or "select";
 * NULL when out of range (static storage). */
const char* pced_step_launch_kind(const pced_step_args* args, int32_t i);

#ifdef __cplusplus
}
#endif
#endif /* PCED_H */
