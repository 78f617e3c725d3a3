// aggregate.cu -- aggregation variants of the experts (appendix "Ablation of
// Expert Aggregation Rule": Mixture-of-Experts, a weighted sum, and
// Product-of-Experts, a weighted product, in probability space, with weights
// from the retrieval scores).  Reading (the paper prints no formula):
//   c_k(v) = (1 + beta_k) lp_k(v) - beta_k lp_0(v)      (Eq. 2 without the prior)
//   p_k = softmax_v c_k,  w_k = r~_k / sum_j r~_j       (r~: r clipped to [1e-8, 1])
//   MoE: agg(v) = log sum_k w_k p_k(v)     PoE: agg(v) = sum_k w_k log p_k(v)
//   token = argmax_v agg (lowest id on ties), score = agg(token),
//   expert = argmax_k w_k p_k(token) (lowest k on ties).
// Two launches over the materialised log-probabilities (S x V fp32, a few MB,
// L2-resident): (1) per (query, expert, chunk) the max and sum of exp of c_k,
// merged into the expert's log-sum-exp by the last chunk to finish; (2) per
// (query, chunk) the best aggregate and the best at another token; the last
// CTA of a query picks the token across chunks, attributes the expert and
// writes the step's results with both near-tie margins.  Every sum runs in a
// fixed order, so results do not depend on timing.
#include <math.h>

#include "aggregate.cuh"
#include "select_key.cuh"

namespace pced {

constexpr int AGG_THREADS = 256;

__device__ __forceinline__ void agg_lse_merge(float& m, float& s, float m2, float s2) {
  if (m2 == -INFINITY) return;
  if (m == -INFINITY) {
    m = m2;
    s = s2;
    return;
  }
  const float M = fmaxf(m, m2);
  s = s * expf(m - M) + s2 * expf(m2 - M);
  m = M;
}

// grid (nchunks, N, B): the chunk's (max, sum exp) of c_k; the last chunk CTA
// of (query, expert) to finish merges them all into lse_k (strided, then a
// fixed tree: the order does not depend on which CTA is last)
__global__ void __launch_bounds__(AGG_THREADS) agg_partials_kernel(AggArgs a) {
  const int c = blockIdx.x, k = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
  const int N = a.N, V = a.V;
  const float* lp0 = a.lp + (int64_t)b * (N + 1) * V;
  const float* lpk = lp0 + (int64_t)(k + 1) * V;
  const float bt = a.beta[b * N + k];
  __shared__ float2 red[AGG_THREADS / 32];
  __shared__ int last;
  auto block_merge = [&](float m, float s) -> float2 {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, m, o), s2 = __shfl_xor_sync(0xffffffffu, s, o);
      agg_lse_merge(m, s, m2, s2);
    }
    if ((tid & 31) == 0) red[tid >> 5] = make_float2(m, s);
    __syncthreads();
    float M = -INFINITY, Sm = 0.f;
    for (int w = 0; w < AGG_THREADS / 32; ++w) agg_lse_merge(M, Sm, red[w].x, red[w].y);
    __syncthreads();
    return make_float2(M, Sm);
  };
  if (a.rec_stats && c == 0) {
    // raw logits: the log-sum-exps of expert k's row (and, for k = 0, the
    // amateur's) from the LM head's tile records, in a fixed order
    for (int r = 0; r < (k == 0 ? 2 : 1); ++r) {
      const int64_t row = (int64_t)b * (N + 1) + (r == 0 ? k + 1 : 0);
      float mm = -INFINITY, ss = 0.f;
      for (int j = tid; j < a.nrec; j += AGG_THREADS) {
        const float2 e = a.rec_stats[row * a.nrec + j];
        agg_lse_merge(mm, ss, e.x, e.y);
      }
      const float2 t = block_merge(mm, ss);
      if (tid == 0) a.lse_rows[row] = t.x + logf(t.y);
    }
  }
  float m = -INFINITY, s = 0.f;
  const int v1 = min(V, (c + 1) * AGG_CHUNK);
  for (int v = c * AGG_CHUNK + tid; v < v1; v += AGG_THREADS) {
    const float ck = (1.f + bt) * lpk[v] - bt * lp0[v];
    agg_lse_merge(m, s, ck, 1.f);
  }
  const float2 ms = block_merge(m, s);
  const int64_t pk = (int64_t)b * N + k;
  if (tid == 0) {
    a.part[pk * a.nchunks + c] = ms;
    __threadfence();
    last = atomicAdd(a.kdone + pk, 1) == a.nchunks - 1;
  }
  __syncthreads();
  if (!last) return;
  __threadfence();  // the other chunks' statistics are visible
  m = -INFINITY;
  s = 0.f;
  for (int j = tid; j < a.nchunks; j += AGG_THREADS) {
    const float2 e = __ldcg(a.part + pk * a.nchunks + j);
    agg_lse_merge(m, s, e.x, e.y);
  }
  const float2 t = block_merge(m, s);
  if (tid == 0) {
    a.lse_k[pk] = t.x + logf(t.y);
    a.kdone[pk] = 0;
  }
}

// (value, token) order: larger value, then lower token
__device__ __forceinline__ bool agg_better(float v2, int t2, float v1, int t1) {
  return v2 > v1 || (v2 == v1 && t2 < t1);
}
// top-2 over disjoint token sets: (b1, t1) best, b2 best value at another token
__device__ __forceinline__ void agg_top2(float& b1, int& t1, float& b2, float r1, int rt, float r2) {
  if (agg_better(r1, rt, b1, t1)) {
    b2 = fmaxf(b1, r2);
    b1 = r1;
    t1 = rt;
  } else {
    b2 = fmaxf(b2, r1);
  }
}

// grid (nchunks, B).  rule 0 is Eq. 3 itself on the materialised
// log-probabilities: per token the best expert's score of Eq. 2 (the first
// step of a dynamic-beta decode selects this way, from the log-probabilities
// it has written for beta anyway); rules 1 and 2 are MoE and PoE.
__global__ void __launch_bounds__(AGG_THREADS) agg_select_kernel(AggArgs a) {
  const int c = blockIdx.x, b = blockIdx.y, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int N = a.N, V = a.V, n1 = N + 1;
  __shared__ float w_s[AGG_MAX_N], lse_s[AGG_MAX_N], beta_s[AGG_MAX_N];
  __shared__ float wsum;
  __shared__ float bv_s[AGG_THREADS / 32], b2_s[AGG_THREADS / 32];
  __shared__ int bt_s[AGG_THREADS / 32];
  __shared__ int last;
  if (c == 0 && b == 0 && tid == 0 && a.tile_ctr) *a.tile_ctr = 0;  // the next LM head claims its tiles from 0
  for (int k = tid; k < N; k += AGG_THREADS) {
    w_s[k] = fminf(fmaxf(a.r[b * N + k], 1e-8f), 1.0f);
    beta_s[k] = a.beta[b * N + k];
    if (a.rule == 0) {
      // the per-expert constant of Eq. 2: gamma log r_k (plus the log-sum-exps
      // when s_k are raw logits: z = lp + L)
      const float btk = beta_s[k];
      lse_s[k] = a.gamma * logf(w_s[k]) +
                 (a.raw_logits ? (1.f + btk) * a.lse[b * n1 + 1 + k] - btk * a.lse[b * n1] : 0.f);
    } else {
      lse_s[k] = a.lse_k[(int64_t)b * N + k];
    }
  }
  __syncthreads();
  if (tid == 0) {
    float t = 0.f;
    for (int k = 0; k < N; ++k) t += w_s[k];
    wsum = t;
  }
  __syncthreads();
  const float inv_w = 1.0f / wsum;
  const float* lp0 = a.lp + (int64_t)b * n1 * V;
  // the chunk's best aggregate and token, and the best at another token
  float bv = -INFINITY, b2 = -INFINITY;
  int bt = 0x7fffffff;
  const int v1 = min(V, (c + 1) * AGG_CHUNK);
  for (int v = c * AGG_CHUNK + tid; v < v1; v += AGG_THREADS) {
    const float l0 = lp0[v];
    float acc = a.rule == 0 ? -INFINITY : 0.f;
    for (int k = 0; k < N; ++k) {
      if (a.rule == 0) {
        acc = fmaxf(acc, (1.f + beta_s[k]) * lp0[(int64_t)(k + 1) * V + v] - beta_s[k] * l0 + lse_s[k]);
        continue;
      }
      const float lpk = (1.f + beta_s[k]) * lp0[(int64_t)(k + 1) * V + v] - beta_s[k] * l0 - lse_s[k];  // log p_k(v)
      acc += a.rule == 1 ? w_s[k] * inv_w * expf(lpk) : w_s[k] * inv_w * lpk;
    }
    const float agg = a.rule == 1 ? logf(acc) : acc;
    agg_top2(bv, bt, b2, agg, v, -INFINITY);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float v2 = __shfl_xor_sync(0xffffffffu, bv, o), s2 = __shfl_xor_sync(0xffffffffu, b2, o);
    const int t2 = __shfl_xor_sync(0xffffffffu, bt, o);
    agg_top2(bv, bt, b2, v2, t2, s2);
  }
  if (lane == 0) {
    bv_s[warp] = bv;
    bt_s[warp] = bt;
    b2_s[warp] = b2;
  }
  __syncthreads();
  if (tid == 0) {
    for (int w = 1; w < AGG_THREADS / 32; ++w) agg_top2(bv, bt, b2, bv_s[w], bt_s[w], b2_s[w]);
    a.best[(int64_t)b * a.nchunks + c] = make_float2(bv, __int_as_float(bt));
    a.best2[(int64_t)b * a.nchunks + c] = b2;
    __threadfence();
    last = atomicAdd(a.qdone + b, 1) == a.nchunks - 1;
  }
  __syncthreads();
  if (!last || warp != 0) return;
  __threadfence();  // the other chunks' results of query b are visible
  // best over the chunks (one warp, lanes over chunks, then a tree)
  float sv = -INFINITY, sv2 = -INFINITY;
  int st = 0x7fffffff;
  for (int j = lane; j < a.nchunks; j += 32) {
    const float2 e = __ldcg(a.best + (int64_t)b * a.nchunks + j);
    agg_top2(sv, st, sv2, e.x, __float_as_int(e.y), __ldcg(a.best2 + (int64_t)b * a.nchunks + j));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float v2 = __shfl_xor_sync(0xffffffffu, sv, o), s2 = __shfl_xor_sync(0xffffffffu, sv2, o);
    const int t2 = __shfl_xor_sync(0xffffffffu, st, o);
    agg_top2(sv, st, sv2, v2, t2, s2);
  }
  if (st >= V) st = 0;  // no finite aggregate (degenerate rows): token 0
  // the expert: for Eq. 3 the best score at the token, for MoE / PoE the
  // one that puts the most weighted mass on it (log(w p)); lowest k on
  // ties, and the margin to the next one
  float bp = -INFINITY, bp2 = -INFINITY;
  int bk = 0x7fffffff;
  for (int k = lane; k < N; k += 32) {
    const float ck = (1.f + beta_s[k]) * lp0[(int64_t)(k + 1) * V + st] - beta_s[k] * lp0[st];
    agg_top2(bp, bk, bp2, a.rule == 0 ? ck + lse_s[k] : logf(w_s[k]) + ck - lse_s[k], k, -INFINITY);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float v2 = __shfl_xor_sync(0xffffffffu, bp, o), s2 = __shfl_xor_sync(0xffffffffu, bp2, o);
    const int t2 = __shfl_xor_sync(0xffffffffu, bk, o);
    agg_top2(bp, bk, bp2, v2, t2, s2);
  }
  if (bk >= N) bk = 0;
  if (lane != 0) return;
  a.qdone[b] = 0;
  if (a.lse_out)
    for (int j = 0; j < n1; ++j) a.lse_out[b * n1 + j] = a.lse[b * n1 + j];
  if (a.key_out) {  // expert-partitioned step (rule 0): the reduction and the append come after
    a.key_out[b] = select_key(sv, st, a.expert_base + bk + 1);
    return;
  }
  if (a.token) a.token[b] = st;
  if (a.expert) a.expert[b] = bk + 1;
  if (a.score) a.score[b] = sv;
  if (a.step) {
    const int t = *a.step;
    if (t >= 0 && t < a.max_steps) {
      a.history[(int64_t)b * a.max_steps + t] = st;
      if (a.expert_trace) a.expert_trace[(int64_t)b * a.max_steps + t] = bk + 1;
      if (a.score_trace) a.score_trace[(int64_t)b * a.max_steps + t] = sv;
      if (a.gap_trace) a.gap_trace[(int64_t)b * a.max_steps + t] = make_float2(sv - sv2, bp - bp2);
    } else {
      dev_flag(a.status, PCED_DEV_STEP_LIMIT);
    }
    __threadfence();
    if (atomicAdd(a.done_counter, 1) == a.B - 1) {
      if (t >= 0 && t < a.max_steps) *a.step = t + 1;  // at the limit t stays (as the commit does)
      *a.done_counter = 0;
      __threadfence();
    }
  }
}

cudaError_t agg_partials_launch(const AggArgs& a, cudaStream_t stream) {
  agg_partials_kernel<<<dim3(a.nchunks, a.N, a.B), AGG_THREADS, 0, stream>>>(a);
  return cudaGetLastError();
}

cudaError_t agg_select_launch(const AggArgs& a, cudaStream_t stream) {
  agg_select_kernel<<<dim3(a.nchunks, a.B), AGG_THREADS, 0, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace pced
