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
// L2-resident): (1) per (query, expert, chunk) the max and sum of exp of c_k;
// (2) per (query, chunk) the best aggregate, every CTA first merging the
// chunk statistics of its query into log-sum-exps; the last CTA of a query
// picks the token across chunks and writes the step's results.  Every sum
// runs in a fixed order, so results do not depend on timing.
#include <math.h>

#include "aggregate.cuh"

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

// grid (nchunks, N, B)
__global__ void __launch_bounds__(AGG_THREADS) agg_partials_kernel(AggArgs a) {
  const int c = blockIdx.x, k = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
  const int N = a.N, V = a.V;
  const float* lp0 = a.lp + (int64_t)b * (N + 1) * V;
  const float* lpk = lp0 + (int64_t)(k + 1) * V;
  const float bt = a.beta[b * N + k];
  float m = -INFINITY, s = 0.f;
  const int v1 = min(V, (c + 1) * AGG_CHUNK);
  for (int v = c * AGG_CHUNK + tid; v < v1; v += AGG_THREADS) {
    const float ck = (1.f + bt) * lpk[v] - bt * lp0[v];
    agg_lse_merge(m, s, ck, 1.f);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o), s2 = __shfl_xor_sync(0xffffffffu, s, o);
    agg_lse_merge(m, s, m2, s2);
  }
  __shared__ float2 red[AGG_THREADS / 32];
  if ((tid & 31) == 0) red[tid >> 5] = make_float2(m, s);
  __syncthreads();
  if (tid == 0) {
    float M = -INFINITY, Sm = 0.f;
    for (int w = 0; w < AGG_THREADS / 32; ++w) agg_lse_merge(M, Sm, red[w].x, red[w].y);
    a.part[((int64_t)b * N + k) * a.nchunks + c] = make_float2(M, Sm);
  }
}

// (value, token) order: larger value, then lower token
__device__ __forceinline__ bool agg_better(float v2, int t2, float v1, int t1) {
  return v2 > v1 || (v2 == v1 && t2 < t1);
}

// grid (nchunks, B)
__global__ void __launch_bounds__(AGG_THREADS) agg_select_kernel(AggArgs a) {
  const int c = blockIdx.x, b = blockIdx.y, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int N = a.N, V = a.V, n1 = N + 1;
  __shared__ float w_s[AGG_MAX_N], lse_s[AGG_MAX_N], beta_s[AGG_MAX_N];
  __shared__ float wsum;
  __shared__ float bv_s[AGG_THREADS / 32];
  __shared__ int bt_s[AGG_THREADS / 32];
  __shared__ int last;
  if (c == 0 && b == 0 && tid == 0 && a.tile_ctr) *a.tile_ctr = 0;  // the next LM head claims its tiles from 0
  for (int k = tid; k < N; k += AGG_THREADS) {
    w_s[k] = fminf(fmaxf(a.r[b * N + k], 1e-8f), 1.0f);
    beta_s[k] = a.beta[b * N + k];
    float m = -INFINITY, s = 0.f;
    const float2* pk = a.part + ((int64_t)b * N + k) * a.nchunks;
    for (int j = 0; j < a.nchunks; ++j) agg_lse_merge(m, s, pk[j].x, pk[j].y);
    lse_s[k] = m + logf(s);
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
  float bv = -INFINITY;
  int bt = 0x7fffffff;
  const int v1 = min(V, (c + 1) * AGG_CHUNK);
  for (int v = c * AGG_CHUNK + tid; v < v1; v += AGG_THREADS) {
    const float l0 = lp0[v];
    float acc = 0.f;
    for (int k = 0; k < N; ++k) {
      const float lpk = (1.f + beta_s[k]) * lp0[(int64_t)(k + 1) * V + v] - beta_s[k] * l0 - lse_s[k];  // log p_k(v)
      acc += a.rule == 1 ? w_s[k] * inv_w * expf(lpk) : w_s[k] * inv_w * lpk;
    }
    const float agg = a.rule == 1 ? logf(acc) : acc;
    if (agg_better(agg, v, bv, bt)) {
      bv = agg;
      bt = v;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float v2 = __shfl_xor_sync(0xffffffffu, bv, o);
    const int t2 = __shfl_xor_sync(0xffffffffu, bt, o);
    if (agg_better(v2, t2, bv, bt)) {
      bv = v2;
      bt = t2;
    }
  }
  if (lane == 0) {
    bv_s[warp] = bv;
    bt_s[warp] = bt;
  }
  __syncthreads();
  if (tid == 0) {
    for (int w = 1; w < AGG_THREADS / 32; ++w)
      if (agg_better(bv_s[w], bt_s[w], bv, bt)) {
        bv = bv_s[w];
        bt = bt_s[w];
      }
    a.best[(int64_t)b * a.nchunks + c] = make_float2(bv, __int_as_float(bt));
    __threadfence();
    last = atomicAdd(a.qdone + b, 1) == a.nchunks - 1;
  }
  __syncthreads();
  if (!last || tid != 0) return;
  __threadfence();  // the other chunks' results of query b are visible
  float sv = -INFINITY;
  int st = 0x7fffffff;
  for (int j = 0; j < a.nchunks; ++j) {
    const float2 e = __ldcg(a.best + (int64_t)b * a.nchunks + j);
    if (agg_better(e.x, __float_as_int(e.y), sv, st)) {
      sv = e.x;
      st = __float_as_int(e.y);
    }
  }
  if (st >= V) st = 0;  // no finite aggregate (degenerate rows): token 0
  int bk = 0;
  float bp = -INFINITY;
  for (int k = 0; k < N; ++k) {  // the expert that puts the most weighted mass on the token
    const float lpk = (1.f + beta_s[k]) * lp0[(int64_t)(k + 1) * V + st] - beta_s[k] * lp0[st] - lse_s[k];
    const float pw = logf(w_s[k]) + lpk;
    if (pw > bp) {
      bp = pw;
      bk = k;
    }
  }
  a.qdone[b] = 0;
  if (a.lse_out)
    for (int j = 0; j < n1; ++j) a.lse_out[b * n1 + j] = a.lse[b * n1 + j];
  if (a.token) a.token[b] = st;
  if (a.expert) a.expert[b] = bk + 1;
  if (a.score) a.score[b] = sv;
  if (a.step) {
    const int t = *a.step;
    if (t >= 0 && t < a.max_steps) {
      a.history[(int64_t)b * a.max_steps + t] = st;
      if (a.expert_trace) a.expert_trace[(int64_t)b * a.max_steps + t] = bk + 1;
      if (a.score_trace) a.score_trace[(int64_t)b * a.max_steps + t] = sv;
    } else {
      dev_flag(a.status, PCED_DEV_STEP_LIMIT);
    }
    __threadfence();
    if (atomicAdd(a.done_counter, 1) == a.B - 1) {
      *a.step = t + 1;
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
