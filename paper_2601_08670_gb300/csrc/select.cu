// select.cu -- Eq. 2 and Eq. 3 on materialised log-probabilities (the unfused
// path behind pced_contrastive_select).
//   shat_k(v) = (1 + beta_k) lp_k(v) - beta_k lp_0(v) + gamma log r_k,  k = 1..N
//   y = argmax_v max_k shat_k(v)
// Pass 1: one CTA per (vocabulary chunk, query) scans its tokens, taking the
// max over experts per token and the best token of the chunk.  Pass 2: one
// CTA per query reduces the chunk records.  Ties: highest score, then lowest
// token id, then lowest expert index (the amateur, row 0, never competes).
#include <math.h>

#include "common.cuh"

namespace pced {

constexpr int SEL_THREADS = 256;
constexpr int SEL_CHUNK = 4096;
constexpr int SEL_MAX_N = 255;

struct Cand {
  float s;
  int v, k;
};
__device__ __forceinline__ bool cand_better(const Cand& x, const Cand& y) {
  return x.s > y.s || (x.s == y.s && (x.v < y.v || (x.v == y.v && x.k < y.k)));
}
__device__ __forceinline__ Cand warp_best(Cand c) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    Cand d;
    d.s = __shfl_xor_sync(0xffffffffu, c.s, o);
    d.v = __shfl_xor_sync(0xffffffffu, c.v, o);
    d.k = __shfl_xor_sync(0xffffffffu, c.k, o);
    if (cand_better(d, c)) c = d;
  }
  return c;
}
__device__ __forceinline__ Cand block_best(Cand c) {
  __shared__ Cand red[SEL_THREADS / 32];
  c = warp_best(c);
  const int tid = threadIdx.x;
  if ((tid & 31) == 0) red[tid >> 5] = c;
  __syncthreads();
  if (tid < 32) {
    Cand d = tid < SEL_THREADS / 32 ? red[tid] : Cand{-INFINITY, 0x7fffffff, 0x7fffffff};
    d = warp_best(d);
    if (tid == 0) red[0] = d;
  }
  __syncthreads();
  return red[0];
}

__global__ void __launch_bounds__(SEL_THREADS)
    select_dense_kernel(const float* __restrict__ lp, const float* __restrict__ beta, const float* __restrict__ r,
                        float gamma, int N, int V, Cand* rec) {
  const int b = blockIdx.y, tid = threadIdx.x, n1 = N + 1;
  __shared__ float bt[SEL_MAX_N], bias[SEL_MAX_N];
  for (int k = tid; k < N; k += SEL_THREADS) {
    bt[k] = beta[b * N + k];
    bias[k] = gamma * logf(fminf(fmaxf(r[b * N + k], 1e-8f), 1.0f));
  }
  __syncthreads();
  const float* lp0 = lp + (int64_t)b * n1 * V;
  Cand best{-INFINITY, 0x7fffffff, 0x7fffffff};
  const int v0 = blockIdx.x * SEL_CHUNK, v1 = min(V, v0 + SEL_CHUNK);
  for (int v = v0 + tid; v < v1; v += SEL_THREADS) {
    const float a0 = lp0[v];
    for (int k = 1; k <= N; ++k) {
      const float x = (1.f + bt[k - 1]) * lp0[(int64_t)k * V + v] - bt[k - 1] * a0 + bias[k - 1];
      const Cand c{x, v, k};
      if (cand_better(c, best)) best = c;
    }
  }
  best = block_best(best);
  if (tid == 0) rec[(int64_t)b * gridDim.x + blockIdx.x] = best;
}

__global__ void __launch_bounds__(SEL_THREADS)
    select_reduce_kernel(const Cand* rec, int nchunks, int32_t* token, int32_t* expert, float* score) {
  const int b = blockIdx.x;
  Cand best{-INFINITY, 0x7fffffff, 0x7fffffff};
  for (int i = threadIdx.x; i < nchunks; i += SEL_THREADS) {
    const Cand c = rec[(int64_t)b * nchunks + i];
    if (cand_better(c, best)) best = c;
  }
  best = block_best(best);
  if (threadIdx.x == 0) {
    token[b] = best.v;
    expert[b] = best.k;
    score[b] = best.s;
  }
}

}  // namespace pced

using namespace pced;
using namespace pced_host;

extern "C" size_t pced_contrastive_select_workspace_size(int32_t B, int32_t N, int32_t V) {
  if (B < 1 || N < 1 || V < 1) return 0;
  const int64_t nchunks = (V + SEL_CHUNK - 1) / SEL_CHUNK;
  Carver c(nullptr);
  c.take<Cand>((size_t)(B * nchunks));
  return 256 + c.used();
}

extern "C" pced_status pced_contrastive_select(const float* logprobs, const float* beta, const float* r, float gamma,
                                               int32_t B, int32_t N, int32_t V, int32_t* token, int32_t* expert,
                                               float* score, void* workspace, size_t workspace_bytes, void* stream) {
  if (!logprobs || !beta || !r || !token || !expert || !score || !workspace)
    return fail(PCED_ERR_INVALID_ARG, "pced_contrastive_select: null pointer");
  if (B < 1 || N < 1 || V < 1 || B > 65535) return fail(PCED_ERR_INVALID_ARG, "pced_contrastive_select: bad sizes");
  if (N > SEL_MAX_N) return fail(PCED_ERR_UNSUPPORTED, "pced_contrastive_select: N > %d", SEL_MAX_N);
  if (!isfinite(gamma)) return fail(PCED_ERR_INVALID_ARG, "pced_contrastive_select: gamma not finite");
  if (((uintptr_t)workspace) & 255u || workspace_bytes < pced_contrastive_select_workspace_size(B, N, V))
    return fail(PCED_ERR_WORKSPACE, "pced_contrastive_select: workspace too small or misaligned");
  if (num_sms() <= 0) return fail(PCED_ERR_NO_DEVICE, "pced_contrastive_select: no CUDA device");
  const int nchunks = (V + SEL_CHUNK - 1) / SEL_CHUNK;
  Carver cv((char*)workspace + 256);
  Cand* rec = cv.take<Cand>((size_t)B * nchunks);
  cudaStream_t s = (cudaStream_t)stream;
  select_dense_kernel<<<dim3(nchunks, B), SEL_THREADS, 0, s>>>(logprobs, beta, r, gamma, N, V, rec);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_status(e, "select launch");
  select_reduce_kernel<<<B, SEL_THREADS, 0, s>>>(rec, nchunks, token, expert, score);
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_status(e, "select reduce launch");
  return PCED_OK;
}
