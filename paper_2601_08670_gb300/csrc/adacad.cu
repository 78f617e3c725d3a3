// adacad.cu -- dynamic contrast strength for the first generated token
// (paper Sec. 3 after Eq. 2: beta_0 is computed as in AdaCAD for the first
// generated token and kept fixed thereafter).  Reading: one beta per
// contextual expert, the Jensen-Shannon divergence in bits between the
// expert's next-token distribution p_k = exp(lp_k) and the amateur's
// p_0 = exp(lp_0):
//   beta[b][k-1] = 1/2 sum_v [ p_k log2(p_k / m) + p_0 log2(p_0 / m) ],  m = (p_k + p_0) / 2,
// in [0, 1].  CTAs of 8192 vocabulary entries per (expert, query) stream both
// rows once; each term uses log m = logaddexp(lp_k, lp_0) - ln 2 in fp32 and
// is summed in fp64 in a fixed order (thread t takes v = t, t + 256, ... of
// its chunk, then a fixed tree, then the chunks in order by the last CTA of
// the pair to finish), so the result does not depend on timing.
#include <math.h>

#include "adacad.cuh"

namespace pced {

constexpr int ADA_THREADS = 256;
constexpr int ADA_CHUNK = 2048;  // vocabulary entries per CTA (about 500 CTAs at llama8: every SM busy)

int32_t adacad_chunks(int32_t V) { return (V + ADA_CHUNK - 1) / ADA_CHUNK; }

// grid (chunks, N, B): CTA (c, k-1, b) sums the terms of v in chunk c; the
// last CTA of (b, k) to finish adds the chunk sums in chunk order
__global__ void __launch_bounds__(ADA_THREADS) adacad_beta_kernel(const float* lp, int32_t N, int32_t V, float* beta,
                                                                  double* part, int* cnt, int* reset_ctr) {
  const int c = blockIdx.x, k = blockIdx.y + 1, b = blockIdx.z, tid = threadIdx.x;
  const int nch = gridDim.x;
  if (reset_ctr && c == 0 && k == 1 && b == 0 && tid == 0) *reset_ctr = 0;
  const float* l0 = lp + (int64_t)b * (N + 1) * V;
  const float* lk = l0 + (int64_t)k * V;
  const float ln2 = 0.69314718055994531f;
  const int v1 = min(V, (c + 1) * ADA_CHUNK);
  double acc = 0.0;
  for (int v = c * ADA_CHUNK + tid; v < v1; v += ADA_THREADS) {
    const float a = lk[v], cc = l0[v];
    const float hi = fmaxf(a, cc), lo = fminf(a, cc);
    if (hi == -INFINITY) continue;  // p_k = p_0 = 0
    const float lm = hi + log1pf(expf(lo - hi)) - ln2;  // log of the midpoint
    float t = 0.f;
    if (a > -INFINITY) t += expf(a) * (a - lm);
    if (cc > -INFINITY) t += expf(cc) * (cc - lm);
    acc += (double)t;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  __shared__ double red[ADA_THREADS / 32];
  __shared__ int last;
  if ((tid & 31) == 0) red[tid >> 5] = acc;
  __syncthreads();
  const int64_t bk = (int64_t)b * N + (k - 1);
  if (tid == 0) {
    double s = 0.0;
    for (int w = 0; w < ADA_THREADS / 32; ++w) s += red[w];
    part[bk * nch + c] = s;
    __threadfence();
    last = atomicAdd(cnt + bk, 1) == nch - 1;
    if (last) {
      __threadfence();
      double tot = 0.0;
      for (int j = 0; j < nch; ++j) tot += __ldcg(part + bk * nch + j);
      beta[bk] = (float)(0.5 * tot / 0.69314718055994531);
      cnt[bk] = 0;
    }
  }
}

size_t adacad_scratch_bytes(int32_t B, int32_t N, int32_t V) {
  pced_host::Carver c(nullptr);
  c.take<double>((size_t)B * N * adacad_chunks(V));
  c.take<int>((size_t)B * N);
  return c.used();
}

cudaError_t adacad_beta_launch(const float* lp, int32_t B, int32_t N, int32_t V, float* beta, void* scratch,
                               int* reset_ctr, cudaStream_t stream) {
  pced_host::Carver cv(scratch);
  double* part = cv.take<double>((size_t)B * N * adacad_chunks(V));
  int* cnt = cv.take<int>((size_t)B * N);
  adacad_beta_kernel<<<dim3(adacad_chunks(V), N, B), ADA_THREADS, 0, stream>>>(lp, N, V, beta, part, cnt,
                                                                                reset_ctr);
  return cudaGetLastError();
}

int* adacad_counters(void* scratch, int32_t B, int32_t N, int32_t V) {
  pced_host::Carver cv(scratch);
  cv.take<double>((size_t)B * N * adacad_chunks(V));
  return cv.take<int>((size_t)B * N);
}

}  // namespace pced

using namespace pced;
using namespace pced_host;

extern "C" size_t pced_adacad_beta_workspace_size(int32_t B, int32_t N, int32_t V) {
  if (B < 1 || N < 1 || V < 1) return 0;
  return adacad_scratch_bytes(B, N, V);
}

extern "C" pced_status pced_adacad_beta(const float* logprobs, int32_t B, int32_t N, int32_t V, float* beta,
                                        void* workspace, size_t workspace_bytes, void* stream) {
  if (!logprobs || !beta || !workspace) return fail(PCED_ERR_INVALID_ARG, "pced_adacad_beta: null pointer");
  if (B < 1 || N < 1 || V < 1 || B > 65535 || N > 65535)
    return fail(PCED_ERR_INVALID_ARG, "pced_adacad_beta: bad sizes (B=%d N=%d V=%d)", B, N, V);
  if (((uintptr_t)logprobs | (uintptr_t)beta) & 3u)
    return fail(PCED_ERR_INVALID_ARG, "pced_adacad_beta: pointers must be 4-byte aligned");
  if (((uintptr_t)workspace) & 255u || workspace_bytes < pced_adacad_beta_workspace_size(B, N, V))
    return fail(PCED_ERR_WORKSPACE, "pced_adacad_beta: workspace too small or misaligned");
  if (num_sms() <= 0) return fail(PCED_ERR_NO_DEVICE, "pced_adacad_beta: no CUDA device");
  cudaStream_t s = (cudaStream_t)stream;
  // the per-(query, expert) arrival counters start at zero (the kernel leaves them at zero)
  cudaError_t e = cudaMemsetAsync(adacad_counters(workspace, B, N, V), 0, sizeof(int) * (size_t)B * N, s);
  if (e == cudaSuccess) e = adacad_beta_launch(logprobs, B, N, V, beta, workspace, nullptr, s);
  if (e != cudaSuccess) return cuda_status(e, "pced_adacad_beta launch");
  return PCED_OK;
}
