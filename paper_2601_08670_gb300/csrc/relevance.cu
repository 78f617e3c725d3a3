// relevance.cu -- relevance scores r_k in [0, 1) for the retrieval prior of
// Eq. 2, from a retriever's raw scores and a reranker's logits (Sec. 3
// "Retrieval and relevance scoring"; App. "Normalization of Retrieval and
// Reranker Scores"):
//   dense / ColBERT (mode 0): r_ret = clip((s + 1)/2, 0, 1 - eps)
//   sparse (mode 1):          r_ret = clip((2/pi) atan(max(s, 0)), 0, 1 - eps)
//   reranker:                 r_rer = clip(sigmoid(z), 0, 1 - eps)
//   fusion:                   r = 2 r_ret r_rer / (r_ret + r_rer + eps)   (harmonic mean, appendix form)
// Elementwise, evaluated in fp64 and rounded to fp32 once.  Runs once per
// query (not per token); a few hundred scores at most.
#include <math.h>

#include "common.cuh"

namespace pced {

constexpr int REL_THREADS = 256;

__device__ __forceinline__ double rel_clip(double x, double eps) { return x < 0.0 ? 0.0 : fmin(x, 1.0 - eps); }

__global__ void __launch_bounds__(REL_THREADS) relevance_kernel(const float* s, int32_t mode, const float* z,
                                                                int32_t n, double eps, float* r) {
  const int k = blockIdx.x * REL_THREADS + threadIdx.x;
  if (k >= n) return;
  const double sk = s[k];
  const double rr = mode == 0 ? rel_clip((sk + 1.0) * 0.5, eps)
                              : rel_clip(0.63661977236758134308 * atan(fmax(sk, 0.0)), eps);  // 2/pi
  double out = rr;
  if (z) {
    const double rz = rel_clip(1.0 / (1.0 + exp(-(double)z[k])), eps);
    out = 2.0 * rr * rz / (rr + rz + eps);
  }
  r[k] = (float)out;
}

}  // namespace pced

using namespace pced;
using namespace pced_host;

extern "C" pced_status pced_relevance(const float* ret_scores, int32_t ret_mode, const float* rer_logits, int32_t n,
                                      double eps, float* r, void* stream) {
  if (n < 0) return fail(PCED_ERR_INVALID_ARG, "pced_relevance: n=%d", n);
  if (ret_mode != PCED_RET_DENSE && ret_mode != PCED_RET_SPARSE)
    return fail(PCED_ERR_INVALID_ARG, "pced_relevance: retrieval mode %d (0 dense/ColBERT, 1 sparse)", ret_mode);
  if (!(eps >= 0.0 && eps < 0.5)) return fail(PCED_ERR_INVALID_ARG, "pced_relevance: eps must be in [0, 0.5)");
  if (n == 0) return PCED_OK;
  if (!ret_scores || !r) return fail(PCED_ERR_INVALID_ARG, "pced_relevance: null pointer");
  if (((uintptr_t)ret_scores | (uintptr_t)r | (uintptr_t)rer_logits) & 3u)
    return fail(PCED_ERR_INVALID_ARG, "pced_relevance: pointers must be 4-byte aligned");
  if (num_sms() <= 0) return fail(PCED_ERR_NO_DEVICE, "pced_relevance: no CUDA device");
  relevance_kernel<<<(n + REL_THREADS - 1) / REL_THREADS, REL_THREADS, 0, (cudaStream_t)stream>>>(
      ret_scores, ret_mode, rer_logits, n, eps, r);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_status(e, "pced_relevance launch");
  return PCED_OK;
}
