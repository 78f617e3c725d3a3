// partition.cu -- the expert-partitioned decode step.  Eq. 3 couples a
// query's experts only through the maximum over them (Sec. 3: the experts
// run as independent streams; the choice is one max), so experts can live on
// different GPUs: each holds the amateur, a replica of W_U and some of the
// experts, runs pced_step with key_out set (its experts' best choice as a
// packed key, nothing appended), the keys meet in one all-reduce-max
// (NCCL or any other max reduction of int64), and pced_step_commit appends
// the common token on every one of them.
#include "common.cuh"
#include "select_key.cuh"

namespace pced {

// one CTA: each query's token, expert and score from its reduced key, then
// the step counter advances
__global__ void step_commit_kernel(const int64_t* keys, int32_t B, int32_t* step, int32_t* history,
                                   int32_t* expert_trace, float* score_trace, int32_t max_steps, int* status) {
  const int t = *step;
  const bool in_range = t >= 0 && t < max_steps;
  for (int b = threadIdx.x; b < B; b += blockDim.x) {
    float sc;
    int32_t tok, ex;
    select_key_unpack(keys[b], &sc, &tok, &ex);
    if (!in_range) continue;
    history[(int64_t)b * max_steps + t] = tok;
    if (expert_trace) expert_trace[(int64_t)b * max_steps + t] = ex;
    if (score_trace) score_trace[(int64_t)b * max_steps + t] = sc;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    if (in_range) *step = t + 1;
    else dev_flag(status, PCED_DEV_STEP_LIMIT);
  }
}

}  // namespace pced

using namespace pced;
using namespace pced_host;

extern "C" int64_t pced_select_key(float score, int32_t token, int32_t expert) {
  return select_key(score, token, expert);
}

extern "C" void pced_select_key_unpack(int64_t key, float* score, int32_t* token, int32_t* expert) {
  float s;
  int32_t t, e;
  select_key_unpack(key, &s, &t, &e);
  if (score) *score = s;
  if (token) *token = t;
  if (expert) *expert = e;
}

extern "C" pced_status pced_step_commit(const int64_t* keys, int32_t B, int32_t* step, int32_t* history,
                                        int32_t* expert_trace, float* score_trace, int32_t max_steps, int* status,
                                        void* stream) {
  if (!keys || !step || !history) return fail(PCED_ERR_INVALID_ARG, "pced_step_commit: null pointer");
  if (B < 1 || max_steps < 1) return fail(PCED_ERR_INVALID_ARG, "pced_step_commit: B=%d max_steps=%d", B, max_steps);
  if (num_sms() <= 0) return fail(PCED_ERR_NO_DEVICE, "pced_step_commit: no CUDA device");
  step_commit_kernel<<<1, 256, 0, (cudaStream_t)stream>>>(keys, B, step, history, expert_trace, score_trace,
                                                          max_steps, status);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? PCED_OK : cuda_status(e, "step commit launch");
}
