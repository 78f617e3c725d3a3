// adacad.cuh -- dynamic contrast strength from materialised log-probabilities.
#pragma once
#include "common.cuh"

namespace pced {

// beta[b][k-1] = Jensen-Shannon divergence in bits between rows b*(N+1)+k and
// b*(N+1) of lp [B*(N+1)][V]; reset_ctr (optional) is set to 0.  scratch
// (adacad_scratch_bytes, 256-byte aligned) holds chunk sums and per-(query,
// expert) counters that must be zero at launch (the kernel leaves them zero).
size_t adacad_scratch_bytes(int32_t B, int32_t N, int32_t V);
int* adacad_counters(void* scratch, int32_t B, int32_t N, int32_t V);
cudaError_t adacad_beta_launch(const float* lp, int32_t B, int32_t N, int32_t V, float* beta, void* scratch,
                               int* reset_ctr, cudaStream_t stream);

}  // namespace pced
