// select_key.cuh -- the choice of Eq. 3 packed into one int64 whose signed
// order is Eq. 3's order: the higher score first, then the lower token id,
// then the lower expert index.  The maximum of such keys over disjoint sets
// of a query's experts is the choice over their union, so ranks that each
// hold some experts (with the amateur and W_U replicated) agree on a token
// through one all-reduce-max, the only cross-expert coupling of Eq. 3.
//
// Layout (as unsigned, then the top bit flipped so that signed order equals
// unsigned order): bits 63-32 the fp32 score mapped to an order-preserving
// unsigned code, bits 31-12 (2^20 - 1 - token), bits 11-0 (4095 - (expert - 1)).
#pragma once
#include <stdint.h>
#include <string.h>

namespace pced {

constexpr int32_t KEY_MAX_TOKENS = 1 << 20;   // token ids below 2^20
constexpr int32_t KEY_MAX_EXPERTS = 1 << 12;  // global expert indices 1..4096

__host__ __device__ inline uint32_t key_score_code(float score) {
  uint32_t b;
#ifdef __CUDA_ARCH__
  b = __float_as_uint(score);
#else
  memcpy(&b, &score, 4);
#endif
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

__host__ __device__ inline float key_score_value(uint32_t code) {
  const uint32_t b = (code & 0x80000000u) ? (code & 0x7FFFFFFFu) : ~code;
#ifdef __CUDA_ARCH__
  return __uint_as_float(b);
#else
  float f;
  memcpy(&f, &b, 4);
  return f;
#endif
}

// token in [0, 2^20), expert (1-based, global) in [1, 4096]
__host__ __device__ inline int64_t select_key(float score, int32_t token, int32_t expert) {
  const uint64_t u = ((uint64_t)key_score_code(score) << 32) |
                     ((uint64_t)(uint32_t)(KEY_MAX_TOKENS - 1 - token) << 12) |
                     (uint64_t)(uint32_t)(KEY_MAX_EXPERTS - expert);
  return (int64_t)(u ^ 0x8000000000000000ull);
}

__host__ __device__ inline void select_key_unpack(int64_t key, float* score, int32_t* token, int32_t* expert) {
  const uint64_t u = (uint64_t)key ^ 0x8000000000000000ull;
  *score = key_score_value((uint32_t)(u >> 32));
  *token = KEY_MAX_TOKENS - 1 - (int32_t)((u >> 12) & 0xFFFFFu);
  *expert = KEY_MAX_EXPERTS - (int32_t)(u & 0xFFFu);
}

}  // namespace pced
