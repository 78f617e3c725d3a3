/*
 * synth.h -- seeded synthetic inputs for PCED decode-step workloads.
 *
 * This module defines the INPUTS only (KV-cache prefixes, token embedding,
 * unembedding weights).  It holds none of the decoding method's arithmetic.
 * Both the CPU oracle and the CUDA path receive their inputs from here, so
 * that both see bit-identical bf16 tensors.
 *
 * Generator: splitmix64 (S. Vigna, public domain), used as a counter-based
 * generator: output i of a stream with state `key` is
 *     fmix64(key + (i + 1) * 0x9E3779B97F4A7C15)
 * where fmix64 is splitmix64's finaliser.  Stream keys are derived by chaining
 * splitmix64 over (seed, tensor, layer, sequence, head).
 *
 * Value: an Irwin-Hall(4) approximation of N(0, sigma^2): the four 16-bit
 * fields u_j of one 64-bit output give
 *     x = (u_0 + u_1 + u_2 + u_3 - 131070) * scale,  scale = sigma*sqrt(3)/65536
 * (unit variance for sigma = 1, support +-3.46 sigma).  The integer sum is
 * exact, the single fp32 multiply is IEEE round-to-nearest on every target,
 * and the bf16 conversion is integer round-to-nearest-even, so host and device
 * produce the same bits.  `scale` is passed in as an fp32 value.
 */
#ifndef PCED_SYNTH_H
#define PCED_SYNTH_H

#include <stdint.h>

#if defined(__CUDACC__)
#define SYNTH_HD __host__ __device__ __forceinline__
#else
#define SYNTH_HD static inline
#endif

#define SYNTH_GOLDEN 0x9E3779B97F4A7C15ull

/* tensor tags of the stream-key derivation */
enum { SYNTH_T_KCACHE = 1, SYNTH_T_VCACHE = 2, SYNTH_T_EMBED = 3, SYNTH_T_UNEMBED = 4 };

SYNTH_HD uint64_t synth_fmix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

/* i-th output of a splitmix64 stream whose state is `key` */
SYNTH_HD uint64_t synth_bits(uint64_t key, uint64_t i) {
  return synth_fmix64(key + (i + 1ull) * SYNTH_GOLDEN);
}

SYNTH_HD uint64_t synth_stream_key(uint64_t seed, uint32_t tensor, uint32_t layer,
                                   uint32_t seq, uint32_t head) {
  uint64_t k = synth_bits(seed, tensor);
  k = synth_bits(k, layer);
  k = synth_bits(k, seq);
  return synth_bits(k, head);
}

SYNTH_HD float synth_u32_as_float(uint32_t u) {
  union { uint32_t u; float f; } c;
  c.u = u;
  return c.f;
}
SYNTH_HD uint32_t synth_float_as_u32(float f) {
  union { uint32_t u; float f; } c;
  c.f = f;
  return c.u;
}

/* fp32 sample of stream `key`, element i */
SYNTH_HD float synth_normal(uint64_t key, uint64_t i, float scale) {
  uint64_t b = synth_bits(key, i);
  int32_t s = (int32_t)(b & 0xFFFFu) + (int32_t)((b >> 16) & 0xFFFFu) +
              (int32_t)((b >> 32) & 0xFFFFu) + (int32_t)(b >> 48) - 131070;
  return (float)s * scale;
}

/* fp32 -> bf16 bits, round to nearest even (inputs are finite) */
SYNTH_HD uint16_t synth_f32_to_bf16(float f) {
  uint32_t u = synth_float_as_u32(f);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

SYNTH_HD uint16_t synth_normal_bf16(uint64_t key, uint64_t i, float scale) {
  return synth_f32_to_bf16(synth_normal(key, i, scale));
}

#endif /* PCED_SYNTH_H */
