// synth_dev.cu -- device-side fills of the seeded synthetic inputs (synth.h).
// Same element definition as synth_host.c, so the device tensors are
// bit-identical to the host ones.  Input generation only: this library is
// not part of the decoding path and the decoding library does not link it.
#include <cuda_runtime.h>
#include <stdint.h>

#include "synth.h"

namespace {

__global__ void fill_cache_kernel(uint16_t* __restrict__ cache, int64_t layer_elems,
                                  const int64_t* __restrict__ kv_offset, const int32_t* __restrict__ cap,
                                  const int32_t* __restrict__ base_len, const int32_t* __restrict__ seq_ids,
                                  int32_t S, int32_t L, int32_t Hkv, int32_t D, uint64_t seed,
                                  uint32_t tensor, float scale) {
  const int64_t nslab = (int64_t)L * S * Hkv;
  for (int64_t w = blockIdx.x; w < nslab; w += gridDim.x) {
    const int32_t h = (int32_t)(w % Hkv);
    const int32_t s = (int32_t)((w / Hkv) % S);
    const int32_t l = (int32_t)(w / ((int64_t)Hkv * S));
    const uint64_t key = synth_stream_key(seed, tensor, (uint32_t)l, (uint32_t)seq_ids[s], (uint32_t)h);
    uint16_t* slab = cache + (int64_t)l * layer_elems + kv_offset[s] + (int64_t)h * cap[s] * D;
    const int64_t n = (int64_t)base_len[s] * D;  // multiple of 8 because D is
    for (int64_t i = (int64_t)threadIdx.x * 8; i < n; i += (int64_t)blockDim.x * 8) {
      uint32_t packed[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        uint32_t lo = synth_normal_bf16(key, (uint64_t)(i + 2 * e), scale);
        uint32_t hi = synth_normal_bf16(key, (uint64_t)(i + 2 * e + 1), scale);
        packed[e] = lo | (hi << 16);
      }
      *reinterpret_cast<uint4*>(slab + i) = make_uint4(packed[0], packed[1], packed[2], packed[3]);
    }
  }
}

// Paged layout: the pool of one layer is num_blocks blocks of [Hkv][P][D];
// row pos of (sequence s, kv-head h) lives in block table[s][pos / P] at row
// pos % P.  Same element values as fill_cache_kernel (element index pos*D + dim
// of the (layer, sequence, head) stream).
__global__ void fill_cache_paged_kernel(uint16_t* __restrict__ pool, int64_t layer_elems,
                                        const int32_t* __restrict__ table, int32_t max_blocks, int32_t P,
                                        const int32_t* __restrict__ base_len, const int32_t* __restrict__ seq_ids,
                                        int32_t S, int32_t L, int32_t Hkv, int32_t D, uint64_t seed,
                                        uint32_t tensor, float scale) {
  const int64_t nslab = (int64_t)L * S * Hkv;
  for (int64_t w = blockIdx.x; w < nslab; w += gridDim.x) {
    const int32_t h = (int32_t)(w % Hkv);
    const int32_t s = (int32_t)((w / Hkv) % S);
    const int32_t l = (int32_t)(w / ((int64_t)Hkv * S));
    const uint64_t key = synth_stream_key(seed, tensor, (uint32_t)l, (uint32_t)seq_ids[s], (uint32_t)h);
    const int64_t n = (int64_t)base_len[s] * D;
    for (int64_t i = (int64_t)threadIdx.x * 8; i < n; i += (int64_t)blockDim.x * 8) {
      const int64_t pos = i / D, dim = i % D;
      const int32_t blk = table[(int64_t)s * max_blocks + pos / P];
      uint16_t* dst = pool + (int64_t)l * layer_elems + (((int64_t)blk * Hkv + h) * P + pos % P) * D + dim;
      uint32_t packed[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        uint32_t lo = synth_normal_bf16(key, (uint64_t)(i + 2 * e), scale);
        uint32_t hi = synth_normal_bf16(key, (uint64_t)(i + 2 * e + 1), scale);
        packed[e] = lo | (hi << 16);
      }
      *reinterpret_cast<uint4*>(dst) = make_uint4(packed[0], packed[1], packed[2], packed[3]);
    }
  }
}

__global__ void fill_matrix_kernel(uint16_t* __restrict__ out, int64_t row0, int64_t n, int64_t cols,
                                   uint64_t key, float scale) {
  const uint64_t base = (uint64_t)(row0 * cols);
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
    out[i] = synth_normal_bf16(key, base + (uint64_t)i, scale);
}

}  // namespace

extern "C" {

// Device version of synth_fill_cache (all table pointers are device pointers,
// D must be a multiple of 8 and the cache 16-byte aligned).  Returns a
// cudaError_t value.
int synth_dev_fill_cache(void* cache, int64_t layer_elems, const int64_t* kv_offset, const int32_t* cap,
                         const int32_t* base_len, const int32_t* seq_ids, int32_t S, int32_t L, int32_t Hkv,
                         int32_t D, uint64_t seed, uint32_t tensor, float scale, void* stream) {
  if (D % 8 != 0 || ((uintptr_t)cache & 15u) != 0) return (int)cudaErrorInvalidValue;
  int64_t nslab = (int64_t)L * S * Hkv;
  int grid = (int)(nslab < 4096 ? nslab : 4096);
  if (grid < 1) return 0;
  fill_cache_kernel<<<grid, 256, 0, (cudaStream_t)stream>>>((uint16_t*)cache, layer_elems, kv_offset, cap,
                                                            base_len, seq_ids, S, L, Hkv, D, seed, tensor, scale);
  return (int)cudaGetLastError();
}

// Paged version of synth_dev_fill_cache (table: device int32 [S][max_blocks]).
int synth_dev_fill_cache_paged(void* pool, int64_t layer_elems, const int32_t* table, int32_t max_blocks, int32_t P,
                               const int32_t* base_len, const int32_t* seq_ids, int32_t S, int32_t L, int32_t Hkv,
                               int32_t D, uint64_t seed, uint32_t tensor, float scale, void* stream) {
  if (D % 8 != 0 || P < 1 || ((uintptr_t)pool & 15u) != 0) return (int)cudaErrorInvalidValue;
  int64_t nslab = (int64_t)L * S * Hkv;
  int grid = (int)(nslab < 4096 ? nslab : 4096);
  if (grid < 1) return 0;
  fill_cache_paged_kernel<<<grid, 256, 0, (cudaStream_t)stream>>>((uint16_t*)pool, layer_elems, table, max_blocks, P,
                                                                  base_len, seq_ids, S, L, Hkv, D, seed, tensor,
                                                                  scale);
  return (int)cudaGetLastError();
}

// Device version of synth_fill_matrix.
int synth_dev_fill_matrix(void* out, int64_t row0, int64_t rows, int64_t cols, uint64_t seed, uint32_t tensor,
                          float scale, void* stream) {
  int64_t n = rows * cols;
  if (n <= 0) return 0;
  uint64_t key = synth_stream_key(seed, tensor, 0, 0, 0);
  int64_t blocks = (n + 255) / 256;
  int grid = (int)(blocks < 65536 ? blocks : 65536);
  fill_matrix_kernel<<<grid, 256, 0, (cudaStream_t)stream>>>((uint16_t*)out, row0, n, cols, key, scale);
  return (int)cudaGetLastError();
}

}  // extern "C"
