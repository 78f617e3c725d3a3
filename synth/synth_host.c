/*
 * synth_host.c -- host-side fills of the seeded synthetic inputs (synth.h).
 * Input generation only; no part of the decoding method lives here.
 * Threads split the output range; every element depends only on its own
 * (stream, index), so the result does not depend on the thread count.
 */
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>

#include "synth.h"

typedef struct {
  uint16_t* cache;
  int64_t layer_elems;
  const int64_t* kv_offset;
  const int32_t* cap;
  const int32_t* base_len;
  const int32_t* seq_ids;
  int32_t S, L, Hkv, D;
  uint64_t seed;
  uint32_t tensor;
  float scale;
  int32_t nthreads;
  int32_t tid;
} cache_job;

static void* cache_worker(void* p) {
  cache_job* j = (cache_job*)p;
  int64_t nslab = (int64_t)j->L * j->S * j->Hkv;
  for (int64_t w = j->tid; w < nslab; w += j->nthreads) {
    int32_t h = (int32_t)(w % j->Hkv);
    int32_t s = (int32_t)((w / j->Hkv) % j->S);
    int32_t l = (int32_t)(w / ((int64_t)j->Hkv * j->S));
    uint64_t key = synth_stream_key(j->seed, j->tensor, (uint32_t)l, (uint32_t)j->seq_ids[s], (uint32_t)h);
    uint16_t* slab = j->cache + (int64_t)l * j->layer_elems + j->kv_offset[s] + (int64_t)h * j->cap[s] * j->D;
    int64_t n = (int64_t)j->base_len[s] * j->D;
    for (int64_t i = 0; i < n; ++i) slab[i] = synth_normal_bf16(key, (uint64_t)i, j->scale);
  }
  return NULL;
}

/* Fill positions [0, base_len[s]) of every (layer, sequence, kv-head) slab.
 * Slab (l, s, h) starts at element l*layer_elems + kv_offset[s] + h*cap[s]*D
 * and holds cap[s] rows of D elements.  seq_ids[s] is the global sequence id
 * that keys the stream, so a subset of sequences can be generated alone.
 * Positions >= base_len[s] are left untouched. */
void synth_fill_cache(uint16_t* cache, int64_t layer_elems, const int64_t* kv_offset,
                      const int32_t* cap, const int32_t* base_len, const int32_t* seq_ids,
                      int32_t S, int32_t L, int32_t Hkv, int32_t D, uint64_t seed,
                      uint32_t tensor, float scale, int32_t nthreads) {
  if (nthreads < 1) nthreads = 1;
  if (nthreads > 256) nthreads = 256;
  pthread_t th[256];
  cache_job jobs[256];
  for (int32_t t = 0; t < nthreads; ++t) {
    cache_job j = {cache, layer_elems, kv_offset, cap, base_len, seq_ids, S, L, Hkv, D,
                   seed, tensor, scale, nthreads, t};
    jobs[t] = j;
    pthread_create(&th[t], NULL, cache_worker, &jobs[t]);
  }
  for (int32_t t = 0; t < nthreads; ++t) pthread_join(th[t], NULL);
}

typedef struct {
  uint16_t* out;
  int64_t row0, rows, cols;
  uint64_t key;
  float scale;
  int32_t nthreads, tid;
} mat_job;

static void* mat_worker(void* p) {
  mat_job* j = (mat_job*)p;
  int64_t n = j->rows * j->cols;
  int64_t per = (n + j->nthreads - 1) / j->nthreads;
  int64_t a = per * j->tid, b = a + per < n ? a + per : n;
  uint64_t base = (uint64_t)(j->row0 * j->cols);
  for (int64_t i = a; i < b; ++i) j->out[i] = synth_normal_bf16(j->key, base + (uint64_t)i, j->scale);
  return NULL;
}

/* Fill rows [row0, row0 + rows) of a dense [*, cols] bf16 matrix whose
 * element (r, c) is stream (seed, tensor, 0, 0, 0) element r*cols + c.
 * out[0] receives element (row0, 0). */
void synth_fill_matrix(uint16_t* out, int64_t row0, int64_t rows, int64_t cols, uint64_t seed,
                       uint32_t tensor, float scale, int32_t nthreads) {
  if (nthreads < 1) nthreads = 1;
  if (nthreads > 256) nthreads = 256;
  uint64_t key = synth_stream_key(seed, tensor, 0, 0, 0);
  pthread_t th[256];
  mat_job jobs[256];
  for (int32_t t = 0; t < nthreads; ++t) {
    mat_job j = {out, row0, rows, cols, key, scale, nthreads, t};
    jobs[t] = j;
    pthread_create(&th[t], NULL, mat_worker, &jobs[t]);
  }
  for (int32_t t = 0; t < nthreads; ++t) pthread_join(th[t], NULL);
}

/* single values, for spot checks */
uint64_t synth_key(uint64_t seed, uint32_t tensor, uint32_t layer, uint32_t seq, uint32_t head) {
  return synth_stream_key(seed, tensor, layer, seq, head);
}
uint16_t synth_value_bf16(uint64_t key, uint64_t i, float scale) { return synth_normal_bf16(key, i, scale); }
float synth_value_f32(uint64_t key, uint64_t i, float scale) { return synth_normal(key, i, scale); }
