// attention_noalloc.cu -- pced_decode_attention_noalloc: the same split-KV
// decode attention as pced_decode_attention (same split and combine kernels,
// same partition, same results), with the partial-record scratch held in a
// fixed device array of this library instead of a caller workspace.
//
// Some callers cannot allocate device memory at the point where they need one
// layer of attention: code running while an allocator is locked or being
// torn down, a host callback that must not call into the CUDA allocator,
// or an embedding runtime whose memory pool is owned and capped by someone
// else.  They still own their inputs and outputs; this entry point asks them
// for nothing more.
//
// The array is a file-scope __device__ variable, so every GPU that loads the
// library reserves PCED_NOALLOC_SCRATCH_BYTES for it until the process exits.
// Host code cannot use the array's name as a device address: the first call
// on each device (with that device current) asks the runtime for the real
// address with cudaGetSymbolAddress and caches it per device.
#include <mutex>

#include "attention.cuh"

namespace {

static __device__ __align__(256) unsigned char g_att_scratch[PCED_NOALLOC_SCRATCH_BYTES];

constexpr int NOALLOC_MAX_DEVICES = 64;
std::mutex g_scratch_mu;
void* g_scratch_ptr[NOALLOC_MAX_DEVICES];

// Device address of g_att_scratch on the current device (looked up once per
// device).  Returns nullptr after recording the error.
void* scratch_address(pced_status* st) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    cudaGetLastError();
    *st = pced_host::fail(PCED_ERR_NO_DEVICE, "pced_decode_attention_noalloc: no CUDA device (%s)",
                          cudaGetErrorString(e));
    return nullptr;
  }
  if (dev < 0 || dev >= NOALLOC_MAX_DEVICES) {
    *st = pced_host::fail(PCED_ERR_UNSUPPORTED, "pced_decode_attention_noalloc: device index %d >= %d", dev,
                          NOALLOC_MAX_DEVICES);
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_att_scratch);
    if (e != cudaSuccess || !p) {
      cudaGetLastError();
      *st = pced_host::cuda_status(e, "pced_decode_attention_noalloc: cudaGetSymbolAddress of the scratch array");
      return nullptr;
    }
    g_scratch_ptr[dev] = p;
  }
  return g_scratch_ptr[dev];
}

}  // namespace

using namespace pced;
using namespace pced_host;

extern "C" pced_status pced_decode_attention_noalloc(const void* q, const void* k_cache, const void* v_cache,
                                                     int64_t cache_elems, const int64_t* kv_offset,
                                                     const int32_t* cap, const int32_t* seq_len, int32_t S,
                                                     int32_t Hq, int32_t Hkv, int32_t D, int64_t total_cap,
                                                     float scale, float* out, int32_t* status, void* stream) {
  if (!q || !k_cache || !v_cache || !kv_offset || !cap || !seq_len || !out)
    return fail(PCED_ERR_INVALID_ARG, "pced_decode_attention_noalloc: null pointer");
  if (S < 1 || Hq < 1 || Hkv < 1 || Hq % Hkv != 0 || cache_elems < D || total_cap < S)
    return fail(PCED_ERR_INVALID_ARG, "pced_decode_attention_noalloc: bad sizes (S=%d Hq=%d Hkv=%d)", S, Hq, Hkv);
  if (D != 64 && D != 128)
    return fail(PCED_ERR_UNSUPPORTED, "pced_decode_attention_noalloc: D=%d (supported: 64, 128)", D);
  if (Hq / Hkv > ATT_MAX_G) return fail(PCED_ERR_UNSUPPORTED, "pced_decode_attention_noalloc: Hq/Hkv > %d", ATT_MAX_G);
  if (S > ATT_MAX_S) return fail(PCED_ERR_UNSUPPORTED, "pced_decode_attention_noalloc: S > %d", ATT_MAX_S);
  if (Hq * D > 8192) return fail(PCED_ERR_UNSUPPORTED, "pced_decode_attention_noalloc: Hq*D > 8192");
  if (cache_elems % D != 0 || cache_elems / D >= (int64_t)1 << 31)
    return fail(PCED_ERR_UNSUPPORTED, "pced_decode_attention_noalloc: cache of %lld elements",
                (long long)cache_elems);
  if ((((uintptr_t)k_cache) | ((uintptr_t)v_cache)) & 15u)
    return fail(PCED_ERR_INVALID_ARG, "pced_decode_attention_noalloc: caches must be 16-byte aligned");
  if (((uintptr_t)q) & 3u) return fail(PCED_ERR_INVALID_ARG, "pced_decode_attention_noalloc: q must be 4-byte aligned");
  if (((uintptr_t)status) & 3u)
    return fail(PCED_ERR_INVALID_ARG, "pced_decode_attention_noalloc: status must be 4-byte aligned");
  if (num_sms() <= 0) return fail(PCED_ERR_NO_DEVICE, "pced_decode_attention_noalloc: no CUDA device");

  // Scratch layout (256-byte aligned pieces): status sink | rec_o | rec_ml |
  // plan_pre | plan_per.  Record slot c + h*S + s for CTA c < ctas.
  const int32_t G = Hq / Hkv;
  const int ctas = att_grid(total_cap * Hkv);
  const int64_t slots = (int64_t)ctas + (int64_t)S * Hkv;
  Carver sizer(nullptr);
  sizer.take<int32_t>(1);
  sizer.take<float>((size_t)(slots * G * D));
  sizer.take<float2>((size_t)(slots * G));
  sizer.take<int64_t>((size_t)S + 1);
  sizer.take<int64_t>(1);
  if (sizer.used() > (size_t)PCED_NOALLOC_SCRATCH_BYTES)
    return fail(PCED_ERR_UNSUPPORTED,
                "pced_decode_attention_noalloc: needs %zu bytes of scratch for S=%d Hkv=%d G=%d D=%d on %d CTAs, "
                "above the fixed maximum of %zu bytes (use pced_decode_attention with a workspace)",
                sizer.used(), S, Hkv, G, D, ctas, (size_t)PCED_NOALLOC_SCRATCH_BYTES);

  pced_status st = PCED_OK;
  void* scratch = scratch_address(&st);
  if (!scratch) return st;

  CUtensorMap kmap, vmap;
  const uint64_t rows = (uint64_t)(cache_elems / D);
  st = make_tmap_kv(&kmap, k_cache, rows, (uint32_t)D, ATT_BLOCK_N);
  if (st != PCED_OK) return st;
  st = make_tmap_kv(&vmap, v_cache, rows, (uint32_t)D, ATT_BLOCK_N);
  if (st != PCED_OK) return st;

  // Nothing here has to start at zero: every record and plan entry the combine
  // kernel reads is written by the split kernel of the same call, and the
  // status sink (used when the caller passes no status word) is write-only.
  Carver cv(scratch);
  int* sink = cv.take<int>(1);
  AttArgs a;
  a.q = (const __nv_bfloat16*)q;
  a.kv_offset = kv_offset;
  a.cap = cap;
  a.seq_len = seq_len;
  a.S = S;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.G = G;
  a.row_base = 0;
  a.scale_log2 = scale * 1.4426950408889634f;
  a.rec_o = cv.take<float>((size_t)(slots * G * D));
  a.rec_ml = cv.take<float2>((size_t)(slots * G));
  a.plan_pre = cv.take<int64_t>((size_t)S + 1);
  a.plan_per = cv.take<int64_t>(1);
  a.status = status ? (int*)status : sink;
  cudaStream_t s = (cudaStream_t)stream;
  cudaError_t e = att_split_launch(D, kmap, vmap, a, ctas, s);
  if (e != cudaSuccess) return cuda_status(e, "pced_decode_attention_noalloc: split launch");

  CombineArgs c = {};
  c.S = S;
  c.Hq = Hq;
  c.Hkv = Hkv;
  c.G = G;
  c.D = D;
  c.rec_o = a.rec_o;
  c.rec_ml = a.rec_ml;
  c.plan_pre = a.plan_pre;
  c.plan_per = a.plan_per;
  c.out = out;
  c.status = a.status;
  e = att_combine_launch(c, s);
  if (e != cudaSuccess) return cuda_status(e, "pced_decode_attention_noalloc: combine launch");
  return PCED_OK;
}
