// host.cu -- host-side plumbing of the C ABI: error strings, device queries and
// TMA tensor-map encoding (driver entry point fetched through the runtime, so
// the library needs no link-time dependency on libcuda).
#include <stdarg.h>
#include <stdio.h>

#include "common.cuh"

namespace pced_host {

static thread_local char g_err[512] = "";

void set_error(const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
}

pced_status fail(pced_status st, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return st;
}

pced_status cuda_status(cudaError_t e, const char* what) {
  set_error("%s: %s", what, cudaGetErrorString(e));
  return PCED_ERR_CUDA;
}

int num_sms() {
  static int cache[64];
  static bool init[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    cudaGetLastError();
    return 0;
  }
  if (!init[dev]) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
      cudaGetLastError();
      return 0;
    }
    cache[dev] = n;
    init[dev] = true;
  }
  return cache[dev];
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = (EncodeTiledFn)ptr;
    else
      cudaGetLastError();
  }
  return fn;
}

pced_status make_tmap_2d(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows,
                         uint32_t box_cols, bool l2_promote_256) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return fail(PCED_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
  if (box_cols * 2 != 128 || box_rows < 1 || box_rows > 256 || rows < 1 || rows > (1ull << 32) ||
      (cols * 2) % 16 != 0 || ((uintptr_t)base & 15u))
    return fail(PCED_ERR_INVALID_ARG, "tensor map: unsupported geometry");
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {cols * 2};
  const cuuint32_t box[2] = {box_cols, box_rows};
  const cuuint32_t es[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  l2_promote_256 ? CU_TENSOR_MAP_L2_PROMOTION_L2_256B : CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(PCED_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
  return PCED_OK;
}

// Tensor map over a cache of `rows` rows of D bf16 (D = 64 or 128) whose box
// is a whole 64-row K or V tile in one copy: dimension 0 is 64 elements
// (128 bytes, the swizzle span), dimension 1 the rows, dimension 2 the D/64
// column blocks of a row.  Shared memory receives [D/64][box_rows][128 B] with
// the 128-byte swizzle, the layout of D/64 separate 64-column boxes.
pced_status make_tmap_kv(CUtensorMap* map, const void* base, uint64_t rows, uint32_t D, uint32_t box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return fail(PCED_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
  if ((D != 64 && D != 128) || box_rows < 1 || box_rows > 256 || rows < 1 || rows > (1ull << 32) ||
      ((uintptr_t)base & 15u))
    return fail(PCED_ERR_INVALID_ARG, "kv tensor map: unsupported geometry");
  const cuuint64_t dims[3] = {64, rows, D / 64};
  const cuuint64_t strides[2] = {(cuuint64_t)D * 2, 128};
  const cuuint32_t box[3] = {64, box_rows, D / 64};
  const cuuint32_t es[3] = {1, 1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(PCED_ERR_CUDA, "cuTensorMapEncodeTiled (kv tile) failed (%d)", (int)r);
  return PCED_OK;
}

}  // namespace pced_host

extern "C" const char* pced_status_string(int32_t status) {
  switch (status) {
    case PCED_OK: return "ok";
    case PCED_ERR_INVALID_ARG: return "invalid argument";
    case PCED_ERR_WORKSPACE: return "workspace too small or misaligned";
    case PCED_ERR_UNSUPPORTED: return "unsupported shape";
    case PCED_ERR_CUDA: return "CUDA error";
    case PCED_ERR_NO_DEVICE: return "no CUDA device";
    default: return "unknown status";
  }
}

extern "C" const char* pced_last_error(void) { return pced_host::g_err; }
