// attention.cuh -- split-KV decode attention over per-expert caches (declarations
// shared by the attention translation unit and the step orchestration).
#pragma once
#include "common.cuh"

namespace pced {

constexpr int ATT_BLOCK_N = 64;     // keys per pipeline stage
constexpr int ATT_CONSUMERS = 4;    // consumer warps; warp w owns keys [16w, 16w+16) of every stage
constexpr int ATT_THREADS = (ATT_CONSUMERS + 1) * 32;
constexpr int ATT_MAX_S = 1024;     // sequences per launch (prefix table lives in shared memory)
constexpr int ATT_MAX_G = 8;        // query heads per kv-head (mma N = 8)
constexpr int ATT_MAX_CTAS = 1024;  // upper bound of the grid (sizes the partial-record pool)

// Partition of all (sequence, kv-head, key) positions into equal contiguous
// ranges, one per CTA.  Position of key k of kv-head h of sequence s:
//   pre[s] + h * len[s] + k,   pre[s] = Hkv * sum_{s' < s} len[s'].
// A CTA's range is cut into pieces at (s, h) boundaries; the partial result of
// CTA c over segment seg = s*Hkv + h is stored in record slot c + seg (slots
// are unique: each step along the position axis crosses either a CTA or a
// segment boundary).
struct AttPlan {
  int64_t total;  // sum over segments of their lengths
  int64_t per;    // keys per CTA (last CTA may get fewer)
  int32_t ctas;
};

struct AttArgs {
  const __nv_bfloat16* q;     // [S][Hq][D]
  const int64_t* kv_offset;   // [S]
  const int32_t* cap;         // [S]
  const int32_t* seq_len;     // [S]
  int32_t S, Hq, Hkv, G;
  int64_t row_base;           // row of this layer's region in the tensor maps
  float scale_log2;           // softmax scale * log2(e)
  float* rec_o;               // [slots][G][D] unnormalised partial outputs
  float2* rec_ml;             // [slots][G] (running max in log2 units, sum of exp2)
  int64_t* plan_pre;          // [S+1] written by CTA 0 (prefix of Hkv*len)
  int64_t* plan_per;          // [1]   written by CTA 0
  int* status;
};

size_t att_records_bytes(int32_t S, int32_t Hq, int32_t Hkv, int32_t D);
int att_grid(int64_t total_cap_keys);
// launch the split kernel for head dim D (64 or 128)
cudaError_t att_split_launch(int D, const CUtensorMap& kmap, const CUtensorMap& vmap, const AttArgs& a, int ctas,
                             cudaStream_t stream);

// Combine partial records of one layer.
//   mode 0: out[s][hq][dd] = o (fp32)
//   mode 1: resid[s] += o; u = bf16(rmsnorm(resid[s])); then either write u to
//           q_next and append K/V rows of layer `next_layer` at seq_len[s]-1,
//           or (last layer) write u to hidden (and hidden_copy if non-null).
struct CombineArgs {
  int mode;
  int32_t S, Hq, Hkv, G, D;
  const float* rec_o;
  const float2* rec_ml;
  const int64_t* plan_pre;
  const int64_t* plan_per;
  const int32_t* seq_len;
  float* out;                 // mode 0
  float* resid;               // mode 1 [S][d]
  float rms_eps;
  __nv_bfloat16* q_next;      // mode 1, not last layer
  __nv_bfloat16* hidden;      // mode 1, last layer
  __nv_bfloat16* hidden_copy; // optional
  __nv_bfloat16* k_cache;     // mode 1: caches and geometry for the append
  __nv_bfloat16* v_cache;
  const int64_t* kv_offset;
  const int32_t* cap;
  int64_t next_layer_elem_base;  // element offset of the next layer's region
  int append;                 // 1: append into the next layer (not last layer)
  int* status;
};
cudaError_t att_combine_launch(const CombineArgs& a, cudaStream_t stream);

}  // namespace pced
