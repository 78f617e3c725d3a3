// attention.cuh -- split-KV decode attention over per-expert caches (declarations
// shared by the attention translation unit and the step orchestration).
#pragma once
#include "common.cuh"

namespace pced {

constexpr int ATT_BLOCK_N = 64;     // keys per pipeline stage
constexpr int ATT_CONSUMERS = 8;    // two warpgroups of four warps; warpgroup g takes the CTA's tiles with
                                    // index = g (mod 2), warp w of a group owns keys [16w, 16w+16) of a tile
constexpr int ATT_THREADS = (ATT_CONSUMERS + 1) * 32;
constexpr int ATT_MAX_S = 1024;     // sequences per launch (prefix table lives in shared memory)
constexpr int ATT_MAX_G = 8;        // query heads per kv-head (mma N = 8)
constexpr int ATT_MAX_CTAS = 1024;  // upper bound of the grid (sizes the partial-record pool)

// Partition of all (kv-head, sequence, key) positions into equal contiguous
// ranges, one per CTA.  Position of key k of kv-head h of sequence s:
//   h * T + pre[s] + k,   pre[s] = sum_{s' < s} len[s'],  T = pre[S].
// Head-major order spreads short segments (the amateurs) across CTAs.  A
// CTA's range is cut into pieces at segment boundaries; the partial result of
// CTA c over segment seg = h*S + s is stored in record slot c + seg (slots are
// unique: each step along the position axis crosses a CTA boundary or a
// segment boundary, or both).
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
  int64_t* plan_pre;          // [S+1] written by CTA 0 (prefix of len)
  int64_t* plan_per;          // [1]   written by CTA 0: keys per CTA
  int* status;
};

size_t att_records_bytes(int32_t S, int32_t Hq, int32_t Hkv, int32_t D);
int att_grid(int64_t total_cap_keys);
// launch the split kernel for head dim D (64 or 128)
cudaError_t att_split_launch(int D, const CUtensorMap& kmap, const CUtensorMap& vmap, const AttArgs& a, int ctas,
                             cudaStream_t stream);

// Combine the partial records of one layer; one CTA per (kv-head, sequence).
//   mode 0: out[s][hq][dd] = o (fp32)
//   mode 1: resid[s] += o for the CTA's heads; the last CTA of a sequence
//           then forms u = bf16(rmsnorm(resid[s])) and either writes u to
//           q_next and appends the next layer's K/V rows at seq_len[s]-1, or
//           (last layer) writes u to hidden (and hidden_copy if non-null).
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
  float* part_ss;             // mode 1 [S][Hkv] partial sums of squares
  int32_t* counters;          // mode 1 [S] arrival counters (zero between launches)
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
