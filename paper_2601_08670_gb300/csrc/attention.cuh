// attention.cuh -- split-KV decode attention over per-expert caches (declarations
// shared by the attention translation units and the step orchestration).
#pragma once
#include "common.cuh"

namespace pced {

constexpr int ATT_BLOCK_N = 64;     // keys per pipeline stage
constexpr int ATT_CONSUMERS = 8;    // two warpgroups of four warps; warpgroup g takes the CTA's tiles with
                                    // index = g (mod 2), warp w of a group owns keys [16w, 16w+16) of a tile
constexpr int ATT_THREADS = (ATT_CONSUMERS + 1) * 32;
constexpr int ATT_CT = ATT_CONSUMERS * 32;  // consumer threads
constexpr int ATT_MAX_S = 1024;     // sequences per launch (prefix table lives in shared memory)
constexpr int ATT_MAX_G = 8;        // query heads per kv-head (mma N = 8)
constexpr int ATT_MAX_CTAS = 1024;  // upper bound of the grid (sizes the partial-record pool)
constexpr float ATT_RESCALE_SLACK = 8.f;  // log2 units the online-softmax reference may trail the max
constexpr int ATT_MAX_GROUPS = 4;   // sequence groups of the step kernel
constexpr int ATT_PTAB = 1024;       // block-table entries a step-kernel CTA keeps in shared memory

// ---------------------------------------------------------------- one layer
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

// Combine the partial records of one layer; one CTA per (kv-head, sequence):
// out[s][hq][dd] = o (fp32).
struct CombineArgs {
  int32_t S, Hq, Hkv, G, D;
  const float* rec_o;
  const float2* rec_ml;
  const int64_t* plan_pre;
  const int64_t* plan_per;
  float* out;
  int* status;
};
cudaError_t att_combine_launch(const CombineArgs& a, cudaStream_t stream);

// ------------------------------------------------------- whole decode step
// One cooperative launch runs the embedding and every layer of the step.
//
// Partition: head-major positions as above, but each segment (h, s) spans
// len[s] + seg_cost positions; the last seg_cost hold no keys and stand for
// the fixed cost of a piece (query formation, partial merge, record), so CTAs
// that cover many short segments get fewer keys.  With paged caches the
// extents are rounded up to whole 64-key tiles and the CTA boundaries down to
// multiples of 64 positions, so every piece starts on a tile boundary and no
// tile straddles two blocks (blocks hold a multiple of 64 rows).  The partition is the same
// at every layer, so the producer warp streams K/V tiles straight through all
// layers (a shared-memory ring plus L2 prefetch ahead of it) while the
// consumers wait for the layer dependency.
//
// Roles inside a CTA (warp-specialised, hand-offs through double-buffered
// shared-memory slots guarded by mbarriers): a producer warp (TMA), an input
// warp that prepares each piece's query bf16(x_l * inv_rms(x_l)) and the row
// appended this step, and eight consumer warps that run the attention math and
// then combine their partials through shared memory (each thread ends up
// owning four consecutive outputs of one head).  K and V tiles arrive as one
// 3-D tensor copy each.
//
// Sequence groups: the sequences are cut into `groups` contiguous ranges of
// about equal weight and every range is partitioned over all CTAs as above.
// A CTA takes layer l of group 0, then of group 1, ..., then layer l+1 of
// group 0: while one group's layer dependency resolves (merges, residual
// update, next query), the CTAs stream the next group's keys.  Record slots of
// group g start at g * (gridDim.x + S * Hkv).
//
// Layer dependency: a segment split over CTAs c0..c1 is completed by c0 (for
// which it is the last piece of the layer); c0+1..c1 publish their records
// for it.  The completing CTA adds the head group's attention output to the
// residual stream, x_{l+1} = x_l + o (double buffered by layer parity), and
// stores the group's sum of squares.  A piece of layer l waits for its head
// group of x_l[s] and all group sums of x_l[s].  Everything exchanged between
// CTAs is a tagged 64-bit word (see attention.cu).  After the last layer each
// completing CTA writes its head group of the final hidden state; the last
// CTA to finish advances seq_len and the epoch.
struct StepAttArgs {
  int32_t S, Hq, Hkv, G, L, n1, V, bos, max_steps;
  int64_t rows_per_layer;     // rows (of D elements) of one layer's region in the tensor maps
  int64_t layer_elems;
  float scale_log2, rms_eps;
  int32_t seg_cost;           // partition weight of a piece, in keys
  int32_t seg_lead;           // how many of the seg_cost positions come before the keys (the rest after)
  int32_t pf_tiles;           // tiles prefetched into L2 ahead of the shared-memory ring
  int32_t groups;             // sequence groups (1..ATT_MAX_GROUPS), each partitioned over all CTAs
  const int64_t* kv_offset;   // [S] (slab layout)
  const int32_t* cap;         // [S]
  const int32_t* block_table; // [S][max_blocks] (paged layout) or null
  int32_t block_rows, max_blocks, num_blocks;
  int32_t block_shift;        // log2(block_rows) when it is a power of two, else -1
  float rope_theta;           // rotary base (0: no rotary embedding)
  int32_t* seq_len;           // [S] +1 per launch for every sequence with room
  const int32_t* step;        // [1] step counter t (token y_{t-1} = history[b][t-1])
  const int32_t* history;     // [B][max_steps]
  const __nv_bfloat16* embed; // [V][d]
  __nv_bfloat16* k_cache;
  __nv_bfloat16* v_cache;
  uint64_t* resid;            // [2][S][d] tagged residual stream x_l (buffer l % 2)
  uint64_t* part_ss;          // [2][S][Hkv][8] tagged sums of squares of x_l per head group and consumer warp
  uint64_t* rec_o;            // [slots][G*D] tagged partial outputs
  uint64_t* rec_ml;           // [slots][G][2] tagged (max, sum)
  int32_t* epoch;             // [1] launches completed (tags name the launch)
  int32_t* done_cnt;          // [1] CTAs finished (zero between launches)
  __nv_bfloat16* hidden;      // [S][d] final hidden state
  __nv_bfloat16* hidden_copy; // optional copy of `hidden`
  unsigned long long wait_ns; // limit of the kernel's waits on other warps and CTAs (PCED_DEV_TIMEOUT after it)
  int* status;
};
constexpr int ATT_MAX_LAYERS = 1000;  // layer index fits the 10-bit field of the tags
int64_t att_step_slots(int32_t S, int32_t Hkv);
// tuning of the partition and the prefetch distance (PCED_ATT_SEGCOST /
// PCED_ATT_PF in the environment override the defaults)
int att_step_seg_cost(int D);
int att_step_pf_tiles();
int att_step_groups();
int att_step_seg_lead(int seg_cost);
cudaError_t att_step_launch(int D, const CUtensorMap& kmap, const CUtensorMap& vmap, const StepAttArgs& a, int ctas,
                            cudaStream_t stream);

}  // namespace pced
