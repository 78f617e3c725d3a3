// attention.cu -- decode attention of every expert over its own KV cache
// (paper Sec. 3: N+1 parallel streams, each with an independently encoded
// cache; grouped-query heads).
//
// Split-KV flash decoding on sm_103a, shared by both kernels of this file:
//   * all (kv-head, sequence, key) positions are cut into equal contiguous
//     ranges, one per CTA, so ragged caches load-balance without a host plan;
//   * a producer warp streams 64-key K and V tiles through a multi-stage
//     shared-memory ring with TMA (2-D tensor copies, 128-byte swizzle),
//     completion tracked by mbarriers;
//   * two warpgroups of consumer warps take alternate tiles; each warp owns 16
//     keys of a tile and computes, for the G query heads sharing the kv-head,
//     S^T = K Q^T and O^T += V^T P^T with bf16 mma.sync (fp32 accumulate),
//     online softmax in base 2 with warp shuffles; P is split into bf16 hi +
//     lo parts so the PV product keeps ~16 significant bits;
//   * per piece, the eight warps' partials are merged in shared memory into one
//     unnormalised record (max, sum, o); records of a segment split across
//     CTAs are merged by a combine kernel (one layer) or by the last CTA to
//     finish the segment (whole decode step, see att_step_kernel).
#include <math.h>
#include <stdlib.h>

#include "attention.cuh"

namespace pced {

template <int D>
struct AttCfg {
  static constexpr int BOXES = D / 64;                  // 64-element TMA boxes per row
  static constexpr int BOX_BYTES = ATT_BLOCK_N * 128;   // 64 rows x 128 B
  static constexpr int TILE_BYTES = BOXES * BOX_BYTES;  // K (or V) part of a stage
  static constexpr int STAGE_BYTES = 2 * TILE_BYTES;
  static constexpr int STAGES = D == 128 ? 5 : 7;       // odd: consecutive uses of a stage alternate warpgroups
  static constexpr int KSTEPS = D / 16;
  static constexpr int MTILES = D / 16;
  static constexpr int OPAD = 9;                        // padded head stride of the merge scratch
  static constexpr int OROW = D + 4;                    // padded row (one head of one warp) of the step kernel's partials
  static constexpr int OPT = ATT_MAX_G * D / ATT_CT;   // outputs of a piece per consumer thread (G <= 8)
  static constexpr int MERGE_FLOATS = 2 * ATT_CONSUMERS * ATT_MAX_G + ATT_CONSUMERS * D * OPAD + ATT_CONSUMERS + 8;
  static constexpr size_t BARS = (2 * STAGES + 2) * 8;
  static constexpr size_t SMEM = 1024 + (size_t)STAGES * STAGE_BYTES + BARS + (size_t)MERGE_FLOATS * 4 +
                                 (ATT_MAX_S + 1) * 8 + ATT_MAX_S * 4 + ATT_MAX_S + 128;
};

// shared-memory scratch of the consumers (after the stages and barriers)
struct Scratch {
  float* ms;      // [8][8] per-warp running max of a piece
  float* ls;      // [8][8] per-warp sum
  float* os;      // [8][D][OPAD] per-warp o
  float* red;     // [8] per-warp partial sums
  int* flag;      // [8] broadcast flags
  int64_t* pre;   // [S+1] prefix of the segment extents
  int32_t* lens;  // [S] live lengths
  uint8_t* apnd;  // [S] 1 if this step appends a row to sequence s
};

template <int D>
__device__ __forceinline__ Scratch carve_scratch(uint8_t* p) {
  using C = AttCfg<D>;
  Scratch sc;
  float* f = reinterpret_cast<float*>(p);
  sc.ms = f;
  sc.ls = f + ATT_CONSUMERS * ATT_MAX_G;
  sc.os = f + 2 * ATT_CONSUMERS * ATT_MAX_G;
  sc.red = sc.os + ATT_CONSUMERS * D * C::OPAD;
  sc.flag = reinterpret_cast<int*>(sc.red + ATT_CONSUMERS);
  sc.pre = reinterpret_cast<int64_t*>(f + C::MERGE_FLOATS);
  sc.lens = reinterpret_cast<int32_t*>(sc.pre + ATT_MAX_S + 1);
  sc.apnd = reinterpret_cast<uint8_t*>(sc.lens + ATT_MAX_S);
  return sc;
}

// Non-negative 64-bit quotient through the 32-bit divider when both operands
// fit (positions of any realistic step do); 64-bit division is a long
// software sequence.
__device__ __forceinline__ int64_t udiv_pos(int64_t a, int64_t b) {
  if ((((uint64_t)a | (uint64_t)b) >> 32) == 0) return (int64_t)((uint32_t)a / (uint32_t)b);
  return a / b;
}

struct Piece {
  int32_t s, h, k0, k1;  // real keys [k0, k1) of kv-head h of sequence s (k0 == k1: no keys)
  int64_t adv;           // positions the piece spans
};

// Piece that starts at position p of the position space of sequences
// [s_lo, s_hi) and ends at the next segment boundary or at `end`.  Segment
// (h, s) spans positions [h*T + pre[s] - pre[s_lo], h*T + pre[s+1] - pre[s_lo])
// with T = pre[s_hi] - pre[s_lo]; positions lead .. lead + lens[s] - 1 of it
// are its keys, the others (if any) only weight the partition.
__device__ __forceinline__ Piece find_piece(const int64_t* pre, const int32_t* lens, int32_t s_lo, int32_t s_hi,
                                            int64_t T, int64_t p, int64_t end, int32_t lead = 0) {
  Piece pc;
  pc.h = (int32_t)udiv_pos(p, T);
  const int64_t r = p - (int64_t)pc.h * T + pre[s_lo];
  int32_t lo = s_lo, hi = s_hi - 1;
  while (lo < hi) {
    const int32_t mid = (lo + hi + 1) >> 1;
    if (pre[mid] <= r) lo = mid;
    else hi = mid - 1;
  }
  pc.s = lo;
  const int64_t off = r - pre[lo] - lead;  // key index of position p (negative in the leading part)
  const int64_t seg_end = (int64_t)pc.h * T + pre[lo + 1] - pre[s_lo];
  const int64_t e = seg_end < end ? seg_end : end;
  pc.adv = e - p;
  const int64_t len = lens[lo];
  const int64_t k0 = off < 0 ? 0 : off, k1 = off + pc.adv < len ? off + pc.adv : len;
  if (k0 < k1) {
    pc.k0 = (int32_t)k0;
    pc.k1 = (int32_t)k1;
  } else {
    pc.k0 = pc.k1 = 0;
  }
  return pc;
}

// The piece after prev when prev ended at its segment's end p (< end): the
// next segment of the same position space, so no search is needed (find_piece
// at p gives the same piece, as every segment spans at least one position).
__device__ __forceinline__ Piece next_piece(const Piece& prev, const int64_t* pre, const int32_t* lens,
                                            int32_t s_lo, int32_t s_hi, int64_t T, int64_t p, int64_t end,
                                            int32_t lead = 0) {
  Piece pc;
  pc.s = prev.s + 1;
  pc.h = prev.h;
  if (pc.s >= s_hi) {
    pc.s = s_lo;
    ++pc.h;
  }
  const int64_t seg_end = (int64_t)pc.h * T + pre[pc.s + 1] - pre[s_lo];
  const int64_t e = seg_end < end ? seg_end : end;
  pc.adv = e - p;
  const int64_t len = lens[pc.s];
  const int64_t k1 = pc.adv - lead < len ? pc.adv - lead : len;  // keys start at offset lead
  if (k1 > 0) {
    pc.k0 = 0;
    pc.k1 = (int32_t)k1;
  } else {
    pc.k0 = pc.k1 = 0;
  }
  return pc;
}

// exclusive prefix of ext[i] = roundup(lens[i], align) + extra into pre[0..S]
// (one warp; align a power of two)
__device__ __forceinline__ void prefix_extents(const int32_t* lens, int32_t S, int32_t extra, int64_t* pre, int lane,
                                               int32_t align = 1) {
  const int chunk = (S + 31) / 32;
  const int b0 = lane * chunk, b1 = min(S, b0 + chunk);
  const int64_t am = align - 1;
  int64_t sum = 0;
  for (int i = b0; i < b1; ++i) sum += (((int64_t)lens[i] + am) & ~am) + extra;
  int64_t incl = sum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int64_t v = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += v;
  }
  int64_t run = incl - sum;
  for (int i = b0; i < b1; ++i) {
    pre[i] = run;
    run += (((int64_t)lens[i] + am) & ~am) + extra;
  }
  if (lane == 31) pre[S] = incl;
}

// ------------------------------------------------------------ consumer math
// Online-softmax state of one consumer warp over its keys of a piece.
template <int D>
struct WarpAcc {
  float m0, m1, l0, l1;  // heads 2tq and 2tq+1 of this thread
  float o[D / 16][4];    // O^T fragments: dims 16i + g (+8), heads 2tq, 2tq+1
};

template <int D>
__device__ __forceinline__ void acc_reset(WarpAcc<D>& A) {
  A.m0 = A.m1 = -INFINITY;
  A.l0 = A.l1 = 0.f;
#pragma unroll
  for (int i = 0; i < D / 16; ++i) A.o[i][0] = A.o[i][1] = A.o[i][2] = A.o[i][3] = 0.f;
}

// This warp's 16 keys [kb, kb+16) of the 64-key K/V tiles at sk / sv (TMA
// 128-byte swizzle, D/64 boxes of 64 rows x 128 B); keys at or past nvalid
// are masked.  qf: B operand of S^T = K Q^T (dims x heads).
//
// P enters the P V product as bf16 hi + lo parts.  With PK (at most four
// heads) both parts share one MMA: accumulator columns 0-3 take the hi parts
// of heads 0-3 and columns 4-7 the lo parts of the same heads (qf repeats
// heads 0-3 in columns 4-7, so the threads owning those columns, tq >= 2,
// hold the same scores as lane ^ 2), and o of head h is column h plus column
// h + 4 (summed once per piece, see pack_fold).
template <int D, bool PK = false>
__device__ __forceinline__ void tile_math(WarpAcc<D>& A, const uint32_t (&qf)[D / 16][2], uint32_t sk, uint32_t sv,
                                          int kb, int nvalid, float scale_log2, int lane) {
  using C = AttCfg<D>;
  const int g = lane >> 2, tq = lane & 3, mat = lane >> 3, mr = lane & 7;
  // ---- scores S^T (16 keys x 8 heads), four independent accumulation chains
  float sc4[4][4] = {};
  {
    const int key = kb + (mat & 1) * 8 + mr;
    const uint32_t rowa = sk + key * 128;
    const uint32_t sw = key & 7;
#pragma unroll
    for (int j = 0; j < C::KSTEPS; ++j) {
      const int chunk = 2 * j + (mat >> 1);
      const uint32_t addr = rowa + (chunk >> 3) * C::BOX_BYTES + (((chunk & 7) ^ sw) << 4);
      uint32_t a0, a1, a2, a3;
      ldsm_x4(addr, a0, a1, a2, a3);
      mma_bf16(sc4[j & 3], a0, a1, a2, a3, qf[j][0], qf[j][1]);
    }
  }
  const bool v0 = kb + g < nvalid, v1 = kb + g + 8 < nvalid;
  const float s0 = v0 ? ((sc4[0][0] + sc4[1][0]) + (sc4[2][0] + sc4[3][0])) * scale_log2 : -INFINITY;
  const float s1 = v0 ? ((sc4[0][1] + sc4[1][1]) + (sc4[2][1] + sc4[3][1])) * scale_log2 : -INFINITY;
  const float s2 = v1 ? ((sc4[0][2] + sc4[1][2]) + (sc4[2][2] + sc4[3][2])) * scale_log2 : -INFINITY;
  const float s3 = v1 ? ((sc4[0][3] + sc4[1][3]) + (sc4[2][3] + sc4[3][3])) * scale_log2 : -INFINITY;
  // The reference max only moves when a score exceeds it by more than
  // ATT_RESCALE_SLACK (log2 units): exp2 of the others stays below
  // 2^ATT_RESCALE_SLACK, and the rescale of o, l (and the max reduction across
  // the warp) is skipped for most tiles.  Any reference gives the same o / l.
  float x0 = fmaxf(s0, s2), x1 = fmaxf(s1, s3);
  if (__any_sync(0xffffffffu, x0 > A.m0 + ATT_RESCALE_SLACK || x1 > A.m1 + ATT_RESCALE_SLACK)) {
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
      x0 = fmaxf(x0, __shfl_xor_sync(0xffffffffu, x0, off));
      x1 = fmaxf(x1, __shfl_xor_sync(0xffffffffu, x1, off));
    }
    const float n0 = fmaxf(A.m0, x0), n1 = fmaxf(A.m1, x1);
    const float al0 = A.m0 == -INFINITY ? 0.f : exp2f(A.m0 - n0);
    const float al1 = A.m1 == -INFINITY ? 0.f : exp2f(A.m1 - n1);
    A.l0 *= al0;
    A.l1 *= al1;
#pragma unroll
    for (int i = 0; i < C::MTILES; ++i) {
      A.o[i][0] *= al0;
      A.o[i][2] *= al0;
      A.o[i][1] *= al1;
      A.o[i][3] *= al1;
    }
    A.m0 = n0;
    A.m1 = n1;
  }
  const float u0 = A.m0 == -INFINITY ? 0.f : A.m0, u1 = A.m1 == -INFINITY ? 0.f : A.m1;
  const float p0 = exp2f(s0 - u0), p1 = exp2f(s1 - u1), p2 = exp2f(s2 - u0), p3 = exp2f(s3 - u1);
  A.l0 += p0 + p2;
  A.l1 += p1 + p3;
  // ---- P^T as the B operand (keys x heads), split into bf16 hi + lo
  const uint32_t h01 = pack_bf16(p0, p1), h23 = pack_bf16(p2, p3);
  const uint32_t q01 = pack_bf16(p0 - bf16_lo(h01), p1 - bf16_hi(h01));
  const uint32_t q23 = pack_bf16(p2 - bf16_lo(h23), p3 - bf16_hi(h23));
  const bool lo_cols = PK && tq >= 2;
  const uint32_t bh0 = movmatrix_t(lo_cols ? q01 : h01), bh1 = movmatrix_t(lo_cols ? q23 : h23);
  const uint32_t bl0 = PK ? 0u : movmatrix_t(q01), bl1 = PK ? 0u : movmatrix_t(q23);
  // ---- O^T += V^T P^T; rows of V past the live length are zeroed
  const bool partial = kb + 16 > nvalid;
  const int klo = kb + 2 * tq, khi = klo + 8;
  const int key = kb + (mat >> 1) * 8 + mr;
  const uint32_t rowa = sv + key * 128;
  const uint32_t sw = key & 7;
#pragma unroll
  for (int i = 0; i < C::MTILES; ++i) {
    const int chunk = 2 * i + (mat & 1);
    const uint32_t addr = rowa + (chunk >> 3) * C::BOX_BYTES + (((chunk & 7) ^ sw) << 4);
    uint32_t a0, a1, a2, a3;
    ldsm_x4_t(addr, a0, a1, a2, a3);
    if (partial) {
      const uint32_t mlo = (klo < nvalid ? 0xFFFFu : 0u) | (klo + 1 < nvalid ? 0xFFFF0000u : 0u);
      const uint32_t mhi = (khi < nvalid ? 0xFFFFu : 0u) | (khi + 1 < nvalid ? 0xFFFF0000u : 0u);
      a0 &= mlo;
      a1 &= mlo;
      a2 &= mhi;
      a3 &= mhi;
    }
    mma_bf16(A.o[i], a0, a1, a2, a3, bh0, bh1);
    if (!PK) mma_bf16(A.o[i], a0, a1, a2, a3, bl0, bl1);
  }
}

// After tile_math<D, true>: o of heads 2tq, 2tq+1 in the threads with tq < 2
// (hi columns plus the lo columns held by lane ^ 2).
template <int D>
__device__ __forceinline__ void pack_fold(WarpAcc<D>& A) {
#pragma unroll
  for (int i = 0; i < D / 16; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) A.o[i][j] += __shfl_xor_sync(0xffffffffu, A.o[i][j], 2);
}

// Merge the eight consumer warps' accumulators of a piece through shared
// memory.  Afterwards this thread holds, for outputs idx = ctid + k*ATT_CT
// (idx = hh*D + dd < G*D), the piece's running max mx[k] (log2 units), sum
// ls[k] and unnormalised output acc[k].
template <int D>
__device__ __forceinline__ bool cta_merge(const WarpAcc<D>& A, const Scratch& sc, int G, int warp, int lane, int ctid,
                                          uint32_t bar, uint32_t& ph, int* status, float (&mx)[AttCfg<D>::OPT],
                                          float (&ls)[AttCfg<D>::OPT], float (&acc)[AttCfg<D>::OPT]) {
  using C = AttCfg<D>;
  const int g = lane >> 2, tq = lane & 3;
  float l0 = A.l0, l1 = A.l1;
#pragma unroll
  for (int off = 4; off < 32; off <<= 1) {
    l0 += __shfl_xor_sync(0xffffffffu, l0, off);
    l1 += __shfl_xor_sync(0xffffffffu, l1, off);
  }
  // every consumer is done with the previous piece's scratch
  if (!warps_sync(bar, ph, status)) return false;
  if (g == 0) {
    sc.ms[warp * ATT_MAX_G + 2 * tq] = A.m0;
    sc.ms[warp * ATT_MAX_G + 2 * tq + 1] = A.m1;
    sc.ls[warp * ATT_MAX_G + 2 * tq] = l0;
    sc.ls[warp * ATT_MAX_G + 2 * tq + 1] = l1;
  }
  float* ow = sc.os + warp * D * C::OPAD;
#pragma unroll
  for (int i = 0; i < C::MTILES; ++i) {
    const int d0 = 16 * i + g, d1 = d0 + 8;
    ow[d0 * C::OPAD + 2 * tq] = A.o[i][0];
    ow[d0 * C::OPAD + 2 * tq + 1] = A.o[i][1];
    ow[d1 * C::OPAD + 2 * tq] = A.o[i][2];
    ow[d1 * C::OPAD + 2 * tq + 1] = A.o[i][3];
  }
  if (!warps_sync(bar, ph, status)) return false;
#pragma unroll
  for (int k = 0; k < C::OPT; ++k) {
    const int idx = ctid + k * ATT_CT;
    mx[k] = -INFINITY;
    ls[k] = 0.f;
    acc[k] = 0.f;
    if (idx >= G * D) continue;
    const int hh = idx / D, dd = idx - hh * D;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < ATT_CONSUMERS; ++w) M = fmaxf(M, sc.ms[w * ATT_MAX_G + hh]);
    float a = 0.f, l = 0.f;
#pragma unroll
    for (int w = 0; w < ATT_CONSUMERS; ++w) {
      const float mw = sc.ms[w * ATT_MAX_G + hh];
      if (mw == -INFINITY) continue;
      const float e = exp2f(mw - M);
      a += sc.os[(w * D + dd) * C::OPAD + hh] * e;
      l += sc.ls[w * ATT_MAX_G + hh] * e;
    }
    mx[k] = M;
    ls[k] = l;
    acc[k] = a;
  }
  return true;
}

// =================================================================== one layer
template <int D>
__global__ void __launch_bounds__(ATT_THREADS, 1)
    att_split_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap, AttArgs a) {
  using C = AttCfg<D>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  // layout: stages | full[STAGES] | empty[STAGES] | consumer barrier | spare | scratch
  const uint32_t bar_full = base + C::STAGES * C::STAGE_BYTES;
  const uint32_t bar_empty = bar_full + C::STAGES * 8;
  const uint32_t bar_c = bar_empty + C::STAGES * 8;
  const Scratch sc = carve_scratch<D>(gbase + C::STAGES * C::STAGE_BYTES + C::BARS);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int32_t S = a.S, G = a.G;

  if (tid == 0) {
    for (int i = 0; i < C::STAGES; ++i) {
      mbar_init(bar_full + 8 * i, 1);
      mbar_init(bar_empty + 8 * i, 4);  // the four warps of the consuming warpgroup
    }
    mbar_init(bar_c, ATT_CONSUMERS);
    mbar_fence_init();
  }
  if (warp == ATT_CONSUMERS && lane == 0) {
    tma_prefetch_desc(&kmap);
    tma_prefetch_desc(&vmap);
  }
  // live lengths, clamped into [1, cap] (out-of-range lengths are flagged)
  for (int i = tid; i < S; i += ATT_THREADS) {
    int32_t L = a.seq_len[i], c = a.cap[i];
    if (L < 1 || L > c) {
      dev_flag(a.status, PCED_DEV_BAD_LENGTH);
      L = L < 1 ? 1 : (L > c ? (c < 1 ? 1 : c) : L);
    }
    sc.lens[i] = L;
  }
  __syncthreads();
  if (warp == 0) prefix_extents(sc.lens, S, 0, sc.pre, lane);
  __syncthreads();
  const int64_t* pre = sc.pre;
  const int32_t* lens = sc.lens;
  const int64_t T = pre[S];
  const int64_t total = T * a.Hkv;
  const int64_t per = (total + gridDim.x - 1) / gridDim.x;
  if (blockIdx.x == 0) {
    for (int i = tid; i <= S; i += ATT_THREADS) a.plan_pre[i] = pre[i];
    if (tid == 0) *a.plan_per = per;
  }
  const int64_t r_begin = min(total, (int64_t)blockIdx.x * per);
  const int64_t r_end = min(total, r_begin + per);

  if (warp == ATT_CONSUMERS) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      uint32_t it = 0;
      bool ok = true;
      for (int64_t p = r_begin; p < r_end && ok;) {
        const Piece pc = find_piece(pre, lens, 0, S, T, p, r_end);
        p += pc.adv;
        const int64_t slab_row = a.row_base + (a.kv_offset[pc.s] + (int64_t)pc.h * a.cap[pc.s] * D) / D;
        for (int32_t kt = pc.k0; kt < pc.k1; kt += ATT_BLOCK_N, ++it) {
          const uint32_t st = it % C::STAGES, ph = (it / C::STAGES) & 1u;
          if (!mbar_wait(bar_empty + 8 * st, ph ^ 1u, a.status)) {
            ok = false;
            break;
          }
          const uint32_t fb = bar_full + 8 * st;
          const uint32_t sk = base + st * C::STAGE_BYTES, sv = sk + C::TILE_BYTES;
          mbar_arrive_expect_tx(fb, C::STAGE_BYTES);
          const int32_t row = (int32_t)(slab_row + kt);
          tma_load_3d(sk, &kmap, fb, 0, row, 0, pol);
          tma_load_3d(sv, &vmap, fb, 0, row, 0, pol);
        }
      }
      if (!ok) {
        // let copies already in flight land before the CTA exits
        for (uint32_t j = (it >= C::STAGES ? it - C::STAGES : 0); j < it; ++j)
          mbar_wait(bar_full + 8 * (j % C::STAGES), (j / C::STAGES) & 1u, a.status);
      }
    }
    return;
  }

  // -------------------------------------------------------------- consumers
  const int wg = warp >> 2, wl = warp & 3;
  const int g = lane >> 2, tq = lane & 3;
  const int kb = 16 * wl;
  uint32_t it = 0, cph = 0;
  bool ok = true;
  for (int64_t p = r_begin; p < r_end && ok;) {
    const Piece pc = find_piece(pre, lens, 0, S, T, p, r_end);
    p += pc.adv;
    uint32_t qf[C::KSTEPS][2];
    {
      const bool hv = g < G;
      const uint32_t* qrow = reinterpret_cast<const uint32_t*>(
          a.q + ((int64_t)pc.s * a.Hq + (int64_t)pc.h * G + (hv ? g : 0)) * D);
#pragma unroll
      for (int j = 0; j < C::KSTEPS; ++j) {
        qf[j][0] = hv ? qrow[8 * j + tq] : 0u;
        qf[j][1] = hv ? qrow[8 * j + 4 + tq] : 0u;
      }
    }
    WarpAcc<D> A;
    acc_reset(A);
    for (int32_t kt = pc.k0; kt < pc.k1; kt += ATT_BLOCK_N, ++it) {
      if ((int)(it & 1u) != wg) continue;
      const uint32_t use = it / C::STAGES, st = it % C::STAGES, ph = use & 1u;
      // Consecutive uses of a stage belong to different warpgroups.  Waiting for
      // the release of the previous use first guarantees that the full barrier
      // has completed that use's phase, so the parity test below refers to this
      // tile's phase and not to the older one with the same parity.
      if (use > 0 && !mbar_wait(bar_empty + 8 * st, (use - 1u) & 1u, a.status)) {
        ok = false;
        break;
      }
      if (!mbar_wait(bar_full + 8 * st, ph, a.status)) {
        ok = false;
        break;
      }
      const int nvalid = min(ATT_BLOCK_N, pc.k1 - kt);
      if (kb < nvalid) {
        const uint32_t sk = base + st * C::STAGE_BYTES;
        tile_math<D>(A, qf, sk, sk + C::TILE_BYTES, kb, nvalid, a.scale_log2, lane);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(bar_empty + 8 * st);
    }
    if (!ok) break;
    float mx[C::OPT], ls[C::OPT], acc[C::OPT];
    if (!cta_merge<D>(A, sc, G, warp, lane, tid, bar_c, cph, a.status, mx, ls, acc)) break;
    const int64_t slot = (int64_t)blockIdx.x + (int64_t)pc.h * S + pc.s;
#pragma unroll
    for (int k = 0; k < C::OPT; ++k) {
      const int idx = tid + k * ATT_CT;
      if (idx >= G * D) continue;
      a.rec_o[slot * G * D + idx] = acc[k];
      if (idx % D == 0) a.rec_ml[slot * G + idx / D] = make_float2(mx[k], ls[k]);
    }
    if (!warps_sync(bar_c, cph, a.status)) break;
  }
}

// One CTA per (kv-head h, sequence s): weights of the records that cover the
// segment are formed once in shared memory, then every output element sums
// its records with independent loads.
constexpr int CMB_THREADS = 128;
constexpr int CMB_SLOTS = 64;                                  // records weighted per pass
constexpr int CMB_PER_THREAD = ATT_MAX_G * 128 / CMB_THREADS;  // G*D <= 1024 outputs per CTA

__global__ void __launch_bounds__(CMB_THREADS) att_combine_kernel(CombineArgs a) {
  const int h = blockIdx.x, s = blockIdx.y, tid = threadIdx.x;
  const int32_t Hq = a.Hq, G = a.G, D = a.D, S = a.S, d = Hq * D;
  __shared__ float wts[CMB_SLOTS][ATT_MAX_G];
  const int64_t per = *a.plan_per;
  const int64_t T = a.plan_pre[S];
  const int64_t pre_s = a.plan_pre[s];
  const int64_t len = a.plan_pre[s + 1] - pre_s;
  const int64_t seg = (int64_t)h * S + s;
  const int64_t pa = (int64_t)h * T + pre_s;
  const int64_t c0 = pa / per, c1 = (pa + len - 1) / per;
  const int GD = G * D;

  // global max and total of each head over all records of the segment
  float Mh = -INFINITY, Lh = 0.f;
  if (tid < G) {
    for (int64_t c = c0; c <= c1; ++c) Mh = fmaxf(Mh, a.rec_ml[(c + seg) * G + tid].x);
    for (int64_t c = c0; c <= c1; ++c) {
      const float2 ml = a.rec_ml[(c + seg) * G + tid];
      if (ml.x != -INFINITY) Lh += ml.y * exp2f(ml.x - Mh);
    }
  }
  __shared__ float Msh[ATT_MAX_G], Lsh[ATT_MAX_G];
  if (tid < G) {
    Msh[tid] = Mh;
    Lsh[tid] = Lh;
  }
  float acc[CMB_PER_THREAD];
#pragma unroll
  for (int j = 0; j < CMB_PER_THREAD; ++j) acc[j] = 0.f;
  for (int64_t cb = c0; cb <= c1; cb += CMB_SLOTS) {
    const int64_t rem = c1 + 1 - cb;
    const int n = (int)(rem < CMB_SLOTS ? rem : CMB_SLOTS);
    __syncthreads();
    for (int i = tid; i < n * G; i += CMB_THREADS) {
      const int ci = i / G, gh = i - ci * G;
      const float2 ml = a.rec_ml[(cb + ci + seg) * G + gh];
      wts[ci][gh] = ml.x == -INFINITY ? 0.f : exp2f(ml.x - Msh[gh]) / Lsh[gh];
    }
    __syncthreads();
    for (int ci = 0; ci < n; ++ci) {
      const float* ro = a.rec_o + (cb + ci + seg) * GD;
#pragma unroll
      for (int j = 0; j < CMB_PER_THREAD; ++j) {
        const int idx = tid + j * CMB_THREADS;
        if (idx < GD) acc[j] += wts[ci][idx / D] * ro[idx];
      }
    }
  }
#pragma unroll
  for (int j = 0; j < CMB_PER_THREAD; ++j) {
    const int idx = tid + j * CMB_THREADS;
    if (idx < GD) a.out[(int64_t)s * d + (int64_t)h * GD + idx] = acc[j];
  }
}

// ============================================================ whole step
// Values exchanged between CTAs inside the step kernel are 64-bit words
// (fp32 value, 32-bit tag) written and read with single relaxed gpu-scope
// accesses, so a reader that sees the expected tag also sees the value: no
// fences or arrival counters are needed, and a wait is a poll on the data
// itself.  tag(l) = (epoch << 10) | (l + 1) names the launch and the layer
// whose input the word belongs to (never 0, so zeroed memory never matches).
__device__ __forceinline__ uint32_t step_tag(int32_t epoch, int l) {
  return ((uint32_t)epoch << 10) | (uint32_t)(l + 1);
}
__device__ __forceinline__ void st_tagged(uint64_t* p, float v, uint32_t tag) {
  const uint64_t w = ((uint64_t)tag << 32) | (uint64_t)__float_as_uint(v);
  asm volatile("st.relaxed.gpu.global.b64 [%0], %1;" ::"l"(p), "l"(w) : "memory");
}
__device__ __forceinline__ uint64_t ld_tagged(const uint64_t* p) {
  uint64_t w;
  asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(w) : "l"(p) : "memory");
  return w;
}
__device__ __forceinline__ float tv_value(uint64_t w) { return __uint_as_float((uint32_t)w); }
__device__ __forceinline__ bool tv_ok(uint64_t w, uint32_t tag) { return (uint32_t)(w >> 32) == tag; }

// Bounded poll used by the tagged waits: false once the time limit is spent.
__device__ __forceinline__ bool poll_again(uint64_t& t0, int* status, unsigned long long limit_ns = kWaitLimitNs) {
  const uint64_t now = globaltimer_ns();
  if (t0 == 0) t0 = now;
  if (now - t0 > limit_ns) {
    dev_flag(status, PCED_DEV_TIMEOUT);
    return false;
  }
  __nanosleep(128);  // fewer polls of L2 while the data is on its way (measured 1-4 us faster per step than 32 ns)
  return true;
}

// Sequence groups of the step kernel and this CTA's range in each (shared
// memory, written once by thread 0).
struct GroupPlan {
  int32_t n;
  int32_t s_lo[ATT_MAX_GROUPS + 1];  // group g holds sequences [s_lo[g], s_lo[g+1])
  int64_t T[ATT_MAX_GROUPS];         // positions per kv-head
  int64_t P[ATT_MAX_GROUPS];         // positions per CTA
  int64_t cb[ATT_MAX_GROUPS], ce[ATT_MAX_GROUPS];
};

// Cut the sequences into min(want, S) contiguous groups of about equal weight
// (pre: prefix of the extents) and partition each over the grid.  align (a
// power of two dividing every extent): CTA c of a group takes positions
// [c*P, (c+1)*P) rounded down to multiples of align, with P at least align,
// so every CTA range is a whole number of tiles and none inside a segment is
// empty (the CTAs holding a segment's keys stay consecutive).
__device__ __forceinline__ void plan_groups(GroupPlan& gp, const int64_t* pre, int32_t S, int32_t Hkv, int want,
                                            int64_t grid, int64_t cta, int32_t align = 1) {
  int ng = want < 1 ? 1 : (want > ATT_MAX_GROUPS ? ATT_MAX_GROUPS : want);
  if (ng > S) ng = S;
  const int64_t T = pre[S];
  gp.s_lo[0] = 0;
  for (int g = 1; g < ng; ++g) {
    const int64_t target = T * g / ng;
    int32_t s = gp.s_lo[g - 1] + 1;
    while (s < S - (ng - g) && pre[s] < target) ++s;
    gp.s_lo[g] = s;
  }
  gp.s_lo[ng] = S;
  for (int g = 0; g < ng; ++g) {
    const int64_t Tg = pre[gp.s_lo[g + 1]] - pre[gp.s_lo[g]];
    const int64_t tot = (int64_t)Hkv * Tg;
    int64_t Pg = (tot + grid - 1) / grid;
    if (Pg < align) Pg = align;
    const int64_t am = ~(int64_t)(align - 1);
    gp.T[g] = Tg;
    gp.P[g] = Pg;
    gp.cb[g] = min(tot, cta * Pg) & am;
    gp.ce[g] = min(tot, (cta + 1) * Pg) & am;
  }
  gp.n = ng;
}

// Block index of key x (paged caches).
__device__ __forceinline__ int32_t block_of(const StepAttArgs& a, int32_t x) {
  return a.block_shift >= 0 ? x >> a.block_shift : (int32_t)((uint32_t)x / (uint32_t)a.block_rows);
}

// Row, within a layer's region of the tensor maps, of key 0 of kv-head h in
// block blk (of [Hkv][P][D]); -1 for a block id outside the pool (flagged).
__device__ __forceinline__ int32_t block_base_of(const StepAttArgs& a, int32_t blk, int32_t h) {
  if (blk < 0 || blk >= a.num_blocks) {
    dev_flag(a.status, PCED_DEV_BAD_BLOCK);
    return -1;
  }
  return (blk * a.Hkv + h) * a.block_rows;  // below rows_per_layer < 2^31
}

// block_base_of for block j of (sequence s, kv-head h): entry i of the CTA's
// shared copy (built once per launch for the pieces of one layer, ptab_n
// entries) or, past the copy, from the table in global memory.
__device__ __forceinline__ int32_t block_base(const StepAttArgs& a, int32_t s, int32_t h, int32_t j, int32_t i,
                                              const int32_t* ptab, int32_t ptab_n) {
  if (i < ptab_n) return ptab[i];
  return block_base_of(a, j < a.max_blocks ? __ldg(a.block_table + (int64_t)s * a.max_blocks + j) : -1, h);
}

// The CTA whose range (as plan_groups cuts it) holds position x.
__device__ __forceinline__ int64_t part_cta(int64_t x, int64_t Pg, int32_t align) {
  return udiv_pos((x & ~(int64_t)(align - 1)) + align - 1, Pg);
}

// Tile cursor over a CTA's ranges through all layers and groups (the
// producer's order: layer by layer, group by group).  Slab caches: the tile's
// tensor-map row is the slab's first row + kt.  Paged caches (PAGED): pieces
// start on 64-key boundaries (tile-aligned partition), so a tile never
// straddles two blocks; the row, row kt % P of block table[s][kt / P], is
// advanced without a division, the block is looked up once (in the CTA's
// shared copy) and the next piece is found without a search.  A bad block id
// (flagged) points the tile past the last row of the tensor map, where the
// loads read zeros.
template <bool PAGED>
struct TileCursor {
  int32_t l, g, kt;
  int64_t p, row0;  // slab caches: tensor-map row of key 0 of the current piece
  int32_t row;      // paged caches: tensor-map row of the tile
  bool bad;         // paged caches: the tile's block id is outside the pool
  int32_t kin, bj;  // paged caches: key offset of the tile in its block, the block's index
  int32_t bi, ptn;  // paged caches: block-table copy entry of block bj; of the next piece's first block
  Piece pc;
  bool ok;
  __device__ __forceinline__ int32_t tile_row() const { return PAGED ? row : (int32_t)(row0 + kt); }
};

// cont (paged caches): c.pc is the piece before position c.p in the same group
template <bool PAGED>
__device__ __forceinline__ void cursor_seek(TileCursor<PAGED>& c, const StepAttArgs& a, const int64_t* pre,
                                            const int32_t* lens, const GroupPlan& gp, int D, const int32_t* ptab,
                                            int32_t ptab_n, bool cont) {
  while (true) {
    if (c.p >= gp.ce[c.g]) {
      if (++c.g >= gp.n) {
        c.g = 0;
        if (++c.l >= a.L) {
          c.ok = false;
          return;
        }
        c.ptn = 0;  // every layer visits the same pieces
      }
      c.p = gp.cb[c.g];
      cont = false;
      continue;
    }
    if (PAGED && cont)
      c.pc = next_piece(c.pc, pre, lens, gp.s_lo[c.g], gp.s_lo[c.g + 1], gp.T[c.g], c.p, gp.ce[c.g], a.seg_lead);
    else
      c.pc = find_piece(pre, lens, gp.s_lo[c.g], gp.s_lo[c.g + 1], gp.T[c.g], c.p, gp.ce[c.g], a.seg_lead);
    cont = true;
    if (c.pc.k0 < c.pc.k1) {
      c.kt = c.pc.k0;
      if (!PAGED) {
        c.row0 = (int64_t)c.l * a.rows_per_layer + (a.kv_offset[c.pc.s] + (int64_t)c.pc.h * a.cap[c.pc.s] * D) / D;
        return;
      }
      c.bj = block_of(a, c.kt);  // kt is a multiple of 64 (tile-aligned partition)
      c.kin = c.kt - c.bj * a.block_rows;
      c.bi = c.ptn;
      c.ptn += block_of(a, c.pc.k1 - 1) - c.bj + 1;
      const int32_t b0 = block_base(a, c.pc.s, c.pc.h, c.bj, c.bi, ptab, ptab_n);
      c.bad = b0 < 0;
      c.row = (int32_t)(c.bad ? (int64_t)a.L * a.rows_per_layer : (int64_t)c.l * a.rows_per_layer + b0 + c.kin);
      return;
    }
    c.p += c.pc.adv;
  }
}
template <bool PAGED>
__device__ __forceinline__ void cursor_begin(TileCursor<PAGED>& c, const StepAttArgs& a, const int64_t* pre,
                                             const int32_t* lens, const GroupPlan& gp, int D, const int32_t* ptab,
                                             int32_t ptab_n) {
  c.l = 0;
  c.g = 0;
  c.p = gp.cb[0];
  c.ptn = 0;
  c.bad = false;
  c.ok = a.L > 0;
  if (c.ok) cursor_seek(c, a, pre, lens, gp, D, ptab, ptab_n, false);
}
template <bool PAGED>
__device__ __forceinline__ void cursor_next(TileCursor<PAGED>& c, const StepAttArgs& a, const int64_t* pre,
                                            const int32_t* lens, const GroupPlan& gp, int D, const int32_t* ptab,
                                            int32_t ptab_n) {
  c.kt += ATT_BLOCK_N;
  if (c.kt < c.pc.k1) {
    if (PAGED) {
      c.kin += ATT_BLOCK_N;
      if (c.kin == a.block_rows) {
        c.kin = 0;
        ++c.bj;
        ++c.bi;
        const int32_t b0 = block_base(a, c.pc.s, c.pc.h, c.bj, c.bi, ptab, ptab_n);
        c.bad = b0 < 0;
        c.row = (int32_t)(c.bad ? (int64_t)a.L * a.rows_per_layer : (int64_t)c.l * a.rows_per_layer + b0);
      } else if (!c.bad) {
        c.row += ATT_BLOCK_N;
      }
    }
    return;
  }
  c.p += c.pc.adv;
  cursor_seek(c, a, pre, lens, gp, D, ptab, ptab_n, true);
}

// The producer: K/V tiles of every layer in consumption order into the
// NST-stage ring; the L2 prefetch cursor runs pf_tiles ahead so HBM keeps
// streaming while the ring is full.  One thread.
template <int D, bool PAGED>
__device__ __forceinline__ void produce_tiles(const CUtensorMap* kmap, const CUtensorMap* vmap, const StepAttArgs& a,
                                              const int64_t* pre, const int32_t* lens, const GroupPlan& gp,
                                              const int32_t* ptab, int32_t ptab_n, uint32_t base, uint32_t NST,
                                              uint32_t bar_full, uint32_t bar_empty) {
  using C = AttCfg<D>;
  const uint64_t pol = policy_evict_first();
  TileCursor<PAGED> ld, pf;
  cursor_begin(ld, a, pre, lens, gp, D, ptab, ptab_n);
  cursor_begin(pf, a, pre, lens, gp, D, ptab, ptab_n);
  for (int i = 0; i < a.pf_tiles && pf.ok; ++i) {
    if (!pf.bad) {
      tma_prefetch_l2_3d(kmap, 0, pf.tile_row(), 0);
      tma_prefetch_l2_3d(vmap, 0, pf.tile_row(), 0);
    }
    cursor_next(pf, a, pre, lens, gp, D, ptab, ptab_n);
  }
  uint32_t it = 0, st = 0, ph = 0;
  bool ok = true;
  while (ld.ok) {
    if (!mbar_wait(bar_empty + 8 * st, ph ^ 1u, a.status, a.wait_ns)) {
      ok = false;
      break;
    }
    const uint32_t fb = bar_full + 8 * st;
    const uint32_t sk = base + st * C::STAGE_BYTES, sv = sk + C::TILE_BYTES;
    mbar_arrive_expect_tx(fb, C::STAGE_BYTES);
    const int32_t row = ld.tile_row();
    tma_load_3d(sk, kmap, fb, 0, row, 0, pol);
    tma_load_3d(sv, vmap, fb, 0, row, 0, pol);
    ++it;
    if (++st == NST) {
      st = 0;
      ph ^= 1u;
    }
    cursor_next(ld, a, pre, lens, gp, D, ptab, ptab_n);
    if (pf.ok) {
      if (!pf.bad) {
        tma_prefetch_l2_3d(kmap, 0, pf.tile_row(), 0);
        tma_prefetch_l2_3d(vmap, 0, pf.tile_row(), 0);
      }
      cursor_next(pf, a, pre, lens, gp, D, ptab, ptab_n);
    }
  }
  if (!ok) {
    for (uint32_t j = (it >= NST ? it - NST : 0); j < it; ++j)
      mbar_wait(bar_full + 8 * (j % NST), (j / NST) & 1u, a.status);
  }
}

// 1/rms of x_l[s] from its Hkv per-group sums of squares (waits for all of
// them): the same order in every warp and CTA, so every user gets the same
// value bit for bit.  Whole warp.
__device__ __forceinline__ bool wait_inv_rms(const uint64_t* part, int n, uint32_t tag, int d, float eps, int lane,
                                             int* status, unsigned long long limit_ns, float& inv) {
  uint64_t t0 = 0;
  while (true) {
    float t = 0.f;
    bool ok = true;
    for (int i = lane; i < n; i += 32) {
      const uint64_t w = ld_tagged(part + i);
      ok &= tv_ok(w, tag);
      t += tv_value(w);
    }
    if (__all_sync(0xffffffffu, ok)) {
      t = warp_sum(t);
      t = __shfl_sync(0xffffffffu, t, 0);
      inv = 1.0f / sqrtf(t / (float)d + eps);
      return true;
    }
    if (!poll_again(t0, status, limit_ns)) return false;
  }
}

// Rotary embedding of two rotate-half pairs: (a0, b0) at frequency f and
// (a1, b1) at f + 1 (elements f, f + 1 and their partners f + D/2,
// f + 1 + D/2); r = (cos, sin) of the two angles fp32(pos * inv_freq).
struct RopePair {
  float c0, s0, c1, s1;
};
__device__ __forceinline__ RopePair rope_angles(int f, float posf, const float* rope_f) {
  RopePair r;
  sincosf(__fmul_rn(posf, rope_f[f]), &r.s0, &r.c0);
  sincosf(__fmul_rn(posf, rope_f[f + 1]), &r.s1, &r.c1);
  return r;
}
__device__ __forceinline__ void rope_rotate(float& a0, float& a1, float& b0, float& b1, const RopePair& r) {
  const float x0 = a0, x1 = a1;
  a0 = x0 * r.c0 - b0 * r.s0;
  b0 = b0 * r.c0 + x0 * r.s0;
  a1 = x1 * r.c1 - b1 * r.s1;
  b1 = b1 * r.c1 + x1 * r.s1;
}

// What the input warp tells the consumers about the piece in a hand-off slot
// (the consumers take their pieces from the slots, in the input warp's order).
struct PieceDesc {
  int32_t s, h, k0, k1;  // keys [k0, k1) of kv-head h of sequence s
  int32_t l, gi;         // layer, sequence group
  int32_t c0, c1;        // CTAs holding the segment's keys (c0 completes it)
  int32_t app_row;       // key appended this step if it falls in the piece, else -1
  int32_t end;           // no more pieces
  int32_t pad[2];
};

// Shared-memory layout of the step kernel (byte offsets from the 1024-byte
// aligned base), a function of the head dim and group size only.
struct StepSmem {
  uint32_t stages;      // K/V ring stages
  uint32_t bar;         // full[st] empty[st] qfull[2] qempty[2] pfull[2] pempty[2] msync
  uint32_t qbuf, qslot; // [2] hand-off slots: q words [8][D/2+4], K row, V row (bf16), x_l of the head group (fp32),
                        // PieceDesc (at qdesc)
  uint32_t qdesc;
  uint32_t pbuf, pslot; // [2] partial hand-off slots: ms[8][8], ls[8][8], os[8][G][D + 4]
  uint32_t misc;        // flags
  uint32_t tables;      // pre[ATT_MAX_S+1] int64, GroupPlan, lens[ATT_MAX_S] int32, apnd[ATT_MAX_S] u8
  uint32_t ptab;        // block-table copy: ptab[ATT_PTAB] int32, its entry count, ptab_h[ATT_PTAB] u8
  uint32_t rope;        // rotary inverse frequencies [D/2] fp32
  uint32_t total;       // bytes to request, alignment slack included
};
__host__ __device__ inline StepSmem step_smem(int D, int G) {
  StepSmem L;
  const uint32_t stage_bytes = 2u * (uint32_t)(D / 64) * (ATT_BLOCK_N * 128u);
  L.qdesc = 8u * (uint32_t)(D / 2 + 4) * 4u + 4u * (uint32_t)D + 4u * (uint32_t)(G * D);
  L.qslot = L.qdesc + (uint32_t)sizeof(PieceDesc);
  L.pslot = 2u * ATT_CONSUMERS * ATT_MAX_G * 4u + (uint32_t)ATT_CONSUMERS * G * (D + 4) * 4u;
  const uint32_t tables = (ATT_MAX_S + 1) * 8u + (uint32_t)((sizeof(GroupPlan) + 7) & ~(size_t)7) + ATT_MAX_S * 4u + ATT_MAX_S;
  const uint32_t max_st = D == 128 ? 5u : 7u;
  for (L.stages = max_st; L.stages >= 2u; --L.stages) {
    L.bar = L.stages * stage_bytes;
    L.qbuf = L.bar + (2u * L.stages + 9u) * 8u;
    L.qbuf = (L.qbuf + 15u) & ~15u;
    L.pbuf = L.qbuf + 2u * L.qslot;
    L.misc = L.pbuf + 2u * L.pslot;
    L.tables = L.misc + 64u;
    L.ptab = L.tables + ((tables + 15u) & ~15u);
    L.rope = (L.ptab + ATT_PTAB * 5u + 16u + 15u) & ~15u;
    L.total = 1024u + L.rope + 4u * (uint32_t)(D / 2);
    if (L.total <= 227u * 1024u) break;
  }
  return L;
}

// x_0[s] = E[y_{t-1}] for every sequence (tagged, residual buffer 0) and its
// per-group sums of squares.  The rows are cut into (sequence, kv-head group,
// eighth) slices of GD / 8 elements, spread over the CTAs' input warps: each
// lane loads one 16-byte chunk, so a warp's share is one memory round trip
// (one warp embedding a whole row waited on the load traffic of the whole
// grid at the start of a launch), and each slice's sum of squares goes to its
// own partial-sum slot (ATT_CONSUMERS per head group, the layout the layers'
// merges use).  Whole warp.
template <int D>
__device__ void embed_slices(const StepAttArgs& a, uint32_t tag, int lane) {
  const int d = a.Hq * D, GD = a.G * D, S = a.S, Hkv = a.Hkv;
  const int cps = GD / (8 * ATT_CONSUMERS);  // chunks of a slice: G*D/64, in [2, 16]
  int lps = 1;                               // lanes per slice: cps rounded up to a power of two
  while (lps < cps) lps <<= 1;
  const int per_pass = 32 / lps;             // slices a warp covers at once
  const int nslices = S * Hkv * ATT_CONSUMERS;
  const int t = *a.step;
  if (blockIdx.x == 0 && lane == 0 && t >= a.max_steps) dev_flag(a.status, PCED_DEV_STEP_LIMIT);
  for (int q0 = blockIdx.x * per_pass; q0 < nslices; q0 += gridDim.x * per_pass) {
    const int q = q0 + lane / lps, k = lane % lps;
    const bool on = q < nslices && k < cps;
    const int s = on ? q / (Hkv * ATT_CONSUMERS) : 0, h = on ? (q / ATT_CONSUMERS) % Hkv : 0, j = q % ATT_CONSUMERS;
    int tok = a.bos;
    if (t > 0 && t <= a.max_steps) tok = a.history[(int64_t)(s / a.n1) * a.max_steps + t - 1];
    if (tok < 0 || tok >= a.V) {
      if (on) dev_flag(a.status, PCED_DEV_BAD_TOKEN);
      tok = 0;
    }
    const int64_t e0 = (int64_t)h * GD + (int64_t)j * (GD / ATT_CONSUMERS) + 8 * k;  // first element of the chunk
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (on) v = __ldg(reinterpret_cast<const uint4*>(a.embed + (int64_t)tok * d + e0));
    float ss = 0.f;
    if (on) {
      uint64_t* x = a.resid + (int64_t)s * d + e0;
      const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float lo = bf16_lo(w[i]), hi = bf16_hi(w[i]);
        st_tagged(x + 2 * i, lo, tag);
        st_tagged(x + 2 * i + 1, hi, tag);
        ss += lo * lo + hi * hi;
      }
    }
    // the slice's lanes are an aligned group of lps: a xor tree over them
    for (int o = 1; o < lps; o <<= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    if (on && k == 0) st_tagged(a.part_ss + ((int64_t)s * Hkv + h) * ATT_CONSUMERS + j, ss, tag);
  }
}

constexpr int STEP_PRODUCER = ATT_CONSUMERS;      // warp 8: TMA
constexpr int STEP_INPUT = ATT_CONSUMERS + 1;     // warp 9: queries, appended rows, x_l hand-off
constexpr int STEP_THREADS = (ATT_CONSUMERS + 2) * 32;

template <int D, bool PK>
__global__ void __launch_bounds__(STEP_THREADS, 1)
    att_step_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                    StepAttArgs a) {
  using C = AttCfg<D>;
  constexpr int QW = D / 2 + 4;  // padded words per query row in the hand-off slot
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  const int32_t S = a.S, G = a.G, Hkv = a.Hkv, GD = G * D, d = a.Hq * D;
  const StepSmem SL = step_smem(D, G);
  const uint32_t NST = SL.stages;
  const uint32_t bar_full = base + SL.bar, bar_empty = bar_full + 8 * NST;
  const uint32_t bar_qfull = bar_empty + 8 * NST, bar_qempty = bar_qfull + 16;
  const uint32_t bar_pfull = bar_qempty + 16, bar_pempty = bar_pfull + 16, bar_m = bar_pempty + 16;
  int* flag = reinterpret_cast<int*>(gbase + SL.misc + 32);
  int64_t* pre = reinterpret_cast<int64_t*>(gbase + SL.tables);
  GroupPlan& gp = *reinterpret_cast<GroupPlan*>(pre + ATT_MAX_S + 1);
  int32_t* lens = reinterpret_cast<int32_t*>(reinterpret_cast<uint8_t*>(&gp) + ((sizeof(GroupPlan) + 7) & ~(size_t)7));
  uint8_t* apnd = reinterpret_cast<uint8_t*>(lens + ATT_MAX_S);
  int32_t* ptab = reinterpret_cast<int32_t*>(gbase + SL.ptab);
  int32_t* ptab_cnt = ptab + ATT_PTAB;
  uint8_t* ptab_h = reinterpret_cast<uint8_t*>(ptab_cnt + 4);  // kv-head of each entry (while building)
  float* rope_f = reinterpret_cast<float*>(gbase + SL.rope);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int32_t epoch = *a.epoch;

  if (tid == 0) {
    for (uint32_t i = 0; i < NST; ++i) {
      mbar_init(bar_full + 8 * i, 1);
      mbar_init(bar_empty + 8 * i, 4);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar_qfull + 8 * i, 1);
      mbar_init(bar_qempty + 8 * i, ATT_CONSUMERS);
      mbar_init(bar_pfull + 8 * i, ATT_CONSUMERS);
      mbar_init(bar_pempty + 8 * i, ATT_CONSUMERS);
    }
    mbar_init(bar_m, ATT_CONSUMERS);
    mbar_fence_init();
  }
  if (warp == STEP_PRODUCER && lane == 0) {
    tma_prefetch_desc(&kmap);
    tma_prefetch_desc(&vmap);
  }
  // the next grid (LM head) may be scheduled as SMs free up; it waits for
  // this grid's completion before reading the hidden states
  pdl_launch_dependents();
  // rotary inverse frequencies theta^(-2f/D), rounded to fp32
  if (a.rope_theta > 0.f && tid < D / 2) rope_f[tid] = (float)pow((double)a.rope_theta, -2.0 * tid / D);
  // lengths after this step's append (a full cache appends nothing)
  for (int i = tid; i < S; i += STEP_THREADS) {
    int32_t n = a.seq_len[i];
    const int32_t c = a.cap[i];
    if (n < 0 || n > c) {
      dev_flag(a.status, PCED_DEV_BAD_LENGTH);
      n = n < 0 ? 0 : c;
    }
    const bool ap = n < c;
    if (!ap) dev_flag(a.status, PCED_DEV_CACHE_FULL);
    int32_t len = ap ? n + 1 : n;
    if (len < 1) {
      dev_flag(a.status, PCED_DEV_BAD_LENGTH);
      len = 1;
    }
    lens[i] = len;
    apnd[i] = ap ? 1 : 0;
  }
  __syncthreads();
  const int32_t align = a.block_table ? ATT_BLOCK_N : 1;
  if (warp == 0) prefix_extents(lens, S, a.seg_cost, pre, lane, align);
  __syncthreads();
  if (tid == 0) plan_groups(gp, pre, S, Hkv, a.groups, gridDim.x, blockIdx.x, align);
  __syncthreads();
  if (a.block_table) {
    // paged caches: for the blocks of this CTA's pieces (the same in every
    // layer), in the cursor's order, keep the block's row base for the
    // piece's kv-head (block_base_of) in shared memory, so the producer and
    // the input warp never wait on a table read in the loop
    if (warp == 0) {
      if (lane == 0) {
        int32_t n = 0;
        for (int gi = 0; gi < gp.n && n < ATT_PTAB; ++gi) {
          Piece pc;
          pc.adv = -1;  // none yet
          for (int64_t pp = gp.cb[gi]; pp < gp.ce[gi] && n < ATT_PTAB;) {
            pc = pc.adv < 0
                     ? find_piece(pre, lens, gp.s_lo[gi], gp.s_lo[gi + 1], gp.T[gi], pp, gp.ce[gi], a.seg_lead)
                     : next_piece(pc, pre, lens, gp.s_lo[gi], gp.s_lo[gi + 1], gp.T[gi], pp, gp.ce[gi], a.seg_lead);
            pp += pc.adv;
            if (pc.k0 == pc.k1) continue;
            const int32_t j0 = block_of(a, pc.k0), j1 = block_of(a, pc.k1 - 1);
            for (int32_t j = j0; j <= j1 && n < ATT_PTAB; ++j) {
              ptab_h[n] = (uint8_t)pc.h;
              ptab[n++] = j < a.max_blocks ? pc.s * a.max_blocks + j : -1;
            }
          }
        }
        *ptab_cnt = n;
      }
      __syncwarp();
      const int32_t n = *ptab_cnt;
      for (int32_t i = lane; i < n; i += 32)
        ptab[i] = block_base_of(a, ptab[i] < 0 ? -1 : __ldg(a.block_table + ptab[i]), ptab_h[i]);
    }
    __syncthreads();
  }
  const int32_t ptab_n = a.block_table ? *ptab_cnt : 0;

  if (warp == STEP_PRODUCER) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      if (a.block_table)
        produce_tiles<D, true>(&kmap, &vmap, a, pre, lens, gp, ptab, ptab_n, base, NST, bar_full, bar_empty);
      else
        produce_tiles<D, false>(&kmap, &vmap, a, pre, lens, gp, ptab, ptab_n, base, NST, bar_full, bar_empty);
    }
    return;
  }

  if (warp == STEP_INPUT) {
    // ---------------------------------------------------------- input warp
    // For every piece, in order: wait for head group h of x_l[s] and the
    // group sums of x_l[s], then hand the consumers q = bf16(x_l * inv_rms)
    // (and, for the piece holding the row appended this step, that row's K
    // and V, also written to the caches) through a double-buffered slot.
    embed_slices<D>(a, step_tag(epoch, 0), lane);
    uint32_t p = 0;
    bool ok = true;
    for (int l = 0; l < a.L && ok; ++l) {
      const int par = l & 1;
      const uint32_t tag = step_tag(epoch, l);
      int32_t ptn = 0;  // block-table copy: entry of the next piece's first block (as the producer's cursor)
      for (int gi = 0; gi < gp.n && ok; ++gi) {
      Piece pc;
      pc.adv = -1;  // none yet
      for (int64_t pp = gp.cb[gi]; pp < gp.ce[gi] && ok;) {
        pc = pc.adv < 0 ? find_piece(pre, lens, gp.s_lo[gi], gp.s_lo[gi + 1], gp.T[gi], pp, gp.ce[gi], a.seg_lead)
                        : next_piece(pc, pre, lens, gp.s_lo[gi], gp.s_lo[gi + 1], gp.T[gi], pp, gp.ce[gi], a.seg_lead);
        pp += pc.adv;
        if (pc.k0 == pc.k1) continue;
        int32_t pt = 0, j0 = 0;
        if (a.block_table) {
          if (pc.k0 & (ATT_BLOCK_N - 1)) dev_flag(a.status, PCED_DEV_BAD_BLOCK);  // the partition guarantees it
          j0 = block_of(a, pc.k0);
          pt = ptn;
          ptn += block_of(a, pc.k1 - 1) - j0 + 1;
        }
        const uint32_t slot = p & 1u, u = p >> 1;
        ++p;
        if (u > 0 && !mbar_wait(bar_qempty + 8 * slot, (u - 1u) & 1u, a.status, a.wait_ns)) {
          ok = false;
          break;
        }
        const uint64_t* xs = a.resid + ((int64_t)par * S + pc.s) * d;
        const uint64_t* xq = xs + (int64_t)pc.h * GD;
        const bool app = apnd[pc.s] && pc.k1 == lens[pc.s];
        const uint64_t* ps = a.part_ss + ((int64_t)par * S + pc.s) * Hkv * ATT_CONSUMERS;
        uint32_t* qw = reinterpret_cast<uint32_t*>(gbase + SL.qbuf + slot * SL.qslot);
        float* xr = reinterpret_cast<float*>(qw + 8 * QW + D);  // x_l of the head group, for the completing CTA
        float inv = 0.f;
        // query elements by rotary quads: lane takes elements 2k, 2k+1 of head
        // g and their rotate-half partners 2k + D/2, 2k + 1 + D/2 (quad
        // m = g*D/4 + k); the first chunk's poll also covers the group sums
        // (one round trip)
        const bool rope = a.rope_theta > 0.f;
        // this lane's two rotary frequencies are 2k, 2k + 1 with k = lane mod D/4
        // for every quad it takes (D/4 divides 32); their angles only depend
        // on the position, so they are found before the wait for x_l
        static_assert(32 % (D / 4) == 0, "rotary quads per lane assume D/4 divides 32");
        RopePair rp = {1.f, 0.f, 1.f, 0.f};
        if (rope) rp = rope_angles(2 * (lane % (D / 4)), (float)(lens[pc.s] - apnd[pc.s]), rope_f);
        for (int m0 = 0; m0 < GD / 4 && ok; m0 += 32 * 4) {
          float v[4][4], t = 0.f;
          uint64_t t0 = 0;
          while (true) {
            bool good = true;
            t = 0.f;
            if (m0 == 0)
              for (int i = lane; i < Hkv * ATT_CONSUMERS; i += 32) {
                const uint64_t w = ld_tagged(ps + i);
                good &= tv_ok(w, tag);
                t += tv_value(w);
              }
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              const int m = m0 + lane + 32 * j;
              v[j][0] = v[j][1] = v[j][2] = v[j][3] = 0.f;
              if (m >= GD / 4) continue;
              const int e = (m / (D / 4)) * D + 2 * (m % (D / 4));
              const uint64_t w0 = ld_tagged(xq + e), w1 = ld_tagged(xq + e + 1);
              const uint64_t w2 = ld_tagged(xq + e + D / 2), w3 = ld_tagged(xq + e + D / 2 + 1);
              good &= tv_ok(w0, tag) && tv_ok(w1, tag) && tv_ok(w2, tag) && tv_ok(w3, tag);
              v[j][0] = tv_value(w0);
              v[j][1] = tv_value(w1);
              v[j][2] = tv_value(w2);
              v[j][3] = tv_value(w3);
            }
            if (__all_sync(0xffffffffu, good)) break;
            if (!poll_again(t0, a.status, a.wait_ns)) {
              ok = false;
              break;
            }
          }
          if (!ok) break;
          if (m0 == 0) {
            // same summation order as every other user of these sums
            t = warp_sum(t);
            t = __shfl_sync(0xffffffffu, t, 0);
            inv = 1.0f / sqrtf(t / (float)d + a.rms_eps);
          }
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int m = m0 + lane + 32 * j;
            if (m >= GD / 4) continue;
            const int g = m / (D / 4), k = m % (D / 4), e = g * D + 2 * k;
            float a0 = v[j][0] * inv, a1 = v[j][1] * inv, b0 = v[j][2] * inv, b1 = v[j][3] * inv;
            if (rope) rope_rotate(a0, a1, b0, b1, rp);
            qw[g * QW + k] = pack_bf16(a0, a1);
            qw[g * QW + k + D / 4] = pack_bf16(b0, b1);
            xr[e] = v[j][0];
            xr[e + 1] = v[j][1];
            xr[e + D / 2] = v[j][2];
            xr[e + D / 2 + 1] = v[j][3];
          }
        }
        if (ok && app) {
          // K row = head h of u (rotated like the queries), V row = head Hkv + h of u
          const uint64_t* xk = xs + (int64_t)pc.h * D;
          const uint64_t* xv = xs + ((int64_t)Hkv + pc.h) * D;
          uint32_t* kr = qw + 8 * QW;
          uint32_t* vr = kr + D / 2;
          int64_t arow;
          if (a.block_table) {
            const int32_t key = lens[pc.s] - 1, j = block_of(a, key);
            const int32_t b0 = block_base(a, pc.s, pc.h, j, pt + (j - j0), ptab, ptab_n);
            arow = b0 < 0 ? -1 : (int64_t)l * a.rows_per_layer + b0 + (key - j * a.block_rows);
          } else {
            arow = (int64_t)l * a.rows_per_layer + (a.kv_offset[pc.s] + (int64_t)pc.h * a.cap[pc.s] * D) / D +
                   lens[pc.s] - 1;
          }
          // a bad block id was flagged: keep the cache untouched
          const bool wrow = arow >= 0 &&
                            PCED_IN_BOUNDS(arow >= (int64_t)l * a.rows_per_layer &&
                                               arow < (int64_t)(l + 1) * a.rows_per_layer &&
                                               (a.block_table || lens[pc.s] - 1 < a.cap[pc.s]),
                                           a.status);
          const int64_t grow = (wrow ? arow : 0) * D;
          constexpr int RQ = (D / 4 + 31) / 32;  // rotary quads per lane (as for the queries)
          float kx[RQ][4], vx[RQ][4];
          uint64_t t0 = 0;
          while (true) {
            bool good = true;
#pragma unroll
            for (int j = 0; j < RQ; ++j) {
              const int k = lane + 32 * j;
#pragma unroll
              for (int c = 0; c < 4; ++c) kx[j][c] = vx[j][c] = 0.f;
              if (k >= D / 4) continue;
              const int e[4] = {2 * k, 2 * k + 1, 2 * k + D / 2, 2 * k + 1 + D / 2};
#pragma unroll
              for (int c = 0; c < 4; ++c) {
                const uint64_t wk = ld_tagged(xk + e[c]), wv = ld_tagged(xv + e[c]);
                good &= tv_ok(wk, tag) && tv_ok(wv, tag);
                kx[j][c] = tv_value(wk);
                vx[j][c] = tv_value(wv);
              }
            }
            if (__all_sync(0xffffffffu, good)) break;
            if (!poll_again(t0, a.status, a.wait_ns)) {
              ok = false;
              break;
            }
          }
#pragma unroll
          for (int j = 0; j < RQ; ++j) {
            const int k = lane + 32 * j;
            if (!ok || k >= D / 4) continue;
            float a0 = kx[j][0] * inv, a1 = kx[j][1] * inv, b0 = kx[j][2] * inv, b1 = kx[j][3] * inv;
            if (rope) rope_rotate(a0, a1, b0, b1, rp);  // keys rotate, values do not
            const uint32_t ka = pack_bf16(a0, a1), kb = pack_bf16(b0, b1);
            const uint32_t va = pack_bf16(vx[j][0] * inv, vx[j][1] * inv), vb = pack_bf16(vx[j][2] * inv, vx[j][3] * inv);
            kr[k] = ka;
            kr[k + D / 4] = kb;
            vr[k] = va;
            vr[k + D / 4] = vb;
            if (wrow) {
              uint32_t* gk = reinterpret_cast<uint32_t*>(a.k_cache + grow);
              uint32_t* gv = reinterpret_cast<uint32_t*>(a.v_cache + grow);
              gk[k] = ka;
              gk[k + D / 4] = kb;
              gv[k] = va;
              gv[k + D / 4] = vb;
            }
          }
        }
        if (lane == 0) {
          const int64_t pa = (int64_t)pc.h * gp.T[gi] + pre[pc.s] - pre[gp.s_lo[gi]] + a.seg_lead;  // first key
          PieceDesc* dsc = reinterpret_cast<PieceDesc*>(reinterpret_cast<uint8_t*>(qw) + SL.qdesc);
          dsc->s = pc.s;
          dsc->h = pc.h;
          dsc->k0 = pc.k0;
          dsc->k1 = pc.k1;
          dsc->l = l;
          dsc->gi = gi;
          dsc->c0 = (int32_t)part_cta(pa, gp.P[gi], align);
          dsc->c1 = (int32_t)part_cta(pa + lens[pc.s] - 1, gp.P[gi], align);
          dsc->app_row = app ? lens[pc.s] - 1 : -1;
          dsc->end = 0;
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(bar_qfull + 8 * slot);
      }
      }
    }
    // end marker for the consumers
    if (ok) {
      const uint32_t slot = p & 1u, u = p >> 1;
      if (u == 0 || mbar_wait(bar_qempty + 8 * slot, (u - 1u) & 1u, a.status, a.wait_ns)) {
        if (lane == 0) {
          PieceDesc* dsc = reinterpret_cast<PieceDesc*>(gbase + SL.qbuf + slot * SL.qslot + SL.qdesc);
          dsc->end = 1;
          mbar_arrive(bar_qfull + 8 * slot);
        }
      }
    }
    return;
  }

  // -------------------------------------------------------------- consumers
  const int wg = warp >> 2, wl = warp & 3;
  const int g = lane >> 2, tq = lane & 3;
  const int kb = 16 * wl;
  // B column g of S^T = K Q^T is head g; with PK columns 4-7 repeat heads 0-3,
  // so the threads owning those columns compute the scores they mirror
  const int qh = PK ? (g & 3) : g;
  const bool hv = qh < G;
  uint32_t it = 0, p = 0, cst = 0, cuse = 0;  // tile counter; its stage and use count (it % NST, it / NST)
  bool ok = true;
  for (;;) {
    const uint32_t slot = p & 1u, u = p >> 1;
    ++p;
    if (!mbar_wait(bar_qfull + 8 * slot, u & 1u, a.status, a.wait_ns)) {
      ok = false;
      break;
    }
    const uint32_t* qw = reinterpret_cast<const uint32_t*>(gbase + SL.qbuf + slot * SL.qslot);
    const PieceDesc dsc = *reinterpret_cast<const PieceDesc*>(gbase + SL.qbuf + slot * SL.qslot + SL.qdesc);
    if (dsc.end) break;
    const int l = dsc.l;
    const int64_t rbase = (int64_t)dsc.gi * ((int64_t)gridDim.x + (int64_t)S * Hkv);  // the group's record slots
    Piece pc;
    pc.s = dsc.s;
    pc.h = dsc.h;
    pc.k0 = dsc.k0;
    pc.k1 = dsc.k1;
    uint32_t qf[C::KSTEPS][2];
#pragma unroll
    for (int j = 0; j < C::KSTEPS; ++j) {
      qf[j][0] = hv ? qw[qh * QW + 8 * j + tq] : 0u;
      qf[j][1] = hv ? qw[qh * QW + 8 * j + 4 + tq] : 0u;
    }
    const int32_t app_row = dsc.app_row;

    WarpAcc<D> A;
    acc_reset(A);
    for (int32_t kt = pc.k0; kt < pc.k1; kt += ATT_BLOCK_N, ++it, cst = cst + 1 == NST ? (++cuse, 0u) : cst + 1) {
      if ((int)(it & 1u) != wg) continue;
      const uint32_t use = cuse, st = cst, ph = use & 1u;
      if (use > 0 && !mbar_wait(bar_empty + 8 * st, (use - 1u) & 1u, a.status, a.wait_ns)) {
        ok = false;
        break;
      }
      if (!mbar_wait(bar_full + 8 * st, ph, a.status, a.wait_ns)) {
        ok = false;
        break;
      }
      const int nvalid = min(ATT_BLOCK_N, pc.k1 - kt);
      const uint32_t sk = base + st * C::STAGE_BYTES, sv = sk + C::TILE_BYTES;
      if (app_row >= kt && app_row < kt + ATT_BLOCK_N && ((app_row - kt) >> 4) == wl) {
        // the appended row (prepared by the input warp) replaces whatever
        // the cache held there when the tile was loaded
        const int r = app_row - kt;
        const uint32_t src = base + SL.qbuf + slot * SL.qslot + 8 * QW * 4;
        for (int c = lane; c < 2 * (D / 8); c += 32) {
          const int cc = c % (D / 8);
          const uint32_t dst = (c < D / 8 ? sk : sv) + (cc >> 3) * C::BOX_BYTES + r * 128 +
                               ((((uint32_t)cc & 7u) ^ ((uint32_t)r & 7u)) << 4);
          uint32_t w0, w1, w2, w3;
          asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                       : "=r"(w0), "=r"(w1), "=r"(w2), "=r"(w3)
                       : "r"(src + 16 * c));
          asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(dst), "r"(w0), "r"(w1), "r"(w2), "r"(w3)
                       : "memory");
        }
        fence_proxy_async_smem();
        __syncwarp();
      }
      if (kb < nvalid) tile_math<D, PK>(A, qf, sk, sv, kb, nvalid, a.scale_log2, lane);
      __syncwarp();
      if (lane == 0) mbar_arrive(bar_empty + 8 * st);
    }
    if (!ok) break;
    const int64_t seg = (int64_t)pc.h * S + pc.s;
    const int64_t c0 = dsc.c0, c1 = dsc.c1;
    const bool merges = c0 == (int64_t)blockIdx.x;  // the segment's first CTA completes it
    if (!merges) {
      __syncwarp();
      if (lane == 0) mbar_arrive(bar_qempty + 8 * slot);
    }
    // combine the eight warps' partials through a double-buffered slot;
    // afterwards thread tid < G*D/4 owns outputs idx0..idx0+3 (head hh)
    if (u > 0 && !mbar_wait(bar_pempty + 8 * slot, (u - 1u) & 1u, a.status, a.wait_ns)) {
      ok = false;
      break;
    }
    float l0 = A.l0, l1 = A.l1;
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
      l0 += __shfl_xor_sync(0xffffffffu, l0, off);
      l1 += __shfl_xor_sync(0xffffffffu, l1, off);
    }
    if (PK) pack_fold<D>(A);
    float* ms = reinterpret_cast<float*>(gbase + SL.pbuf + slot * SL.pslot);  // [ATT_MAX_G][8 warps]
    float* ls = ms + ATT_MAX_G * ATT_CONSUMERS;                                // [ATT_MAX_G][8 warps]
    float* os = ls + ATT_MAX_G * ATT_CONSUMERS;                                // [8 warps][G][D + 4]
    if (g == 0) {
      ms[(2 * tq) * ATT_CONSUMERS + warp] = A.m0;
      ms[(2 * tq + 1) * ATT_CONSUMERS + warp] = A.m1;
      ls[(2 * tq) * ATT_CONSUMERS + warp] = l0;
      ls[(2 * tq + 1) * ATT_CONSUMERS + warp] = l1;
    }
    {
      float* ow = os + warp * G * C::OROW;
      const bool h0 = 2 * tq < G, h1 = 2 * tq + 1 < G;
#pragma unroll
      for (int i = 0; i < C::MTILES; ++i) {
        const int d0 = 16 * i + g, d1 = d0 + 8;
        if (h0) {
          ow[(2 * tq) * C::OROW + d0] = A.o[i][0];
          ow[(2 * tq) * C::OROW + d1] = A.o[i][2];
        }
        if (h1) {
          ow[(2 * tq + 1) * C::OROW + d0] = A.o[i][1];
          ow[(2 * tq + 1) * C::OROW + d1] = A.o[i][3];
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(bar_pfull + 8 * slot);
    if (!mbar_wait(bar_pfull + 8 * slot, u & 1u, a.status, a.wait_ns)) {
      ok = false;
      break;
    }
    const uint32_t tag = step_tag(epoch, l);
    const bool own = tid < GD / 4;
    const int hh = own ? tid / (D / 4) : 0, idx0 = own ? 4 * tid : 0;
    float mx = -INFINITY, lsum = 0.f, acc[4] = {0.f, 0.f, 0.f, 0.f};
    if (own) {
      float mw[ATT_CONSUMERS], lw[ATT_CONSUMERS];
      const float4* m4 = reinterpret_cast<const float4*>(ms + hh * ATT_CONSUMERS);
      const float4* l4 = reinterpret_cast<const float4*>(ls + hh * ATT_CONSUMERS);
      *reinterpret_cast<float4*>(mw) = m4[0];
      *reinterpret_cast<float4*>(mw + 4) = m4[1];
      *reinterpret_cast<float4*>(lw) = l4[0];
      *reinterpret_cast<float4*>(lw + 4) = l4[1];
      float M = mw[0];
#pragma unroll
      for (int w = 1; w < ATT_CONSUMERS; ++w) M = fmaxf(M, mw[w]);
      const float* oc = os + hh * C::OROW + (idx0 - hh * D);
#pragma unroll
      for (int w = 0; w < ATT_CONSUMERS; ++w) {
        if (mw[w] == -INFINITY) continue;  // a warp without live keys in this piece
        const float e = exp2f(mw[w] - M);
        const float4 o4 = *reinterpret_cast<const float4*>(oc + w * G * C::OROW);
        acc[0] += o4.x * e;
        acc[1] += o4.y * e;
        acc[2] += o4.z * e;
        acc[3] += o4.w * e;
        lsum += lw[w] * e;
      }
      mx = M;
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(bar_pempty + 8 * slot);
    if (!merges) {
      // the segment continues in an earlier CTA: publish this CTA's record
      const int64_t rs = rbase + (int64_t)blockIdx.x + seg;
      if (own && PCED_IN_BOUNDS(rs >= 0 && rs < (int64_t)a.groups * (gridDim.x + S * Hkv), a.status)) {
        uint64_t* ro = a.rec_o + rs * GD + idx0;
#pragma unroll
        for (int j = 0; j < 4; ++j) st_tagged(ro + j, acc[j], tag);
        if (idx0 % D == 0) {
          st_tagged(a.rec_ml + (rs * G + hh) * 2, mx, tag);
          st_tagged(a.rec_ml + (rs * G + hh) * 2 + 1, lsum, tag);
        }
      }
      continue;
    }
    // complete the segment: the records of CTAs c0+1..c1 in order (RB at a
    // time, one round trip when they are there)
    constexpr int RB = 4;
    for (int64_t c = c0 + 1; c <= c1 && ok; c += RB) {
      float mv[RB], lv[RB], ov[RB][4];
      uint64_t t0 = 0;
      while (true) {
        bool good = true;
#pragma unroll
        for (int q = 0; q < RB; ++q) {
          mv[q] = -INFINITY;
          lv[q] = 0.f;
#pragma unroll
          for (int j = 0; j < 4; ++j) ov[q][j] = 0.f;
          if (!own || c + q > c1) continue;
          const int64_t rs = rbase + c + q + seg;
          if (!PCED_IN_BOUNDS(rs >= 0 && rs < (int64_t)a.groups * (gridDim.x + S * Hkv), a.status)) continue;
          const uint64_t wm = ld_tagged(a.rec_ml + (rs * G + hh) * 2);
          const uint64_t wl = ld_tagged(a.rec_ml + (rs * G + hh) * 2 + 1);
          uint64_t wo[4];
#pragma unroll
          for (int j = 0; j < 4; ++j) wo[j] = ld_tagged(a.rec_o + rs * GD + idx0 + j);
          good &= tv_ok(wm, tag) && tv_ok(wl, tag);
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            good &= tv_ok(wo[j], tag);
            ov[q][j] = tv_value(wo[j]);
          }
          mv[q] = tv_value(wm);
          lv[q] = tv_value(wl);
        }
        if (__all_sync(0xffffffffu, good)) break;
        if (!poll_again(t0, a.status, a.wait_ns)) {
          ok = false;
          break;
        }
      }
#pragma unroll
      for (int q = 0; q < RB; ++q) {
        if (mv[q] == -INFINITY) continue;
        const float Mn = fmaxf(mx, mv[q]);
        const float f = mx == -INFINITY ? 0.f : exp2f(mx - Mn), e = exp2f(mv[q] - Mn);
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[j] = acc[j] * f + ov[q][j] * e;
        lsum = lsum * f + lv[q] * e;
        mx = Mn;
      }
    }
    if (!ok) break;
    // x_{l+1} = x_l + o for head group h (x_l from the input warp's slot)
    const int nx = (l + 1) & 1;
    const uint32_t ntag = step_tag(epoch, l + 1);
    const float* xr = reinterpret_cast<const float*>(qw + 8 * QW + D);
    uint64_t* xn = a.resid + ((int64_t)nx * S + pc.s) * d + (int64_t)pc.h * GD;
    float xv[4] = {0.f, 0.f, 0.f, 0.f};
    float ss = 0.f;
    if (own && PCED_IN_BOUNDS(pc.s >= 0 && pc.s < S && (int64_t)pc.h * GD + idx0 + 4 <= d, a.status)) {
      const float4 x4 = *reinterpret_cast<const float4*>(xr + idx0);
      const float xo[4] = {x4.x, x4.y, x4.z, x4.w};
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        xv[j] = xo[j] + (lsum > 0.f ? acc[j] / lsum : 0.f);
        st_tagged(xn + idx0 + j, xv[j], ntag);
        ss += xv[j] * xv[j];
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(bar_qempty + 8 * slot);
    ss = warp_sum(ss);
    uint64_t* ps = a.part_ss + ((int64_t)nx * S + pc.s) * Hkv * ATT_CONSUMERS;
    if (lane == 0) st_tagged(ps + pc.h * ATT_CONSUMERS + warp, ss, ntag);
  }
  // Final hidden state, head group h of every segment this CTA completed at
  // the last layer.  It needs the sums of all the sequence's head groups, so
  // it waits here, after this CTA has done all its merges: a wait inside the
  // loop could close a cycle (two CTAs each waiting for a merge the other
  // would only do later).  The CTA's pieces are walked again to find them.
  if (ok && a.L > 0) {
    const int nx = a.L & 1;
    const uint32_t ntag = step_tag(epoch, a.L);
    const bool own = tid < GD / 4;
    const int idx0 = own ? 4 * tid : 0;
    for (int gi = 0; gi < gp.n && ok; ++gi) {
      Piece pc;
      pc.adv = -1;  // none yet
      for (int64_t pp = gp.cb[gi]; pp < gp.ce[gi] && ok;) {
        pc = pc.adv < 0 ? find_piece(pre, lens, gp.s_lo[gi], gp.s_lo[gi + 1], gp.T[gi], pp, gp.ce[gi], a.seg_lead)
                        : next_piece(pc, pre, lens, gp.s_lo[gi], gp.s_lo[gi + 1], gp.T[gi], pp, gp.ce[gi], a.seg_lead);
        pp += pc.adv;
        if (pc.k0 == pc.k1) continue;
        const int64_t pa = (int64_t)pc.h * gp.T[gi] + pre[pc.s] - pre[gp.s_lo[gi]] + a.seg_lead;  // first key
        if (part_cta(pa, gp.P[gi], align) != (int64_t)blockIdx.x) continue;  // completed by another CTA
        const uint64_t* ps = a.part_ss + ((int64_t)nx * S + pc.s) * Hkv * ATT_CONSUMERS;
        float inv;
        if (!wait_inv_rms(ps, Hkv * ATT_CONSUMERS, ntag, d, a.rms_eps, lane, a.status, a.wait_ns, inv)) {
          ok = false;
          break;
        }
        if (own) {
          // x_L as this thread stored it when it completed the segment
          const uint64_t* xn = a.resid + ((int64_t)nx * S + pc.s) * d + (int64_t)pc.h * GD + idx0;
          __nv_bfloat16* hs = a.hidden + (int64_t)pc.s * d + (int64_t)pc.h * GD + idx0;
          __nv_bfloat16* hc = a.hidden_copy ? a.hidden_copy + (int64_t)pc.s * d + (int64_t)pc.h * GD + idx0 : nullptr;
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const __nv_bfloat16 hv2 = __float2bfloat16_rn(tv_value(xn[j]) * inv);
            hs[j] = hv2;
            if (hc) hc[j] = hv2;
          }
        }
      }
    }
  }
  // ---- the last CTA to finish advances seq_len and the epoch
  uint32_t cph = 0;
  if (tid == 0) {
    const int prev = atom_acq_rel_gpu_add(a.done_cnt, 1);
    flag[0] = prev == (int)gridDim.x - 1;
  }
  if (warps_sync(bar_m, cph, a.status) && flag[0]) {
    for (int i = tid; i < S; i += ATT_CT)
      if (apnd[i]) a.seq_len[i] = lens[i];
    if (tid == 0) {
      *a.done_cnt = 0;
      *a.epoch = epoch + 1;
    }
  }
}

// ------------------------------------------------------------------- host
size_t att_records_bytes(int32_t S, int32_t Hq, int32_t Hkv, int32_t D) {
  const int64_t G = Hq / (Hkv > 0 ? Hkv : 1);
  const int64_t slots = ATT_MAX_CTAS + (int64_t)S * Hkv;
  pced_host::Carver c(nullptr);
  c.take<float>((size_t)(slots * G * D));
  c.take<float2>((size_t)(slots * G));
  c.take<int64_t>((size_t)S + 1);
  c.take<int64_t>(1);
  return c.used();
}

int att_grid(int64_t total_cap_keys) {
  int64_t want = (total_cap_keys + 255) / 256;
  int64_t sms = pced_host::num_sms();
  int64_t g = want < sms ? want : sms;
  if (g > ATT_MAX_CTAS) g = ATT_MAX_CTAS;
  return (int)(g < 1 ? 1 : g);
}

int64_t att_step_slots(int32_t S, int32_t Hkv) { return ATT_MAX_GROUPS * (ATT_MAX_CTAS + (int64_t)S * Hkv); }

static int env_int(const char* name, int dflt, int lo, int hi) {
  const char* e = getenv(name);
  if (!e || !*e) return dflt;
  const int v = atoi(e);
  return v < lo ? lo : (v > hi ? hi : v);
}
int att_step_seg_cost(int D) { return env_int("PCED_ATT_SEGCOST", 512, 0, 1 << 20); }
int att_step_pf_tiles() { return env_int("PCED_ATT_PF", 6, 0, 64); }
int att_step_groups() { return env_int("PCED_ATT_GROUPS", 2, 1, ATT_MAX_GROUPS); }
int att_step_seg_lead(int seg_cost) { return env_int("PCED_ATT_LEAD", seg_cost / 2, 0, seg_cost); }

// cudaFuncSetAttribute once per kernel and device
template <typename K>
static cudaError_t set_smem_once(K kernel, size_t bytes, bool* done) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!done[dev]) {
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e != cudaSuccess) return e;
    done[dev] = true;
  }
  return cudaSuccess;
}

template <int D>
static cudaError_t launch_split(const CUtensorMap& kmap, const CUtensorMap& vmap, const AttArgs& a, int ctas,
                                cudaStream_t stream) {
  static bool configured[64];
  cudaError_t e = set_smem_once(att_split_kernel<D>, AttCfg<D>::SMEM, configured);
  if (e != cudaSuccess) return e;
  att_split_kernel<D><<<ctas, ATT_THREADS, AttCfg<D>::SMEM, stream>>>(kmap, vmap, a);
  return cudaGetLastError();
}

cudaError_t att_split_launch(int D, const CUtensorMap& kmap, const CUtensorMap& vmap, const AttArgs& a, int ctas,
                             cudaStream_t stream) {
  if (D == 128) return launch_split<128>(kmap, vmap, a, ctas, stream);
  if (D == 64) return launch_split<64>(kmap, vmap, a, ctas, stream);
  return cudaErrorInvalidValue;
}

cudaError_t att_combine_launch(const CombineArgs& a, cudaStream_t stream) {
  att_combine_kernel<<<dim3(a.Hkv, a.S), CMB_THREADS, 0, stream>>>(a);
  return cudaGetLastError();
}

template <int D, bool PK>
static cudaError_t launch_step(const CUtensorMap& kmap, const CUtensorMap& vmap, const StepAttArgs& a, int ctas,
                               cudaStream_t stream) {
  static bool configured[64];
  const StepSmem SL = step_smem(D, a.G);
  cudaError_t e = set_smem_once(att_step_kernel<D, PK>, 227 * 1024, configured);
  if (e != cudaSuccess) return e;
  // every CTA waits for the others' layer results, so all must be resident at
  // once: a cooperative launch guarantees it (or fails)
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(ctas);
  cfg.blockDim = dim3(STEP_THREADS);
  cfg.dynamicSmemBytes = SL.total;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, att_step_kernel<D, PK>, kmap, vmap, a);
}

cudaError_t att_step_launch(int D, const CUtensorMap& kmap, const CUtensorMap& vmap, const StepAttArgs& a, int ctas,
                            cudaStream_t stream) {
  const bool pk = a.G <= 4;  // hi and lo parts of P share one MMA
  if (D == 128) return pk ? launch_step<128, true>(kmap, vmap, a, ctas, stream)
                          : launch_step<128, false>(kmap, vmap, a, ctas, stream);
  if (D == 64) return pk ? launch_step<64, true>(kmap, vmap, a, ctas, stream)
                         : launch_step<64, false>(kmap, vmap, a, ctas, stream);
  return cudaErrorInvalidValue;
}

}  // namespace pced

// ------------------------------------------------------------------ C ABI
using namespace pced;
using namespace pced_host;

extern "C" size_t pced_decode_attention_workspace_size(int32_t S, int32_t Hq, int32_t Hkv, int32_t D) {
  if (S < 1 || Hq < 1 || Hkv < 1 || D < 1) return 0;
  return 256 + att_records_bytes(S, Hq, Hkv, D);
}

extern "C" pced_status pced_decode_attention(const void* q, const void* k_cache, const void* v_cache,
                                             int64_t cache_elems, const int64_t* kv_offset, const int32_t* cap,
                                             const int32_t* seq_len, int32_t S, int32_t Hq, int32_t Hkv,
                                             int32_t D, int64_t total_cap, float scale, float* out,
                                             void* workspace, size_t workspace_bytes, void* stream) {
  if (!q || !k_cache || !v_cache || !kv_offset || !cap || !seq_len || !out || !workspace)
    return fail(PCED_ERR_INVALID_ARG, "pced_decode_attention: null pointer");
  if (S < 1 || Hq < 1 || Hkv < 1 || Hq % Hkv != 0 || cache_elems < D || total_cap < S)
    return fail(PCED_ERR_INVALID_ARG, "pced_decode_attention: bad sizes (S=%d Hq=%d Hkv=%d)", S, Hq, Hkv);
  if (D != 64 && D != 128) return fail(PCED_ERR_UNSUPPORTED, "pced_decode_attention: D=%d (supported: 64, 128)", D);
  if (Hq / Hkv > ATT_MAX_G) return fail(PCED_ERR_UNSUPPORTED, "pced_decode_attention: Hq/Hkv > %d", ATT_MAX_G);
  if (S > ATT_MAX_S) return fail(PCED_ERR_UNSUPPORTED, "pced_decode_attention: S > %d", ATT_MAX_S);
  if (Hq * D > 8192) return fail(PCED_ERR_UNSUPPORTED, "pced_decode_attention: Hq*D > 8192");
  if (cache_elems % D != 0 || cache_elems / D >= (int64_t)1 << 31)
    return fail(PCED_ERR_UNSUPPORTED, "pced_decode_attention: cache of %lld elements", (long long)cache_elems);
  if ((((uintptr_t)k_cache) | ((uintptr_t)v_cache)) & 15u)
    return fail(PCED_ERR_INVALID_ARG, "pced_decode_attention: caches must be 16-byte aligned");
  if (((uintptr_t)q) & 3u) return fail(PCED_ERR_INVALID_ARG, "pced_decode_attention: q must be 4-byte aligned");
  if (((uintptr_t)workspace) & 255u || workspace_bytes < pced_decode_attention_workspace_size(S, Hq, Hkv, D))
    return fail(PCED_ERR_WORKSPACE, "pced_decode_attention: workspace too small or misaligned");
  if (num_sms() <= 0) return fail(PCED_ERR_NO_DEVICE, "pced_decode_attention: no CUDA device");

  CUtensorMap kmap, vmap;
  const uint64_t rows = (uint64_t)(cache_elems / D);
  pced_status st = make_tmap_kv(&kmap, k_cache, rows, (uint32_t)D, ATT_BLOCK_N);
  if (st != PCED_OK) return st;
  st = make_tmap_kv(&vmap, v_cache, rows, (uint32_t)D, ATT_BLOCK_N);
  if (st != PCED_OK) return st;

  const int32_t G = Hq / Hkv;
  Carver cv((char*)workspace + 256);
  const int64_t slots = ATT_MAX_CTAS + (int64_t)S * Hkv;
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
  a.status = (int*)workspace;
  const int ctas = att_grid(total_cap * Hkv);
  cudaStream_t s = (cudaStream_t)stream;
  cudaError_t e = att_split_launch(D, kmap, vmap, a, ctas, s);
  if (e != cudaSuccess) return cuda_status(e, "attention split launch");

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
  if (e != cudaSuccess) return cuda_status(e, "attention combine launch");
  return PCED_OK;
}
