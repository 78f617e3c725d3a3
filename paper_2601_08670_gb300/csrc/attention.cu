// attention.cu -- decode attention of every expert over its own KV cache
// (paper Sec. 3: N+1 parallel streams, each with an independently encoded
// cache; grouped-query heads).
//
// Split-KV flash decoding on sm_103a:
//   * all (sequence, kv-head, key) positions are cut into equal contiguous
//     ranges, one per CTA, so ragged caches load-balance without a host plan;
//   * a producer warp streams 64-key K and V tiles through a multi-stage
//     shared-memory ring with TMA (2-D tensor copies, 128-byte swizzle),
//     completion tracked by mbarriers;
//   * four consumer warps each own 16 keys of every tile and compute, for the
//     G query heads sharing the kv-head, S^T = K Q^T and O^T += V^T P^T with
//     bf16 mma.sync (fp32 accumulate), online softmax in base 2 with warp
//     shuffles; P is split into bf16 hi + lo parts so the PV product keeps
//     ~16 significant bits;
//   * per piece, the four warps' partials are merged in shared memory and
//     written as one unnormalised record (max, sum, o); a combine kernel
//     merges records across CTAs and either writes o or, on the step path,
//     updates the residual stream, normalises it and appends the next layer's
//     K/V rows.
#include <math.h>

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
  static constexpr int OPAD = 9;  // padded head stride of the merge scratch
  static constexpr int MERGE_FLOATS = 2 * ATT_CONSUMERS * ATT_MAX_G + ATT_CONSUMERS * D * OPAD;
  static constexpr size_t SMEM = 1024 + (size_t)STAGES * STAGE_BYTES + (2 * STAGES + 1) * 8 +
                                 (size_t)MERGE_FLOATS * 4 + (ATT_MAX_S + 1) * 8 + ATT_MAX_S * 4 + 128;
};

struct Piece {
  int32_t s, h, k0, k1;
};

// (sequence, head, key range) of the piece that starts at global position p
// and ends at the next segment boundary or at `end`.
__device__ __forceinline__ Piece find_piece(const int64_t* pre, const int32_t* lens, int32_t S, int64_t T, int64_t p,
                                            int64_t end) {
  Piece pc;
  pc.h = (int32_t)(p / T);
  const int64_t r = p - (int64_t)pc.h * T;
  int32_t lo = 0, hi = S - 1;
  while (lo < hi) {
    const int32_t mid = (lo + hi + 1) >> 1;
    if (pre[mid] <= r) lo = mid;
    else hi = mid - 1;
  }
  pc.s = lo;
  pc.k0 = (int32_t)(r - pre[lo]);
  const int64_t seg_end = (int64_t)pc.h * T + pre[lo] + lens[lo];
  const int64_t e = seg_end < end ? seg_end : end;
  pc.k1 = pc.k0 + (int32_t)(e - p);
  return pc;
}

template <int KSTEPS>
__device__ __forceinline__ void load_q_frag(uint32_t (&qf)[KSTEPS][2], const AttArgs& a, const Piece& pc, int g,
                                            int tq, int D) {
  const bool hv = g < a.G;
  const __nv_bfloat16* qrow = a.q + ((int64_t)pc.s * a.Hq + (int64_t)pc.h * a.G + (hv ? g : 0)) * D;
#pragma unroll
  for (int j = 0; j < KSTEPS; ++j) {
    qf[j][0] = hv ? *reinterpret_cast<const uint32_t*>(qrow + 16 * j + 2 * tq) : 0u;
    qf[j][1] = hv ? *reinterpret_cast<const uint32_t*>(qrow + 16 * j + 8 + 2 * tq) : 0u;
  }
}

template <int D>
__global__ void __launch_bounds__(ATT_THREADS, 1)
    att_split_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap, AttArgs a) {
  using C = AttCfg<D>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  // layout: stages | full[STAGES] | empty[STAGES] | merge | merge scratch | pre[S+1] | lens[S]
  const uint32_t bar_full = base + C::STAGES * C::STAGE_BYTES;
  const uint32_t bar_empty = bar_full + C::STAGES * 8;
  const uint32_t bar_merge = bar_empty + C::STAGES * 8;
  float* mscr = reinterpret_cast<float*>(gbase + C::STAGES * C::STAGE_BYTES + (2 * C::STAGES + 1) * 8);
  float* ms = mscr;                                  // [8][8]
  float* ls = mscr + ATT_CONSUMERS * ATT_MAX_G;      // [8][8]
  float* os = mscr + 2 * ATT_CONSUMERS * ATT_MAX_G;  // [8][D][OPAD]
  int64_t* pre = reinterpret_cast<int64_t*>(mscr + C::MERGE_FLOATS);
  int32_t* lens = reinterpret_cast<int32_t*>(pre + ATT_MAX_S + 1);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int32_t S = a.S, G = a.G;

  if (tid == 0) {
    for (int i = 0; i < C::STAGES; ++i) {
      mbar_init(bar_full + 8 * i, 1);
      mbar_init(bar_empty + 8 * i, 4);  // one warpgroup consumes each stage
    }
    mbar_init(bar_merge, ATT_CONSUMERS * 32);
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
    lens[i] = L;
  }
  __syncthreads();
  if (warp == 0) {  // exclusive prefix of len
    const int chunk = (S + 31) / 32;
    const int b0 = lane * chunk, b1 = min(S, b0 + chunk);
    int64_t sum = 0;
    for (int i = b0; i < b1; ++i) sum += lens[i];
    int64_t incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int64_t v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    int64_t run = incl - sum;
    for (int i = b0; i < b1; ++i) {
      pre[i] = run;
      run += lens[i];
    }
    if (lane == 31) pre[S] = incl;
  }
  __syncthreads();
  const int64_t T = pre[S];
  const int64_t total = T * a.Hkv;
  const int64_t per = (total + gridDim.x - 1) / gridDim.x;
  if (blockIdx.x == 0) {
    for (int i = tid; i <= S; i += ATT_THREADS) a.plan_pre[i] = pre[i];
    if (tid == 0) *a.plan_per = per;
  }
  const int64_t r_begin = (int64_t)blockIdx.x * per;
  const int64_t r_end = min(total, r_begin + per);

  if (warp == ATT_CONSUMERS) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      uint32_t it = 0;
      bool ok = true;
      for (int64_t p = r_begin; p < r_end && ok;) {
        const Piece pc = find_piece(pre, lens, S, T, p, r_end);
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
#pragma unroll
          for (int b = 0; b < C::BOXES; ++b) {
            tma_load_2d(sk + b * C::BOX_BYTES, &kmap, fb, b * 64, row, pol);
            tma_load_2d(sv + b * C::BOX_BYTES, &vmap, fb, b * 64, row, pol);
          }
        }
        p += pc.k1 - pc.k0;
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
  const int wg = warp >> 2, wl = warp & 3;  // warpgroup, warp within the group
  const int g = lane >> 2, tq = lane & 3;   // mma group id / thread in group
  const int mat = lane >> 3, mr = lane & 7;
  const int kb = 16 * wl;                   // first key of this warp's slice of a tile
  uint32_t it = 0, mphase = 0;
  bool ok = true;
  uint32_t qn[C::KSTEPS][2];
  if (r_begin < r_end) load_q_frag<C::KSTEPS>(qn, a, find_piece(pre, lens, S, T, r_begin, r_end), g, tq, D);
  for (int64_t p = r_begin; p < r_end && ok;) {
    const Piece pc = find_piece(pre, lens, S, T, p, r_end);
    p += pc.k1 - pc.k0;
    // B operand of S^T = K Q^T (rows: head dim, cols: the G query heads);
    // the next piece's query is fetched now so its latency overlaps this piece
    uint32_t qf[C::KSTEPS][2];
#pragma unroll
    for (int j = 0; j < C::KSTEPS; ++j) {
      qf[j][0] = qn[j][0];
      qf[j][1] = qn[j][1];
    }
    if (p < r_end) load_q_frag<C::KSTEPS>(qn, a, find_piece(pre, lens, S, T, p, r_end), g, tq, D);

    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
    float o[C::MTILES][4];
#pragma unroll
    for (int i = 0; i < C::MTILES; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;

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
        const uint32_t sk = base + st * C::STAGE_BYTES, sv = sk + C::TILE_BYTES;
        // ---- scores S^T (16 keys x 8 heads), two independent accumulation chains
        float sa[4] = {0.f, 0.f, 0.f, 0.f}, sb[4] = {0.f, 0.f, 0.f, 0.f};
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
            mma_bf16((j & 1) ? sb : sa, a0, a1, a2, a3, qf[j][0], qf[j][1]);
          }
        }
        const bool v0 = kb + g < nvalid, v1 = kb + g + 8 < nvalid;
        const float s0 = v0 ? (sa[0] + sb[0]) * a.scale_log2 : -INFINITY;
        const float s1 = v0 ? (sa[1] + sb[1]) * a.scale_log2 : -INFINITY;
        const float s2 = v1 ? (sa[2] + sb[2]) * a.scale_log2 : -INFINITY;
        const float s3 = v1 ? (sa[3] + sb[3]) * a.scale_log2 : -INFINITY;
        float x0 = fmaxf(s0, s2), x1 = fmaxf(s1, s3);
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
          x0 = fmaxf(x0, __shfl_xor_sync(0xffffffffu, x0, off));
          x1 = fmaxf(x1, __shfl_xor_sync(0xffffffffu, x1, off));
        }
        const float n0 = fmaxf(m0, x0), n1 = fmaxf(m1, x1);
        const float u0 = n0 == -INFINITY ? 0.f : n0, u1 = n1 == -INFINITY ? 0.f : n1;
        const float al0 = exp2f(m0 - u0), al1 = exp2f(m1 - u1);
        const float p0 = exp2f(s0 - u0), p1 = exp2f(s1 - u1), p2 = exp2f(s2 - u0), p3 = exp2f(s3 - u1);
        l0 = l0 * al0 + p0 + p2;
        l1 = l1 * al1 + p1 + p3;
        m0 = n0;
        m1 = n1;
#pragma unroll
        for (int i = 0; i < C::MTILES; ++i) {
          o[i][0] *= al0;
          o[i][2] *= al0;
          o[i][1] *= al1;
          o[i][3] *= al1;
        }
        // ---- P^T as the B operand (keys x heads), split into bf16 hi + lo
        const uint32_t h01 = pack_bf16(p0, p1), h23 = pack_bf16(p2, p3);
        const uint32_t q01 = pack_bf16(p0 - bf16_lo(h01), p1 - bf16_hi(h01));
        const uint32_t q23 = pack_bf16(p2 - bf16_lo(h23), p3 - bf16_hi(h23));
        const uint32_t bh0 = movmatrix_t(h01), bh1 = movmatrix_t(h23);
        const uint32_t bl0 = movmatrix_t(q01), bl1 = movmatrix_t(q23);
        // ---- O^T += V^T P^T; rows of V past the live length are zeroed
        const bool partial = kb + 16 > nvalid;
        const int klo = kb + 2 * tq, khi = klo + 8;
        {
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
            mma_bf16(o[i], a0, a1, a2, a3, bh0, bh1);
            mma_bf16(o[i], a0, a1, a2, a3, bl0, bl1);
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(bar_empty + 8 * st);
    }
    if (!ok) break;

    // ---- merge the eight warps' partials of this piece and write the record
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
      l0 += __shfl_xor_sync(0xffffffffu, l0, off);
      l1 += __shfl_xor_sync(0xffffffffu, l1, off);
    }
    if (g == 0) {
      ms[warp * ATT_MAX_G + 2 * tq] = m0;
      ms[warp * ATT_MAX_G + 2 * tq + 1] = m1;
      ls[warp * ATT_MAX_G + 2 * tq] = l0;
      ls[warp * ATT_MAX_G + 2 * tq + 1] = l1;
    }
    float* ow = os + warp * D * C::OPAD;
#pragma unroll
    for (int i = 0; i < C::MTILES; ++i) {
      const int d0 = 16 * i + g, d1 = d0 + 8;
      ow[d0 * C::OPAD + 2 * tq] = o[i][0];
      ow[d0 * C::OPAD + 2 * tq + 1] = o[i][1];
      ow[d1 * C::OPAD + 2 * tq] = o[i][2];
      ow[d1 * C::OPAD + 2 * tq + 1] = o[i][3];
    }
    if (!bar_sync_bounded(bar_merge, mphase, a.status)) break;
    const int64_t slot = (int64_t)blockIdx.x + (int64_t)pc.h * S + pc.s;
    for (int idx = tid; idx < G * D; idx += ATT_CONSUMERS * 32) {
      const int hh = idx / D, dd = idx - hh * D;
      float M = -INFINITY;
#pragma unroll
      for (int w = 0; w < ATT_CONSUMERS; ++w) M = fmaxf(M, ms[w * ATT_MAX_G + hh]);
      float acc = 0.f, lsum = 0.f;
#pragma unroll
      for (int w = 0; w < ATT_CONSUMERS; ++w) {
        const float mw = ms[w * ATT_MAX_G + hh];
        if (mw == -INFINITY) continue;
        const float e = exp2f(mw - M);
        acc += os[(w * D + dd) * C::OPAD + hh] * e;
        lsum += ls[w * ATT_MAX_G + hh] * e;
      }
      a.rec_o[(slot * G + hh) * D + dd] = acc;
      if (dd == 0) a.rec_ml[slot * G + hh] = make_float2(M, lsum);
    }
    if (!bar_sync_bounded(bar_merge, mphase, a.status)) break;
  }
}

// ------------------------------------------------------------------ combine
// One CTA per (kv-head h, sequence s): weights of the records that cover the
// segment are formed once in shared memory, then every output element sums
// its records with independent loads.
constexpr int CMB_THREADS = 128;
constexpr int CMB_SLOTS = 64;                        // records weighted per pass
constexpr int CMB_PER_THREAD = ATT_MAX_G * 128 / CMB_THREADS;  // G*D <= 1024 outputs per CTA

__global__ void __launch_bounds__(CMB_THREADS) att_combine_kernel(CombineArgs a) {
  const int h = blockIdx.x, s = blockIdx.y, tid = threadIdx.x;
  const int32_t Hq = a.Hq, Hkv = a.Hkv, G = a.G, D = a.D, S = a.S, d = Hq * D;
  __shared__ float wts[CMB_SLOTS][ATT_MAX_G];
  __shared__ float red[CMB_THREADS / 32];
  __shared__ int last;
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
  if (a.mode == 0) {
#pragma unroll
    for (int j = 0; j < CMB_PER_THREAD; ++j) {
      const int idx = tid + j * CMB_THREADS;
      if (idx < GD) a.out[(int64_t)s * d + (int64_t)h * GD + idx] = acc[j];
    }
    return;
  }
  // residual update of this CTA's heads and their sum of squares
  float ss = 0.f;
  float* xr = a.resid + (int64_t)s * d + (int64_t)h * GD;
#pragma unroll
  for (int j = 0; j < CMB_PER_THREAD; ++j) {
    const int idx = tid + j * CMB_THREADS;
    if (idx < GD) {
      const float x = xr[idx] + acc[j];
      xr[idx] = x;
      ss += x * x;
    }
  }
  ss = warp_sum(ss);
  if ((tid & 31) == 0) red[tid >> 5] = ss;
  __syncthreads();
  if (tid == 0) {
    float t = 0.f;
    for (int w = 0; w < CMB_THREADS / 32; ++w) t += red[w];
    a.part_ss[(int64_t)s * Hkv + h] = t;
    __threadfence();
    const int prev = atomicAdd(&a.counters[s], 1);
    last = prev == Hkv - 1;
    if (last) a.counters[s] = 0;
  }
  __syncthreads();
  if (!last) return;
  // last CTA of sequence s: normalise the whole residual row (sums in head order)
  __threadfence();
  __shared__ float inv_sh;
  if (tid == 0) {
    float t = 0.f;
    for (int hh = 0; hh < Hkv; ++hh) t += __ldcg(&a.part_ss[(int64_t)s * Hkv + hh]);
    inv_sh = 1.0f / sqrtf(t / (float)d + a.rms_eps);
  }
  __syncthreads();
  const float inv = inv_sh;
  const int32_t pos = a.seq_len[s] - 1;
  const int32_t capv = a.cap[s];
  const bool can_append = a.append && pos >= 0 && pos < capv;
  const float* xs = a.resid + (int64_t)s * d;
  for (int idx = tid; idx < d; idx += CMB_THREADS) {
    const __nv_bfloat16 u = __float2bfloat16_rn(__ldcg(xs + idx) * inv);
    if (a.append) {
      a.q_next[(int64_t)s * d + idx] = u;
      if (can_append && idx < 2 * Hkv * D) {
        const int hh = idx / D, dd = idx - hh * D;
        const bool isv = hh >= Hkv;
        const int hk = isv ? hh - Hkv : hh;
        const int64_t e = a.next_layer_elem_base + a.kv_offset[s] + ((int64_t)hk * capv + pos) * D + dd;
        (isv ? a.v_cache : a.k_cache)[e] = u;
      }
    } else {
      a.hidden[(int64_t)s * d + idx] = u;
      if (a.hidden_copy) a.hidden_copy[(int64_t)s * d + idx] = u;
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

template <int D>
static cudaError_t launch_split(const CUtensorMap& kmap, const CUtensorMap& vmap, const AttArgs& a, int ctas,
                                cudaStream_t stream) {
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(att_split_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)AttCfg<D>::SMEM);
    if (e != cudaSuccess) return e;
    configured = true;
  }
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
  pced_status st = make_tmap_2d(&kmap, k_cache, rows, (uint64_t)D, ATT_BLOCK_N, 64, true);
  if (st != PCED_OK) return st;
  st = make_tmap_2d(&vmap, v_cache, rows, (uint64_t)D, ATT_BLOCK_N, 64, true);
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
  c.mode = 0;
  c.S = S;
  c.Hq = Hq;
  c.Hkv = Hkv;
  c.G = G;
  c.D = D;
  c.rec_o = a.rec_o;
  c.rec_ml = a.rec_ml;
  c.plan_pre = a.plan_pre;
  c.plan_per = a.plan_per;
  c.seq_len = seq_len;
  c.out = out;
  c.status = a.status;
  e = att_combine_launch(c, s);
  if (e != cudaSuccess) return cuda_status(e, "attention combine launch");
  return PCED_OK;
}
