// lm_head.cu -- per-expert vocabulary scores (paper Sec. 3, "per-expert logits
// s_k"; Eq. 2 mixes them as log-probabilities) on the 5th-generation tensor
// cores.
//
// Swap-AB skinny GEMM: Z^T[V x S] = W[V x d] * H^T[d x S].  The vocabulary is
// the UMMA M dimension (128-row tiles), the S hidden rows are the N dimension,
// so the bf16 unembedding matrix streams from HBM exactly once per step while
// the tiny H operand is re-read from L2.  Persistent CTAs, one per SM:
//   warp 0  TMA producer (W tile 128x64 + H slab S_pad x 64 per stage, 128B swizzle)
//   warp 1  TMEM allocator and single-thread tcgen05.mma issuer (fp32 accumulators
//           in TMEM, double-buffered when 2*S_pad <= 512 columns)
//   warps 2-9 epilogue: tcgen05.ld of the 128 x S accumulator (warp w reads TMEM lane
//           quarter w % 4; warps 2-5 take the first half of the columns, 6-9 the rest);
//           per column the tile's (max, sum exp) for the log-softmax and, for each
//           contextual expert k of query b, the tile's max and argmax of
//           u_k(v) = (1+beta_k) z_k(v) - beta_k z_0(v), reduced over the rows with
//           transposed butterflies (one shuffle per column and reduction).
// Because shat_k(v) = u_k(v) + c_k with c_k = -(1+beta_k) L_k + beta_k L_0 + gamma log r_k
// constant in v, Eq. 3 only needs these per-tile maxima and the log-sum-exps L:
// the [S x V] logits never reach HBM on the fused path.
#include <math.h>
#include <stdlib.h>

#include "lm_head.cuh"
#include "select_key.cuh"

namespace pced {

constexpr int LM_A_BYTES = LM_TILE_V * LM_TILE_K * 2;  // 16 KB
constexpr size_t LM_SMEM_BUDGET = 227 * 1024;

bool lm_geometry(int32_t S, int32_t d, int32_t V, LmGeom* g) {
  if (S < 1 || S > LM_MAX_S || d < LM_TILE_K || d % LM_TILE_K != 0 || V < 1) return false;
  g->S = S;
  g->d = d;
  g->V = V;
  g->nchunk = (S + 255) / 256;
  const int per = (S + g->nchunk - 1) / g->nchunk;
  g->chunk_n = ((per < 16 ? 16 : per) + 15) / 16 * 16;
  g->S_pad = g->nchunk * g->chunk_n;
  if (g->S_pad > 512) return false;
  g->acc_bufs = 2 * g->S_pad <= 512 ? 2 : 1;
  uint32_t cols = 32;
  while (cols < (uint32_t)(g->acc_bufs * g->S_pad)) cols <<= 1;
  g->tmem_cols = cols;
  g->ntiles = (V + LM_TILE_V - 1) / LM_TILE_V;
  g->nks = d / LM_TILE_K;
  const size_t slab = LM_A_BYTES + (size_t)g->S_pad * 128;
  const size_t fixed = 1024 + 64 * 8 + 16 + (size_t)2 * 4 * g->S_pad * sizeof(float2) +
                       (size_t)2 * g->S_pad * sizeof(float2) + (size_t)g->S_pad * sizeof(float2) + 32 * 4 + 8 * 64 * 4 + 64 + 128;
  // several consecutive K-slabs per stage so each row is fetched in longer
  // runs and the tensor cores get longer bursts per stage; keep at least
  // three stages in flight
  g->slabs = 1;
  for (int sl = 4; sl >= 2; sl >>= 1)
    if (g->nks % sl == 0 && fixed + 3 * sl * slab <= LM_SMEM_BUDGET) {
      g->slabs = sl;
      break;
    }
  const size_t stage = (size_t)g->slabs * slab;
  int st = (int)((LM_SMEM_BUDGET - fixed) / stage);
  if (st > 8) st = 8;
  if (st < 2) return false;
  g->stages = st;
  g->nst = g->nks / g->slabs;
  g->smem = fixed + (size_t)st * stage;
  int sms = pced_host::num_sms();
  g->grid = g->ntiles < sms ? g->ntiles : sms;
  if (g->grid < 1) g->grid = 1;
  return true;
}

// Top-2 over tokens of (value, token) candidates whose token sets are
// disjoint: (b1, t1) the best (larger value, then lower token), b2 the best
// value at another token; merges the candidate set (r1, rt, r2) into it.
__device__ __forceinline__ void top2_merge(float& b1, int& t1, float& b2, float r1, int rt, float r2) {
  if (r1 > b1 || (r1 == b1 && rt < t1)) {
    b2 = fmaxf(b1, r2);
    b1 = r1;
    t1 = rt;
  } else {
    b2 = fmaxf(b2, r1);
  }
}

struct FMax {
  __device__ __forceinline__ float operator()(float x, float y) const { return fmaxf(x, y); }
};
struct FAdd {
  __device__ __forceinline__ float operator()(float x, float y) const { return x + y; }
};

// Reduce NB columns held one per register over the 32 lanes (vocabulary rows)
// of a warp in transposed form: every exchange hands half of the columns still
// held to the partner lane, so NB columns cost NB - 1 shuffles instead of
// 5 NB.  The pairing (lane bit 4 first, bit 0 last) is that of a per-column
// xor tree, so sums round identically.  NB = 32: lane l ends with column l;
// NB = 16 or 8: full exchanges across the lane bits at and above NB first, so
// every lane l ends with column l & (NB - 1).
template <int NB, class Op>
__device__ __forceinline__ float bfly_reduce(float (&x)[NB], int lane, Op op) {
#pragma unroll
  for (int w = 16; w >= NB; w >>= 1) {
#pragma unroll
    for (int i = 0; i < NB; ++i) x[i] = op(x[i], __shfl_xor_sync(0xffffffffu, x[i], w));
  }
#pragma unroll
  for (int w = NB / 2; w >= 1; w >>= 1) {
    const bool hi = (lane & w) != 0;
#pragma unroll
    for (int i = 0; i < w; ++i) {
      const float send = hi ? x[i] : x[i + w];
      const float keep = hi ? x[i + w] : x[i];
      x[i] = op(keep, __shfl_xor_sync(0xffffffffu, send, w));
    }
  }
  return x[0];
}

// Top-2 over the 32 lanes (vocabulary rows) of NB columns held one per
// register, in the transposed form of bfly_reduce: (best value, its token,
// best value at another token) travel together, ties to the lower token.
// Lane l ends with column l & (NB - 1).  `tok` is this lane's token.
template <int NB>
__device__ __forceinline__ void bfly_top2(const float (&u)[NB], int tok, int lane, float& r1, int& rt, float& r2) {
  constexpr int K = NB == 32 ? 16 : NB;  // slots after the first level
  float b1[K], b2[K];
  int bt[K];
  const int ptok = tok + ((lane ^ 16) - lane);  // the row across lane bit 4
  const bool hi16 = (lane & 16) != 0;
#pragma unroll
  for (int i = 0; i < K; ++i) {
    // NB = 32: the first halving level; NB <= 16: a full exchange
    const float send = NB == 32 ? (hi16 ? u[i] : u[(i + 16) % NB]) : u[i];
    const float keep = NB == 32 ? (hi16 ? u[(i + 16) % NB] : u[i]) : u[i];
    const float o = __shfl_xor_sync(0xffffffffu, send, 16);
    const bool take = o > keep || (o == keep && ptok < tok);
    b1[i] = take ? o : keep;
    bt[i] = take ? ptok : tok;
    b2[i] = take ? keep : o;
  }
  // NB = 8: one more full exchange, across lane bit 3
#pragma unroll
  for (int w = 8; w >= NB; w >>= 1) {
#pragma unroll
    for (int i = 0; i < K; ++i) {
      const float o1 = __shfl_xor_sync(0xffffffffu, b1[i], w), o2 = __shfl_xor_sync(0xffffffffu, b2[i], w);
      const int ot = __shfl_xor_sync(0xffffffffu, bt[i], w);
      top2_merge(b1[i], bt[i], b2[i], o1, ot, o2);
    }
  }
#pragma unroll
  for (int w = (NB == 32 ? 8 : NB / 2); w >= 1; w >>= 1) {
    const bool hi = (lane & w) != 0;
#pragma unroll
    for (int i = 0; i < w; ++i) {
      const float s1 = hi ? b1[i] : b1[i + w], s2 = hi ? b2[i] : b2[i + w];
      const int st = hi ? bt[i] : bt[i + w];
      float k1 = hi ? b1[i + w] : b1[i], k2 = hi ? b2[i + w] : b2[i];
      int kt = hi ? bt[i + w] : bt[i];
      const float o1 = __shfl_xor_sync(0xffffffffu, s1, w), o2 = __shfl_xor_sync(0xffffffffu, s2, w);
      const int ot = __shfl_xor_sync(0xffffffffu, st, w);
      top2_merge(k1, kt, k2, o1, ot, o2);
      b1[i] = k1;
      bt[i] = kt;
      b2[i] = k2;
    }
  }
  r1 = b1[0];
  rt = bt[0];
  r2 = b2[0];
}

// Epilogue of NB accumulator columns c0.. (c0 a multiple of NB) of one
// warp's 32 vocabulary rows: mode 0 stores the logits; both modes record the
// per-column (max, sum of exp) of the 32 rows; mode 1 also records per expert
// column the max of u_k = (1 + beta) z_k - beta z_0, its first (lowest)
// vocabulary index and the best value at another index.  `bc` is this warp's
// broadcast buffer; z_am carries the row's amateur logit from its query's
// first column to the expert columns; ccoef / cmask hold each column's
// (1 + beta, beta) and the amateur / expert column bits of each 32-column
// block (the same for every tile).
template <int NB>
__device__ __forceinline__ void epi_block(const LmArgs& a, uint32_t taddr, int c0, int v, bool valid, int lane,
                                          int q, float* bc, float2* wst, float2* wag, float* wu2, const float2* ccoef,
                                          const uint32_t* cmask, float& z_am) {
  const int S = a.S, S_pad = a.S_pad;
  float z[NB], t[NB];
  if (NB == 32)
    tmem_ld32(taddr, z);
  else if (NB == 16)
    tmem_ld16(taddr, z);
  else
    tmem_ld8(taddr, z);
  if (a.mode == 0 && valid) {
#pragma unroll
    for (int i = 0; i < NB; ++i)
      if (c0 + i < S) a.logits[(int64_t)(c0 + i) * a.V + v] = z[i];
  }
#pragma unroll
  for (int i = 0; i < NB; ++i) t[i] = valid ? z[i] : -INFINITY;
  float u[NB];
  const uint32_t em = a.mode == 1 ? cmask[16 + (c0 >> 5)] >> (c0 & 31) : 0u;
  if (a.mode == 1) {
    const uint32_t am = cmask[c0 >> 5] >> (c0 & 31);
    float za = z_am;
#pragma unroll
    for (int i = 0; i < NB; ++i) {
      if ((am >> i) & 1u) za = z[i];
      const float2 cf = ccoef[c0 + i];
      u[i] = valid && ((em >> i) & 1u) ? cf.x * z[i] - cf.y * za : -INFINITY;
    }
    z_am = za;
  }
  const float m = bfly_reduce<NB>(t, lane, FMax());
  float b1 = -INFINITY, b2 = -INFINITY;
  int bt = 0;
  if (a.mode == 1) bfly_top2<NB>(u, v, lane, b1, bt, b2);
  const int li = lane & (NB - 1), mycol = c0 + li;
  if (lane < NB) bc[lane] = m;
  __syncwarp();
#pragma unroll
  for (int i = 0; i < NB; ++i) t[i] = valid ? __expf(z[i] - bc[i]) : 0.f;
  const float sm = bfly_reduce<NB>(t, lane, FAdd());
  if (lane < NB && mycol < S) {
    wst[q * S_pad + mycol] = make_float2(m, sm);
    if ((em >> li) & 1u) {
      wag[q * S_pad + mycol] = make_float2(b1, __int_as_float(bt));
      wu2[q * S_pad + mycol] = b2;
    }
  }
  __syncwarp();
}

// The MMAs of one stage of SL K-slabs (single N chunk), fully unrolled: the
// start-address field of a K-major SW128 descriptor advances by 2 per 16-wide
// K-step and by the slab size >> 4 per slab.
template <int SL>
__device__ __forceinline__ void umma_slabs(uint32_t dcol, uint64_t ad0, uint64_t bd0, uint32_t bstep, uint32_t idesc,
                                           bool first) {
#pragma unroll
  for (int j = 0; j < SL; ++j)
#pragma unroll
    for (int k = 0; k < LM_TILE_K / 16; ++k)
      umma_bf16(dcol, ad0 + (uint64_t)(j * (LM_A_BYTES >> 4) + 2 * k), bd0 + (uint64_t)(j * bstep + 2 * k), idesc,
                !(first && j == 0 && k == 0));
}

__global__ void __launch_bounds__(LM_THREADS, 1)
    lm_head_kernel(const __grid_constant__ CUtensorMap wmap, const __grid_constant__ CUtensorMap hmap, LmArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  const int SL = a.slabs, S_pad = a.S_pad;
  const uint32_t b_bytes = (uint32_t)S_pad * 128u;
  const uint32_t st_bytes = (uint32_t)SL * (LM_A_BYTES + b_bytes);  // SL A slabs, then SL B slabs
  const int stages = a.stages;
  // layout: stages | full | empty | tfull[2] | tempty[2] | tid[2] | epi | drain |
  //         tmem slot, tile ring, accumulator tiles | scratch
  const uint32_t bar_full = base + stages * st_bytes;
  const uint32_t bar_empty = bar_full + 8 * stages;
  const uint32_t bar_tfull = bar_empty + 8 * stages;
  const uint32_t bar_tempty = bar_tfull + 16;
  const uint32_t bar_tid = bar_tempty + 16;
  const uint32_t bar_epi = bar_tid + 16;
  const uint32_t bar_drain = bar_epi + 8;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(gbase + (bar_drain + 8 - base));
  int32_t* tring = reinterpret_cast<int32_t*>(tmem_slot + 4);  // [LM_TRING] claimed tiles, producer -> MMA warp
  int32_t* acc_tile = tring + LM_TRING;                        // [2] tile of each accumulator, MMA warp -> epilogue
  float2* wst = reinterpret_cast<float2*>(gbase + (bar_drain + 8 - base) + 96);  // [4][S_pad] per-warp stats
  float2* wag = wst + 4 * S_pad;                                                  // [4][S_pad] per-warp argmax
  float* wu2 = reinterpret_cast<float*>(wag + 4 * S_pad);                         // [4][S_pad] per-warp runner-up
  float2* ccoef = wag + 6 * S_pad;                                 // [S_pad] (1 + beta, beta) per column
  uint32_t* cmask = reinterpret_cast<uint32_t*>(ccoef + S_pad);     // [2][16] amateur / expert column bits
  float* bc = reinterpret_cast<float*>(cmask + 32);                // [8][64] per-warp column broadcast

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int i = 0; i < stages; ++i) {
      mbar_init(bar_full + 8 * i, 1);
      mbar_init(bar_empty + 8 * i, 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar_tfull + 8 * i, 1);
      mbar_init(bar_tempty + 8 * i, LM_EPI_THREADS);
      mbar_init(bar_tid + 8 * i, 1);
    }
    mbar_init(bar_epi, LM_EPI_THREADS);
    mbar_init(bar_drain, 1);
    mbar_fence_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&wmap);
    tma_prefetch_desc(&hmap);
  }
  if (a.pdl) pdl_launch_dependents();
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), a.tmem_cols);
    tmem_relinquish();
  }
  if (a.mode == 1) {
    // per column: expert columns carry (1 + beta_k, beta_k), the amateur
    // column of each query starts its group; bit i of block kb is column 32 kb + i
    const int n1 = a.N + 1;
    for (int c = tid; c < S_pad; c += LM_THREADS) {
      const int j = c % n1, bq = c / n1;
      const float bt = c < a.S && j > 0 ? a.beta[bq * a.N + j - 1] : 0.f;
      ccoef[c] = make_float2(1.f + bt, bt);
    }
    if (warp == 0)
      for (int kb = 0; kb < 16; ++kb) {
        const int c = 32 * kb + lane;
        const bool in = c < a.S;
        const uint32_t am = __ballot_sync(0xffffffffu, in && c % n1 == 0);
        const uint32_t em = __ballot_sync(0xffffffffu, in && c % n1 != 0);
        if (lane == 0) {
          cmask[kb] = am;
          cmask[16 + kb] = em;
        }
      }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int ntiles = a.ntiles, nst = a.nst;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA
    if (lane == 0) {
      const uint64_t pol_w = policy_evict_first(), pol_h = policy_evict_last();
      // Tiles are claimed from a global counter, so CTAs that start early (as
      // the previous kernel's CTAs leave their SMs) take more of them.  The
      // claimed ids reach the MMA warp through tring (written before the
      // arrive on the full barrier of the tile's first stage); -1 ends.
      int tile = -1, ks = 0;
      uint32_t tseq = 0;
      auto claim = [&]() {
        const int t = atomicAdd(a.tile_ctr, 1);
        tile = t < ntiles ? t : -1;
        tring[tseq % LM_TRING] = tile;
        ++tseq;
        ks = 0;
      };
      auto load_w = [&](uint32_t st) {
        const uint32_t fb = bar_full + 8 * st, sa = base + st * st_bytes;
        mbar_arrive_expect_tx(fb, st_bytes);
        // consecutive K-slabs of the same 128 rows back to back: longer runs per row
        for (int j = 0; j < SL; ++j)
          tma_load_2d(sa + j * LM_A_BYTES, &wmap, fb, (ks * SL + j) * LM_TILE_K, tile * LM_TILE_V, pol_w);
      };
      auto load_h = [&](uint32_t st, int kss) {
        const uint32_t fb = bar_full + 8 * st, sb = base + st * st_bytes + SL * LM_A_BYTES;
        for (int j = 0; j < SL; ++j)
          for (int c = 0; c < a.nchunk; ++c)
            tma_load_2d(sb + j * b_bytes + c * a.chunk_n * 128, &hmap, fb, (kss * SL + j) * LM_TILE_K,
                        c * a.chunk_n, pol_h);
      };
      claim();
      uint32_t it = 0;
      // With programmatic dependent launch the weights of the first stages
      // stream while the previous kernel (which writes H) finishes.
      if (a.pdl) {
        int pre_ks[8];
        while (tile >= 0 && it < (uint32_t)stages) {
          load_w(it);
          pre_ks[it++] = ks;
          if (++ks == nst) claim();
        }
        pdl_wait();
        for (uint32_t i = 0; i < it; ++i) load_h(i, pre_ks[i]);
      }
      bool ok = true;
      while (tile >= 0) {
        const uint32_t st = it % stages, ph = (it / stages) & 1u;
        if (!mbar_wait(bar_empty + 8 * st, ph ^ 1u, a.status)) {
          ok = false;
          break;
        }
        load_w(st);
        load_h(st, ks);
        ++it;
        if (++ks == nst) claim();
      }
      if (ok) {
        // end marker: a phase of the next stage's full barrier without data
        const uint32_t st = it % stages, ph = (it / stages) & 1u;
        if (mbar_wait(bar_empty + 8 * st, ph ^ 1u, a.status)) mbar_arrive(bar_full + 8 * st);
      } else {
        for (uint32_t j = (it >= (uint32_t)stages ? it - stages : 0); j < it; ++j)
          mbar_wait(bar_full + 8 * (j % stages), (j / stages) & 1u, a.status);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA
    if (lane == 0) {
      const uint32_t idesc = umma_idesc_bf16(LM_TILE_V, a.chunk_n);
      uint32_t it = 0, acc = 0, tseq = 0;
      bool ok = true;
      for (;; ++acc) {
        const uint32_t buf = acc % a.acc_bufs, aph = (acc / a.acc_bufs) & 1u;
        // the next tile's first stage (or the end marker) tells which tile it is
        {
          const uint32_t st = it % stages, ph = (it / stages) & 1u;
          if (!mbar_wait(bar_full + 8 * st, ph, a.status)) {
            ok = false;
            break;
          }
        }
        const int tile = tring[tseq % LM_TRING];
        ++tseq;
        if (!mbar_wait(bar_tempty + 8 * buf, aph ^ 1u, a.status)) {
          ok = false;
          break;
        }
        acc_tile[buf] = tile;
        mbar_arrive(bar_tid + 8 * buf);
        if (tile < 0) break;
        tc_fence_after();
        const uint32_t dcol = tmem_base + buf * S_pad;
        for (int ks = 0; ks < nst; ++ks, ++it) {
          const uint32_t st = it % stages, ph = (it / stages) & 1u;
          if (ks > 0 && !mbar_wait(bar_full + 8 * st, ph, a.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = base + st * st_bytes, sb = sa + SL * LM_A_BYTES;
          // descriptors are built once per stage; a K-step moves the start
          // address field (bytes >> 4) by 2, a slab by its size >> 4
          const uint64_t ad0 = umma_desc_sw128(sa), bd0 = umma_desc_sw128(sb);
          if (a.nchunk == 1 && (SL == 4 || SL == 2 || SL == 1)) {
            const uint32_t bstep = b_bytes >> 4;
            const bool first = ks == 0;
            if (SL == 4)
              umma_slabs<4>(dcol, ad0, bd0, bstep, idesc, first);
            else if (SL == 2)
              umma_slabs<2>(dcol, ad0, bd0, bstep, idesc, first);
            else
              umma_slabs<1>(dcol, ad0, bd0, bstep, idesc, first);
          } else if (a.nchunk == 2 && SL == 1) {
            // more than 256 hidden rows: two N chunks per K-step, unrolled
            // (the issuing thread, not the data, set the pace with a loop here)
            const uint32_t coff = (uint32_t)(a.chunk_n * 128) >> 4, dc1 = dcol + a.chunk_n;
#pragma unroll
            for (int k = 0; k < LM_TILE_K / 16; ++k) {
              umma_bf16(dcol, ad0 + 2 * k, bd0 + 2 * k, idesc, (ks | k) != 0);
              umma_bf16(dc1, ad0 + 2 * k, bd0 + coff + 2 * k, idesc, (ks | k) != 0);
            }
          } else {
            for (int j = 0; j < SL; ++j) {
#pragma unroll
              for (int k = 0; k < LM_TILE_K / 16; ++k) {
                const uint64_t ad = ad0 + (uint64_t)(j * (LM_A_BYTES >> 4) + 2 * k);
                for (int c = 0; c < a.nchunk; ++c)
                  umma_bf16(dcol + c * a.chunk_n, ad, bd0 + (uint64_t)((j * b_bytes + c * a.chunk_n * 128) >> 4) + 2 * k,
                            idesc, (ks | j | k) != 0);
              }
            }
          }
          umma_commit(bar_empty + 8 * st);
        }
        if (!ok) break;
        umma_commit(bar_tfull + 8 * buf);
      }
      // all issued MMAs complete before TMEM is released
      umma_commit(bar_drain);
      mbar_wait(bar_drain, 0, a.status);
    }
    __syncwarp();
  } else {
    // ----------------------------------------------------------- epilogue
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    const int etid = tid - 64, half = (warp - 2) >> 2;
    const int S = a.S, n1 = a.N + 1;
    uint32_t ephase = 0;
    for (uint32_t acc = 0;; ++acc) {
      const uint32_t buf = acc % a.acc_bufs, aph = (acc / a.acc_bufs) & 1u;
      if (!mbar_wait(bar_tid + 8 * buf, aph, a.status)) break;
      const int tile = acc_tile[buf];
      if (tile < 0) break;
      if (!mbar_wait(bar_tfull + 8 * buf, aph, a.status)) break;
      tc_fence_after();
      const int v = tile * LM_TILE_V + 32 * q + lane;
      const bool valid = v < a.V;
      const uint32_t trow = tmem_base + ((uint32_t)(32 * q) << 16) + buf * S_pad;
      // column blocks of W = 32 (the last one may be 16 wide), or of S_pad / 2
      // when S_pad <= 32 so that both warp halves work; the first half of the
      // blocks goes to warps 2-5, the rest to warps 6-9
      const int W = S_pad <= 32 ? S_pad / 2 : 32;
      const int nb = (S + W - 1) / W, kb0 = half ? (nb + 1) / 2 : 0, kb1 = half ? nb : (nb + 1) / 2;
      float z_am = 0.f;
      if (a.mode == 1 && kb0 < kb1 && (W * kb0) % n1 != 0)
        z_am = tmem_ld1(trow + W * kb0 - (W * kb0) % n1);  // the row's amateur logit of the open query
      float* wbc = bc + 64 * (warp - 2);
      for (int kb = kb0; kb < kb1; ++kb) {
        const int c0 = W * kb;
        if (W == 8)
          epi_block<8>(a, trow + c0, c0, v, valid, lane, q, wbc, wst, wag, wu2, ccoef, cmask, z_am);
        else if (c0 + 32 <= S_pad && W == 32)
          epi_block<32>(a, trow + c0, c0, v, valid, lane, q, wbc, wst, wag, wu2, ccoef, cmask, z_am);
        else
          epi_block<16>(a, trow + c0, c0, v, valid, lane, q, wbc, wst, wag, wu2, ccoef, cmask, z_am);
      }
      tc_fence_before();
      mbar_arrive(bar_tempty + 8 * buf);
      if (!bar_sync_bounded(bar_epi, ephase, a.status)) break;
      // this tile's records: the four lane quarters' results folded in a fixed
      // order, stored per tile so the cross-tile merge order does not depend
      // on which CTA took the tile
      const bool tile_ok = PCED_IN_BOUNDS(tile < ntiles, a.status);
      for (int col = etid; col < S && tile_ok; col += LM_EPI_THREADS) {
        float cm = -INFINITY, cs = 0.f;
#pragma unroll
        for (int qq = 0; qq < 4; ++qq) {
          const float2 r = wst[qq * S_pad + col];
          lse_merge(cm, cs, r.x, r.y);
        }
        a.rec_stats[(int64_t)col * ntiles + tile] = make_float2(cm, cs);
        if (a.mode == 1 && col % n1 != 0) {
          float bu = -INFINITY, b2 = -INFINITY;
          int bv = 0x7fffffff;
#pragma unroll
          for (int qq = 0; qq < 4; ++qq) {
            const float2 r = wag[qq * S_pad + col];
            top2_merge(bu, bv, b2, r.x, __float_as_int(r.y), wu2[qq * S_pad + col]);
          }
          a.rec_arg[(int64_t)col * ntiles + tile] = make_float2(bu, __int_as_float(bv));
          a.rec_u2[(int64_t)col * ntiles + tile] = b2;
        }
      }
      if (!bar_sync_bounded(bar_epi, ephase, a.status)) break;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, a.tmem_cols);
  }
}

cudaError_t lm_head_launch(const CUtensorMap& wmap, const CUtensorMap& hmap, const LmGeom& g, const LmArgs& a,
                           cudaStream_t stream) {
  // the shared-memory limit is an attribute of the kernel on each device
  static bool configured[64];
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!configured[dev]) {
    e = cudaFuncSetAttribute(lm_head_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)LM_SMEM_BUDGET);
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(g.grid);
  cfg.blockDim = dim3(LM_THREADS);
  cfg.dynamicSmemBytes = g.smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = a.pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, lm_head_kernel, wmap, hmap, a);
}

// ------------------------------------------------------------ mode-0 finish
// grid (chunks, S): every CTA of row s forms lse[s] from the row's tile
// records (the same fixed order in each) and turns its chunk of logits into
// log-probabilities in place; chunk 0 stores lse.
constexpr int LSE_CHUNK = 8192;  // (144 CTAs for 9 rows of 128K entries)

__global__ void __launch_bounds__(256) lm_lse_finalize_kernel(float* logits, const float2* rec_stats, float* lse,
                                                              int32_t V, int32_t nrec) {
  const int c = blockIdx.x, s = blockIdx.y, tid = threadIdx.x;
  __shared__ float2 red[8];
  __shared__ float Ls;
  float M = -INFINITY, sum = 0.f;
  for (int t = tid; t < nrec; t += 256) {
    const float2 r = rec_stats[(int64_t)s * nrec + t];
    lse_merge(M, sum, r.x, r.y);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, M, o), s2 = __shfl_xor_sync(0xffffffffu, sum, o);
    lse_merge(M, sum, m2, s2);
  }
  if ((tid & 31) == 0) red[tid >> 5] = make_float2(M, sum);
  __syncthreads();
  if (tid == 0) {
    float m = -INFINITY, su = 0.f;
    for (int w = 0; w < 8; ++w) lse_merge(m, su, red[w].x, red[w].y);
    Ls = m + logf(su);
    if (c == 0) lse[s] = Ls;
  }
  __syncthreads();
  const float L = Ls;
  float* row = logits + (int64_t)s * V;
  const int v1 = min(V, (c + 1) * LSE_CHUNK);
  for (int v = c * LSE_CHUNK + tid; v < v1; v += 256) row[v] -= L;
}

cudaError_t lm_lse_finalize_launch(float* logits, const float2* rec_stats, float* lse, int32_t S, int32_t V,
                                   int32_t nrec, cudaStream_t stream) {
  lm_lse_finalize_kernel<<<dim3((V + LSE_CHUNK - 1) / LSE_CHUNK, S), 256, 0, stream>>>(logits, rec_stats, lse, V,
                                                                                      nrec);
  return cudaGetLastError();
}

// ------------------------------------------- Eq. 2 + Eq. 3 from tile records
// One CTA per row s = b*(N+1) + j: L_s from the row's tile records and, for an
// expert row (j > 0), the best tile record of u_k; the last CTA of query b to
// finish forms score_k = u_k* + c_k and picks the best (score desc, token
// asc, expert asc).  Every reduction runs in a fixed order (thread t takes
// records t, t + 256, ... in four interleaved chains, then a fixed tree), so
// the result does not depend on timing.
constexpr int SEL_R_THREADS = 256;
constexpr int SEL_ZROWS = 12;  // hidden rows per block of the near-tie dot products

__device__ __forceinline__ void lse_block(const float2* rec, int T, int tid, float2* red, float& L) {
  float m[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY}, su[4] = {0.f, 0.f, 0.f, 0.f};
  int t = tid;
  for (; t + 3 * SEL_R_THREADS < T; t += 4 * SEL_R_THREADS) {
    float2 r[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) r[k] = rec[t + k * SEL_R_THREADS];
#pragma unroll
    for (int k = 0; k < 4; ++k) lse_merge(m[k], su[k], r[k].x, r[k].y);
  }
  for (; t < T; t += SEL_R_THREADS) {
    const float2 r = rec[t];
    lse_merge(m[0], su[0], r.x, r.y);
  }
#pragma unroll
  for (int k = 1; k < 4; ++k) lse_merge(m[0], su[0], m[k], su[k]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m[0], o), s2 = __shfl_xor_sync(0xffffffffu, su[0], o);
    lse_merge(m[0], su[0], m2, s2);
  }
  if ((tid & 31) == 0) red[tid >> 5] = make_float2(m[0], su[0]);
  __syncthreads();
  if (tid == 0) {
    float M = -INFINITY, Sm = 0.f;
    for (int w = 0; w < SEL_R_THREADS / 32; ++w) lse_merge(M, Sm, red[w].x, red[w].y);
    L = M + logf(Sm);
  }
}

__global__ void __launch_bounds__(SEL_R_THREADS) select_from_records_kernel(SelectArgs a) {
  const int j = blockIdx.x, b = blockIdx.y, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int N = a.N, n1 = N + 1, s = b * n1 + j, T = a.nrec;
  if (!PCED_IN_BOUNDS(s < a.B * n1, a.status)) return;
  if (a.pdl) pdl_wait();  // the LM head's records are complete and visible
  if (j == 0 && b == 0 && tid == 0 && a.tile_ctr) *a.tile_ctr = 0;  // the next LM head claims its tiles from 0
  __shared__ float2 red[SEL_R_THREADS / 32];
  __shared__ float sv[SEL_R_THREADS / 32], sv2[SEL_R_THREADS / 32];
  __shared__ int si[SEL_R_THREADS / 32];
  __shared__ int last;
  __shared__ int pick[2];   // token, expert of the query (last CTA)
  __shared__ float zy[LM_MAX_N1];  // z_s(token) of the query's rows (last CTA)
  __shared__ float zpart[SEL_R_THREADS / 32][SEL_ZROWS];
  float L = 0.f;
  lse_block(a.rec_stats + (int64_t)s * T, T, tid, red, L);
  if (j > 0) {
    // the row's best u_k and its token, and the best u_k at any other token
    const float2* rec = a.rec_arg + (int64_t)s * T;
    const float* rec2 = a.rec_u2 + (int64_t)s * T;
    float bu = -INFINITY, b2 = -INFINITY;
    int bv = 0x7fffffff;
    for (int t = tid; t < T; t += SEL_R_THREADS) {
      const float2 r = rec[t];
      top2_merge(bu, bv, b2, r.x, __float_as_int(r.y), rec2[t]);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float r1 = __shfl_xor_sync(0xffffffffu, bu, o), r2 = __shfl_xor_sync(0xffffffffu, b2, o);
      const int rt = __shfl_xor_sync(0xffffffffu, bv, o);
      top2_merge(bu, bv, b2, r1, rt, r2);
    }
    if (lane == 0) {
      sv[warp] = bu;
      si[warp] = bv;
      sv2[warp] = b2;
    }
    __syncthreads();
    if (tid == 0) {
      for (int w = 1; w < SEL_R_THREADS / 32; ++w) top2_merge(bu, bv, b2, sv[w], si[w], sv2[w]);
      a.sel_u[s] = bu;
      a.sel_tok[s] = bv;
      a.sel_u2[s] = b2;
    }
  }
  if (tid == 0) {
    a.sel_L[s] = L;
    if (a.lse_out) a.lse_out[s] = L;
    __threadfence();
    last = atomicAdd(a.qdone + b, 1) == n1 - 1;
  }
  __syncthreads();
  if (!last) return;
  __threadfence();  // the other rows' results of query b are visible
  const float L0 = __ldcg(a.sel_L + b * n1);
  float bs = -INFINITY;
  int bt = 0x7fffffff, bk = 0x7fffffff;
  if (warp == 0) {
    for (int k = lane; k < N; k += 32) {
      const int sk = b * n1 + 1 + k;
      const float btk = a.beta[b * N + k];
      const float rr = fminf(fmaxf(a.r[b * N + k], 1e-8f), 1.0f);
      const float c = (a.raw_logits ? 0.f : -(1.f + btk) * __ldcg(a.sel_L + sk) + btk * L0) + a.gamma * logf(rr);
      const float sc = __ldcg(a.sel_u + sk) + c;
      const int tk = __ldcg(a.sel_tok + sk);
      if (sc > bs || (sc == bs && (tk < bt || (tk == bt && k < bk)))) {
        bs = sc;
        bt = tk;
        bk = k;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float s2 = __shfl_xor_sync(0xffffffffu, bs, o);
      const int t2 = __shfl_xor_sync(0xffffffffu, bt, o), k2 = __shfl_xor_sync(0xffffffffu, bk, o);
      if (s2 > bs || (s2 == bs && (t2 < bt || (t2 == bt && k2 < bk)))) {
        bs = s2;
        bt = t2;
        bk = k2;
      }
    }
    if (lane == 0) {
      pick[0] = bt;
      pick[1] = bk;
    }
  }
  float2 gaps = make_float2(INFINITY, INFINITY);
  if (a.gap_trace && !a.key_out) {
    __syncthreads();
    const int y = pick[0] >= 0 && pick[0] < a.V ? pick[0] : 0;
    // z_s(y) = h_s . W[y] for the query's rows.  Thread t takes the 16-byte
    // chunks i = t, t + 256 of W[y] and the same chunks of up to 16 rows at a
    // time, all loads of a row block in flight together (one round trip for
    // d <= 4096); per row the partial sums meet in a fixed order (warp tree,
    // then the warps in order).
    const int nv = a.d / 8;  // 16-byte chunks of a row (d % 64 == 0)
    const uint4* wy = reinterpret_cast<const uint4*>(a.w_unembed + (int64_t)y * a.d);
    const uint4* h0 = reinterpret_cast<const uint4*>(a.hidden + (int64_t)b * n1 * a.d);
    for (int r0 = 0; r0 < n1; r0 += SEL_ZROWS) {
      float acc[SEL_ZROWS];
#pragma unroll
      for (int r = 0; r < SEL_ZROWS; ++r) acc[r] = 0.f;
      for (int i0 = tid; i0 < nv; i0 += 2 * SEL_R_THREADS) {
        uint4 wv[2], hv[2][SEL_ZROWS];
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          const int i = i0 + u * SEL_R_THREADS;
          if (i < nv) wv[u] = __ldg(wy + i);
#pragma unroll
          for (int r = 0; r < SEL_ZROWS; ++r)
            if (i < nv && r0 + r < n1) hv[u][r] = __ldcg(h0 + (int64_t)(r0 + r) * nv + i);
        }
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          if (i0 + u * SEL_R_THREADS >= nv) continue;
          const uint32_t ww[4] = {wv[u].x, wv[u].y, wv[u].z, wv[u].w};
#pragma unroll
          for (int r = 0; r < SEL_ZROWS; ++r) {
            if (r0 + r >= n1) continue;
            const uint32_t hw[4] = {hv[u][r].x, hv[u][r].y, hv[u][r].z, hv[u][r].w};
            float p = 0.f;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              p = fmaf(bf16_lo(hw[q]), bf16_lo(ww[q]), p);
              p = fmaf(bf16_hi(hw[q]), bf16_hi(ww[q]), p);
            }
            acc[r] += p;
          }
        }
      }
#pragma unroll
      for (int r = 0; r < SEL_ZROWS; ++r) {
        const float t = warp_sum(acc[r]);
        if (lane == 0) zpart[warp][r] = t;
      }
      __syncthreads();
      if (tid < SEL_ZROWS && r0 + tid < n1) {
        float z = 0.f;
        for (int w = 0; w < SEL_R_THREADS / 32; ++w) z += zpart[w][tid];
        zy[r0 + tid] = z;
      }
      __syncthreads();
    }
    if (warp == 0) {
      // token gap: the best score at another token, over all experts
      float other = -INFINITY, se_best = -INFINITY, se_other = -INFINITY;
      for (int k = lane; k < N; k += 32) {
        const int sk = b * n1 + 1 + k;
        const float btk = a.beta[b * N + k];
        const float rr = fminf(fmaxf(a.r[b * N + k], 1e-8f), 1.0f);
        const float Lk = __ldcg(a.sel_L + sk);
        const float c = (a.raw_logits ? 0.f : -(1.f + btk) * Lk + btk * L0) + a.gamma * logf(rr);
        const float cand = __ldcg(a.sel_tok + sk) != bt ? __ldcg(a.sel_u + sk) : __ldcg(a.sel_u2 + sk);
        other = fmaxf(other, cand + c);
        // expert gap: every expert's score at the chosen token, from the recomputed logits
        const float se = (1.f + btk) * zy[1 + k] - btk * zy[0] + c;
        if (k == bk) se_best = se;
        else se_other = fmaxf(se_other, se);
      }
      other = warp_max(other);
      se_best = warp_max(se_best);
      se_other = warp_max(se_other);
      gaps = make_float2(bs - other, se_best - se_other);
    }
  }
  if (warp != 0) return;
  if (lane == 0 && a.key_out) {
    // expert-partitioned step: this GPU's best, the reduction over GPUs and
    // the append come after
    a.qdone[b] = 0;
    a.key_out[b] = select_key(bs, bt, a.expert_base + bk + 1);
    return;
  }
  if (lane == 0) {
    a.qdone[b] = 0;
    if (a.token) a.token[b] = bt;
    if (a.expert) a.expert[b] = bk + 1;
    if (a.score) a.score[b] = bs;
    if (a.step) {
      const int t = *a.step;
      if (t >= 0 && t < a.max_steps) {
        a.history[(int64_t)b * a.max_steps + t] = bt;
        if (a.expert_trace) a.expert_trace[(int64_t)b * a.max_steps + t] = bk + 1;
        if (a.score_trace) a.score_trace[(int64_t)b * a.max_steps + t] = bs;
        if (a.gap_trace) a.gap_trace[(int64_t)b * a.max_steps + t] = gaps;
      } else {
        dev_flag(a.status, PCED_DEV_STEP_LIMIT);
      }
      __threadfence();
      if (atomicAdd(a.done_counter, 1) == a.B - 1) {
        if (t >= 0 && t < a.max_steps) *a.step = t + 1;  // at the limit t stays (as the commit does)
        *a.done_counter = 0;
        __threadfence();
      }
    }
  }
}

cudaError_t select_from_records_launch(const SelectArgs& a, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.N + 1, a.B);
  cfg.blockDim = dim3(SEL_R_THREADS);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = a.pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, select_from_records_kernel, a);
}

}  // namespace pced

// ------------------------------------------------------------------ C ABI
using namespace pced;
using namespace pced_host;

extern "C" size_t pced_lm_head_workspace_size(int32_t S, int32_t V) {
  if (S < 1 || V < 1) return 0;
  const int64_t ntiles = (V + LM_TILE_V - 1) / LM_TILE_V;
  Carver c(nullptr);
  c.take<float2>((size_t)(S * ntiles));
  return 256 + c.used();
}

extern "C" pced_status pced_lm_head_logprobs(const void* hidden, const void* w_unembed, int32_t S, int32_t d,
                                             int32_t V, float* logprobs, float* lse, void* workspace,
                                             size_t workspace_bytes, void* stream) {
  if (!hidden || !w_unembed || !logprobs || !lse || !workspace)
    return fail(PCED_ERR_INVALID_ARG, "pced_lm_head_logprobs: null pointer");
  if (S < 1 || d < 1 || V < 1) return fail(PCED_ERR_INVALID_ARG, "pced_lm_head_logprobs: bad sizes");
  LmGeom g;
  if (!lm_geometry(S, d, V, &g) || d > 16384)
    return fail(PCED_ERR_UNSUPPORTED, "pced_lm_head_logprobs: S=%d d=%d (need S<=512, d%%64==0, d<=16384)", S, d);
  if ((((uintptr_t)hidden) | ((uintptr_t)w_unembed)) & 15u)
    return fail(PCED_ERR_INVALID_ARG, "pced_lm_head_logprobs: operands must be 16-byte aligned");
  if (((uintptr_t)workspace) & 255u || workspace_bytes < pced_lm_head_workspace_size(S, V))
    return fail(PCED_ERR_WORKSPACE, "pced_lm_head_logprobs: workspace too small or misaligned");
  if (num_sms() <= 0) return fail(PCED_ERR_NO_DEVICE, "pced_lm_head_logprobs: no CUDA device");
  CUtensorMap wmap, hmap;
  pced_status st = make_tmap_2d(&wmap, w_unembed, (uint64_t)V, (uint64_t)d, LM_TILE_V, LM_TILE_K, true);
  if (st != PCED_OK) return st;
  st = make_tmap_2d(&hmap, hidden, (uint64_t)S, (uint64_t)d, (uint32_t)g.chunk_n, LM_TILE_K, false);
  if (st != PCED_OK) return st;
  Carver cv((char*)workspace + 256);
  LmArgs a = {};
  a.mode = 0;
  a.S = S;
  a.N = 0;
  a.V = V;
  a.ntiles = g.ntiles;
  a.nks = g.nks;
  a.slabs = g.slabs;
  a.nst = g.nst;
  a.stages = g.stages;
  a.acc_bufs = g.acc_bufs;
  a.S_pad = g.S_pad;
  a.nchunk = g.nchunk;
  a.chunk_n = g.chunk_n;
  a.tmem_cols = g.tmem_cols;
  a.logits = logprobs;
  a.rec_stats = cv.take<float2>((size_t)S * g.ntiles);
  a.rec_arg = nullptr;
  a.beta = nullptr;
  a.status = (int*)workspace;
  a.tile_ctr = (int*)workspace + 1;  // tile counter, zeroed here
  cudaStream_t s = (cudaStream_t)stream;
  cudaError_t e = cudaMemsetAsync(a.tile_ctr, 0, sizeof(int), s);
  if (e != cudaSuccess) return cuda_status(e, "lm head tile counter");
  e = lm_head_launch(wmap, hmap, g, a, s);
  if (e != cudaSuccess) return cuda_status(e, "lm head launch");
  e = lm_lse_finalize_launch(logprobs, a.rec_stats, lse, S, V, g.ntiles, s);
  if (e != cudaSuccess) return cuda_status(e, "lse finalize launch");
  return PCED_OK;
}
