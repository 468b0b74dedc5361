// The tcgen05 pipeline shared by the one-shot GEMM kernel (tc_gemm.cu) and
// the persistent drafting kernel (draft_gru.cu).
//
// A "phase" is one batched skinny GEMM: Y[b, o] = sum_k X[b, k] W[o, k] with
// the batch on the MMA's M = 128 (rows past B are never used), weight rows on
// N (n_tile per tile) and K in 64-element chunks with the 128-byte swizzle
// (both operands K-major). Four roles run it, each on its own thread(s):
//
//  * producer (one thread): TMA loads of weight tiles (B operand) and
//    activation tiles (A operand) into a ring of S stages (a stage may hold
//    two consecutive K chunks, the weights' loaded as one 3-D box:
//    b_chunks = 2). Weight tiles do not
//    depend on anything computed earlier, so `prod_prefetch` issues the next
//    phase's first weight stages early (their barriers get the weight bytes as
//    expected transactions; the arrival, with any activation bytes, comes from
//    `prod_run` once the activations exist).
//  * MMA issuer (one thread): tcgen05.mma into double-buffered TMEM
//    accumulators; tcgen05.commit frees stages and publishes accumulators.
//  * logits producer (one thread, combine phases only): TMA loads of the
//    DFlash-logit tile of each vocabulary tile, double-buffered.
//  * epilogue (8 warps): TMEM -> registers; either stores (optionally with an
//    activation, f32 split partials or bf16) or the fused combine.
//  * noise (8 warps, temperature-1 combine launches only): the Gumbel
//    variates of each tile, written to a second pair of TMEM buffers ahead
//    of the epilogue (they depend on nothing computed earlier), so that the
//    epilogue's work per element is that of temperature 0 plus one add.
//
// Every role keeps running counters across phases so mbarrier parities stay
// consistent when one CTA runs many phases (the persistent kernel).
#pragma once

#include "dels_device.cuh"

namespace dels {
namespace tce {

constexpr int kBlockK = 64;                     // bf16 per 128-byte row
constexpr int kUmmaK = 16;
constexpr int kATileBytes = 128 * 128;          // 128 rows x 128 B
constexpr int kEpiWarps = 8;
constexpr int kMaxStages = 12;

// CTA-wide pipeline resources.
struct Ctx {
  uint8_t* sA;              // S activation stages (a_stage_bytes apart); also the resident-A area
  uint8_t* sB;              // S weight stage tiles
  uint8_t* sL;              // 2 DFlash-logit tiles
  float* sP;                // prior slice of this CTA's vocabulary range
  RowAcc* red;              // [256] epilogue merge scratch
  float* tr;                // [8 warps][32][33] store transpose scratch (EPI_STORE), or null
  uint64_t* full;           // [S]
  uint64_t* empty;          // [S]
  uint64_t* accf;           // [2]
  uint64_t* acce;           // [2]
  uint64_t* lfull;          // [2]
  uint64_t* lempty;         // [2]
  uint64_t* afull;          // [1] resident activations
  uint64_t* nfull;          // [2] noise buffers written (temperature-1 launches)
  uint64_t* nempty;         // [2] noise buffers read
  uint32_t noise_col;       // TMEM column of noise buffer 0 (buffer 1 follows at n_tile)
  uint32_t tmem_base;
  int S;
  uint32_t a_stage_bytes;   // pitch of the activation stages (>= the rows actually loaded; the MMA
                            // reads 128 rows from each, rows past the loaded ones feed unused outputs)
  uint32_t b_stage_bytes;   // bytes reserved per weight stage
  uint32_t l_buf_bytes;     // bytes reserved per logits tile
  volatile int* abort_flag;
  uint64_t deadline;
};

// One phase as seen by this CTA.
struct Phase {
  const TcGemmArgs* a;
  const CUtensorMap* mA0;
  const CUtensorMap* mB0;
  const CUtensorMap* mA1;
  const CUtensorMap* mB1;
  const CUtensorMap* mL;
  int first, count, stride;  // this CTA's items
  int j;                     // block position (combine: coordinate into the DFlash-logit map)
};

// An item is one output tile over one K range. Its chunks are visited in a
// rotated order (starting at chunk `rot` of the range) so that the CTAs that
// share a K range — and so read the same activation chunks — do not all
// request the same lines of L2 at the same moment.
struct Item {
  int o0, seg, kb, ke, split, rot;
  __device__ __forceinline__ int chunk(int i) const {
    const int len = ke - kb;
    const int r = i + rot;
    return kb + (r >= len ? r - len : r);
  }
};

__device__ __forceinline__ Item get_item(const TcGemmArgs& a, int i) {
  Item it;
  const int ot = i % a.num_o_tiles;
  it.split = i / a.num_o_tiles;
  it.o0 = ot * a.n_tile;
  it.seg = (it.split < a.seg_splits[0]) ? 0 : 1;
  const int ls = it.seg ? it.split - a.seg_splits[0] : it.split;
  const int nch = a.seg_chunks[it.seg];
  const int ns = a.seg_splits[it.seg];
  const int per = (nch + ns - 1) / ns;
  it.kb = ls * per;
  it.ke = min(nch, it.kb + per);
  const int len = it.ke - it.kb;
  // two chunks per stage: the rotation keeps pairs of consecutive chunks
  if (a.b_chunks == 2)
    it.rot = len >= 2 ? (ot % (len >> 1)) * 2 : 0;
  else
    it.rot = len > 0 ? ot % len : 0;
  return it;
}

// Items of CTA `cta` of `ncta`: a contiguous range for the combine (one
// RowAcc per CTA covers them all), a strided set otherwise.
__device__ __forceinline__ void item_range(const TcGemmArgs& a, int cta, int ncta, int& first, int& count,
                                           int& stride) {
  const int total = a.num_o_tiles * a.total_splits;
  if (a.cluster_k > 1) {
    // one item per CTA: the tile is the cluster's index, the K split its rank
    const int ck = a.cluster_k;
    first = (cta % ck) * a.num_o_tiles + cta / ck;
    count = (cta / ck < a.num_o_tiles && cta % ck < a.total_splits) ? 1 : 0;
    stride = ncta;
    return;
  }
  if (a.epi == EPI_COMBINE) {
    const long long lo = (long long)cta * total / ncta;
    const long long hi = (long long)(cta + 1) * total / ncta;
    first = (int)lo;
    count = (int)(hi - lo);
    stride = 1;
  } else {
    first = cta;
    count = (cta < total) ? (total - 1 - cta) / ncta + 1 : 0;
    stride = ncta;
  }
}

// Activation of a 32-value accumulator chunk. The branch sits outside the
// unrolled loops: inside them the compiler predicates every activation's
// arithmetic for every value, which costs microseconds per tile.
__device__ __forceinline__ void act_apply32(int act, float (&x)[32]) {
  if (act == ACT_SILU) {
#pragma unroll
    for (int i = 0; i < 32; ++i) x[i] = __fdividef(x[i], 1.f + __expf(-x[i]));
  } else if (act == ACT_GELU) {
#pragma unroll
    for (int i = 0; i < 32; ++i) x[i] = 0.5f * x[i] * (1.f + erff(x[i] * 0.70710678118654752f));
  }
}

// ------------------------------------------------------------------ producer

struct ProdState {
  int fills = 0;      // stage fills completed (arrived)
  int pre_end = 0;    // fills [fills, pre_end) have their weights in flight, arrival pending
  int afull_uses = 0;
};

// Weights of the stage that starts at visit index i of the item: one 2-D box
// (one K chunk), or one 3-D box of C consecutive K chunks.
template <int C>
__device__ __forceinline__ void load_w(const Ctx& c, const Phase& p, const Item& it, int i, int s, uint64_t pol_w) {
  const CUtensorMap* mB = it.seg ? p.mB1 : p.mB0;
  if constexpr (C > 1)
    tma_load_3d(c.sB + s * c.b_stage_bytes, mB, &c.full[s], 0, it.o0, it.chunk(i), pol_w);
  else
    tma_load_2d(c.sB + s * c.b_stage_bytes, mB, &c.full[s], it.chunk(i) * kBlockK, it.o0, pol_w);
}

// Issue the weight tiles of the phase's first stages (up to S) ahead of the
// activations. Only waits for stages freed by already-issued MMAs.
template <int C>
__device__ __forceinline__ bool prod_prefetch_c(const Ctx& c, const Phase& p, ProdState& st, uint64_t pol_w) {
  const TcGemmArgs& a = *p.a;
  const uint32_t b_bytes = (uint32_t)a.n_tile * 128u * (uint32_t)C;
  int f = max(st.fills, st.pre_end);
  int t = 0;
  int done = f - st.fills;   // stages already prefetched for this phase
  // skip the chunks already prefetched
  Item it = p.count > 0 ? get_item(a, p.first) : Item{0, 0, 0, 0, 0, 0};
  int i = 0;   // chunk index within the item (visit order)
  for (int skip = done; skip > 0 && t < p.count;) {
    if (i >= it.ke - it.kb) {
      if (++t >= p.count) break;
      it = get_item(a, p.first + t * p.stride);
      i = 0;
      continue;
    }
    i += C;
    --skip;
  }
  while (f - st.fills < c.S && t < p.count) {
    if (i >= it.ke - it.kb) {
      if (++t >= p.count) break;
      it = get_item(a, p.first + t * p.stride);
      i = 0;
      continue;
    }
    const int s = f % c.S;
    if (!mbar_wait(&c.empty[s], ((f / c.S) & 1) ^ 1, c.deadline, c.abort_flag)) return false;
    mbar_expect_tx(&c.full[s], b_bytes);
    load_w<C>(c, p, it, i, s, pol_w);
    ++f;
    i += C;
  }
  st.pre_end = f;
  return true;
}
__device__ __forceinline__ bool prod_prefetch(const Ctx& c, const Phase& p, ProdState& st, uint64_t pol_w) {
  return p.a->b_chunks == 2 ? prod_prefetch_c<2>(c, p, st, pol_w) : prod_prefetch_c<1>(c, p, st, pol_w);
}

// Load the activations (and the remaining weights) of the phase.
template <int C>
__device__ __forceinline__ bool prod_run_c(const Ctx& c, const Phase& p, ProdState& st, uint64_t pol_w,
                                           uint64_t pol_act) {
  const TcGemmArgs& a = *p.a;
  const uint32_t b_bytes = (uint32_t)a.n_tile * 128u * (uint32_t)C;
  const uint32_t a_copy_bytes = (uint32_t)a.a_box_rows * 128u;
  const uint32_t a_bytes = a_copy_bytes * (uint32_t)a.a_copies;
  if (a.a_resident && p.count > 0) {
    // every CTA loads the same activations here: start at a CTA-dependent chunk
    const int nch = a.seg_chunks[0];
    mbar_arrive_expect_tx(c.afull, (uint32_t)nch * a_bytes);
    for (int i = 0; i < nch; ++i) {
      const int ch = (i + (int)blockIdx.x) % nch;
      for (int cp = 0; cp < a.a_copies; ++cp)
        tma_load_2d(c.sA + ch * kATileBytes + cp * a_copy_bytes, p.mA0, c.afull, ch * kBlockK, 0, pol_act);
    }
    ++st.afull_uses;
  }
  int f = st.fills;
  for (int t = 0; t < p.count; ++t) {
    const Item it = get_item(a, p.first + t * p.stride);
    const CUtensorMap* mA = it.seg ? p.mA1 : p.mA0;
    for (int i = 0; i < it.ke - it.kb; i += C, ++f) {
      const int kc = it.chunk(i);
      const int s = f % c.S;
      // staged activations: chunk kc + cc of the stage at sA + s * a_stage_bytes + cc * kATileBytes
      if (f < st.pre_end) {
        if (a.a_resident) {
          mbar_arrive(&c.full[s]);
        } else {
          mbar_arrive_expect_tx(&c.full[s], (uint32_t)C * a_bytes);
#pragma unroll
          for (int cc = 0; cc < C; ++cc)
            for (int cp = 0; cp < a.a_copies; ++cp)
              tma_load_2d(c.sA + s * c.a_stage_bytes + cc * kATileBytes + cp * a_copy_bytes, mA, &c.full[s],
                          (kc + cc) * kBlockK, 0, pol_act);
        }
        continue;
      }
      if (!mbar_wait(&c.empty[s], ((f / c.S) & 1) ^ 1, c.deadline, c.abort_flag)) {
        st.fills = f;
        return false;
      }
      mbar_arrive_expect_tx(&c.full[s], b_bytes + (a.a_resident ? 0u : (uint32_t)C * a_bytes));
      if (!a.a_resident) {
#pragma unroll
        for (int cc = 0; cc < C; ++cc)
          for (int cp = 0; cp < a.a_copies; ++cp)
            tma_load_2d(c.sA + s * c.a_stage_bytes + cc * kATileBytes + cp * a_copy_bytes, mA, &c.full[s],
                        (kc + cc) * kBlockK, 0, pol_act);
      }
      load_w<C>(c, p, it, i, s, pol_w);
    }
  }
  st.fills = f;
  st.pre_end = max(st.pre_end, f);
  return true;
}
__device__ __forceinline__ bool prod_run(const Ctx& c, const Phase& p, ProdState& st, uint64_t pol_w,
                                         uint64_t pol_act) {
  return p.a->b_chunks == 2 ? prod_run_c<2>(c, p, st, pol_w, pol_act) : prod_run_c<1>(c, p, st, pol_w, pol_act);
}

// ------------------------------------------------------------- logits producer

struct LState {
  int tiles = 0;      // logits tiles issued
  int pre = 0;        // tiles of the current phase already issued ahead
};

// Issue up to `max_tiles` logits tiles of the phase (continuing after the
// `st.pre` already issued for it). Waits only for buffers freed by the epilogue.
__device__ __forceinline__ bool lprod_issue(const Ctx& c, const Phase& p, LState& st, int max_tiles,
                                            uint64_t pol_stream) {
  const TcGemmArgs& a = *p.a;
  const uint32_t box_bytes = (uint32_t)a.l_box_rows * 128u;
  const uint32_t tile_bytes = box_bytes * (uint32_t)a.l_boxes;
  int issued = 0;
  for (int t = st.pre; t < p.count && issued < max_tiles; ++t, ++issued) {
    const Item it = get_item(a, p.first + t * p.stride);
    const int buf = st.tiles & 1;
    if (!mbar_wait(&c.lempty[buf], ((st.tiles >> 1) & 1) ^ 1, c.deadline, c.abort_flag)) return false;
    mbar_arrive_expect_tx(&c.lfull[buf], tile_bytes);
    for (int bx = 0; bx < a.l_boxes; ++bx)
      tma_load_3d(c.sL + buf * c.l_buf_bytes + bx * box_bytes, p.mL, &c.lfull[buf], it.o0 + bx * a.l_box_cols, p.j,
                  0, pol_stream);
    ++st.tiles;
  }
  st.pre += issued;
  return true;
}

// ------------------------------------------------------------------- MMA

struct MmaState {
  int fills = 0;
  int tiles = 0;
  int afull_uses = 0;
};

template <int C>
__device__ __forceinline__ bool mma_run_c(const Ctx& c, const Phase& p, MmaState& st) {
  const TcGemmArgs& a = *p.a;
  const uint32_t idesc = idesc_bf16_f32(128, a.n_tile);
  if (a.a_resident && p.count > 0) {
    if (!mbar_wait(c.afull, st.afull_uses & 1, c.deadline, c.abort_flag)) return false;
    ++st.afull_uses;
  }
  for (int t = 0; t < p.count; ++t) {
    const Item it = get_item(a, p.first + t * p.stride);
    const int buf = st.tiles & 1;
    if (!mbar_wait(&c.acce[buf], ((st.tiles >> 1) & 1) ^ 1, c.deadline, c.abort_flag)) return false;
    tc_fence_after();
    const uint32_t d_tmem = c.tmem_base + (uint32_t)(buf * a.n_tile);
    for (int i = 0; i < it.ke - it.kb; i += C, ++st.fills) {
      const int s = st.fills % c.S;
      if (!mbar_wait(&c.full[s], (st.fills / c.S) & 1, c.deadline, c.abort_flag)) return false;
      tc_fence_after();
#pragma unroll
      for (int cc = 0; cc < C; ++cc) {
        const int kc = it.chunk(i + cc);
        const uint32_t a_addr =
            smem_u32(a.a_resident ? c.sA + kc * kATileBytes : c.sA + s * c.a_stage_bytes + cc * kATileBytes);
        const uint32_t b_addr = smem_u32(c.sB + s * c.b_stage_bytes + cc * a.n_tile * 128);
#pragma unroll
        for (int kk = 0; kk < kBlockK / kUmmaK; ++kk) {
          tc_mma_f16(d_tmem, smem_desc_sw128(a_addr + kk * kUmmaK * 2), smem_desc_sw128(b_addr + kk * kUmmaK * 2),
                     idesc, (i > 0 || cc > 0 || kk > 0) ? 1u : 0u);
        }
      }
      tc_commit(&c.empty[s]);
    }
    tc_commit(&c.accf[buf]);
    ++st.tiles;
  }
  return true;
}
__device__ __forceinline__ bool mma_run(const Ctx& c, const Phase& p, MmaState& st) {
  return p.a->b_chunks == 2 ? mma_run_c<2>(c, p, st) : mma_run_c<1>(c, p, st);
}

// ----------------------------------------------------------------- epilogue

// One 32-column chunk of the combine epilogue: fused = l_L + alpha*acc - beta*prior,
// then top-1/top-2 and the online log-sum-exp. `lrow` is this row's 128-byte
// line of the logits box holding the chunk, `half` selects the chunk's
// 64-byte half (bf16) and `ptile` the prior of the chunk's columns.
template <bool KEYS = false>
__device__ __forceinline__ void combine_chunk(const float (&acc)[32], const uint8_t* lrow, int half, int swz,
                                              bool long_f32, const float* ptile, int cbase, int V, float alpha,
                                              float nbeta, float& best, float& second, int& idx, float& m,
                                              float& ssum, const float (&g)[32]) {
  float f[32];
  if (!long_f32) {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const uint4 w = *reinterpret_cast<const uint4*>(lrow + (((half * 4 + k) ^ swz) << 4));
      const float4 p0 = *reinterpret_cast<const float4*>(ptile + k * 8);
      const float4 p1 = *reinterpret_cast<const float4*>(ptile + k * 8 + 4);
      f[k * 8 + 0] = fmaf(nbeta, p0.x, fmaf(alpha, acc[k * 8 + 0], bf16lo(w.x)));
      f[k * 8 + 1] = fmaf(nbeta, p0.y, fmaf(alpha, acc[k * 8 + 1], bf16hi(w.x)));
      f[k * 8 + 2] = fmaf(nbeta, p0.z, fmaf(alpha, acc[k * 8 + 2], bf16lo(w.y)));
      f[k * 8 + 3] = fmaf(nbeta, p0.w, fmaf(alpha, acc[k * 8 + 3], bf16hi(w.y)));
      f[k * 8 + 4] = fmaf(nbeta, p1.x, fmaf(alpha, acc[k * 8 + 4], bf16lo(w.z)));
      f[k * 8 + 5] = fmaf(nbeta, p1.y, fmaf(alpha, acc[k * 8 + 5], bf16hi(w.z)));
      f[k * 8 + 6] = fmaf(nbeta, p1.z, fmaf(alpha, acc[k * 8 + 6], bf16lo(w.w)));
      f[k * 8 + 7] = fmaf(nbeta, p1.w, fmaf(alpha, acc[k * 8 + 7], bf16hi(w.w)));
    }
  } else {
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const float4 w = *reinterpret_cast<const float4*>(lrow + ((k ^ swz) << 4));
      const float4 p = *reinterpret_cast<const float4*>(ptile + k * 4);
      f[k * 4 + 0] = fmaf(nbeta, p.x, fmaf(alpha, acc[k * 4 + 0], w.x));
      f[k * 4 + 1] = fmaf(nbeta, p.y, fmaf(alpha, acc[k * 4 + 1], w.y));
      f[k * 4 + 2] = fmaf(nbeta, p.z, fmaf(alpha, acc[k * 4 + 2], w.z));
      f[k * 4 + 3] = fmaf(nbeta, p.w, fmaf(alpha, acc[k * 4 + 3], w.w));
    }
  }
  if (cbase + 32 > V) {
#pragma unroll
    for (int i = 0; i < 32; ++i)
      if (cbase + i >= V) f[i] = -INFINITY;
  }
  if constexpr (KEYS) {
    // temperature 1: the top-2 over the keys f + g (g: the Gumbel variates);
    // keys at or below the runner-up change neither the top-1 nor the top-2
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      float k[8], km = -INFINITY;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        k[i] = f[t * 8 + i] + g[t * 8 + i];
        km = fmaxf(km, k[i]);
      }
      if (km > second) {
#pragma unroll
        for (int i = 0; i < 8; ++i) top2_push(k[i], cbase + t * 8 + i, best, second, idx);
      }
    }
  } else {
#pragma unroll
    for (int i = 0; i < 32; ++i) top2_push(f[i], cbase + i, best, second, idx);
  }
  lse_chunk_ex2<32>(f, best, m, ssum);
}

struct EpiState {
  int tiles = 0;      // accumulator tiles consumed
  int ltiles = 0;     // logits tiles consumed
  int ntiles = 0;     // noise tiles consumed (temperature 1)
};

// The epilogue's quadrant / copy / worker mapping of a combine phase (see
// epi_run): the noise warps write exactly the values the epilogue reads.
struct EpiMap {
  int q, qpc, cpy, b, workers, quad_live;
};
__device__ __forceinline__ EpiMap epi_map(const TcGemmArgs& a, int warp, int lane) {
  EpiMap m;
  m.q = warp & 3;
  m.qpc = (a.a_box_rows + 31) / 32;
  m.cpy = m.q / m.qpc;
  m.b = (m.q % m.qpc) * 32 + lane;
  m.workers = 2 * a.a_copies;
  m.quad_live = m.cpy < a.a_copies && ((m.q % m.qpc) * 32) < a.B;
  return m;
}

// Noise warp of TMEM lane quadrant warp % 4 (temperature-1 combine phases;
// two per quadrant, g = 0, 1): for every tile of the phase, the Gumbel
// variates of the columns that epilogue warp g of the quadrant combines,
// written to noise buffer (tile & 1) once the epilogue has released it.
__device__ __forceinline__ bool noise_run(const Ctx& c, const Phase& p, int warp, int lane, int g) {
  const TcGemmArgs& a = *p.a;
  const EpiMap mp = epi_map(a, warp, lane);
  const int nchunk = a.n_tile / 32;
  for (int t = 0; t < p.count; ++t) {
    const Item it = get_item(a, p.first + t * p.stride);
    const int nb = t & 1;
    if (!mbar_wait(&c.nempty[nb], ((t >> 1) & 1) ^ 1, c.deadline, c.abort_flag)) return false;
    tc_fence_after();
    if (mp.quad_live) {
      const uint32_t base = c.tmem_base + ((uint32_t)(mp.q * 32) << 16) + c.noise_col + (uint32_t)(nb * a.n_tile);
      {
#pragma unroll 1
        for (int cc = mp.cpy * 2 + g; cc < nchunk; cc += mp.workers) {
#pragma unroll 1
          for (int grp = 0; grp < 4; ++grp) {
            float gv[8];
            gumbel8(a.seed, a.step, mp.b, a.j, kStreamDraft, ((it.o0 + cc * 32) >> 3) + grp, gv);
            tmem_st_32x32b_x8(base + (uint32_t)(cc * 32 + grp * 8), gv);
          }
        }
      }
      tmem_st_wait();
    }
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(&c.nfull[nb]);
  }
  return true;
}

// Stage the prior of this CTA's vocabulary range for a combine phase
// (called by the 256 epilogue threads; ends with an epilogue-only barrier).
__device__ __forceinline__ void epi_stage_prior(const Ctx& c, const Phase& p, int ep) {
  const TcGemmArgs& a = *p.a;
  const int n = p.count * a.n_tile;
  const int v0 = p.first * a.n_tile;
  for (int i = ep; i < n; i += kEpiWarps * 32) {
    const int v = v0 + i;
    c.sP[i] = v < a.V ? __ldg(a.prior + v) : 0.f;
  }
  named_bar_sync<2>(kEpiWarps * 32);
}

// Epilogue of one phase; `warp` is the CTA warp index (2..9), `cta` the
// index under which combine partials are published.
// COMB: the phase is a combine phase (EPI_COMBINE); a compile-time flag so
// that a store-only kernel carries none of the combine's registers.
template <bool COMB, bool SAMPLE = false>
__device__ __forceinline__ bool epi_run(const Ctx& c, const Phase& p, EpiState& st, int warp, int lane, int cta) {
  const TcGemmArgs& a = *p.a;
  constexpr bool comb = COMB;
  const int q = warp & 3;                      // TMEM lane quadrant
  const int g = (warp - 2) >> 2;               // column-chunk parity
  const int nchunk = a.n_tile / 32;
  // The A tile holds a_copies stacked copies of the activation rows (each
  // a_box_rows rows, a multiple of 32 for the combine): quadrant q holds copy
  // cpy, rows 32*(q % qpc)..; the copies split the tile's 32-column chunks
  // between them, so every row's columns are covered exactly once.
  const int qpc = comb ? (a.a_box_rows + 31) / 32 : 4;
  const int cpy = q / qpc;
  const int b = (q % qpc) * 32 + lane;
  const int workers = 2 * (comb ? a.a_copies : 1);
  const int worker = (comb ? cpy : 0) * 2 + g;
  const bool quad_live = (comb ? cpy < a.a_copies : true) && ((q % qpc) * 32) < a.B;
  float best = -INFINITY, second = -INFINITY, m = -INFINITY, ssum = 0.f;
  int idx = 0x7FFFFFFF;
  const float alpha = a.alpha, nbeta = -a.beta;
  const int br = comb ? min(b, a.l_box_rows - 1) : 0;   // logits-box rows past B are never used
  const int swz = br & 7;
  const uint32_t box_bytes = (uint32_t)a.l_box_rows * 128u;
  bool ok = true;
  for (int t = 0; t < p.count; ++t) {
    const Item it = get_item(a, p.first + t * p.stride);
    const int buf = st.tiles & 1;
    ok = mbar_wait(&c.accf[buf], (st.tiles >> 1) & 1, c.deadline, c.abort_flag);
    if (!ok) break;
    tc_fence_after();
    const int lbuf_i = st.ltiles & 1;
    if (comb) {
      ok = mbar_wait(&c.lfull[lbuf_i], (st.ltiles >> 1) & 1, c.deadline, c.abort_flag);
      if (!ok) break;
    }
    const uint32_t tbase = c.tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * a.n_tile);
    const int nbuf = st.ntiles & 1;
    if constexpr (SAMPLE) {
      ok = mbar_wait(&c.nfull[nbuf], (st.ntiles >> 1) & 1, c.deadline, c.abort_flag);
      if (!ok) break;
      tc_fence_after();
    }
    const uint32_t gbase = c.tmem_base + ((uint32_t)(q * 32) << 16) + c.noise_col + (uint32_t)(nbuf * a.n_tile);
    if (quad_live && comb) {
      const uint8_t* lbuf = c.sL + lbuf_i * c.l_buf_bytes;
      const float* ptile = c.sP + t * a.n_tile;
      const int c0 = worker, c1 = worker + workers;
      auto run_chunk = [&](const float (&acc)[32], int cc) {
        if (!a.long_f32) {
          // bf16 boxes of 64 columns: chunk cc is half (cc & 1) of box (cc >> 1)
          combine_chunk(acc, lbuf + (cc >> 1) * box_bytes + br * 128, cc & 1, swz, false, ptile + cc * 32,
                        it.o0 + cc * 32, a.V, alpha, nbeta, best, second, idx, m, ssum, acc);
        } else {
          // f32 boxes of 32 columns: chunk cc is box cc
          combine_chunk(acc, lbuf + cc * box_bytes + br * 128, 0, swz, true, ptile + cc * 32,
                        it.o0 + cc * 32, a.V, alpha, nbeta, best, second, idx, m, ssum, acc);
        }
      };
      if constexpr (SAMPLE) {
#pragma unroll 1
        for (int cc = c0; cc < nchunk; cc += workers) {
          float acc[32], g[32];
          tmem_ld_32x32b_x32(tbase + (uint32_t)(cc * 32), acc);
          tmem_ld_32x32b_x32(gbase + (uint32_t)(cc * 32), g);
          tmem_ld_wait();
          if (!a.long_f32)
            combine_chunk<true>(acc, lbuf + (cc >> 1) * box_bytes + br * 128, cc & 1, swz, false, ptile + cc * 32,
                                it.o0 + cc * 32, a.V, alpha, nbeta, best, second, idx, m, ssum, g);
          else
            combine_chunk<true>(acc, lbuf + cc * box_bytes + br * 128, 0, swz, true, ptile + cc * 32,
                                it.o0 + cc * 32, a.V, alpha, nbeta, best, second, idx, m, ssum, g);
        }
      } else {
        // one call site per type: the unrolled chunk is large, and more
        // copies of it cost instruction-cache misses
#pragma unroll 1
        for (int cc = c0; cc < nchunk; cc += workers) {
          float acc0[32];
          tmem_ld_32x32b_x32(tbase + (uint32_t)(cc * 32), acc0);
          tmem_ld_wait();
          run_chunk(acc0, cc);
        }
      }
    } else if (quad_live) {
      for (int cc = g; cc < nchunk; cc += 2) {
        float acc[32];
        tmem_ld_32x32b_x32(tbase + (uint32_t)(cc * 32), acc);
        tmem_ld_wait();
        const int cbase = it.o0 + cc * 32;
        if (a.act != ACT_NONE) act_apply32(a.act, acc);
        if (a.out_f32 && !a.out_bmajor && c.tr && !a.out_bf16) {
          // f32 rows through a shared-memory transpose (all lanes of the
          // warp take part): each store instruction then writes 32
          // consecutive outputs of one row, one 128-byte line
          float* tr = c.tr + (warp - 2) * 32 * 33;
#pragma unroll
          for (int i = 0; i < 32; ++i) tr[lane * 33 + i] = acc[i];
          __syncwarp();
          const int r0 = b - lane;
          const int rows = min(32, a.B - r0);
          float* dst = a.out_f32 + (long long)it.split * a.out_split_stride + cbase + lane;
          if (cbase + lane < a.O)
            for (int r = 0; r < rows; ++r) dst[(long long)(r0 + r) * a.ldo] = tr[r * 33 + lane];
          __syncwarp();
        } else if (b < a.B) {
          if (a.out_f32 && a.out_bmajor) {
            // column-by-column: the warp's 32 rows are 32 consecutive floats
            float* dst = a.out_f32 + (long long)it.split * a.out_split_stride + (long long)cbase * a.ldb + b;
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (cbase + i < a.O) dst[(long long)i * a.ldb] = acc[i];
          } else if (a.out_f32) {
            float* dst = a.out_f32 + (long long)it.split * a.out_split_stride + (long long)b * a.ldo + cbase;
            if (cbase + 32 <= a.O && (a.ldo & 3) == 0) {
#pragma unroll
              for (int k = 0; k < 8; ++k)
                reinterpret_cast<float4*>(dst)[k] =
                    make_float4(acc[k * 4 + 0], acc[k * 4 + 1], acc[k * 4 + 2], acc[k * 4 + 3]);
            } else {
              for (int i = 0; i < 32; ++i)
                if (cbase + i < a.O) dst[i] = acc[i];
            }
          }
          if (a.out_bf16) {
            uint16_t* dst = a.out_bf16 + (long long)b * a.ldo_bf16 + cbase;
            if (cbase + 32 <= a.O && (a.ldo_bf16 & 7) == 0) {
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                uint4 w;
                w.x = (uint32_t)f32_to_bf16_rne(acc[k * 8 + 0]) | ((uint32_t)f32_to_bf16_rne(acc[k * 8 + 1]) << 16);
                w.y = (uint32_t)f32_to_bf16_rne(acc[k * 8 + 2]) | ((uint32_t)f32_to_bf16_rne(acc[k * 8 + 3]) << 16);
                w.z = (uint32_t)f32_to_bf16_rne(acc[k * 8 + 4]) | ((uint32_t)f32_to_bf16_rne(acc[k * 8 + 5]) << 16);
                w.w = (uint32_t)f32_to_bf16_rne(acc[k * 8 + 6]) | ((uint32_t)f32_to_bf16_rne(acc[k * 8 + 7]) << 16);
                reinterpret_cast<uint4*>(dst)[k] = w;
              }
            } else {
              for (int i = 0; i < 32; ++i)
                if (cbase + i < a.O) dst[i] = f32_to_bf16_rne(acc[i]);
            }
          }
        }
      }
    }
    tc_fence_before();
    __syncwarp();
    if (lane == 0) {
      mbar_arrive(&c.acce[buf]);
      if (comb) mbar_arrive(&c.lempty[lbuf_i]);
      if (SAMPLE) mbar_arrive(&c.nempty[nbuf]);
    }
    ++st.tiles;
    if (comb) ++st.ltiles;
    if (SAMPLE) ++st.ntiles;
  }
  if (comb) {
    // merge the workers' states of each row, publish one record per request
    const int rpc = qpc * 32;
    if (quad_live) {
      RowAcc mine;
      mine.m = best; mine.s = ssum; mine.second = second; mine.idx = idx;
      c.red[worker * rpc + b] = mine;
    }
    named_bar_sync<1>(kEpiWarps * 32);
    if (worker == 0 && quad_live && b < a.B && !*c.abort_flag) {
      RowAcc r = rowacc_init();
      if (p.count > 0)
        for (int w = 0; w < workers; ++w) r = rowacc_merge(r, c.red[w * rpc + b]);
      reinterpret_cast<float4*>(a.partials)[(long long)b * a.partial_ld + cta] =
          make_float4(r.m, r.s, r.second, __int_as_float(r.idx));
    }
    named_bar_sync<1>(kEpiWarps * 32);   // red[] is reused by the next phase
  }
  return ok;
}

}  // namespace tce
}  // namespace dels
