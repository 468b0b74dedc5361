// tcgen05 batched skinny GEMM for sm_103a, with two epilogues:
//
//  * EPI_COMBINE — the vocabulary projection l_S = W_vocab r of Appendix A,
//    fused with the Section 4.3 combine: each tile of vocabulary rows is
//    multiplied on the tensor cores into TMEM, then the epilogue adds the
//    DFlash logits (a TMA-loaded tile of l_L[:, j, :]) and the prior term
//    (staged once per CTA in shared memory), and folds the fused values into
//    per-row top-1/top-2/online-LSE state. Only one 16-byte record per
//    (CTA, request) leaves the kernel; the [B, V] short and fused logits are
//    never written.
//  * EPI_STORE — Y[b, o] = act(sum_k X[b, k] W[o, k]) for the local-head
//    products (GRU input/recurrent gates, low-rank projection, MLP and
//    transformer layers), optionally split over K with f32 partial outputs.
//
// Layout: the batch is the MMA's M dimension (M = 128; rows >= B are
// zero-filled by TMA out-of-bounds handling), weight rows are N (n_tile per
// tile), K is streamed in 64-element (128-byte) chunks with the 128-byte
// swizzle. Both operands are K-major, so one 128B-swizzled smem descriptor
// form serves A and B. Accumulators are double-buffered in TMEM so the
// epilogue of tile t overlaps the MMAs of tile t+1.
//
// Warp roles (352 threads): warp 0 = weight/activation TMA producer,
// warp 1 = MMA issuer and TMEM owner, warps 2..9 = epilogue (warp w reads
// TMEM lanes 32*(w%4)..+31, i.e. batch rows 32*(w%4)..+31, and the 32-column
// chunks c with c % 2 == (w-2)/4), warp 10 = DFlash-logit tile producer.
//
// Programmatic dependent launch: the kernel lets its successor launch at
// once, and before waiting for its own predecessor it already allocates TMEM,
// stages the prior, starts the DFlash-logit tiles and the first weight
// stages — everything that does not depend on the previous kernel.
#include <algorithm>

#include "dels_device.cuh"

namespace dels {

namespace {

constexpr int kWarps = 11;
constexpr int kThreads = kWarps * 32;
constexpr int kEpiWarps = 8;
constexpr int kLWarp = 10;
constexpr int kBlockK = 64;                     // bf16 per 128-byte row
constexpr int kUmmaK = 16;
constexpr int kATileBytes = 128 * 128;          // 128 rows x 128 B
constexpr int kMaxStages = 12;

struct Smem {
  uint32_t a_off, b_off, l_off, p_off, bar_off, red_off, total;
  int a_tiles;
};

__host__ __device__ inline Smem smem_layout(const TcGemmArgs& a) {
  Smem s{};
  const int b_tile = a.n_tile * 128;
  const bool comb = a.epi == EPI_COMBINE;
  const int l_tile = comb ? a.l_boxes * a.l_box_rows * 128 : 0;
  s.a_tiles = a.a_resident ? a.seg_chunks[0] : a.stages;
  uint32_t off = 0;
  s.a_off = off;
  off += (uint32_t)s.a_tiles * kATileBytes;
  s.b_off = off;
  off += (uint32_t)a.stages * b_tile;
  s.l_off = off;
  off += 2u * l_tile;
  s.p_off = off;
  off += comb ? (uint32_t)a.max_items_per_cta * a.n_tile * 4 : 0;
  off = (off + 15) / 16 * 16;
  s.bar_off = off;
  off += 64 * 8;                                  // mbarriers + tmem slot + flags
  s.red_off = off;
  off += comb ? 2 * 128 * 16 : 0;
  s.total = off + 1024;                           // slack for 1024-byte alignment
  return s;
}

struct Item {
  int o0, seg, kb, ke, split;
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
  return it;
}

// Items of this CTA: a contiguous range for the combine (one RowAcc per CTA
// covers them all), a strided set otherwise.
__device__ __forceinline__ void item_range(const TcGemmArgs& a, int& first, int& count, int& stride) {
  const int total = a.num_o_tiles * a.total_splits;
  if (a.epi == EPI_COMBINE) {
    const long long lo = (long long)blockIdx.x * total / gridDim.x;
    const long long hi = (long long)(blockIdx.x + 1) * total / gridDim.x;
    first = (int)lo;
    count = (int)(hi - lo);
    stride = 1;
  } else {
    first = blockIdx.x;
    count = (blockIdx.x < total) ? (total - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;
    stride = gridDim.x;
  }
}

__device__ __forceinline__ float act_apply(int act, float x) {
  if (act == ACT_SILU) return x / (1.f + __expf(-x));
  if (act == ACT_GELU) return 0.5f * x * (1.f + erff(x * 0.70710678118654752f));
  return x;
}

// One 32-column chunk of the combine epilogue: fused = l_L + alpha*acc - beta*prior,
// then top-1/top-2 and the online log-sum-exp. `lrow` is this row's 128-byte
// line of the logits box holding the chunk, `half` selects the chunk's
// 64-byte half (bf16) and `ptile` the prior of the chunk's columns.
__device__ __forceinline__ void combine_chunk(const float (&acc)[32], const uint8_t* lrow, int half, int swz,
                                              bool long_f32, const float* ptile, int cbase, int V, float alpha,
                                              float nbeta, float& best, float& second, int& idx, float& m,
                                              float& ssum) {
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
#pragma unroll
  for (int i = 0; i < 32; ++i) top2_push(f[i], cbase + i, best, second, idx);
  lse_chunk_ex2<32>(f, best, m, ssum);
}

__global__ void __launch_bounds__(kThreads, 1)
    k_tc_gemm(const __grid_constant__ CUtensorMap mA0, const __grid_constant__ CUtensorMap mB0,
              const __grid_constant__ CUtensorMap mA1, const __grid_constant__ CUtensorMap mB1,
              const __grid_constant__ CUtensorMap mL, const TcGemmArgs a, uint64_t budget_ns) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  const Smem lay = smem_layout(a);

  uint8_t* sA = smem + lay.a_off;
  uint8_t* sB = smem + lay.b_off;
  uint8_t* sL = smem + lay.l_off;
  float* sP = reinterpret_cast<float*>(smem + lay.p_off);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + lay.bar_off);
  uint64_t* full = bars;                       // [stages]
  uint64_t* empty = bars + kMaxStages;         // [stages]
  uint64_t* accf = bars + 2 * kMaxStages;      // [2]
  uint64_t* acce = accf + 2;                   // [2]
  uint64_t* lfull = acce + 2;                  // [2]
  uint64_t* lempty = lfull + 2;                // [2]
  uint64_t* afull = lempty + 2;                // [1]
  uint64_t* mmadone = afull + 1;               // [1]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mmadone + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  RowAcc* red = reinterpret_cast<RowAcc*>(smem + lay.red_off);   // [2][128]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int S = a.stages;
  const bool comb = a.epi == EPI_COMBINE;
  const uint32_t tmem_cols =
      (a.n_tile * 2 <= 32) ? 32u : (uint32_t)(a.n_tile * 2 <= 64 ? 64 : (a.n_tile * 2 <= 128 ? 128 : 256));
  const uint64_t deadline = globaltimer_ns() + budget_ns;

  if (threadIdx.x == 0) {
    pdl_trigger();
    for (int i = 0; i < S; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&accf[i], 1);
      mbar_init(&acce[i], kEpiWarps);
      mbar_init(&lfull[i], 1);
      mbar_init(&lempty[i], kEpiWarps);
    }
    mbar_init(afull, 1);
    mbar_init(mmadone, 1);
    *abort_flag = 0;
    fence_mbarrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&mA0);
    tma_prefetch_desc(&mB0);
    if (a.seg_splits[1] > 0) {
      tma_prefetch_desc(&mA1);
      tma_prefetch_desc(&mB1);
    }
    if (comb) tma_prefetch_desc(&mL);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  int first, count, stride;
  item_range(a, first, count, stride);
  const uint32_t b_tile_bytes = (uint32_t)a.n_tile * 128u;
  const uint32_t l_box_bytes = (uint32_t)a.l_box_rows * 128u;
  const uint32_t l_tile_bytes = l_box_bytes * (uint32_t)a.l_boxes;

  if (warp == 0) {
    // ------------------------------------------------ weight / activation producer
    if (lane == 0 && !a.debug_skip_producer) {
      const uint64_t pol_act = l2_policy_evict_last();   // small, re-read by every CTA
      const uint64_t pol_w = l2_policy_evict_last();     // weights: re-read every block position
      int fills = 0;
      bool ok = true;
      // The weight stages do not depend on the previous kernel: start up to S
      // of them before waiting for it. Their barriers get the weight bytes as
      // expected transactions now and the arrival (with any activation bytes)
      // after the wait, so no phase can complete early.
      int pre = 0;
      if (count > 0) {
        int t = 0;
        Item it = get_item(a, first);
        int kc = it.kb;
        while (pre < S) {
          if (kc >= it.ke) {
            if (++t >= count) break;
            it = get_item(a, first + t * stride);
            kc = it.kb;
            continue;
          }
          mbar_expect_tx(&full[pre], b_tile_bytes);
          tma_load_2d(sB + pre * b_tile_bytes, it.seg ? &mB1 : &mB0, &full[pre], kc * kBlockK, it.o0, pol_w);
          ++pre;
          ++kc;
        }
      }
      pdl_wait();
      if (a.a_resident) {
        mbar_arrive_expect_tx(afull, (uint32_t)a.seg_chunks[0] * kATileBytes);
        for (int c = 0; c < a.seg_chunks[0]; ++c)
          tma_load_2d(sA + c * kATileBytes, &mA0, afull, c * kBlockK, 0, pol_act);
      }
      for (int t = 0; t < count && ok; ++t) {
        const Item it = get_item(a, first + t * stride);
        const CUtensorMap* mA = it.seg ? &mA1 : &mA0;
        const CUtensorMap* mB = it.seg ? &mB1 : &mB0;
        for (int kc = it.kb; kc < it.ke; ++kc, ++fills) {
          const int s = fills % S;
          if (fills < pre) {
            // weights already in flight: add the activation chunk and arrive
            if (a.a_resident) {
              mbar_arrive(&full[s]);
            } else {
              mbar_arrive_expect_tx(&full[s], (uint32_t)kATileBytes);
              tma_load_2d(sA + s * kATileBytes, mA, &full[s], kc * kBlockK, 0, pol_act);
            }
            continue;
          }
          ok = mbar_wait(&empty[s], ((fills / S) & 1) ^ 1, deadline, abort_flag);
          if (!ok) break;
          mbar_arrive_expect_tx(&full[s], b_tile_bytes + (a.a_resident ? 0u : (uint32_t)kATileBytes));
          if (!a.a_resident) tma_load_2d(sA + s * kATileBytes, mA, &full[s], kc * kBlockK, 0, pol_act);
          tma_load_2d(sB + s * b_tile_bytes, mB, &full[s], kc * kBlockK, it.o0, pol_w);
        }
      }
      // After an abort, wait (bounded) for the copies this thread issued to
      // land before the CTA exits; normally they were all consumed already.
      if (*abort_flag) {
        const uint64_t drain_deadline = globaltimer_ns() + 100000000ull;
        volatile int dummy = 0;
        for (int k = max(0, fills - S); k < fills; ++k)
          mbar_wait(&full[k % S], (k / S) & 1, drain_deadline, &dummy);
        if (a.a_resident) mbar_wait(afull, 0, drain_deadline, &dummy);
      }
    } else if (lane == 0) {
      pdl_wait();
    }
  } else if (warp == kLWarp) {
    // ------------------------------------------------ DFlash-logit tile producer
    if (lane == 0) {
      int l_issued = 0;
      if (comb && !a.debug_skip_producer) {
        const uint64_t pol_stream = l2_policy_evict_first();   // read once
        for (int t = 0; t < count; ++t) {
          const Item it = get_item(a, first + t * stride);
          const int buf = t & 1;
          if (!mbar_wait(&lempty[buf], ((t >> 1) & 1) ^ 1, deadline, abort_flag)) break;
          mbar_arrive_expect_tx(&lfull[buf], l_tile_bytes);
          for (int bx = 0; bx < a.l_boxes; ++bx)
            tma_load_3d(sL + buf * l_tile_bytes + bx * l_box_bytes, &mL, &lfull[buf], it.o0 + bx * a.l_box_cols,
                        a.j, 0, pol_stream);
          ++l_issued;
        }
      }
      pdl_wait();
      if (*abort_flag) {
        const uint64_t drain_deadline = globaltimer_ns() + 100000000ull;
        volatile int dummy = 0;
        for (int t = max(0, l_issued - 2); t < l_issued; ++t)
          mbar_wait(&lfull[t & 1], (t >> 1) & 1, drain_deadline, &dummy);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(128, a.n_tile);
      int fills = 0;
      bool ok = true;
      pdl_wait();
      if (a.a_resident) ok = mbar_wait(afull, 0, deadline, abort_flag);
      for (int t = 0; t < count && ok; ++t) {
        const Item it = get_item(a, first + t * stride);
        const int buf = t & 1;
        ok = mbar_wait(&acce[buf], ((t >> 1) & 1) ^ 1, deadline, abort_flag);
        if (!ok) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(buf * a.n_tile);
        for (int kc = it.kb; kc < it.ke; ++kc, ++fills) {
          const int s = fills % S;
          ok = mbar_wait(&full[s], (fills / S) & 1, deadline, abort_flag);
          if (!ok) break;
          tc_fence_after();
          const uint32_t a_addr = smem_u32(sA + (a.a_resident ? kc : s) * kATileBytes);
          const uint32_t b_addr = smem_u32(sB + s * b_tile_bytes);
#pragma unroll
          for (int kk = 0; kk < kBlockK / kUmmaK; ++kk) {
            tc_mma_f16(d_tmem, smem_desc_sw128(a_addr + kk * kUmmaK * 2), smem_desc_sw128(b_addr + kk * kUmmaK * 2),
                       idesc, (kc > it.kb || kk > 0) ? 1u : 0u);
          }
          tc_commit(&empty[s]);
        }
        if (!ok) break;
        tc_commit(&accf[buf]);
      }
      // every MMA issued by this thread has completed once mmadone fires
      tc_commit(mmadone);
      volatile int dummy = 0;
      mbar_wait(mmadone, 0, globaltimer_ns() + 100000000ull, &dummy);
    }
  } else {
    // ------------------------------------------------ epilogue
    const int ep = threadIdx.x - 64;             // 0..255
    const int q = warp & 3;                      // TMEM lane quadrant
    const int g = (warp - 2) >> 2;               // column-chunk parity
    const int b = q * 32 + lane;                 // batch row of this thread
    const bool quad_live = (q * 32) < a.B;
    const int nchunk = a.n_tile / 32;
    float best = -INFINITY, second = -INFINITY, m = -INFINITY, ssum = 0.f;
    int idx = 0x7FFFFFFF;
    const float alpha = a.alpha, nbeta = -a.beta;
    if (comb) {
      // the prior of this CTA's vocabulary range, once (an input: no wait needed)
      const int n = count * a.n_tile;
      const int v0 = first * a.n_tile;
      for (int i = ep; i < n; i += kEpiWarps * 32) {
        const int v = v0 + i;
        sP[i] = v < a.V ? __ldg(a.prior + v) : 0.f;
      }
      named_bar_sync<2>(kEpiWarps * 32);
    }
    pdl_wait();
    const int br = comb ? min(b, a.l_box_rows - 1) : 0;   // logits-box rows past B are never used
    const int swz = br & 7;
    bool ok = true;
    for (int t = 0; t < count && ok; ++t) {
      const Item it = get_item(a, first + t * stride);
      const int buf = t & 1;
      ok = mbar_wait(&accf[buf], (t >> 1) & 1, deadline, abort_flag);
      if (!ok) break;
      tc_fence_after();
      if (comb) {
        ok = mbar_wait(&lfull[buf], (t >> 1) & 1, deadline, abort_flag);
        if (!ok) break;
      }
      const uint32_t tbase = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * a.n_tile);
      if (quad_live && comb) {
        // n_tile == 128: chunks g and g + 2, both loaded before one wait
        float acc0[32], acc1[32];
        tmem_ld_32x32b_x32(tbase + (uint32_t)(g * 32), acc0);
        tmem_ld_32x32b_x32(tbase + (uint32_t)((g + 2) * 32), acc1);
        tmem_ld_wait();
        const uint8_t* lbuf = sL + buf * l_tile_bytes;
        const float* ptile = sP + t * a.n_tile;
        if (!a.long_f32) {
          // bf16 boxes of 64 columns: chunk cc is half (cc & 1) of box (cc >> 1)
          combine_chunk(acc0, lbuf + (g >> 1) * l_box_bytes + br * 128, g & 1, swz, false, ptile + g * 32,
                        it.o0 + g * 32, a.V, alpha, nbeta, best, second, idx, m, ssum);
          combine_chunk(acc1, lbuf + ((g + 2) >> 1) * l_box_bytes + br * 128, g & 1, swz, false,
                        ptile + (g + 2) * 32, it.o0 + (g + 2) * 32, a.V, alpha, nbeta, best, second, idx, m, ssum);
        } else {
          // f32 boxes of 32 columns: chunk cc is box cc
          combine_chunk(acc0, lbuf + g * l_box_bytes + br * 128, 0, swz, true, ptile + g * 32, it.o0 + g * 32, a.V,
                        alpha, nbeta, best, second, idx, m, ssum);
          combine_chunk(acc1, lbuf + (g + 2) * l_box_bytes + br * 128, 0, swz, true, ptile + (g + 2) * 32,
                        it.o0 + (g + 2) * 32, a.V, alpha, nbeta, best, second, idx, m, ssum);
        }
      } else if (quad_live) {
        for (int cc = g; cc < nchunk; cc += 2) {
          float acc[32];
          tmem_ld_32x32b_x32(tbase + (uint32_t)(cc * 32), acc);
          tmem_ld_wait();
          const int cbase = it.o0 + cc * 32;
          if (b < a.B) {
#pragma unroll
            for (int i = 0; i < 32; ++i) acc[i] = act_apply(a.act, acc[i]);
            if (a.out_f32) {
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
        mbar_arrive(&acce[buf]);
        if (comb) mbar_arrive(&lempty[buf]);
      }
    }
    if (comb) {
      // merge the two column-parity halves of each row, publish one record
      RowAcc mine;
      mine.m = best; mine.s = ssum; mine.second = second; mine.idx = idx;
      red[g * 128 + b] = mine;
      named_bar_sync<1>(kEpiWarps * 32);
      if (g == 0 && b < a.B && !*abort_flag) {
        const RowAcc r = count > 0 ? rowacc_merge(red[b], red[128 + b]) : rowacc_init();
        reinterpret_cast<float4*>(a.partials)[(long long)b * a.partial_ld + blockIdx.x] =
            make_float4(r.m, r.s, r.second, __int_as_float(r.idx));
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0 && *abort_flag) raise_status(a.status, DELS_STATUS_TIMEOUT);
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, tmem_cols);
  }
}

}  // namespace

size_t tc_gemm_smem_bytes(const TcGemmArgs& a) { return smem_layout(a).total; }

cudaError_t launch_tc_gemm(const TcGemmArgs& a, const CUtensorMap* mA0, const CUtensorMap* mB0,
                           const CUtensorMap* mA1, const CUtensorMap* mB1, const CUtensorMap* mL, int grid,
                           size_t smem_bytes, cudaStream_t s) {
  if (grid <= 0) return cudaSuccess;
  // The opt-in shared-memory limit is a per-device function attribute; raise
  // it once per device to the largest request seen.
  static int configured_bytes[64] = {0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if ((int)smem_bytes > configured_bytes[dev]) {
    e = cudaFuncSetAttribute(k_tc_gemm, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_bytes);
    if (e != cudaSuccess) return e;
    configured_bytes[dev] = (int)smem_bytes;
  }
  const uint64_t budget = a.debug_skip_producer ? 100000000ull : kWaitBudgetNs;
  return launch_pdl(k_tc_gemm, dim3(grid), dim3(kThreads), smem_bytes, s, *mA0, *mB0, *mA1, *mB1, *mL, a, budget);
}

}  // namespace dels
