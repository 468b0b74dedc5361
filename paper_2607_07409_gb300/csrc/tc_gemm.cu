// One-shot tcgen05 GEMM kernel (one phase of the engine in tc_engine.cuh):
//
//  * EPI_COMBINE — the vocabulary projection l_S = W_vocab r of Appendix A,
//    fused with the Section 4.3 combine: the epilogue adds the DFlash logits
//    (a TMA-loaded tile of l_L[:, j, :]) and the prior term (staged once per
//    CTA in shared memory) and folds the fused values into per-row
//    top-1/top-2/online-LSE state. Only one 16-byte record per (CTA, request)
//    leaves the kernel; no [B, V] logits are written.
//  * EPI_STORE — Y[b, o] = act(sum_k X[b, k] W[o, k]) for the local-head
//    products, optionally split over K with f32 partial outputs.
//
// Warp roles (352 threads): warp 0 = weight/activation TMA producer, warp 1 =
// MMA issuer and TMEM owner, warps 2..9 = epilogue, warp 10 = DFlash-logit
// tile producer.
//
// Programmatic dependent launch: the kernel lets its successor launch at
// once, and before waiting for its own predecessor it already allocates TMEM,
// stages the prior, starts the DFlash-logit tiles and the first weight
// stages — everything that does not depend on the previous kernel.
#include <algorithm>

#include "tc_engine.cuh"

namespace dels {

namespace {

using namespace tce;

constexpr int kWarps = 11;
constexpr int kThreads = kWarps * 32;
constexpr int kNoiseWarps = 8;                          // temperature-1 combine launches
constexpr int kThreadsSample = (kWarps + kNoiseWarps) * 32;
__host__ __device__ constexpr int threads_for(int mode) { return mode == 2 ? kThreadsSample : kThreads; }
constexpr int kLWarp = 10;

struct Smem {
  uint32_t a_off, b_off, l_off, p_off, bar_off, red_off, clus_off, tr_off, total;
};

// EPI_STORE with f32 rows only: the epilogue stores through a per-warp
// 32 x 33 transpose scratch (kStoreTransposeBytes).
__host__ __device__ inline bool store_transposes(const TcGemmArgs& a) {
  return a.epi == EPI_STORE && a.out_f32 && !a.out_bmajor && !a.out_bf16;
}

__host__ __device__ inline Smem smem_layout(const TcGemmArgs& a) {
  Smem s{};
  const int b_tile = a.n_tile * 128;
  const bool comb = a.epi == EPI_COMBINE;
  const int l_tile = comb ? a.l_boxes * a.l_box_rows * 128 : 0;
  const int a_tiles = a.a_resident ? a.seg_chunks[0] : a.stages * (a.b_chunks > 1 ? a.b_chunks : 1);
  uint32_t off = 0;
  s.a_off = off;
  off += (uint32_t)a_tiles * kATileBytes;
  s.b_off = off;
  off += (uint32_t)a.stages * b_tile * (uint32_t)(a.b_chunks > 1 ? a.b_chunks : 1);
  s.l_off = off;
  off += 2u * l_tile;
  s.p_off = off;
  off += comb ? (uint32_t)a.max_items_per_cta * a.n_tile * 4 : 0;
  off = (off + 15) / 16 * 16;
  s.bar_off = off;
  off += 64 * 8;                                  // mbarriers + tmem slot + flags
  s.red_off = off;
  off += comb ? 2 * 128 * 16 : 0;
  s.clus_off = off;                               // cluster split-K: the other ranks' accumulators
  off += a.cluster_k > 1 ? (uint32_t)(a.cluster_k - 1) * 128u * (uint32_t)a.n_tile * 4u : 0u;
  s.tr_off = off;
  off += store_transposes(a) ? (uint32_t)kStoreTransposeBytes : 0u;
  s.total = off + 1024;                           // slack for 1024-byte alignment
  return s;
}

// Cluster split-K, ranks >= 1: wait for the accumulator, then write it into
// rank 0's buffer slot (rank - 1) through distributed shared memory
// ([slot][128 rows][n_tile] f32). Rank 0 only waits for its accumulator here.
__device__ __forceinline__ void epi_cluster_send(const Ctx& c, const TcGemmArgs& a, uint32_t clus_local, int warp,
                                                 int lane, uint32_t rank) {
  if (!mbar_wait(&c.accf[0], 0, c.deadline, c.abort_flag)) return;
  tc_fence_after();
  if (rank == 0) return;
  const int q = warp & 3, g = (warp - 2) >> 2;
  if (q * 32 >= a.B) return;
  const int row = q * 32 + lane;
  const uint32_t tbase = c.tmem_base + ((uint32_t)(q * 32) << 16);
  for (int cc = g; cc < a.n_tile / 32; cc += 2) {
    float acc[32];
    tmem_ld_32x32b_x32(tbase + (uint32_t)(cc * 32), acc);
    tmem_ld_wait();
    const uint32_t dst = cluster_map(
        clus_local + ((((rank - 1) * 128u + (uint32_t)row) * (uint32_t)a.n_tile) + (uint32_t)cc * 32u) * 4u, 0);
#pragma unroll
    for (int k = 0; k < 8; ++k) st_cluster_v4(dst + k * 16, acc[4 * k], acc[4 * k + 1], acc[4 * k + 2], acc[4 * k + 3]);
  }
  tc_fence_before();
}

// Cluster split-K, rank 0, after the cluster barrier: own accumulator plus
// the other ranks' slots, activation, final store.
__device__ __forceinline__ void epi_cluster_finish(const Ctx& c, const TcGemmArgs& a, const float* clus, int o0,
                                                   int warp, int lane) {
  const int q = warp & 3, g = (warp - 2) >> 2;
  if (q * 32 >= a.B) return;
  const int b = q * 32 + lane;
  tc_fence_after();
  const uint32_t tbase = c.tmem_base + ((uint32_t)(q * 32) << 16);
  for (int cc = g; cc < a.n_tile / 32; cc += 2) {
    float acc[32];
    tmem_ld_32x32b_x32(tbase + (uint32_t)(cc * 32), acc);
    tmem_ld_wait();
    for (int r = 1; r < a.cluster_k; ++r) {
      const float4* src = reinterpret_cast<const float4*>(clus + (((r - 1) * 128 + b) * a.n_tile + cc * 32));
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const float4 v = src[k];
        acc[4 * k] += v.x; acc[4 * k + 1] += v.y; acc[4 * k + 2] += v.z; acc[4 * k + 3] += v.w;
      }
    }
    if (b >= a.B) continue;
    if (a.act != ACT_NONE) act_apply32(a.act, acc);
    const int cbase = o0 + cc * 32;
    if (a.out_f32)
      for (int i = 0; i < 32; ++i)
        if (cbase + i < a.O) a.out_f32[(long long)b * a.ldo + cbase + i] = acc[i];
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

// MODE 1 / 2: combine launches at temperature 0 / 1 (one CTA per SM, the
// combine epilogue's registers; MODE 2 adds the 8 noise warps and their two
// TMEM buffers); MODE 0: store launches, compiled separately
// with at most 2 x 352 threads' worth of registers per SM, so that a store
// launch's CTAs can share an SM with the small kernels around them.
template <int MODE>
__global__ void __launch_bounds__(threads_for(MODE), MODE != 0 ? 1 : 2)
    k_tc_gemm(const __grid_constant__ CUtensorMap mA0, const __grid_constant__ CUtensorMap mB0,
              const __grid_constant__ CUtensorMap mA1, const __grid_constant__ CUtensorMap mB1,
              const __grid_constant__ CUtensorMap mL, const __grid_constant__ TcGemmArgs a0,
              const __grid_constant__ CUtensorMap gA, const __grid_constant__ CUtensorMap gB,
              const __grid_constant__ TcGemmArgs a1, int grid0, uint64_t budget_ns) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  // CTAs past grid0 run the second GEMM of a grouped launch
  const bool second = (int)blockIdx.x >= grid0;
  const TcGemmArgs& a = second ? a1 : a0;
  const int cta = second ? (int)blockIdx.x - grid0 : (int)blockIdx.x;
  const int ncta = second ? (int)gridDim.x - grid0 : grid0;
  const Smem lay = smem_layout(a);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr bool comb = MODE != 0;

  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + lay.bar_off);
  Ctx c;
  c.sA = smem + lay.a_off;
  c.sB = smem + lay.b_off;
  c.sL = smem + lay.l_off;
  c.sP = reinterpret_cast<float*>(smem + lay.p_off);
  c.red = reinterpret_cast<RowAcc*>(smem + lay.red_off);
  c.tr = store_transposes(a) ? reinterpret_cast<float*>(smem + lay.tr_off) : nullptr;
  c.full = bars;
  c.empty = bars + kMaxStages;
  c.accf = bars + 2 * kMaxStages;
  c.acce = c.accf + 2;
  c.lfull = c.acce + 2;
  c.lempty = c.lfull + 2;
  c.afull = c.lempty + 2;
  c.nfull = bars + 48;    // noise barriers (temperature 1): slots past the others'
  c.nempty = bars + 50;
  uint64_t* mmadone = c.afull + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mmadone + 1);
  c.abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  c.S = a.stages;
  c.a_stage_bytes = kATileBytes * (uint32_t)(a.b_chunks > 1 ? a.b_chunks : 1);
  c.b_stage_bytes = (uint32_t)a.n_tile * 128u * (uint32_t)(a.b_chunks > 1 ? a.b_chunks : 1);
  c.l_buf_bytes = comb ? (uint32_t)(a.l_boxes * a.l_box_rows * 128) : 0u;
  c.deadline = globaltimer_ns() + budget_ns;
  // two accumulator buffers; at temperature 1 two noise buffers after them
  const uint32_t acc_cols =
      (a.n_tile * 2 <= 32) ? 32u : (uint32_t)(a.n_tile * 2 <= 64 ? 64 : (a.n_tile * 2 <= 128 ? 128 : 256));
  const uint32_t tmem_cols = MODE == 2 ? 2u * acc_cols : acc_cols;
  c.noise_col = acc_cols;

  if (threadIdx.x == 0) {
    pdl_trigger();
    for (int i = 0; i < c.S; ++i) {
      mbar_init(&c.full[i], 1);
      mbar_init(&c.empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&c.accf[i], 1);
      mbar_init(&c.acce[i], kEpiWarps);
      mbar_init(&c.lfull[i], 1);
      mbar_init(&c.lempty[i], kEpiWarps);
    }
    mbar_init(c.afull, 1);
    mbar_init(mmadone, 1);
    if (MODE == 2) {
      for (int i = 0; i < 2; ++i) {
        mbar_init(&c.nfull[i], kNoiseWarps);
        mbar_init(&c.nempty[i], kEpiWarps);
      }
    }
    *c.abort_flag = 0;
    fence_mbarrier_init();
  }
  const CUtensorMap* pA0 = second ? &gA : &mA0;
  const CUtensorMap* pB0 = second ? &gB : &mB0;
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(pA0);
    tma_prefetch_desc(pB0);
    if (!second && a.seg_splits[1] > 0) {
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
  c.tmem_base = *tmem_slot;
  // cluster split-K: every CTA of the cluster is running before any remote write
  const bool clus = a.cluster_k > 1;
  if (clus) cluster_sync_all();

  Phase p;
  p.a = &a;
  p.mA0 = pA0;
  p.mB0 = pB0;
  p.mA1 = second ? &gA : &mA1;
  p.mB1 = second ? &gB : &mB1;
  p.mL = &mL;
  p.j = a.j;
  item_range(a, cta, ncta, p.first, p.count, p.stride);

  if (warp == 0) {
    if (lane == 0) {
      if (!a.debug_skip_producer) {
        const uint64_t pol_w = l2_policy_evict_first();    // streamed once per launch
        const uint64_t pol_act = l2_policy_evict_last();   // small, re-read by every CTA
        ProdState st;
        prod_prefetch(c, p, st, pol_w);                     // weights: independent of the predecessor
        pdl_wait();
        prod_run(c, p, st, pol_w, pol_act);
        // after an abort, wait (bounded) for the copies issued to land
        if (*c.abort_flag) {
          const uint64_t dd = globaltimer_ns() + 100000000ull;
          volatile int dummy = 0;
          for (int k = max(0, st.fills - c.S); k < st.fills; ++k) mbar_wait(&c.full[k % c.S], (k / c.S) & 1, dd, &dummy);
          if (a.a_resident && st.afull_uses) mbar_wait(c.afull, 0, dd, &dummy);
        }
      } else {
        pdl_wait();
      }
    }
  } else if (warp == kLWarp) {
    if (lane == 0) {
      LState ls;
      if (comb && !a.debug_skip_producer) lprod_issue(c, p, ls, 1 << 30, l2_policy_evict_first());
      pdl_wait();
      if (*c.abort_flag) {
        const uint64_t dd = globaltimer_ns() + 100000000ull;
        volatile int dummy = 0;
        for (int t = max(0, ls.tiles - 2); t < ls.tiles; ++t) mbar_wait(&c.lfull[t & 1], (t >> 1) & 1, dd, &dummy);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      pdl_wait();
      MmaState st;
      mma_run(c, p, st);
      // every MMA issued by this thread has completed once mmadone fires
      tc_commit(mmadone);
      volatile int dummy = 0;
      mbar_wait(mmadone, 0, globaltimer_ns() + 100000000ull, &dummy);
    }
  } else if (MODE == 2 && warp >= kWarps) {
    // the variates depend on the arguments only: no wait for the predecessor
    noise_run(c, p, warp, lane, (warp - kWarps) >> 2);
  } else {
    if (comb) epi_stage_prior(c, p, threadIdx.x - 64);   // an input: no wait needed
    pdl_wait();
    if (clus) {
      if (p.count > 0) epi_cluster_send(c, a, smem_u32(smem + lay.clus_off), warp, lane, cluster_ctarank());
    } else {
      EpiState st;
      epi_run<MODE != 0, MODE == 2>(c, p, st, warp, lane, cta);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (clus) {
    // the other ranks' accumulators have landed in rank 0's buffer
    cluster_sync_all();
    if (warp >= 2 && warp < 2 + kEpiWarps && cluster_ctarank() == 0 && p.count > 0 && !*c.abort_flag)
      epi_cluster_finish(c, a, reinterpret_cast<const float*>(smem + lay.clus_off), get_item(a, p.first).o0, warp,
                         lane);
    tc_fence_before();
    __syncthreads();
  }
  if (threadIdx.x == 0 && *c.abort_flag) raise_status(a.status, DELS_STATUS_TIMEOUT);
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(c.tmem_base, tmem_cols);
  }

}

}  // namespace

size_t tc_gemm_smem_bytes(const TcGemmArgs& a) { return smem_layout(a).total; }

cudaError_t launch_tc_gemm(const TcGemmArgs& a, const CUtensorMap* mA0, const CUtensorMap* mB0,
                           const CUtensorMap* mA1, const CUtensorMap* mB1, const CUtensorMap* mL, int grid,
                           size_t smem_bytes, cudaStream_t s, const TcGemmGroup* second) {
  const bool two = second && second->a && second->grid > 0;
  if (grid <= 0 && !two) return cudaSuccess;
  if (two) smem_bytes = std::max(smem_bytes, tc_gemm_smem_bytes(*second->a));
  // The opt-in shared-memory limit is a per-device function attribute; raise
  // it once per device to the largest request seen.
  const bool comb = a.epi == EPI_COMBINE;
  if (two && (second->a->epi == EPI_COMBINE) != comb) return cudaErrorInvalidValue;
  const int mode = comb ? (a.sample ? 2 : 1) : 0;
  auto kern = mode == 2 ? k_tc_gemm<2> : mode == 1 ? k_tc_gemm<1> : k_tc_gemm<0>;
  const int threads = threads_for(mode);
  cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void*>(kern), smem_bytes);
  if (e != cudaSuccess) return e;
  const uint64_t budget = a.debug_skip_producer ? 100000000ull : kWaitBudgetNs;
  const int g0 = std::max(grid, 0);
  // clusters (split-K through distributed shared memory) cover the whole grid:
  // both groups' grids must be whole clusters
  const int ck = std::max(a.cluster_k, two ? second->a->cluster_k : 1);
  if (ck > 1 && (g0 % ck != 0 || (two && second->grid % ck != 0))) return cudaErrorInvalidValue;
  if (two)
    return launch_pdl_cluster(kern, dim3(g0 + second->grid), dim3(threads), smem_bytes, s, ck, *mA0, *mB0,
                              *mA1, *mB1, *mL, a, *second->mA, *second->mB, *second->a, g0, budget);
  return launch_pdl_cluster(kern, dim3(g0), dim3(threads), smem_bytes, s, ck, *mA0, *mB0, *mA1, *mB1, *mL, a,
                            *mA0, *mB0, a, g0, budget);
}

}  // namespace dels
