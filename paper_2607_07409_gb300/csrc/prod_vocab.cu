// One launch per drafted position j >= 1 of the GRU input-table path: the
// head's two products of h_j followed by the vocabulary projection fused with
// the Section 4.3 combine.
//
//   CTAs [0, rank_ctas)            r_j = SiLU(W_rank h_j): the K splits of an
//                                  output tile are the CTAs of one thread-block
//                                  cluster; the others send their accumulators
//                                  to rank 0 through distributed shared memory,
//                                  rank 0 sums, applies SiLU, stores the bf16
//                                  tile and counts it in r_ready.
//   CTAs [rank_ctas, +hh_ctas)     partials of W_hh h_j (read by the next
//                                  position's gates launch).
//   every CTA                      l_S = W_vocab r_j fused with
//                                  l = l_L + alpha l_S - beta l_P over its
//                                  vocabulary range -> one record per request.
//
// The vocabulary phase needs all of r_j, written by other CTAs of the same
// launch, so the launch is cooperative (every CTA co-resident; clusters of
// cluster_k CTAs over the whole grid) and each CTA's
// producer waits, bounded, until r_ready reaches the count expected for
// position j. Its weight tiles do not depend on r_j: they stream into the
// pipeline ring while the products run, as do the first DFlash-logit tiles
// and the prior; only the resident r tile waits for the counter.
//
// Warp roles and pipeline as in tc_gemm.cu (tc_engine.cuh): warp 0 producer,
// warp 1 MMA issuer / TMEM owner, warps 2..9 epilogue, warp 10 logits
// producer. The ring is one FIFO across the two phases: the products' fills
// come first, then the vocabulary's.
#include <atomic>
#include <climits>

#include "tc_engine.cuh"

namespace dels {

namespace {

using namespace tce;

constexpr int kWarps = 11;
constexpr int kThreads = kWarps * 32;
constexpr int kEpiThreads = kEpiWarps * 32;
constexpr int kLWarp = 10;
constexpr uint32_t kTmemCols = 256;

struct Smem {
  uint32_t a_off, b_off, l_off, p_off, bar_off, red_off, clus_off, total;
};

// Product phases load B activation rows per stage (packed at that size; the
// MMA's 128-row read runs into the next stage, rows it never uses); the
// vocabulary phase keeps its activations resident (one 128-row tile per K
// chunk) in the same area once the products are done.
__host__ __device__ inline uint32_t pv_a_stage_bytes(const ProdVocabArgs& P) {
  return (uint32_t)((P.vocab.B + 7) / 8 * 8) * 128u;
}

__host__ __device__ inline Smem pv_layout(const ProdVocabArgs& P) {
  Smem s{};
  const TcGemmArgs& v = P.vocab;
  const uint32_t staged = (uint32_t)P.stages * pv_a_stage_bytes(P) + kATileBytes - pv_a_stage_bytes(P);
  const uint32_t resident = (uint32_t)v.seg_chunks[0] * kATileBytes;
  const uint32_t a_area = ((staged > resident ? staged : resident) + 1023u) / 1024u * 1024u;
  const uint32_t l_tile = (uint32_t)(v.l_boxes * v.l_box_rows * 128);
  uint32_t off = 0;
  s.a_off = off;
  off += a_area;
  s.b_off = off;
  off += (uint32_t)P.stages * (uint32_t)v.n_tile * 128u;   // the vocabulary tile is the widest
  s.l_off = off;
  off += 2u * l_tile;
  s.p_off = off;
  off += (uint32_t)v.max_items_per_cta * v.n_tile * 4u;
  off = (off + 15) / 16 * 16;
  s.bar_off = off;
  off += 64 * 8;
  s.red_off = off;
  off += 2 * 128 * 16;
  s.clus_off = off;                               // rank splits' accumulators, in the cluster's rank 0
  off += (uint32_t)(P.rank.cluster_k - 1) * 128u * (uint32_t)P.rank.n_tile * 4u;
  s.total = off + 1024;
  return s;
}

// Threads of one rank CTA that hold accumulator rows to send: the live TMEM
// lane quadrants x the epilogue warps that take column chunks.
__host__ __device__ inline int rank_senders(const TcGemmArgs& a) {
  const int quads = (a.B + 31) / 32;
  const int chunks = a.n_tile / 32;
  return quads * (chunks < 2 ? chunks : 2) * 32;
}

// Rank product epilogue for one cluster (the K splits of one output tile,
// split = rank in the cluster). Ranks >= 1 send their accumulator rows into
// rank 0's buffer slot (rank - 1) and arrive on rank 0's barrier; rank 0
// waits for them, sums, applies SiLU, stores its bf16 tile of r and counts
// it in r_ready. Every epilogue warp releases the accumulator buffer.
__device__ __forceinline__ void rank_cluster_epilogue(const Ctx& c, const ProdVocabArgs& P, uint8_t* clus,
                                                      uint64_t* rbar, int o0, int warp, int lane, int ep) {
  const TcGemmArgs& a = P.rank;
  const uint32_t rank = cluster_ctarank();
  const int q = warp & 3, g = (warp - 2) >> 2;
  const int nchunk = a.n_tile / 32;
  const bool sender = q * 32 < a.B && g < nchunk;
  const int row = q * 32 + lane;
  const uint32_t tbase = c.tmem_base + ((uint32_t)(q * 32) << 16);
  const bool ok = mbar_wait(&c.accf[0], 0, c.deadline, c.abort_flag);
  tc_fence_after();
  if (rank != 0) {
    if (sender) {
      if (ok) {
        for (int cc = g; cc < nchunk; cc += 2) {
          float acc[32];
          tmem_ld_32x32b_x32(tbase + (uint32_t)(cc * 32), acc);
          tmem_ld_wait();
          const uint32_t dst = cluster_map(
              smem_u32(clus) + ((((rank - 1) * 128u + (uint32_t)row) * (uint32_t)a.n_tile) + (uint32_t)cc * 32u) * 4u,
              0);
#pragma unroll
          for (int k = 0; k < 8; ++k)
            st_cluster_v4(dst + k * 16, acc[4 * k], acc[4 * k + 1], acc[4 * k + 2], acc[4 * k + 3]);
        }
      }
      mbar_arrive_remote(cluster_map(smem_u32(rbar), 0));   // also on abort: rank 0 must not wait forever
    }
  } else {
    const bool got = mbar_wait_cluster(rbar, 0, c.deadline, c.abort_flag);
    if (ok && got && sender) {
      const float* slots = reinterpret_cast<const float*>(clus);
      for (int cc = g; cc < nchunk; cc += 2) {
        float acc[32];
        tmem_ld_32x32b_x32(tbase + (uint32_t)(cc * 32), acc);
        tmem_ld_wait();
        for (int r = 1; r < a.cluster_k; ++r) {
          const float4* src = reinterpret_cast<const float4*>(slots + (((r - 1) * 128 + row) * a.n_tile + cc * 32));
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const float4 v = src[k];
            acc[4 * k] += v.x; acc[4 * k + 1] += v.y; acc[4 * k + 2] += v.z; acc[4 * k + 3] += v.w;
          }
        }
        const int cbase = o0 + cc * 32;
        if (row < a.B) {
          uint16_t* dst = P.r + (long long)row * P.R + cbase;
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const float x = __fdividef(acc[i], 1.f + __expf(-acc[i]));   // SiLU
            if (cbase + i < a.O) dst[i] = f32_to_bf16_rne(x);
          }
        }
      }
    }
    fence_acq_rel_gpu();
    named_bar_sync<1>(kEpiThreads);
    if (ep == 0) {
      fence_acq_rel_gpu();
      atomicAdd(P.r_ready, 1u);
    }
  }
  tc_fence_before();
  __syncwarp();
  if (lane == 0) mbar_arrive(&c.acce[0]);
}

__global__ void __launch_bounds__(kThreads, 1)
    k_prod_vocab(const __grid_constant__ CUtensorMap m_hb, const __grid_constant__ CUtensorMap m_wrank,
                 const __grid_constant__ CUtensorMap m_whh, const __grid_constant__ CUtensorMap m_r,
                 const __grid_constant__ CUtensorMap m_wvocab, const __grid_constant__ CUtensorMap m_long,
                 const __grid_constant__ ProdVocabArgs P, uint64_t budget_ns) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  const Smem lay = pv_layout(P);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int cta = blockIdx.x;

  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + lay.bar_off);
  Ctx c;
  c.sA = smem + lay.a_off;
  c.sB = smem + lay.b_off;
  c.sL = smem + lay.l_off;
  c.sP = reinterpret_cast<float*>(smem + lay.p_off);
  c.red = reinterpret_cast<RowAcc*>(smem + lay.red_off);
  c.tr = nullptr;
  c.full = bars;
  c.empty = bars + kMaxStages;
  c.accf = bars + 2 * kMaxStages;
  c.acce = c.accf + 2;
  c.lfull = c.acce + 2;
  c.lempty = c.lfull + 2;
  c.afull = c.lempty + 2;
  uint64_t* pdone = c.afull + 1;               // every product MMA of this CTA has completed
  uint64_t* mmadone = pdone + 1;
  uint64_t* rbar = mmadone + 1;                // rank 0: the other splits' accumulators have landed
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(rbar + 1);
  c.abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  c.S = P.stages;
  c.a_stage_bytes = pv_a_stage_bytes(P);
  c.b_stage_bytes = (uint32_t)P.vocab.n_tile * 128u;
  c.l_buf_bytes = (uint32_t)(P.vocab.l_boxes * P.vocab.l_box_rows * 128);
  c.deadline = globaltimer_ns() + budget_ns;

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
    mbar_init(pdone, 1);
    mbar_init(mmadone, 1);
    mbar_init(rbar, (uint32_t)((P.rank.cluster_k - 1) * rank_senders(P.rank)));
    *c.abort_flag = 0;
    fence_mbarrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&m_hb);
    tma_prefetch_desc(&m_wrank);
    tma_prefetch_desc(&m_whh);
    tma_prefetch_desc(&m_r);
    tma_prefetch_desc(&m_wvocab);
    tma_prefetch_desc(&m_long);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  c.tmem_base = *tmem_slot;
  // every CTA of the cluster has initialised its barriers before any remote arrive
  cluster_sync_all();

  // this CTA's product work (rank split, recurrent split or none) and its
  // vocabulary range
  const bool is_rank = cta < P.rank_ctas;
  const bool is_hh = !is_rank && cta < P.rank_ctas + P.hh_ctas;
  Phase pp{is_rank ? &P.rank : &P.hh, &m_hb, is_rank ? &m_wrank : &m_whh, &m_hb, is_rank ? &m_wrank : &m_whh,
           &m_long, 0, 0, 1, 0};
  if (is_rank) {
    item_range(P.rank, cta, P.rank_ctas, pp.first, pp.count, pp.stride);   // tile = cluster, split = rank
  } else if (is_hh) {
    item_range(P.hh, cta - P.rank_ctas, P.hh_ctas, pp.first, pp.count, pp.stride);
  }
  const bool has_prod = (is_rank || is_hh) && pp.count > 0;
  Phase pv{&P.vocab, &m_r, &m_wvocab, &m_r, &m_wvocab, &m_long, 0, 0, 1, P.vocab.j};
  item_range(P.vocab, cta, gridDim.x, pv.first, pv.count, pv.stride);

  if (warp == 0) {
    if (lane == 0) {
      const uint64_t pol_w = l2_policy_evict_first();
      const uint64_t pol_act = l2_policy_evict_last();
      ProdState st;
      if (has_prod) prod_prefetch(c, pp, st, pol_w);
      pdl_wait();
      if (has_prod) prod_run(c, pp, st, pol_w, pol_act);
      // The vocabulary weights do not depend on r_j, but streaming them now
      // competes with the rank path for memory bandwidth (measured: the rank
      // partials' reads took 5 us longer), so they start once r_j is ready.
      // The resident r tile overwrites the product stages' activations, and
      // needs every rank tile of this position.
      volatile int dummy = 0;
      bool ok = mbar_wait(pdone, 0, c.deadline, c.abort_flag);
      if (ok) {
        // poll with a pause: ~150 CTAs polling one line back to back slow down
        // every other access served by the same L2 slice
        uint32_t polls = 0;
        while (ld_acquire_gpu(P.r_ready) < P.r_target) {
          __nanosleep(256);
          if ((++polls & 15u) == 0u && (*c.abort_flag || globaltimer_ns() > c.deadline)) {
            *c.abort_flag = 1;
            ok = false;
            break;
          }
        }
      }
      if (ok) {
        fence_proxy_async_global();               // r was written by other CTAs' generic stores
        prod_prefetch(c, pv, st, pol_w);
        prod_run(c, pv, st, pol_w, pol_act);
      }
      if (*c.abort_flag) {
        const uint64_t dd = globaltimer_ns() + 100000000ull;
        const int issued = max(st.fills, st.pre_end);
        for (int k = max(0, issued - c.S); k < issued; ++k) mbar_wait(&c.full[k % c.S], (k / c.S) & 1, dd, &dummy);
        if (st.afull_uses) mbar_wait(c.afull, 0, dd, &dummy);
      }
    }
  } else if (warp == kLWarp) {
    if (lane == 0) {
      LState ls;
      lprod_issue(c, pv, ls, INT_MAX, l2_policy_evict_first());   // inputs: no wait needed
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
      if (has_prod) mma_run(c, pp, st);
      tc_commit(pdone);                           // arrives once the product MMAs have completed
      if (!*c.abort_flag) mma_run(c, pv, st);
      tc_commit(mmadone);
      volatile int dummy = 0;
      mbar_wait(mmadone, 0, globaltimer_ns() + 100000000ull, &dummy);
    }
  } else {
    const int ep = threadIdx.x - 64;
    epi_stage_prior(c, pv, ep);                   // an input: no wait needed
    pdl_wait();
    EpiState st;
    if (is_rank) {
      if (pp.count > 0) {
        rank_cluster_epilogue(c, P, smem + lay.clus_off, rbar, get_item(P.rank, pp.first).o0, warp, lane, ep);
        st.tiles = 1;
      }
    } else if (has_prod) {
      epi_run<false>(c, pp, st, warp, lane, cta);
    }
    if (!*c.abort_flag) epi_run<true>(c, pv, st, warp, lane, cta);
  }

  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0 && *c.abort_flag) raise_status(P.vocab.status, DELS_STATUS_TIMEOUT);
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(c.tmem_base, kTmemCols);
  }
}

}  // namespace

size_t prod_vocab_smem_bytes(const ProdVocabArgs& P) { return pv_layout(P).total; }

cudaError_t launch_prod_vocab(const ProdVocabArgs& P, const CUtensorMap* maps, int grid, size_t smem,
                              cudaStream_t s) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  e = ensure_dynamic_smem(reinterpret_cast<const void*>(k_prod_vocab), smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  if (P.rank.cluster_k < 1 || grid % P.rank.cluster_k != 0 || P.rank_ctas % P.rank.cluster_k != 0)
    return cudaErrorInvalidValue;
  cudaLaunchAttribute attr[3];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = (unsigned)P.rank.cluster_k;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  attr[2].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[2].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  // programmatic serialization with a cooperative launch where the runtime
  // allows it; plain stream order otherwise (remembered per device)
  static std::atomic<int> coop_pdl[64];   // 0 unknown, 1 allowed, -1 refused (zero-initialised: static)
  cfg.numAttrs = coop_pdl[dev].load() >= 0 ? 3 : 2;
  e = cudaLaunchKernelEx(&cfg, k_prod_vocab, maps[0], maps[1], maps[2], maps[3], maps[4], maps[5], P,
                         (uint64_t)kWaitBudgetNs);
  if (e != cudaSuccess && cfg.numAttrs == 3 && coop_pdl[dev].load() == 0) {
    (void)cudaGetLastError();
    coop_pdl[dev].store(-1);
    cfg.numAttrs = 2;
    e = cudaLaunchKernelEx(&cfg, k_prod_vocab, maps[0], maps[1], maps[2], maps[3], maps[4], maps[5], P,
                           (uint64_t)kWaitBudgetNs);
  } else if (e == cudaSuccess && cfg.numAttrs == 3) {
    coop_pdl[dev].store(1);
  }
  return e;
}

}  // namespace dels
