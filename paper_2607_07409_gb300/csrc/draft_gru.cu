// Persistent per-block drafting kernel for the Appendix A GRU head (bf16).
//
// One cooperative launch drafts a whole block (Algorithm 1): every SM runs
// one CTA for the life of the block, the drafted tokens and every
// intermediate stay on chip or in L2, and the CTAs step through the
// positions together, separated by grid-wide barriers:
//
//   position 0 : row reduction of l_L[:, 0, :] (no head, no prior)  | barrier
//                merge -> x_0; gather E_tgt[x_0]; h_0 = 0           | barrier
//   j = 1..n-1 : GRU gate products (tcgen05, split K)               | barrier
//                gates -> h_j (f32) and its bf16 copy               | barrier
//                r_j = SiLU(W_rank h_j) (tcgen05)                   | barrier
//                W_vocab r_j fused with l_L + a l_S - b l_P         | barrier
//                merge -> x_j; gather E_tgt[x_j]                    | barrier
//
// Between phases nothing is relaunched: TMEM, the mbarrier pipelines and the
// per-CTA prior slice persist. Weights do not depend on the previous phase,
// so each CTA's producer issues the next tensor-core phase's first weight
// stages, and the logits producer the next position's first DFlash-logit
// tiles, before joining the barrier; only the activations wait for it.
//
// Warp roles as in the one-shot GEMM: warp 0 weight/activation producer,
// warp 1 MMA issuer (TMEM owner), warps 2..9 epilogue (which also run the
// element-wise phases), warp 10 DFlash-logit producer.
#include <climits>

#include "tc_engine.cuh"

namespace dels {

namespace {

using namespace tce;

constexpr int kWarps = 11;
constexpr int kThreads = kWarps * 32;
constexpr int kEpiThreads = kEpiWarps * 32;
constexpr uint32_t kTmemCols = 256;

struct Smem {
  uint32_t a_off, b_off, l_off, p_off, bar_off, red_off, total;
};

// Activation stages are packed at the size actually loaded (the GRU and rank
// phases load B rows); the area also holds the vocabulary phase's resident
// activations (one 128-row tile per K chunk) and leaves room for the MMA's
// 128-row read of the last stage.
__host__ __device__ inline uint32_t a_stage_bytes(const PersistGruArgs& P) {
  return (uint32_t)((P.B + 7) / 8 * 8) * 128u;
}
__host__ __device__ inline uint32_t a_area_bytes(const PersistGruArgs& P) {
  const uint32_t staged = (uint32_t)P.stages * a_stage_bytes(P) + kATileBytes - a_stage_bytes(P);
  const uint32_t resident = (uint32_t)P.vocab.seg_chunks[0] * kATileBytes;
  const uint32_t m = staged > resident ? staged : resident;
  return (m + 1023u) / 1024u * 1024u;
}

__host__ __device__ inline Smem smem_layout(const PersistGruArgs& P) {
  Smem s{};
  const TcGemmArgs& v = P.vocab;
  const uint32_t l_tile = (uint32_t)(v.l_boxes * v.l_box_rows * 128);
  uint32_t off = 0;
  s.a_off = off;
  off += a_area_bytes(P);
  s.b_off = off;
  off += (uint32_t)P.stages * 128u * 128u;
  s.l_off = off;
  off += 2u * l_tile;
  s.p_off = off;
  off += (uint32_t)v.max_items_per_cta * v.n_tile * 4u;
  off = (off + 15) / 16 * 16;
  s.bar_off = off;
  off += 64 * 8;
  s.red_off = off;
  off += 2 * 128 * 16;
  s.total = off + 1024;
  return s;
}

__device__ __forceinline__ void load8(const uint16_t* p, float (&x)[8]) {
  const uint4 w = __ldcs(reinterpret_cast<const uint4*>(p));
  x[0] = bf16lo(w.x); x[1] = bf16hi(w.x); x[2] = bf16lo(w.y); x[3] = bf16hi(w.y);
  x[4] = bf16lo(w.z); x[5] = bf16hi(w.z); x[6] = bf16lo(w.w); x[7] = bf16hi(w.w);
}
__device__ __forceinline__ void load8(const float* p, float (&x)[8]) {
  const float4 a = __ldcs(reinterpret_cast<const float4*>(p));
  const float4 b = __ldcs(reinterpret_cast<const float4*>(p) + 1);
  x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w; x[4] = b.x; x[5] = b.y; x[6] = b.z; x[7] = b.w;
}

// Grid-wide barrier (all threads of every CTA call it). Arrival is one
// atomic on a counter; the last CTA to arrive resets the counter and
// publishes the next generation number on a separate 128-byte line, which the
// others poll (so polling never contends with the arrivals). `gen` is this
// CTA's count of barriers passed, seeded from the workspace at kernel start.
// Bounded: gives up at the deadline (or when another CTA gave up).
__device__ __forceinline__ bool grid_sync(unsigned* bar, unsigned& gen, int* abort_g, volatile int* abort_cta,
                                          uint64_t deadline) {
  fence_proxy_async_global();
  __syncthreads();
  if (threadIdx.x == 0 && !*abort_cta) {
    unsigned* count = bar;
    unsigned* flag = bar + 32;   // next 128-byte line
    __threadfence();
    const unsigned ticket = atomicAdd(count, 1u);
    if (ticket == gridDim.x - 1) {
      *reinterpret_cast<volatile unsigned*>(count) = 0u;
      __threadfence();
      st_release_gpu(flag, gen + 1);
    } else {
      unsigned polls = 0;
      while (ld_acquire_gpu(flag) == gen) {
        if ((++polls & 15u) == 0) {
          if (*reinterpret_cast<volatile int*>(abort_g) || globaltimer_ns() > deadline) {
            *abort_cta = 1;
            atomicExch(abort_g, 1);
            break;
          }
        }
      }
    }
    ++gen;
    __threadfence();
  }
  __syncthreads();
  fence_proxy_async_global();
  return *abort_cta == 0;
}

// Reduce this epilogue thread's RowAcc over the 256 epilogue threads; the
// result is valid in epilogue thread 0. Uses red[0..7] and named barrier 3.
__device__ __forceinline__ RowAcc epi_block_reduce(RowAcc x, RowAcc* red, int ep) {
  x = rowacc_warp_reduce(x);
  if ((ep & 31) == 0) red[ep >> 5] = x;
  named_bar_sync<3>(kEpiThreads);
  RowAcc r = rowacc_init();
  if (ep < 32) {
    r = ep < kEpiWarps ? red[ep] : rowacc_init();
    r = rowacc_warp_reduce(r);
  }
  named_bar_sync<3>(kEpiThreads);
  return r;
}

__device__ __forceinline__ void write_decode(const RowAcc& r, long long o, const PersistGruArgs& P) {
  const bool ok = rowacc_valid(r);
  if (!ok) raise_status(P.status, DELS_STATUS_NONFINITE);
  P.tokens[o] = ok ? r.idx : -1;
  P.out_lp[o] = ok ? -logf(r.s) : NAN;
  if (P.out_gap) P.out_gap[o] = ok ? (r.m - r.second) : NAN;
}

// Position 0: this CTA's (row, chunk) of l_L[:, 0, :] -> partials[row][chunk].
template <typename T>
__device__ __forceinline__ void pos0_phase(const PersistGruArgs& P, RowAcc* red, int ep) {
  const int C = P.pos0_chunks;
  if ((int)blockIdx.x >= P.B * C) return;
  const int b = blockIdx.x / C, ch = blockIdx.x % C;
  const int c0 = ch * P.pos0_chunk_cols, c1 = min(P.V, c0 + P.pos0_chunk_cols);
  const T* L = static_cast<const T*>(P.longp) + (long long)b * P.n * P.V;
  float best = -INFINITY, second = -INFINITY, m = -INFINITY, s = 0.f;
  int idx = INT_MAX;
  constexpr int U = 4;
  const int step = kEpiThreads * 8;
  for (int cb = c0 + ep * 8; cb < c1; cb += step * U) {
    float lv[U][8];
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (cb + u * step < c1) load8(L + cb + u * step, lv[u]);
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int c = cb + u * step;
      if (c < c1) {
#pragma unroll
        for (int i = 0; i < 8; ++i) top2_push(lv[u][i], c + i, best, second, idx);
        lse_chunk<8>(lv[u], best, m, s);
      }
    }
  }
  RowAcc x;
  x.m = best; x.s = s; x.second = second; x.idx = idx;
  x = epi_block_reduce(x, red, ep);
  if (ep == 0)
    reinterpret_cast<float4*>(P.partials)[(long long)b * P.partial_ld + ch] =
        make_float4(x.m, x.s, x.second, __int_as_float(x.idx));
}

// Merge of position j for request b = blockIdx.x: emit x_j, then gather the
// GRU input E_tgt[x_j] for the next position (and clear the state at j = 0).
__device__ __forceinline__ void merge_phase(const PersistGruArgs& P, int j, int count, bool gather, RowAcc* red,
                                            int* s_tok, int ep) {
  const int b = blockIdx.x;
  if (b >= P.B) return;
  RowAcc x = rowacc_init();
  for (int k = ep; k < count; k += kEpiThreads) {
    const float4 v = __ldcg(reinterpret_cast<const float4*>(P.partials) + (long long)b * P.partial_ld + k);
    RowAcc y;
    y.m = v.x; y.s = v.y; y.second = v.z; y.idx = __float_as_int(v.w);
    x = rowacc_merge(x, y);
  }
  x = epi_block_reduce(x, red, ep);
  if (ep == 0) {
    write_decode(x, (long long)b * P.n + j, P);
    *s_tok = rowacc_valid(x) ? x.idx : -1;
  }
  named_bar_sync<3>(kEpiThreads);
  const int tok = *s_tok;
  if (j == 0) {
    for (int i = ep; i < P.H; i += kEpiThreads) {
      P.h[(long long)i * P.B + b] = 0.f;
      P.hb[(long long)b * P.H + i] = 0;
    }
  }
  if (gather) {
    const int nv = P.D * 2 / 16;   // 16-byte pieces of one embedding row
    uint4* dst = reinterpret_cast<uint4*>(P.eg + (long long)b * P.D);
    if (tok < 0) {
      for (int i = ep; i < nv; i += kEpiThreads) dst[i] = make_uint4(0, 0, 0, 0);
    } else {
      const uint4* src = reinterpret_cast<const uint4*>(P.emb + (long long)tok * P.D);
      for (int i = ep; i < nv; i += kEpiThreads) dst[i] = __ldg(src + i);
    }
  }
}

__device__ __forceinline__ float sigmoid_(float x) { return 1.f / (1.f + __expf(-x)); }

// GRU gates (PyTorch bias-free form, gate rows r, z, n) over the whole batch,
// spread across every CTA's epilogue threads. Partials and the state are
// batch-fastest ([.., unit, b]), so consecutive threads read and write
// consecutive addresses; the bf16 copy feeds the next products as [b, unit].
__device__ __forceinline__ void gates_phase(const PersistGruArgs& P, int S0, int S1, int ep) {
  const int H = P.H, B = P.B;
  const long long total = (long long)B * H;
  const long long split_stride = (long long)3 * H * B;
  for (long long e = (long long)blockIdx.x * kEpiThreads + ep; e < total; e += (long long)gridDim.x * kEpiThreads) {
    const int i = (int)(e / B), b = (int)(e % B);
    const long long base = (long long)i * B + b;
    const long long gH = (long long)H * B;
    float gir = 0.f, giz = 0.f, gin = 0.f, ghr = 0.f, ghz = 0.f, ghn = 0.f;
    for (int s = 0; s < S0; ++s) {
      const float* p = P.gpart + s * split_stride + base;
      gir += __ldcg(p); giz += __ldcg(p + gH); gin += __ldcg(p + 2 * gH);
    }
    for (int s = S0; s < S0 + S1; ++s) {
      const float* p = P.gpart + s * split_stride + base;
      ghr += __ldcg(p); ghz += __ldcg(p + gH); ghn += __ldcg(p + 2 * gH);
    }
    const float r = sigmoid_(gir + ghr);
    const float z = sigmoid_(giz + ghz);
    const float c = tanhf(gin + r * ghn);
    const float hp = __ldcg(P.h + base);
    const float hn = (1.f - z) * c + z * hp;
    P.h[base] = hn;
    P.hb[(long long)b * H + i] = f32_to_bf16_rne(hn);
  }
}

__global__ void __launch_bounds__(kThreads, 1)
    k_draft_gru(const __grid_constant__ CUtensorMap m_eg, const __grid_constant__ CUtensorMap m_wih,
                const __grid_constant__ CUtensorMap m_hb, const __grid_constant__ CUtensorMap m_whh,
                const __grid_constant__ CUtensorMap m_hb_rank, const __grid_constant__ CUtensorMap m_wrank,
                const __grid_constant__ CUtensorMap m_r, const __grid_constant__ CUtensorMap m_wvocab,
                const __grid_constant__ CUtensorMap m_long, const PersistGruArgs P, uint64_t budget_ns) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  const Smem lay = smem_layout(P);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

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
  uint64_t* mmadone = c.afull + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mmadone + 1);
  c.abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  int* s_tok = const_cast<int*>(c.abort_flag + 1);
  c.S = P.stages;
  c.a_stage_bytes = a_stage_bytes(P);
  c.b_stage_bytes = 128u * 128u;
  c.l_buf_bytes = (uint32_t)(P.vocab.l_boxes * P.vocab.l_box_rows * 128);
  c.deadline = globaltimer_ns() + budget_ns;

  if (threadIdx.x == 0) {
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
    *c.abort_flag = 0;
    fence_mbarrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&m_eg);
    tma_prefetch_desc(&m_wih);
    tma_prefetch_desc(&m_hb);
    tma_prefetch_desc(&m_whh);
    tma_prefetch_desc(&m_hb_rank);
    tma_prefetch_desc(&m_wrank);
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

  Phase pg{&P.gru, &m_eg, &m_wih, &m_hb, &m_whh, &m_long, 0, 0, 1, 0};
  Phase pr{&P.rank, &m_hb_rank, &m_wrank, &m_hb_rank, &m_wrank, &m_long, 0, 0, 1, 0};
  Phase pv{&P.vocab, &m_r, &m_wvocab, &m_r, &m_wvocab, &m_long, 0, 0, 1, 1};
  item_range(P.gru, blockIdx.x, gridDim.x, pg.first, pg.count, pg.stride);
  item_range(P.rank, blockIdx.x, gridDim.x, pr.first, pr.count, pr.stride);
  item_range(P.vocab, blockIdx.x, gridDim.x, pv.first, pv.count, pv.stride);

  const bool is_prod = warp == 0 && lane == 0;
  const bool is_mma = warp == 1 && lane == 0;
  const bool is_lprod = warp == 10 && lane == 0;
  const bool is_epi = warp >= 2 && warp < 2 + kEpiWarps;
  const int ep = threadIdx.x - 64;
  ProdState ps;
  MmaState ms;
  LState ls;
  EpiState es;
  uint64_t pol_w = 0, pol_act = 0, pol_stream = 0;
  if (is_prod) {
    pol_w = l2_policy_evict_first();
    pol_act = l2_policy_evict_last();
  }
  if (is_lprod) pol_stream = l2_policy_evict_first();
  // the next tensor-core phase with work for this CTA after `which`
  // (0 = GRU, 1 = rank, 2 = vocab of the same position, 3 = GRU of the next)
  auto next_phase = [&](int which) -> const Phase* {
    if (which < 1 && pr.count > 0) return &pr;
    if (which < 2) return &pv;
    if (pg.count > 0) return &pg;
    if (pr.count > 0) return &pr;
    return &pv;
  };

  const int n = P.n;
  bool ok = true;
  // barrier generation: no CTA can pass the first barrier before this one
  // arrives, so the value read here is the current generation for everyone
  unsigned bar_gen = 0;
  if (threadIdx.x == 0) bar_gen = ld_acquire_gpu(P.grid_bar + 32);
  // ---- start the weight / logits streams of the first phases
  if (n > 1) {
    if (is_prod) prod_prefetch(c, pg.count > 0 ? pg : *next_phase(0), ps, pol_w);
    if (is_lprod) lprod_issue(c, pv, ls, 2, pol_stream);
    if (is_epi) epi_stage_prior(c, pv, ep);
  }
  // ---- position 0
  if (is_epi) {
    if (P.long_f32) pos0_phase<float>(P, c.red, ep);
    else pos0_phase<uint16_t>(P, c.red, ep);
  }
  ok = grid_sync(P.grid_bar, bar_gen, P.abort_global, c.abort_flag, c.deadline);
  if (ok && is_epi) merge_phase(P, 0, P.pos0_chunks, n > 1, c.red, s_tok, ep);
  for (int j = 1; j < n && ok; ++j) {
    pv.j = j;
    ok = grid_sync(P.grid_bar, bar_gen, P.abort_global, c.abort_flag, c.deadline);
    if (!ok) break;
    // GRU gate products: E_tgt[x_{j-1}] W_ih^T and bf16(h_{j-1}) W_hh^T (split K)
    if (is_prod) {
      prod_run(c, pg, ps, pol_w, pol_act);
      prod_prefetch(c, *next_phase(0), ps, pol_w);
    } else if (is_mma) {
      mma_run(c, pg, ms);
    } else if (is_epi) {
      epi_run<false>(c, pg, es, warp, lane, blockIdx.x);
    }
    if (!(ok = grid_sync(P.grid_bar, bar_gen, P.abort_global, c.abort_flag, c.deadline))) break;
    if (is_epi) gates_phase(P, P.gru.seg_splits[0], P.gru.seg_splits[1], ep);
    if (!(ok = grid_sync(P.grid_bar, bar_gen, P.abort_global, c.abort_flag, c.deadline))) break;
    // r_j = SiLU(W_rank h_j), bf16
    if (is_prod) {
      prod_run(c, pr, ps, pol_w, pol_act);
      if (pr.count > 0) prod_prefetch(c, pv, ps, pol_w);
    } else if (is_mma) {
      mma_run(c, pr, ms);
    } else if (is_epi) {
      epi_run<false>(c, pr, es, warp, lane, blockIdx.x);
    }
    if (!(ok = grid_sync(P.grid_bar, bar_gen, P.abort_global, c.abort_flag, c.deadline))) break;
    // vocabulary projection fused with the combine
    if (is_prod) {
      prod_run(c, pv, ps, pol_w, pol_act);
      if (j + 1 < n) prod_prefetch(c, *next_phase(2), ps, pol_w);
    } else if (is_mma) {
      mma_run(c, pv, ms);
    } else if (is_epi) {
      epi_run<true>(c, pv, es, warp, lane, blockIdx.x);
    } else if (is_lprod) {
      lprod_issue(c, pv, ls, INT_MAX, pol_stream);
      if (j + 1 < n) {
        Phase nx = pv;
        nx.j = j + 1;
        ls.pre = 0;
        lprod_issue(c, nx, ls, 2, pol_stream);
      }
    }
    if (!(ok = grid_sync(P.grid_bar, bar_gen, P.abort_global, c.abort_flag, c.deadline))) break;
    if (is_epi) merge_phase(P, j, gridDim.x, j + 1 < n, c.red, s_tok, ep);
  }

  // ---- teardown: let in-flight tensor-core work and copies finish (bounded)
  if (is_mma) {
    tc_commit(mmadone);
    volatile int dummy = 0;
    mbar_wait(mmadone, 0, globaltimer_ns() + 100000000ull, &dummy);
  }
  if (is_prod && *c.abort_flag) {
    const uint64_t dd = globaltimer_ns() + 100000000ull;
    volatile int dummy = 0;
    const int issued = max(ps.fills, ps.pre_end);
    for (int k = max(0, issued - c.S); k < issued; ++k) mbar_wait(&c.full[k % c.S], (k / c.S) & 1, dd, &dummy);
  }
  if (is_lprod && *c.abort_flag) {
    const uint64_t dd = globaltimer_ns() + 100000000ull;
    volatile int dummy = 0;
    for (int t = max(0, ls.tiles - 2); t < ls.tiles; ++t) mbar_wait(&c.lfull[t & 1], (t >> 1) & 1, dd, &dummy);
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0 && *c.abort_flag) raise_status(P.status, DELS_STATUS_TIMEOUT);
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(c.tmem_base, kTmemCols);
  }
}

}  // namespace

size_t draft_gru_smem_bytes(const PersistGruArgs& P) { return smem_layout(P).total; }

cudaError_t launch_draft_gru(const PersistGruArgs& P, const CUtensorMap* maps, int grid, size_t smem,
                             cudaStream_t s) {
  cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void*>(k_draft_gru), smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k_draft_gru, maps[0], maps[1], maps[2], maps[3], maps[4], maps[5], maps[6],
                            maps[7], maps[8], P, (uint64_t)kWaitBudgetNs);
}

}  // namespace dels
