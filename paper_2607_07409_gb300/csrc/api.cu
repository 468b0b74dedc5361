// C ABI of the drafting hot path: argument validation, workspace layout,
// TMA descriptor encoding, and the per-block orchestration of Algorithm 1
// (position 0 from the long logits alone, then local head -> vocabulary
// projection + fused combine -> merge/feedback for positions 1..n-1).
#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <vector>

#include "dels_internal.h"

namespace dels {

// ---------------------------------------------------------------- utilities

int device_sm_count() {
  int dev = 0, v = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return v;
}

int device_max_smem_optin() {
  int dev = 0, v = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess) return 0;
  return v;
}

cudaError_t ensure_dynamic_smem(const void* kernel, size_t bytes) {
  struct Entry {
    const void* kernel;
    int dev;
    size_t bytes;
  };
  static std::mutex mu;
  static std::vector<Entry> done;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  for (Entry& x : done) {
    if (x.kernel != kernel || x.dev != dev) continue;
    if (x.bytes >= bytes) return cudaSuccess;
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e == cudaSuccess) x.bytes = bytes;
    return e;
  }
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  if (e == cudaSuccess) done.push_back(Entry{kernel, dev, bytes});
  return e;
}

namespace {

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
inline size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

}  // namespace

bool encode_tmap_2d(CUtensorMap* m, const void* base, CUtensorMapDataType dt, int elem_bytes, uint64_t inner,
                    uint64_t outer, uint64_t row_pitch_bytes, uint32_t box_inner, uint32_t box_outer,
                    CUtensorMapSwizzle swz) {
  EncodeTiledFn fn = get_encode_fn();
  if (!fn) return false;
  (void)elem_bytes;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {row_pitch_bytes};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t es[2] = {1, 1};
  return fn(m, dt, 2, const_cast<void*>(base), dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_tmap_3d(CUtensorMap* m, const void* base, CUtensorMapDataType dt, int elem_bytes, uint64_t d0,
                    uint64_t d1, uint64_t d2, uint64_t pitch1_bytes, uint64_t pitch2_bytes, uint32_t b0, uint32_t b1,
                    uint32_t b2, CUtensorMapSwizzle swz) {
  EncodeTiledFn fn = get_encode_fn();
  if (!fn) return false;
  (void)elem_bytes;
  cuuint64_t dims[3] = {d0, d1, d2};
  cuuint64_t strides[2] = {pitch1_bytes, pitch2_bytes};
  cuuint32_t box[3] = {b0, b1, b2};
  cuuint32_t es[3] = {1, 1, 1};
  return fn(m, dt, 3, const_cast<void*>(base), dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}


// ------------------------------------------------------- optional profiler
namespace prof {
bool on = false;
struct Rec {
  int cls;
  cudaEvent_t a, b;
};
std::vector<Rec> recs;
std::vector<cudaEvent_t> pool;

cudaEvent_t take() {
  if (!pool.empty()) {
    cudaEvent_t e = pool.back();
    pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  return cudaEventCreate(&e) == cudaSuccess ? e : nullptr;
}

// Brackets one kernel launch with events on its stream while profiling is on.
struct Scope {
  int cls;
  cudaStream_t s;
  cudaEvent_t a = nullptr;
  Scope(int c, cudaStream_t st) : cls(c), s(st) {
    if (on) {
      a = take();
      if (a && cudaEventRecord(a, s) != cudaSuccess) {
        pool.push_back(a);
        a = nullptr;
      }
    }
  }
  ~Scope() {
    if (!a) return;
    cudaEvent_t b = take();
    if (b && cudaEventRecord(b, s) == cudaSuccess) {
      recs.push_back({cls, a, b});
    } else {
      pool.push_back(a);
      if (b) pool.push_back(b);
    }
  }
};
}  // namespace prof

#define PROF(cls) prof::Scope prof_scope_(cls, s)

namespace {

// ------------------------------------------------------------- tcgen05 plans

struct Gemm {
  TcGemmArgs a{};
  CUtensorMap mA0{}, mB0{}, mA1{}, mB1{}, mL{};
  int grid = 0;
  size_t smem = 0;
};

constexpr int kSmemReserve = 512 + 2 * 128 * 16 + 1024 + 256;   // barriers, reduction scratch, alignment slack
constexpr int kMaxStagesHost = 12;                                 // the engine's ring limit

// A = X [B, K] bf16 (row pitch K*2), boxes of `box_rows` rows; W = [O, K] bf16.
bool map_x(CUtensorMap* m, const void* X, int B, int K, int box_rows) {
  return encode_tmap_2d(m, X, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (uint64_t)K, (uint64_t)B, (uint64_t)K * 2, 64,
                        (uint32_t)box_rows, CU_TENSOR_MAP_SWIZZLE_128B);
}
bool map_w(CUtensorMap* m, const void* W, int O, int K, int n_tile) {
  return encode_tmap_2d(m, W, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (uint64_t)K, (uint64_t)O, (uint64_t)K * 2, 64,
                        (uint32_t)n_tile, CU_TENSOR_MAP_SWIZZLE_128B);
}

int pick_stages(const TcGemmArgs& a, int per_stage, int fixed) {
  const int budget = device_max_smem_optin() - kSmemReserve - fixed;
  int st = budget / per_stage;
  return std::max(2, std::min(st, 12));
}

// Y = act(X0 W0^T) over K split into `splits` pieces (segment 1 optional:
// + X1 W1^T with its own splits, written as separate partials).
bool plan_store(Gemm& g, int B, int O, const void* X0, const void* W0, int K0, const void* X1, const void* W1,
                int K1, int n_tile, int splits0, int splits1, int act, float* out_f32, uint16_t* out_bf16,
                int ldo_bf16, int* status, int sms) {
  TcGemmArgs& a = g.a;
  a.B = B;
  a.O = O;
  a.n_tile = n_tile;
  a.num_o_tiles = (O + n_tile - 1) / n_tile;
  a.seg_chunks[0] = (K0 + 63) / 64;
  a.seg_chunks[1] = K1 > 0 ? (K1 + 63) / 64 : 0;
  // make every split non-empty
  auto fix = [](int nch, int s) {
    if (nch == 0) return 0;
    s = std::max(1, std::min(s, nch));
    const int per = (nch + s - 1) / s;
    return (nch + per - 1) / per;
  };
  a.seg_splits[0] = fix(a.seg_chunks[0], splits0);
  a.seg_splits[1] = fix(a.seg_chunks[1], splits1);
  a.total_splits = a.seg_splits[0] + a.seg_splits[1];
  a.epi = EPI_STORE;
  a.a_resident = 0;
  a.act = act;
  a.out_f32 = out_f32;
  a.out_split_stride = (long long)B * O;
  a.ldo = O;
  a.out_bf16 = out_bf16;
  a.ldo_bf16 = ldo_bf16;
  a.status = status;
  // only the B real rows are loaded; the tile's other rows feed unused outputs
  a.a_box_rows = std::min(128, (B + 7) / 8 * 8);
  a.a_copies = 1;
  a.stages = pick_stages(a, 128 * 128 + n_tile * 128, (out_f32 && !out_bf16) ? kStoreTransposeBytes : 0);
  if (!map_x(&g.mA0, X0, B, K0, a.a_box_rows) || !map_w(&g.mB0, W0, O, K0, n_tile)) return false;
  if (K1 > 0) {
    if (!map_x(&g.mA1, X1, B, K1, a.a_box_rows) || !map_w(&g.mB1, W1, O, K1, n_tile)) return false;
  } else {
    g.mA1 = g.mA0;
    g.mB1 = g.mB0;
  }
  g.mL = g.mA0;
  const int items = a.num_o_tiles * a.total_splits;
  g.grid = std::min(items, std::max(1, sms));
  g.smem = tc_gemm_smem_bytes(a);
  return true;
}

// Splits for `tiles` output tiles when the items (tiles x splits) may take
// more than one wave: the split count with the shortest makespan in item
// time, ceil(tiles s / sms) / s, plus 2 % per split for the partials written
// and re-read (80 tiles on 152 SMs: 5 splits, 0.6 of one tile's time, where
// one split left 72 SMs idle).
int splits_balanced(int O, int n_tile, int K, int sms) {
  const int tiles = (O + n_tile - 1) / n_tile;
  const int nch = (K + 63) / 64;
  const int smax = std::min(nch, 32);
  int best = 1;
  double best_cost = 1e30;
  for (int sp = 1; sp <= smax; ++sp) {
    const long long waves = ((long long)tiles * sp + sms - 1) / std::max(1, sms);
    const double cost = (double)waves / sp + 0.02 * sp;
    if (cost < best_cost - 1e-9) {
      best_cost = cost;
      best = sp;
    }
  }
  return best;
}

// Splits so that tiles x splits roughly fills the GPU once.
int splits_for(int O, int n_tile, int K, int sms) {
  const int tiles = (O + n_tile - 1) / n_tile;
  const int nch = (K + 63) / 64;
  int s = std::max(1, sms / std::max(1, tiles));
  return std::min(s, nch);
}

// Vocabulary projection fused with the combine (l_L tile of position j).
bool plan_combine(Gemm& g, int B, int V, int n, const void* X, int K, const void* Wv, const void* longp,
                  dels_dtype ldt, const float* prior, float alpha, float beta, void* partials, int partial_ld,
                  int* status, int sms, bool pair_stages) {
  TcGemmArgs& a = g.a;
  const int n_tile = 128;
  a.B = B;
  a.O = V;
  a.V = V;
  a.n_tile = n_tile;
  a.num_o_tiles = (V + n_tile - 1) / n_tile;
  a.seg_chunks[0] = (K + 63) / 64;
  a.seg_chunks[1] = 0;
  a.seg_splits[0] = 1;
  a.seg_splits[1] = 0;
  a.total_splits = 1;
  a.epi = EPI_COMBINE;
  a.prior = prior;
  a.alpha = alpha;
  a.beta = beta;
  a.long_f32 = (ldt == DELS_F32);
  a.l_box_cols = a.long_f32 ? 32 : 64;
  a.l_box_rows = std::min(128, (B + 7) / 8 * 8);
  a.l_boxes = n_tile / a.l_box_cols;
  a.partials = partials;
  a.partial_ld = partial_ld;
  a.status = status;
  const int grid = std::min(a.num_o_tiles, std::max(1, sms));
  a.max_items_per_cta = (a.num_o_tiles + grid - 1) / grid;
  const int l_fixed = 2 * a.l_boxes * a.l_box_rows * 128 + a.max_items_per_cta * n_tile * 4;
  a.a_resident = (a.seg_chunks[0] <= 4) ? 1 : 0;
  const int es = a.long_f32 ? 4 : 2;
  // Rows of the A tile: the B requests rounded up to whole TMEM lane
  // quadrants; when that is 32 or 64 rows, 4 or 2 copies fill the tile so
  // every epilogue warp owns live rows (the copies split the columns).
  const int rpc = (B + 31) / 32 * 32;
  a.a_box_rows = rpc;
  a.a_copies = (rpc == 32) ? 4 : (rpc == 64 ? 2 : 1);
  if (!a.a_resident && B <= 32) {
    // Activations staged with every K chunk: load only the live rows, once.
    // The copies (and a 32-row box for a handful of requests) would make
    // every CTA fetch the same few L2 lines four times per stage, while a
    // long K leaves the epilogue ample time for the rows of one quadrant.
    a.a_box_rows = (B + 7) / 8 * 8;
    a.a_copies = 1;
  }
  if (a.a_resident) {
    a.stages = pick_stages(a, n_tile * 128, a.seg_chunks[0] * 128 * 128 + l_fixed);
  } else {
    a.stages = pick_stages(a, 128 * 128 + n_tile * 128, l_fixed);
  }
  // An even number of K chunks: each pipeline stage holds two consecutive
  // chunks, the weights' as one 3-D box (8B-shaped launch 29.2 -> 26.8 us;
  // with staged activations, 0.6B-shaped 59.6 -> 53.9 us, 4B-shaped
  // 130.9 -> 126.5 us).
  if (pair_stages && a.seg_chunks[0] % 2 == 0) {
    a.b_chunks = 2;
    a.stages = std::max(2, a.stages / 2);
  }
  if (!map_x(&g.mA0, X, B, K, a.a_box_rows)) return false;
  if (a.b_chunks == 2) {
    if (!encode_tmap_3d(&g.mB0, Wv, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, 64, (uint64_t)V, (uint64_t)(K / 64),
                        (uint64_t)K * 2, 128, 64, (uint32_t)n_tile, 2, CU_TENSOR_MAP_SWIZZLE_128B))
      return false;
  } else if (!map_w(&g.mB0, Wv, V, K, n_tile)) {
    return false;
  }
  if (!encode_tmap_3d(&g.mL, longp, a.long_f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16,
                      es, (uint64_t)V, (uint64_t)n, (uint64_t)B, (uint64_t)V * es, (uint64_t)n * V * es,
                      (uint32_t)a.l_box_cols, 1, (uint32_t)a.l_box_rows, CU_TENSOR_MAP_SWIZZLE_128B))
    return false;
  g.mA1 = g.mA0;
  g.mB1 = g.mB0;
  g.grid = grid;
  g.smem = tc_gemm_smem_bytes(a);
  return true;
}

cudaError_t run(const Gemm& g, cudaStream_t s) {
  return launch_tc_gemm(g.a, &g.mA0, &g.mB0, &g.mA1, &g.mB1, &g.mL, g.grid, g.smem, s);
}

// bf16 GRU heads have two drafting paths that compute the same block: the
// per-position kernel sequence chained by programmatic dependent launch (the
// default, and the faster one as measured), and one cooperative persistent
// launch per block with grid-wide barriers between phases, selected by
// DELS_DRAFT_PERSISTENT=1 in the environment.
// The input-table path's products of h_j and the vocabulary projection run
// as two launches (default, faster as measured) or as one cooperative launch
// (DELS_DRAFT_FUSED=1 in the environment); both compute the same block.
bool fused_products_enabled() {
  const char* e = std::getenv("DELS_DRAFT_FUSED");
  return e && e[0] == '1';
}

bool persistent_enabled() {
  const char* e = std::getenv("DELS_DRAFT_PERSISTENT");
  return e && e[0] == '1';
}

// A store product over `rows` activation rows that may exceed one 128-row
// tile (the transformer head's three-term rows, 3B): ceil(rows / 128)
// launches over consecutive row blocks, all writing one partial buffer
// [S][rows][O].
struct RowBlocks {
  Gemm g[3];
  int count = 0;
};

bool plan_store_rows(RowBlocks& rb, int rows, int O, const uint16_t* X, const void* W, int K, int splits,
                     float* part, int* status, int sms) {
  rb.count = 0;
  for (int r0 = 0; r0 < rows; r0 += kMaxBatchTile) {
    if (rb.count >= 3) return false;
    const int m = std::min(kMaxBatchTile, rows - r0);
    Gemm& g = rb.g[rb.count++];
    if (!plan_store(g, m, O, X + (size_t)r0 * K, W, K, nullptr, nullptr, 0, 128, splits, 0, ACT_NONE,
                    part + (size_t)r0 * O, nullptr, 0, status, sms))
      return false;
    g.a.out_split_stride = (long long)rows * O;
  }
  return rb.count > 0;
}

cudaError_t run_rows(const RowBlocks& rb, cudaStream_t s) {
  for (int i = 0; i < rb.count; ++i) {
    const cudaError_t e = run(rb.g[i], s);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

// ------------------------------------------------------------ draft layout

// Transformer head: every activation that feeds one of the head's own bf16
// products is passed as its exact three-term bf16 expansion (hi + mid + lo,
// stacked as extra rows of the product), so those products equal float32
// products; only the feature fed to W_vocab is rounded to bf16.
constexpr int kXfmrTerms = 3;

// Input-table GRU path: output tile widths of the rank product and of the
// recurrent product (both split over K).
constexpr int kRankTile = 32;
constexpr int kRankSplits = 4;     // K splits of the rank product (grouped launch)
constexpr int kRankClusterSplits = 2;   // ... in the cooperative products+vocabulary launch (2-CTA clusters)
constexpr size_t kRReadyOff = 128; // workspace header: rank tiles finished in the current block
constexpr int kHhTile = 64;

struct Carve {
  size_t off = kHeaderBytes;
  size_t take(size_t bytes) {
    const size_t o = off;
    off = round_up(off + bytes, 256);
    return o;
  }
};

struct DraftLayout {
  bool ok = false;
  int sms = 0;
  int partial_ld = 0;
  size_t partials = 0;
  // GRU
  size_t eg = 0, h = 0, hb = 0, gpart = 0, r = 0;
  int gru_s0 = 0, gru_s1 = 0;
  int rank_grid = 0, hh_splits = 0;          // input-table path: grouped rank + recurrent product
  // MLP
  size_t u = 0, mpart = 0, h1 = 0, h2 = 0;
  int mlp_s1 = 0, mlp_s2 = 0;
  // XFMR
  size_t ex = 0, t = 0, ab = 0, q = 0, kc = 0, vc = 0, xpart = 0, wqkv = 0, xpqkv = 0, ob = 0, uu = 0, anb = 0, fb = 0,
         y = 0, feat = 0;
  int xs_qkv = 0, xs_o = 0, xs_1 = 0, xs_2 = 0;
  // MARKOV
  size_t mk = 0;
  size_t total = 0;
};

int head_es(const dels_local_head* h) { return h->wdtype == DELS_F32 ? 4 : 2; }

DraftLayout draft_layout(const dels_local_head* hd, int B, int n, int V) {
  DraftLayout L;
  L.sms = device_sm_count();
  if (L.sms <= 0) return L;
  const int sms = L.sms;
  Carve c;
  L.partial_ld = std::max(sms, 16 * sms / std::max(1, B) + 1);
  L.partials = c.take((size_t)B * L.partial_ld * 16);
  const int es = head_es(hd);
  const bool bf = hd->wdtype == DELS_BF16;
  switch (hd->kind) {
    case DELS_HEAD_GRU: {
      const int D = hd->d_model, H = hd->d_hidden, R = hd->d_rank;
      L.eg = c.take((size_t)B * D * es);
      L.h = c.take((size_t)B * H * 4);
      L.hb = c.take((size_t)B * H * 2);
      if (bf) {
        L.gru_s0 = std::max(1, std::min((D + 63) / 64, sms / std::max(1, (3 * H + 127) / 128) - 1));
        L.gru_s1 = 1;
        L.rank_grid = (R + kRankTile - 1) / kRankTile * kRankSplits;
        L.hh_splits = splits_for(3 * H, kHhTile, H, std::max(1, sms - L.rank_grid));
      } else {
        L.gru_s0 = 1;
        L.gru_s1 = 1;
      }
      L.gpart = c.take((size_t)std::max(L.gru_s0 + L.gru_s1, L.hh_splits) * B * 3 * H * 4);

      L.r = c.take((size_t)B * R * es);
      break;
    }
    case DELS_HEAD_MLP: {
      const int D = hd->d_model, Hd = hd->d_hidden, W = hd->window;
      L.u = c.take((size_t)B * W * D * es);
      L.mlp_s1 = bf ? splits_for(Hd, 128, W * D, sms) : 1;
      L.mlp_s2 = bf ? splits_for(Hd, 128, Hd, sms) : 1;
      L.mpart = c.take((size_t)std::max(L.mlp_s1, L.mlp_s2) * B * Hd * 4);
      L.h1 = c.take((size_t)B * Hd * es);
      L.h2 = c.take((size_t)B * Hd * es);
      break;
    }
    case DELS_HEAD_XFMR: {
      // the activations of the head's products are three-term bf16
      // expansions (kXfmrTerms rows per request, see launch_splitk_finish)
      const int D = hd->d_model, F = hd->d_hidden, P = hd->max_pos, T = kXfmrTerms;
      L.ex = c.take((size_t)B * D * 2);
      L.t = c.take((size_t)B * D * 4);
      L.ab = c.take((size_t)T * B * D * 2);
      L.q = c.take((size_t)B * D * 4);
      L.kc = c.take((size_t)B * P * D * 4);
      L.vc = c.take((size_t)B * P * D * 4);
      L.xs_qkv = splits_balanced(3 * D, 128, D, sms);
      L.xs_o = splits_balanced(D, 128, D, sms);
      L.xs_1 = splits_balanced(F, 128, D, sms);
      L.xs_2 = splits_balanced(D, 128, F, sms);
      const int smax = std::max(std::max(L.xs_qkv, L.xs_o), std::max(L.xs_1, L.xs_2));
      L.xpart = c.take((size_t)smax * T * B * std::max(D, F) * 4);
      // W_q, W_k and W_v stacked as one [3 d_model, d_model] matrix (copied
      // here unless the caller's three matrices are already contiguous): the
      // three products of a position are one launch, with their partials
      L.wqkv = c.take((size_t)3 * D * D * 2);
      L.xpqkv = c.take((size_t)L.xs_qkv * T * B * 3 * D * 4);
      L.ob = c.take((size_t)T * B * D * 2);
      L.uu = c.take((size_t)B * D * 4);
      L.anb = c.take((size_t)T * B * D * 2);
      L.fb = c.take((size_t)T * B * F * 2);
      L.y = c.take((size_t)B * D * 4);
      L.feat = c.take((size_t)B * D * 2);
      break;
    }
    case DELS_HEAD_MARKOV: {
      L.mk = c.take((size_t)B * hd->d_rank * es);
      break;
    }
    default:
      return L;
  }
  L.total = c.off;
  L.ok = true;
  return L;
}

int validate_head(const dels_local_head* h, int n) {
  if (!h) return DELS_ERR_NULL_POINTER;
  if (h->wdtype != DELS_F32 && h->wdtype != DELS_BF16) return DELS_ERR_BAD_DTYPE;
  const bool bf = h->wdtype == DELS_BF16;
  auto dim_ok = [&](int d) { return d > 0 && d <= 65536 && (!bf || d % 16 == 0) && (bf || d % 4 == 0); };
  if (!h->emb || !h->w_vocab) return DELS_ERR_NULL_POINTER;
  if (!aligned16(h->emb) || !aligned16(h->w_vocab)) return DELS_ERR_ALIGNMENT;
  for (int i = 0; i < 8; ++i)
    if (h->w[i] && !aligned16(h->w[i])) return DELS_ERR_ALIGNMENT;
  switch (h->kind) {
    case DELS_HEAD_GRU:
      if (!h->w[0] || !h->w[1] || !h->w[2]) return DELS_ERR_NULL_POINTER;
      if (!dim_ok(h->d_model) || !dim_ok(h->d_hidden) || !dim_ok(h->d_rank)) return DELS_ERR_BAD_SHAPE;
      if (h->d_rank > 4096) return DELS_ERR_BAD_SHAPE;
      return DELS_OK;
    case DELS_HEAD_MLP:
      if (!h->w[0] || (h->n_layers == 2 && !h->w[1])) return DELS_ERR_NULL_POINTER;
      if (h->n_layers != 1 && h->n_layers != 2) return DELS_ERR_BAD_SHAPE;
      if (h->window < 1 || h->window > 32) return DELS_ERR_BAD_SHAPE;
      if (!dim_ok(h->d_model) || !dim_ok(h->d_hidden) || h->d_rank != h->d_hidden) return DELS_ERR_BAD_SHAPE;
      return DELS_OK;
    case DELS_HEAD_XFMR:
      if (!bf) return DELS_ERR_UNSUPPORTED;
      for (int i = 0; i < 7; ++i)
        if (!h->w[i]) return DELS_ERR_NULL_POINTER;
      if (!dim_ok(h->d_model) || !dim_ok(h->d_hidden) || h->d_rank != h->d_model) return DELS_ERR_BAD_SHAPE;
      if (h->n_heads < 1 || h->d_model % h->n_heads != 0 || h->max_pos < n) return DELS_ERR_BAD_SHAPE;
      if (h->d_model / h->n_heads > 8192) return DELS_ERR_UNSUPPORTED;   // q of one head in shared memory
      if (h->d_model > 32768) return DELS_ERR_UNSUPPORTED;               // RMSNorm rows: 8 CTAs x 4096 values
      return DELS_OK;
    case DELS_HEAD_MARKOV:
      if (!dim_ok(h->d_rank)) return DELS_ERR_BAD_SHAPE;
      return DELS_OK;
    default:
      return DELS_ERR_UNSUPPORTED;
  }
}

int validate_draft(const dels_local_head* head, const void* long_logits, dels_dtype ldt, const float* prior, int B,
                   int n, int V, const int32_t* tok, const float* lp, const float* gap) {
  if (B < 0 || B > kMaxBatchTile) return DELS_ERR_BAD_SHAPE;
  if (n < 1 || n > 32) return DELS_ERR_BAD_SHAPE;
  if (V < 8 || V % 8 != 0) return DELS_ERR_BAD_SHAPE;
  if (ldt != DELS_F32 && ldt != DELS_BF16) return DELS_ERR_BAD_DTYPE;
  int r = validate_head(head, n);
  if (r != DELS_OK) return r;
  if (B == 0) return DELS_OK;
  if (!long_logits || !prior || !tok || !lp) return DELS_ERR_NULL_POINTER;
  if (!aligned16(long_logits) || !aligned16(prior) || !aligned16(tok) || !aligned16(lp) || (gap && !aligned16(gap)))
    return DELS_ERR_ALIGNMENT;
  return DELS_OK;
}

#define DELS_CUDA(call)                        \
  do {                                         \
    cudaError_t e__ = (call);                  \
    if (e__ != cudaSuccess) return DELS_ERR_CUDA; \
  } while (0)

template <typename T>
T* at(void* ws, size_t off) {
  return reinterpret_cast<T*>(static_cast<uint8_t*>(ws) + off);
}

// Position 0: x_0 = argmax l_L[b, 0, :] as per-chunk records (no merge);
// returns the number of records per request.
int position0_rows(const void* long_logits, dels_dtype ldt, int B, int n, int V, void* partials, int partial_ld,
                   int* status, int sms, cudaStream_t s, int* count, const SampleArgs* smp = nullptr) {
  RowsArgs a{};
  const int es = ldt == DELS_F32 ? 4 : 2;
  RowsPlan p = plan_rows(B, V, es, sms, true, partial_ld);
  if (smp && smp->on) {
    // temperature 1: x_0 is drawn from softmax(l_L^(0)) (Gumbel-max records)
    SampleRowsArgs sa{};
    sa.src = long_logits;
    sa.ld = (long long)n * V;
    sa.rows = B;
    sa.rows_per_request = 1;
    sa.j0 = 0;
    sa.V = V;
    sa.chunk_cols = (int)round_up((size_t)p.chunk_cols, 8);
    sa.nchunks = (V + sa.chunk_cols - 1) / sa.chunk_cols;
    sa.vec = ((sa.ld * es) % 16 == 0 && aligned16(long_logits)) ? 1 : 0;
    sa.seed = smp->seed;
    sa.step = smp->step;
    sa.stream = 0;
    sa.partials = partials;
    sa.partial_ld = partial_ld;
    *count = sa.nchunks;
    { PROF(DELS_KCLASS_POS0); DELS_CUDA(launch_sample_rows(sa, ldt == DELS_F32, s)); }
    return DELS_OK;
  }
  a.longp = long_logits;
  a.rows = B;
  a.V = V;
  a.ld_long = (long long)n * V;
  a.chunk_cols = p.chunk_cols;
  a.nchunks = p.nchunks;
  a.rows_per_cta = 1;
  a.partials = partials;
  a.partial_ld = partial_ld;
  a.status = status;
  *count = p.nchunks;
  { PROF(DELS_KCLASS_POS0); DELS_CUDA(launch_combine_rows(a, ldt, true, false, s)); }
  return DELS_OK;
}

// Position 0 merged (+ the gather of the next input).
int draft_position0(const void* long_logits, dels_dtype ldt, int B, int n, int V, void* partials, int partial_ld,
                    int* status, const MergeArgs& merge_base, int sms, cudaStream_t s) {
  int count = 0;
  const int r = position0_rows(long_logits, ldt, B, n, V, partials, partial_ld, status, sms, s, &count,
                               &merge_base.smp);
  if (r != DELS_OK) return r;
  MergeArgs m = merge_base;
  m.count = count;
  m.j = 0;
  { PROF(DELS_KCLASS_MERGE); DELS_CUDA(launch_draft_merge(m, s)); }
  return DELS_OK;
}

}  // namespace
}  // namespace dels

using namespace dels;

extern "C" {

int dels_version(void) { return 100; }

int dels_profile_enable(int on) {
  prof::on = on != 0;
  return DELS_OK;
}

int dels_profile_reset(void) {
  for (auto& r : prof::recs) {
    cudaEventSynchronize(r.b);
    prof::pool.push_back(r.a);
    prof::pool.push_back(r.b);
  }
  prof::recs.clear();
  return DELS_OK;
}

int dels_profile_read(int kernel_class, int* out_launches, double* out_total_ms) {
  if (!out_launches || !out_total_ms) return DELS_ERR_NULL_POINTER;
  if (kernel_class < 0 || kernel_class >= DELS_KCLASS_COUNT) return DELS_ERR_BAD_SHAPE;
  int nl = 0;
  double ms = 0.0;
  for (auto& r : prof::recs) {
    if (r.cls != kernel_class) continue;
    if (cudaEventSynchronize(r.b) != cudaSuccess) return DELS_ERR_CUDA;
    float t = 0.f;
    if (cudaEventElapsedTime(&t, r.a, r.b) != cudaSuccess) return DELS_ERR_CUDA;
    ms += t;
    ++nl;
  }
  *out_launches = nl;
  *out_total_ms = ms;
  return DELS_OK;
}


const char* dels_status_string(int code) {
  switch (code) {
    case DELS_OK: return "ok";
    case DELS_ERR_NULL_POINTER: return "null pointer";
    case DELS_ERR_BAD_SHAPE: return "size out of supported range";
    case DELS_ERR_BAD_DTYPE: return "unsupported dtype";
    case DELS_ERR_ALIGNMENT: return "pointer or pitch not 16-byte aligned";
    case DELS_ERR_WORKSPACE: return "workspace missing or too small";
    case DELS_ERR_UNSUPPORTED: return "unsupported head configuration";
    case DELS_ERR_CUDA: return "CUDA call failed";
    case DELS_ERR_TOO_LARGE: return "problem exceeds the fixed no-allocation scratch";
    case DELS_STATUS_NONFINITE: return "device: non-finite logits";
    case DELS_STATUS_TIMEOUT: return "device: bounded wait expired";
    case DELS_STATUS_BAD_TOKEN: return "device: draft token out of range";
    default: return "unknown status";
  }
}

int dels_prior_from_counts(const int64_t* counts, int V, double lambda, float* out_log_prior) {
  if (!counts || !out_log_prior) return DELS_ERR_NULL_POINTER;
  if (V < 1 || !(lambda > 0.0)) return DELS_ERR_BAD_SHAPE;
  long double total = 0.0L;
  for (int v = 0; v < V; ++v) {
    if (counts[v] < 0) return DELS_ERR_BAD_SHAPE;
    total += (long double)counts[v] + (long double)lambda;
  }
  for (int v = 0; v < V; ++v) {
    const double p = (double)(((long double)counts[v] + (long double)lambda) / total);
    out_log_prior[v] = (float)std::log(p);
  }
  return DELS_OK;
}

// ------------------------------------------------ unigram prior (Appendix A)

namespace {

struct PriorWs {
  unsigned long long* counts;   // [V] (dels_prior_estimate)
  unsigned long long* tally;    // [2] (dels_prior_estimate)
  unsigned long long* partials; // [kPriorMaxPartials] (sum of the counts)
  unsigned* ticket;
  unsigned long long* total;
  // hot ids on chip (when the plan uses them)
  unsigned* hist;               // [kPriorHistBuckets]
  unsigned* cta_total;          // [select CTAs]
  unsigned* n_hot;
  uint32_t* entries;            // [nent]
  int32_t* slot_id;             // [K]
  int32_t* stage;               // [nent * 15]
  unsigned* hot_partials;       // [ctas][(K + 1) / 2]
  size_t bytes;
};

PriorWs prior_ws_layout(void* ws, int V, const PriorPlan& p) {
  PriorWs w{};
  size_t off = kHeaderBytes;
  w.counts = at<unsigned long long>(ws, off);
  off = round_up(off + (size_t)V * 8, 256);
  w.tally = at<unsigned long long>(ws, off);
  off = round_up(off + 16, 256);
  w.partials = at<unsigned long long>(ws, off);
  off = round_up(off + (size_t)kPriorMaxPartials * 8, 256);
  w.ticket = at<unsigned>(ws, off);
  w.total = at<unsigned long long>(ws, off + 8);
  off = round_up(off + 16, 256);
  if (p.use_hot) {
    w.hist = at<unsigned>(ws, off);
    off = round_up(off + (size_t)kPriorHistBuckets * 4, 256);
    w.cta_total = at<unsigned>(ws, off);
    off = round_up(off + (size_t)p.select_ctas * 4, 256);
    w.n_hot = at<unsigned>(ws, off);
    off = round_up(off + 4, 256);
    w.entries = at<uint32_t>(ws, off);
    off = round_up(off + (size_t)p.nent * 4, 256);
    w.slot_id = at<int32_t>(ws, off);
    off = round_up(off + (size_t)p.K * 4, 256);
    w.stage = at<int32_t>(ws, off);
    off = round_up(off + (size_t)p.nent * 15 * 4, 256);
    w.hot_partials = at<unsigned>(ws, off);
    off = round_up(off + (size_t)p.ctas * ((p.K + 1) / 2) * 4, 256);
  }
  w.bytes = off;
  return w;
}

// Splits [0, N) into a scalar head, a vector range (tokens + head 16-byte
// aligned, mask + head 4-byte aligned, a multiple of 512 positions) and a
// scalar tail; pointers that cannot be aligned together get no vector range.
PriorRange prior_range(const int32_t* tokens, const uint8_t* mask, long long begin, long long n) {
  PriorRange r{};
  r.tokens = tokens + begin;
  r.mask = mask + begin;
  r.n = n;
  r.head = (long long)((16 - (reinterpret_cast<uintptr_t>(r.tokens) & 15u)) & 15u) / 4;
  r.nvec = 0;
  if (r.head >= n || ((reinterpret_cast<uintptr_t>(r.mask) + (uintptr_t)r.head) & 3u) != 0) {
    r.head = 0;
    return r;
  }
  r.nvec = (n - r.head) / 512 * 512;
  return r;
}

// Adds the loss-masked counts of positions [0, N) to `counts` (see the
// kernels' file for the two counting schemes).
int prior_count_impl(const int32_t* tokens, const uint8_t* loss_mask, long long N, int V, unsigned long long* counts,
                     unsigned long long* tally, int* status, const PriorPlan& p, const PriorWs& w, int sms,
                     cudaStream_t s) {
  if (N == 0) return DELS_OK;
  PriorSliceArgs sa{};
  sa.V = V;
  sa.slices = p.slices;
  sa.slice = p.slice;
  sa.counts = counts;
  sa.tally = tally;
  sa.status = status;
  auto slices_over = [&](long long begin, long long n, int max_members) {
    for (long long b = begin; b < begin + n; b += kPriorChunk) {
      sa.range = prior_range(tokens, loss_mask, b, std::min(kPriorChunk, begin + n - b));
      if (launch_prior_slices(sa, p.slice_smem, max_members, sms, s) != cudaSuccess) return false;
    }
    return true;
  };
  if (!p.use_hot) return slices_over(0, N, 1 << 30) ? DELS_OK : DELS_ERR_CUDA;
  // a prefix, exactly, then the hot set from the counts so far
  if (!slices_over(0, p.prefix, 24)) return DELS_ERR_CUDA;
  PriorSelectArgs se{};
  se.counts = counts;
  se.V = V;
  se.K = p.K;
  se.nent = p.nent;
  se.hist = w.hist;
  se.entries = w.entries;
  se.stage = w.stage;
  se.cta_total = w.cta_total;
  se.slot_id = w.slot_id;
  se.n_hot = w.n_hot;
  if (launch_prior_select(se, p.select_ctas, s) != cudaSuccess) return DELS_ERR_CUDA;
  PriorHotArgs ha{};
  ha.V = V;
  ha.K = p.K;
  ha.nent = p.nent;
  ha.ctas = p.ctas;
  ha.entries = w.entries;
  ha.slot_id = w.slot_id;
  ha.n_hot = w.n_hot;
  ha.partials = w.hot_partials;
  ha.counts = counts;
  ha.tally = tally;
  ha.status = status;
  for (long long b = p.prefix; b < N; b += kPriorChunk) {
    ha.range = prior_range(tokens, loss_mask, b, std::min(kPriorChunk, N - b));
    if (launch_prior_hot(ha, p.hot_smem, s) != cudaSuccess) return DELS_ERR_CUDA;
  }
  return DELS_OK;
}

}  // namespace

size_t dels_prior_workspace_bytes(int V, int64_t N) {
  if (V < 1 || N < 0) return 0;
  const int sms = device_sm_count();
  const PriorPlan p = plan_prior(V, N, sms);
  if (!p.ok) return 0;
  return prior_ws_layout(nullptr, V, p).bytes;
}

int dels_prior_count(const int32_t* tokens, const uint8_t* loss_mask, int64_t N, int V, uint64_t* counts,
                     uint64_t* tally, void* workspace, size_t workspace_bytes, dels_stream_t stream) {
  if (N < 0 || V < 1) return DELS_ERR_BAD_SHAPE;
  if (!workspace) return DELS_ERR_WORKSPACE;
  if (!counts || (N > 0 && (!tokens || !loss_mask))) return DELS_ERR_NULL_POINTER;
  if ((reinterpret_cast<uintptr_t>(tokens) & 3u) || (reinterpret_cast<uintptr_t>(counts) & 7u) ||
      (reinterpret_cast<uintptr_t>(tally) & 7u) || !aligned16(workspace))
    return DELS_ERR_ALIGNMENT;
  if (workspace_bytes < (size_t)kHeaderBytes) return DELS_ERR_WORKSPACE;
  if (N == 0) return DELS_OK;
  const int sms = device_sm_count();
  if (sms <= 0) return DELS_ERR_CUDA;
  const PriorPlan p = plan_prior(V, N, sms);
  if (!p.ok) return DELS_ERR_CUDA;
  const PriorWs w = prior_ws_layout(workspace, V, p);
  if (workspace_bytes < w.bytes) return DELS_ERR_WORKSPACE;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  PROF(DELS_KCLASS_PRIOR);
  return prior_count_impl(tokens, loss_mask, N, V, reinterpret_cast<unsigned long long*>(counts),
                          reinterpret_cast<unsigned long long*>(tally), at<int>(workspace, 0), p, w, sms, s);
}

int dels_prior_log(const uint64_t* counts, int V, double lambda, float* out_log_prior, void* workspace,
                   size_t workspace_bytes, dels_stream_t stream) {
  if (V < 1 || !(lambda > 0.0) || !std::isfinite(lambda)) return DELS_ERR_BAD_SHAPE;
  if (!counts || !out_log_prior) return DELS_ERR_NULL_POINTER;
  if (!workspace) return DELS_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(counts) & 7u) || (reinterpret_cast<uintptr_t>(out_log_prior) & 3u) ||
      !aligned16(workspace))
    return DELS_ERR_ALIGNMENT;
  if (workspace_bytes < (size_t)kHeaderBytes + (size_t)V * 8) return DELS_ERR_WORKSPACE;
  const int sms = device_sm_count();
  if (sms <= 0) return DELS_ERR_CUDA;
  const PriorPlan p = plan_prior(V, 0, sms);
  if (!p.ok) return DELS_ERR_CUDA;
  const PriorWs w = prior_ws_layout(workspace, V, p);
  if (workspace_bytes < w.bytes) return DELS_ERR_WORKSPACE;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  PriorLogArgs a{};
  a.counts = reinterpret_cast<const unsigned long long*>(counts);
  a.V = V;
  a.lambda = lambda;
  a.partials = w.partials;
  a.ticket = w.ticket;
  a.total = w.total;
  a.out = out_log_prior;
  PROF(DELS_KCLASS_PRIOR);
  if (launch_prior_total(a, sms, s) != cudaSuccess) return DELS_ERR_CUDA;
  if (launch_prior_log(a, sms, s) != cudaSuccess) return DELS_ERR_CUDA;
  return DELS_OK;
}

int dels_prior_estimate(const int32_t* tokens, const uint8_t* loss_mask, int64_t N, int V, double lambda,
                        float* out_log_prior, uint64_t* out_counts, uint64_t* out_tally, void* workspace,
                        size_t workspace_bytes, dels_stream_t stream) {
  if (N < 0 || V < 1 || !(lambda > 0.0) || !std::isfinite(lambda)) return DELS_ERR_BAD_SHAPE;
  if (!out_log_prior || (N > 0 && (!tokens || !loss_mask))) return DELS_ERR_NULL_POINTER;
  if (!workspace) return DELS_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(tokens) & 3u) || (reinterpret_cast<uintptr_t>(out_log_prior) & 3u) ||
      (reinterpret_cast<uintptr_t>(out_counts) & 7u) || (reinterpret_cast<uintptr_t>(out_tally) & 7u) ||
      !aligned16(workspace))
    return DELS_ERR_ALIGNMENT;
  if (workspace_bytes < (size_t)kHeaderBytes + (size_t)V * 8) return DELS_ERR_WORKSPACE;
  const int sms = device_sm_count();
  if (sms <= 0) return DELS_ERR_CUDA;
  const PriorPlan p = plan_prior(V, N, sms);
  if (!p.ok) return DELS_ERR_CUDA;
  const PriorWs w = prior_ws_layout(workspace, V, p);
  if (workspace_bytes < w.bytes) return DELS_ERR_WORKSPACE;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  PROF(DELS_KCLASS_PRIOR);
  // counts and tally start from zero (they sit next to each other)
  const size_t zero_bytes = reinterpret_cast<uint8_t*>(w.tally + 2) - reinterpret_cast<uint8_t*>(w.counts);
  if (cudaMemsetAsync(w.counts, 0, zero_bytes, s) != cudaSuccess) return DELS_ERR_CUDA;
  const int rc = prior_count_impl(tokens, loss_mask, N, V, w.counts, w.tally, at<int>(workspace, 0), p, w, sms, s);
  if (rc != DELS_OK) return rc;
  PriorLogArgs a{};
  a.counts = w.counts;
  a.V = V;
  a.lambda = lambda;
  a.total = w.tally;   // tally[0] = the number of counted positions = sum_v c(v)
  a.tally = w.tally;
  a.out = out_log_prior;
  a.counts_out = reinterpret_cast<unsigned long long*>(out_counts);
  a.tally_out = reinterpret_cast<unsigned long long*>(out_tally);
  if (launch_prior_log(a, sms, s) != cudaSuccess) return DELS_ERR_CUDA;
  return DELS_OK;
}

int dels_read_status(void* workspace, dels_stream_t stream, int32_t* out_status) {
  if (!workspace || !out_status) return DELS_ERR_NULL_POINTER;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int32_t v = 0;
  if (cudaMemcpyAsync(&v, workspace, sizeof(v), cudaMemcpyDeviceToHost, s) != cudaSuccess) return DELS_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return DELS_ERR_CUDA;
  if (cudaMemsetAsync(workspace, 0, sizeof(v), s) != cudaSuccess) return DELS_ERR_CUDA;
  *out_status = v;
  return DELS_OK;
}

// ----------------------------------------------------------------- combine

size_t dels_combine_workspace_bytes(int rows, int V, dels_dtype dtype) {
  if (rows < 0 || V < 1 || (dtype != DELS_F32 && dtype != DELS_BF16)) return 0;
  const int sms = device_sm_count();
  if (sms <= 0) return 0;
  return combine_layout(rows, V, dtype, sms).total;
}

}  // extern "C"

namespace dels {
// Workspace of dels_combine_argmax: status header, one ticket per row group,
// then the partial records ([rows][partial_ld], 16 bytes each).
CombineLayout combine_layout(int rows, int V, dels_dtype dtype, int sms) {
  CombineLayout L{};
  const int es = dtype == DELS_F32 ? 4 : 2;
  L.vec = (V % 8) == 0;
  L.p = plan_rows(rows, V, 2 * es, sms, L.vec, 1 << 20, true, rows_slots_per_sm(false, dtype));
  const size_t groups = ((size_t)rows + L.p.rows_per_cta - 1) / L.p.rows_per_cta;
  L.tickets_off = kHeaderBytes;
  L.partials_off = round_up(L.tickets_off + groups * 4, 256);
  L.total = round_up(L.partials_off + (size_t)rows * L.p.nchunks * 16, 256);
  return L;
}

int combine_check_inputs(const void* long_logits, const void* short_logits, const float* log_prior,
                         const int32_t* out_token) {
  if (!long_logits || !out_token) return DELS_ERR_NULL_POINTER;
  if (!aligned16(long_logits) || (short_logits && !aligned16(short_logits)) || (log_prior && !aligned16(log_prior)))
    return DELS_ERR_ALIGNMENT;
  return DELS_OK;
}
}  // namespace dels

extern "C" {

int dels_combine_argmax(const void* long_logits, const void* short_logits, dels_dtype dtype, const float* log_prior,
                        float alpha, float beta, int rows, int V, int32_t* out_token, float* out_logprob,
                        float* out_top2_gap, void* workspace, size_t workspace_bytes, dels_stream_t stream) {
  if (dtype != DELS_F32 && dtype != DELS_BF16) return DELS_ERR_BAD_DTYPE;
  if (rows < 0 || V < 1) return DELS_ERR_BAD_SHAPE;
  if (!workspace) return DELS_ERR_WORKSPACE;
  if (rows == 0) return DELS_OK;
  const int chk = combine_check_inputs(long_logits, short_logits, log_prior, out_token);
  if (chk != DELS_OK) return chk;
  if (!aligned16(workspace)) return DELS_ERR_ALIGNMENT;
  const size_t need = dels_combine_workspace_bytes(rows, V, dtype);
  if (need == 0) return DELS_ERR_CUDA;
  if (workspace_bytes < need) return DELS_ERR_WORKSPACE;
  const int sms = device_sm_count();
  const CombineLayout L = combine_layout(rows, V, dtype, sms);
  RowsArgs a{};
  a.longp = long_logits;
  a.shortp = short_logits;
  a.prior = log_prior;
  a.alpha = alpha;
  a.beta = beta;
  a.rows = rows;
  a.V = V;
  a.ld_long = V;
  a.ld_short = V;
  a.chunk_cols = L.p.chunk_cols;
  a.nchunks = L.p.nchunks;
  a.rows_per_cta = L.p.rows_per_cta;
  a.counters = at<int>(workspace, L.tickets_off);
  a.partials = at<void>(workspace, L.partials_off);
  a.partial_ld = L.p.nchunks;
  a.out_token = out_token;
  a.out_lp = out_logprob;
  a.out_gap = out_top2_gap;
  a.status = at<int>(workspace, 0);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  PROF(DELS_KCLASS_COMBINE);
  if (launch_combine_rows(a, dtype, L.vec, true, s) != cudaSuccess) return DELS_ERR_CUDA;
  return DELS_OK;
}

// ------------------------------------------------------------------ verify

// Workspace of dels_verify_block: status header, per-request tickets, then
// the partial records ([B (n + 1)][nchunks]).
struct VerifyLayout {
  bool vec;
  RowsPlan p;
  size_t req_tk, partials, total;
};

VerifyLayout verify_layout(int B, int n, int V, dels_dtype dtype, int sms) {
  VerifyLayout L{};
  const int es = dtype == DELS_F32 ? 4 : 2;
  const size_t rows = (size_t)B * (n + 1);
  L.vec = (V % 8) == 0;
  L.p = plan_rows((int)std::min<size_t>(rows, INT32_MAX), V, es, sms, L.vec, 1 << 20, false,
                  rows_slots_per_sm(true, dtype));
  L.req_tk = kHeaderBytes;
  L.partials = round_up(L.req_tk + (size_t)B * 4, 256);
  L.total = round_up(L.partials + rows * L.p.nchunks * 16, 256);
  return L;
}

size_t dels_verify_workspace_bytes(int B, int n, int V, dels_dtype dtype) {
  if (B < 0 || n < 1 || n > kMaxVerifyBlock || V < 1 || (dtype != DELS_F32 && dtype != DELS_BF16)) return 0;
  if ((long long)B * (n + 1) > INT32_MAX) return 0;
  const int sms = device_sm_count();
  if (sms <= 0) return 0;
  return verify_layout(B, n, V, dtype, sms).total;
}

int dels_verify_block(const int32_t* draft_tokens, const void* target_logits, dels_dtype dtype, int B, int n, int V,
                      int32_t* out_accept_len, int32_t* out_bonus, int32_t* out_target_argmax, void* workspace,
                      size_t workspace_bytes, dels_stream_t stream) {
  if (dtype != DELS_F32 && dtype != DELS_BF16) return DELS_ERR_BAD_DTYPE;
  if (B < 0 || n < 1 || n > kMaxVerifyBlock || V < 1) return DELS_ERR_BAD_SHAPE;
  if ((long long)B * (n + 1) > INT32_MAX) return DELS_ERR_BAD_SHAPE;
  if (!workspace) return DELS_ERR_WORKSPACE;
  if (B == 0) return DELS_OK;
  if (!draft_tokens || !target_logits || !out_accept_len || !out_bonus) return DELS_ERR_NULL_POINTER;
  if (!aligned16(target_logits) || !aligned16(workspace)) return DELS_ERR_ALIGNMENT;
  const size_t need = dels_verify_workspace_bytes(B, n, V, dtype);
  if (need == 0) return DELS_ERR_CUDA;
  if (workspace_bytes < need) return DELS_ERR_WORKSPACE;
  const int sms = device_sm_count();
  const size_t rows = (size_t)B * (n + 1);
  const VerifyLayout L = verify_layout(B, n, V, dtype, sms);
  RowsArgs a{};
  a.longp = target_logits;
  a.rows = (int)rows;
  a.V = V;
  a.ld_long = V;
  a.chunk_cols = L.p.chunk_cols;
  a.nchunks = L.p.nchunks;
  a.rows_per_cta = 1;
  a.counters_b = at<int>(workspace, L.req_tk);
  a.partials = at<void>(workspace, L.partials);
  a.partial_ld = L.p.nchunks;
  a.out_token = out_target_argmax;
  a.draft = draft_tokens;
  a.n = n;
  a.out_accept = out_accept_len;
  a.out_bonus = out_bonus;
  a.status = at<int>(workspace, 0);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  PROF(DELS_KCLASS_VERIFY);
  if (launch_verify_rows(a, dtype, L.vec, s) != cudaSuccess) return DELS_ERR_CUDA;
  return DELS_OK;
}

// ------------------------------------------------------------ self test

int dels_selftest_gumbel(const uint32_t* bits, float* g, long long n, dels_stream_t stream) {
  if (n < 0) return DELS_ERR_BAD_SHAPE;
  if (n > 0 && (!bits || !g)) return DELS_ERR_NULL_POINTER;
  const int sms = device_sm_count();
  if (sms <= 0) return DELS_ERR_CUDA;
  DELS_CUDA(launch_selftest_gumbel(bits, g, n, sms, reinterpret_cast<cudaStream_t>(stream)));
  return DELS_OK;
}

size_t dels_selftest_timeout_bytes(void) { return kHeaderBytes + 4096; }

int dels_selftest_timeout(void* workspace, size_t workspace_bytes, dels_stream_t stream) {
  if (!workspace) return DELS_ERR_WORKSPACE;
  if (workspace_bytes < dels_selftest_timeout_bytes()) return DELS_ERR_WORKSPACE;
  if (!aligned16(workspace)) return DELS_ERR_ALIGNMENT;
  const int sms = device_sm_count();
  if (sms <= 0) return DELS_ERR_CUDA;
  // X [8, 64] and W [16, 64] bf16, Y [8, 16] f32 inside the workspace; the
  // producer never fills a stage, so every wait of the kernel runs out
  uint8_t* base = static_cast<uint8_t*>(workspace) + kHeaderBytes;
  Gemm g;
  if (!plan_store(g, 8, 16, base, base + 1024, 64, nullptr, nullptr, 0, 16, 1, 0, ACT_NONE,
                  reinterpret_cast<float*>(base + 3072), nullptr, 0, at<int>(workspace, 0), sms))
    return DELS_ERR_CUDA;
  g.a.debug_skip_producer = 1;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  DELS_CUDA(run(g, s));
  return DELS_OK;
}

// ------------------------------------------------------- GRU input table

size_t dels_gru_input_table_bytes(const dels_local_head* head, int V) {
  if (!head || head->kind != DELS_HEAD_GRU || head->wdtype != DELS_BF16 || V < 1) return 0;
  if (!head->emb || !head->w[0] || head->d_model <= 0 || head->d_hidden <= 0) return 0;
  return (size_t)V * 3 * (size_t)head->d_hidden * 4;
}

int dels_gru_build_input_table(const dels_local_head* head, int V, float* table, size_t table_bytes,
                               void* workspace, size_t workspace_bytes, dels_stream_t stream) {
  if (!head || !table) return DELS_ERR_NULL_POINTER;
  if (head->kind != DELS_HEAD_GRU || head->wdtype != DELS_BF16) return DELS_ERR_UNSUPPORTED;
  if (!head->emb || !head->w[0]) return DELS_ERR_NULL_POINTER;
  if (!workspace || workspace_bytes < kHeaderBytes) return DELS_ERR_WORKSPACE;
  const int D = head->d_model, H = head->d_hidden;
  if (V < 1 || D < 16 || D % 16 || D > 65536 || H < 16 || H % 16 || H > 65536) return DELS_ERR_BAD_SHAPE;
  if (!aligned16(head->emb) || !aligned16(head->w[0]) || !aligned16(table) || !aligned16(workspace))
    return DELS_ERR_ALIGNMENT;
  if (table_bytes < dels_gru_input_table_bytes(head, V)) return DELS_ERR_WORKSPACE;
  const int sms = device_sm_count();
  if (sms <= 0) return DELS_ERR_CUDA;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int* status = at<int>(workspace, 0);
  const uint16_t* E = static_cast<const uint16_t*>(head->emb);
  // G[v0 : v0 + 128] = E[v0 : v0 + 128] W_ih^T, one 128-row block of the
  // vocabulary per launch (the rows sit on the MMA's M like a batch).
  for (int v0 = 0; v0 < V; v0 += kMaxBatchTile) {
    const int rows = std::min(kMaxBatchTile, V - v0);
    Gemm g;
    if (!plan_store(g, rows, 3 * H, E + (size_t)v0 * D, head->w[0], D, nullptr, nullptr, 0, 128, 1, 0, ACT_NONE,
                    table + (size_t)v0 * 3 * H, nullptr, 0, status, sms))
      return DELS_ERR_CUDA;
    PROF(DELS_KCLASS_HEAD_GEMM);
    DELS_CUDA(run(g, s));
  }
  return DELS_OK;
}

// ------------------------------------------------------------------- draft

size_t dels_draft_workspace_bytes(const dels_local_head* head, int B, int n, int V) {
  if (validate_head(head, n) != DELS_OK || B < 0 || B > kMaxBatchTile || n < 1 || n > 32 || V < 8 || V % 8)
    return 0;
  DraftLayout L = draft_layout(head, std::max(B, 1), n, V);
  return L.ok ? L.total : 0;
}

}  // extern "C"

namespace dels {
namespace {

// dels_draft_block with the fusion weights of position j given by aw(j),
// bw(j): one pair for the block, or per-position arrays.
int draft_block_impl(const dels_local_head* head, const void* long_logits, dels_dtype logit_dtype,
                     const float* log_prior, float alpha, float beta, const float* alpha_j, const float* beta_j,
                     int B, int n, int V, int32_t* out_tokens, float* out_logprob, float* out_top2_gap,
                     void* workspace, size_t workspace_bytes, dels_stream_t stream,
                     const SampleArgs* smp = nullptr) {
  auto aw = [&](int j) { return alpha_j ? alpha_j[j] : alpha; };
  auto bw = [&](int j) { return beta_j ? beta_j[j] : beta; };
  int r = validate_draft(head, long_logits, logit_dtype, log_prior, B, n, V, out_tokens, out_logprob, out_top2_gap);
  if (r != DELS_OK) return r;
  if (!workspace) return DELS_ERR_WORKSPACE;
  if (B == 0) return DELS_OK;
  if (!aligned16(workspace)) return DELS_ERR_ALIGNMENT;
  DraftLayout L = draft_layout(head, B, n, V);
  if (!L.ok) return DELS_ERR_CUDA;
  if (workspace_bytes < L.total) return DELS_ERR_WORKSPACE;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int sms = L.sms;
  const bool bf = head->wdtype == DELS_BF16;
  const int es = bf ? 2 : 4;
  int* status = at<int>(workspace, 0);
  void* partials = at<void>(workspace, L.partials);

  MergeArgs mb{};
  mb.partials = partials;
  mb.partial_ld = L.partial_ld;
  mb.B = B;
  mb.n = n;
  mb.tokens = out_tokens;
  mb.out_lp = out_logprob;
  mb.out_gap = out_top2_gap;
  mb.status = status;
  mb.table = head->emb;
  mb.table_f32 = bf ? 0 : 1;
  mb.window = 1;
  // temperature 1 (the kept inputs' source is set per head below)
  const SampleArgs sm = smp ? *smp : SampleArgs{};
  mb.smp = sm;
  mb.smp.R = head->d_rank;
  mb.smp.r_bytes = es;

  switch (head->kind) {
    case DELS_HEAD_GRU: {
      const int D = head->d_model, H = head->d_hidden, R = head->d_rank;
      void* eg = at<void>(workspace, L.eg);
      float* h = at<float>(workspace, L.h);
      uint16_t* hb = at<uint16_t>(workspace, L.hb);
      float* gpart = at<float>(workspace, L.gpart);
      void* rr = at<void>(workspace, L.r);
      mb.D = D;
      mb.dest = eg;
      mb.smp.src_r = rr;
      if (bf && persistent_enabled() && !alpha_j && !beta_j && !sm.on && B <= sms && R <= 256) {
        // one cooperative launch for the whole block
        Gemm gg, gr, gv;
        if (!plan_store(gg, B, 3 * H, eg, head->w[0], D, hb, head->w[1], H, 128, L.gru_s0, L.gru_s1, ACT_NONE,
                        gpart, nullptr, 0, status, sms) ||
            !plan_store(gr, B, R, hb, head->w[2], H, nullptr, nullptr, 0, 32, 1, 0, ACT_SILU, nullptr,
                        static_cast<uint16_t*>(rr), R, status, sms) ||
            !plan_combine(gv, B, V, n, rr, R, head->w_vocab, long_logits, logit_dtype, log_prior, alpha, beta,
                          partials, L.partial_ld, status, sms, false))
          return DELS_ERR_CUDA;
        PersistGruArgs P{};
        P.B = B; P.n = n; P.V = V; P.D = D; P.H = H; P.R = R;
        P.stages = 12;
        P.gru = gg.a;
        P.gru.out_bmajor = 1;                    // partials as [split][3H][B]
        P.gru.ldb = B;
        P.gru.out_split_stride = (long long)3 * H * B;
        P.rank = gr.a;
        P.vocab = gv.a;
        P.gru.stages = P.rank.stages = P.vocab.stages = P.stages;
        P.vocab.max_items_per_cta = (P.vocab.num_o_tiles + sms - 1) / sms;
        P.emb = static_cast<const uint16_t*>(head->emb);
        P.longp = long_logits;
        P.long_f32 = logit_dtype == DELS_F32;
        P.eg = static_cast<uint16_t*>(eg);
        P.h = h;
        P.hb = hb;
        P.gpart = gpart;
        P.r = static_cast<uint16_t*>(rr);
        P.partials = partials;
        P.partial_ld = L.partial_ld;
        P.pos0_chunks = std::max(1, std::min(sms / B, L.partial_ld));
        P.pos0_chunk_cols = (int)round_up((size_t)((V + P.pos0_chunks - 1) / P.pos0_chunks), 8);
        P.tokens = out_tokens;
        P.out_lp = out_logprob;
        P.out_gap = out_top2_gap;
        P.status = status;
        P.grid_bar = at<unsigned>(workspace, 0) + 16;      // counter at byte 64, generation at byte 192
        P.abort_global = at<int>(workspace, 0) + 4;        // byte 16
        // as many pipeline stages as shared memory holds (at most 12)
        size_t smem = draft_gru_smem_bytes(P);
        while (P.stages > 2 && (int)smem > device_max_smem_optin()) {
          --P.stages;
          smem = draft_gru_smem_bytes(P);
        }
        P.gru.stages = P.rank.stages = P.vocab.stages = P.stages;
        if (P.vocab.a_resident && P.vocab.seg_chunks[0] <= P.stages && (int)smem <= device_max_smem_optin()) {
          const CUtensorMap maps[9] = {gg.mA0, gg.mB0, gg.mA1, gg.mB1, gr.mA0, gr.mB0, gv.mA0, gv.mB0, gv.mL};
          { PROF(DELS_KCLASS_DRAFT_BLOCK); DELS_CUDA(launch_draft_gru(P, maps, sms, smem, s)); }
          return DELS_OK;
        }
      }
      const float* G = static_cast<const float*>(head->w[3]);
      if (bf && G && fused_products_enabled() && !sm.on && B <= 64) {
        // Input-table path, fused variant (DELS_DRAFT_FUSED=1): two launches
        // per position —
        //   gates(j)        merge x_{j-1} from the previous position's records,
        //                   then h_j from G[x_{j-1}], the partials of W_hh h_{j-1}
        //                   and h_{j-1};
        //   prod_vocab(j)   (cooperative) r_j = SiLU(W_rank h_j) and the partials
        //                   of W_hh h_j, then l_S = W_vocab r_j fused with the
        //                   combine -> per-CTA records.
        // A last merge kernel decodes x_{n-1}. h_0 = 0 needs no clearing:
        // gates(1) runs with no recurrent partials and h = 0.
        mb.table = nullptr;
        if (n == 1) return draft_position0(long_logits, logit_dtype, B, n, V, partials, L.partial_ld, status, mb, sms, s);
        unsigned* r_ready = at<unsigned>(workspace, kRReadyOff);
        DELS_CUDA(cudaMemsetAsync(r_ready, 0, sizeof(unsigned), s));
        int count = 0;
        r = position0_rows(long_logits, logit_dtype, B, n, V, partials, L.partial_ld, status, sms, s, &count);
        if (r != DELS_OK) return r;
        Gemm gr, gh, gv;
        if (!plan_store(gr, B, R, hb, head->w[2], H, nullptr, nullptr, 0, kRankTile, kRankClusterSplits, 0,
                        ACT_SILU, nullptr, static_cast<uint16_t*>(rr), R, status, sms) ||
            !plan_store(gh, B, 3 * H, hb, head->w[1], H, nullptr, nullptr, 0, kHhTile, L.hh_splits, 0, ACT_NONE,
                        gpart, nullptr, 0, status, sms) ||
            !plan_combine(gv, B, V, n, rr, R, head->w_vocab, long_logits, logit_dtype, log_prior, alpha, beta,
                          partials, L.partial_ld, status, sms, false))
          return DELS_ERR_CUDA;
        // the rank product's K splits form one cluster per output tile
        gr.a.cluster_k = gr.a.total_splits;
        ProdVocabArgs P{};
        P.rank = gr.a;
        P.hh = gh.a;
        P.vocab = gv.a;
        P.rank_ctas = gr.a.num_o_tiles * gr.a.total_splits;
        const int hh_items = gh.a.num_o_tiles * gh.a.total_splits;
        // one CTA per SM (cooperative); CTAs past the vocabulary tiles only
        // take part in the products (and publish neutral records)
        const int ck = gr.a.cluster_k;
        const int grid = std::min(sms, std::max(gv.grid, P.rank_ctas + std::min(hh_items, sms))) / ck * ck;
        if (P.rank_ctas >= grid || grid > L.partial_ld) return DELS_ERR_UNSUPPORTED;
        P.r_ready = r_ready;
        P.r = static_cast<uint16_t*>(rr);
        P.R = R;
        P.stages = kMaxStagesHost;
        size_t smem = prod_vocab_smem_bytes(P);
        while (P.stages > 2 && (int)smem > device_max_smem_optin()) {
          --P.stages;
          smem = prod_vocab_smem_bytes(P);
        }
        if ((int)smem > device_max_smem_optin()) return DELS_ERR_UNSUPPORTED;
        const CUtensorMap maps[6] = {gr.mA0, gr.mB0, gh.mB0, gv.mA0, gv.mB0, gv.mL};
        GatesTableArgs ga{};
        ga.partials = partials;
        ga.partial_ld = L.partial_ld;
        ga.tokens = out_tokens;
        ga.out_lp = out_logprob;
        ga.out_gap = out_top2_gap;
        ga.n = n;
        ga.G = G;
        ga.V = V;
        ga.part = gpart;
        ga.B = B;
        ga.H = H;
        ga.h = h;
        ga.h_bf16 = hb;
        ga.status = status;
        for (int j = 1; j < n; ++j) {
          ga.count = j == 1 ? count : grid;
          ga.jprev = j - 1;
          ga.S = j == 1 ? 0 : gh.a.total_splits;
          { PROF(DELS_KCLASS_HEAD_MISC); DELS_CUDA(launch_gru_gates_table(ga, s)); }
          P.vocab.j = j;
          P.vocab.alpha = aw(j);
          P.vocab.beta = bw(j);
          P.hh_ctas = j + 1 < n ? std::min(hh_items, grid - P.rank_ctas) : 0;
          P.r_target = (unsigned)(j * gr.a.num_o_tiles);
          { PROF(DELS_KCLASS_VOCAB_COMBINE); DELS_CUDA(launch_prod_vocab(P, maps, grid, smem, s)); }
        }
        MergeArgs m = mb;
        m.count = grid;
        m.j = n - 1;
        { PROF(DELS_KCLASS_MERGE); DELS_CUDA(launch_draft_merge(m, s)); }
        return DELS_OK;
      }
      if (bf && G) {
        // Input-table path (gi = G[x] with G = E W_ih^T precomputed): three
        // launches per position —
        //   gates(j)  merge x_{j-1} from the previous position's records, then
        //             h_j from G[x_{j-1}], the partials of W_hh h_{j-1} and h_{j-1};
        //   products  r_j = SiLU(W_rank h_j) side by side with the partials of
        //             W_hh h_j (consumed by gates(j+1));
        //   vocab(j)  l_S = W_vocab r_j fused with the combine -> per-CTA records.
        // A last merge kernel decodes x_{n-1}. h_0 = 0 needs no clearing:
        // gates(1) runs with no recurrent partials and h = 0.
        mb.table = nullptr;
        if (n == 1) return draft_position0(long_logits, logit_dtype, B, n, V, partials, L.partial_ld, status, mb, sms, s);
        int count = 0;
        r = position0_rows(long_logits, logit_dtype, B, n, V, partials, L.partial_ld, status, sms, s, &count,
                           &mb.smp);
        if (r != DELS_OK) return r;
        Gemm gr, gh, gv;
        if (!plan_store(gr, B, R, hb, head->w[2], H, nullptr, nullptr, 0, kRankTile, kRankSplits, 0, ACT_SILU,
                        nullptr, static_cast<uint16_t*>(rr), R, status, sms) ||
            !plan_store(gh, B, 3 * H, hb, head->w[1], H, nullptr, nullptr, 0, kHhTile, L.hh_splits, 0, ACT_NONE,
                        gpart, nullptr, 0, status, sms) ||
            !plan_combine(gv, B, V, n, rr, R, head->w_vocab, long_logits, logit_dtype, log_prior, alpha, beta,
                          partials, L.partial_ld, status, sms, true))
          return DELS_ERR_CUDA;
        // The rank product's K splits reduce inside a cluster (one cluster per
        // output tile, no partials in HBM); its SiLU needs the whole sum.
        const int ck = gr.a.total_splits;
        if (ck > 1) {
          gr.a.cluster_k = ck;
          gr.grid = gr.a.num_o_tiles * ck;
          const int per = (gr.a.seg_chunks[0] + ck - 1) / ck;
          gr.a.stages = std::max(2, std::min(gr.a.stages, per));
          gr.smem = tc_gemm_smem_bytes(gr.a);
        }
        // both products fit one wave next to each other; whole clusters only
        gh.grid = std::min(gh.grid, std::max(ck, sms - gr.grid));
        gh.grid = std::max(ck, gh.grid / ck * ck);
        const TcGemmGroup hh{&gh.a, &gh.mA0, &gh.mB0, gh.grid};
        GatesTableArgs ga{};
        ga.partials = partials;
        ga.partial_ld = L.partial_ld;
        ga.tokens = out_tokens;
        ga.out_lp = out_logprob;
        ga.out_gap = out_top2_gap;
        ga.n = n;
        ga.G = G;
        ga.V = V;
        ga.part = gpart;
        ga.B = B;
        ga.H = H;
        ga.h = h;
        ga.h_bf16 = hb;
        ga.status = status;
        ga.smp = mb.smp;
        for (int j = 1; j < n; ++j) {
          ga.count = j == 1 ? count : gv.grid;
          ga.jprev = j - 1;
          ga.S = j == 1 ? 0 : gh.a.total_splits;
          { PROF(DELS_KCLASS_HEAD_MISC); DELS_CUDA(launch_gru_gates_table(ga, s)); }
          { PROF(DELS_KCLASS_HEAD_GEMM);
            DELS_CUDA(launch_tc_gemm(gr.a, &gr.mA0, &gr.mB0, &gr.mA1, &gr.mB1, &gr.mL, gr.grid, gr.smem, s,
                                     j + 1 < n ? &hh : nullptr)); }
          gv.a.j = j;
          gv.a.sample = sm.on;
          gv.a.seed = sm.seed;
          gv.a.step = sm.step;
          gv.a.alpha = aw(j);
          gv.a.beta = bw(j);
          { PROF(DELS_KCLASS_VOCAB_COMBINE); DELS_CUDA(run(gv, s)); }
        }
        MergeArgs m = mb;
        m.count = gv.grid;
        m.j = n - 1;
        { PROF(DELS_KCLASS_MERGE); DELS_CUDA(launch_draft_merge(m, s)); }
        return DELS_OK;
      }
      // h_0 = 0: the position-0 merge clears the recurrent state
      mb.zero_f32 = h;
      mb.zero_bf16 = hb;
      mb.zero_len = H;
      r = draft_position0(long_logits, logit_dtype, B, n, V, partials, L.partial_ld, status, mb, sms, s);
      mb.zero_f32 = nullptr;
      mb.zero_bf16 = nullptr;
      mb.zero_len = 0;
      if (r != DELS_OK || n == 1) return r;
      if (bf) {
        Gemm gg, gr, gv;
        if (!plan_store(gg, B, 3 * H, eg, head->w[0], D, hb, head->w[1], H, 128, L.gru_s0, L.gru_s1, ACT_NONE,
                        gpart, nullptr, 0, status, sms))
          return DELS_ERR_CUDA;
        if (!plan_store(gr, B, R, hb, head->w[2], H, nullptr, nullptr, 0, 32, 1, 0, ACT_SILU, nullptr,
                        static_cast<uint16_t*>(rr), R, status, sms))
          return DELS_ERR_CUDA;
        if (!plan_combine(gv, B, V, n, rr, R, head->w_vocab, long_logits, logit_dtype, log_prior, alpha, beta,
                          partials, L.partial_ld, status, sms, true))
          return DELS_ERR_CUDA;
        for (int j = 1; j < n; ++j) {
          { PROF(DELS_KCLASS_HEAD_GEMM); DELS_CUDA(run(gg, s)); }
          { PROF(DELS_KCLASS_HEAD_MISC); DELS_CUDA(launch_gru_gates(gpart, gg.a.seg_splits[0], gg.a.seg_splits[1], B, H, h, hb, s)); }
          { PROF(DELS_KCLASS_HEAD_GEMM); DELS_CUDA(run(gr, s)); }
          gv.a.j = j;
          gv.a.sample = sm.on;
          gv.a.seed = sm.seed;
          gv.a.step = sm.step;
          gv.a.alpha = aw(j);
          gv.a.beta = bw(j);
          { PROF(DELS_KCLASS_VOCAB_COMBINE); DELS_CUDA(run(gv, s)); }
          MergeArgs m = mb;
          m.count = gv.grid;
          m.j = j;
          if (j == n - 1) m.table = nullptr;
          { PROF(DELS_KCLASS_MERGE); DELS_CUDA(launch_draft_merge(m, s)); }
        }
      } else {
        const float* E = static_cast<const float*>(eg);
        const float* Wih = static_cast<const float*>(head->w[0]);
        const float* Whh = static_cast<const float*>(head->w[1]);
        const float* Wr = static_cast<const float*>(head->w[2]);
        float* feat = static_cast<float*>(rr);
        const int nch = std::max(1, std::min(L.partial_ld, (V + 255) / 256));
        for (int j = 1; j < n; ++j) {
          { PROF(DELS_KCLASS_HEAD_MISC); DELS_CUDA(launch_gemv_f32(E, D, Wih, B, 3 * H, D, ACT_NONE, gpart, 3 * H, s)); }
          { PROF(DELS_KCLASS_HEAD_MISC); DELS_CUDA(launch_gemv_f32(h, H, Whh, B, 3 * H, H, ACT_NONE, gpart + (size_t)B * 3 * H, 3 * H, s)); }
          { PROF(DELS_KCLASS_HEAD_MISC); DELS_CUDA(launch_gru_gates(gpart, 1, 1, B, H, h, hb, s)); }
          { PROF(DELS_KCLASS_HEAD_MISC); DELS_CUDA(launch_gemv_f32(h, H, Wr, B, R, H, ACT_SILU, feat, R, s)); }
          { PROF(DELS_KCLASS_VOCAB_COMBINE); DELS_CUDA(launch_vocab_combine_f32(feat, R, static_cast<const float*>(head->w_vocab),
                                             static_cast<const uint8_t*>(long_logits) +
                                                 (size_t)j * V * (logit_dtype == DELS_F32 ? 4 : 2),
                                             logit_dtype == DELS_F32, (long long)n * V, log_prior, aw(j), bw(j), B, V,
                                             partials, L.partial_ld, nch, status, s, &sm, j)); }
          MergeArgs m = mb;
          m.count = nch;
          m.j = j;
          if (j == n - 1) m.table = nullptr;
          { PROF(DELS_KCLASS_MERGE); DELS_CUDA(launch_draft_merge(m, s)); }
        }
      }
      return DELS_OK;
    }
    case DELS_HEAD_MLP: {
      const int D = head->d_model, Hd = head->d_hidden, W = head->window, K1 = W * D;
      void* u = at<void>(workspace, L.u);
      float* mpart = at<float>(workspace, L.mpart);
      void* h1 = at<void>(workspace, L.h1);
      void* h2 = at<void>(workspace, L.h2);
      void* feat = head->n_layers == 2 ? h2 : h1;
      mb.D = D;
      mb.window = W;
      mb.dest = u;
      mb.smp.src_r = feat;
      r = draft_position0(long_logits, logit_dtype, B, n, V, partials, L.partial_ld, status, mb, sms, s);
      if (r != DELS_OK || n == 1) return r;
      if (bf) {
        Gemm g1, g2, gv;
        if (!plan_store(g1, B, Hd, u, head->w[0], K1, nullptr, nullptr, 0, 128, L.mlp_s1, 0, ACT_NONE, mpart,
                        nullptr, 0, status, sms))
          return DELS_ERR_CUDA;
        if (head->n_layers == 2 &&
            !plan_store(g2, B, Hd, h1, head->w[1], Hd, nullptr, nullptr, 0, 128, L.mlp_s2, 0, ACT_NONE, mpart,
                        nullptr, 0, status, sms))
          return DELS_ERR_CUDA;
        if (!plan_combine(gv, B, V, n, feat, Hd, head->w_vocab, long_logits, logit_dtype, log_prior, alpha, beta,
                          partials, L.partial_ld, status, sms, true))
          return DELS_ERR_CUDA;
        // a few requests: each layer is one CUDA-core launch (product, GELU and
        // bf16 rounding together) instead of a split-K product plus its reduction
        const bool gemv = gemv_bf16_ok(B, K1) && gemv_bf16_ok(B, Hd);
        for (int j = 1; j < n; ++j) {
          if (gemv) {
            { PROF(DELS_KCLASS_HEAD_GEMM); DELS_CUDA(launch_gemv_bf16(static_cast<const uint16_t*>(u), K1,
                                             static_cast<const uint16_t*>(head->w[0]), B, Hd, K1, ACT_GELU,
                                             static_cast<uint16_t*>(h1), Hd, s)); }
            if (head->n_layers == 2)
              { PROF(DELS_KCLASS_HEAD_GEMM); DELS_CUDA(launch_gemv_bf16(static_cast<const uint16_t*>(h1), Hd,
                                               static_cast<const uint16_t*>(head->w[1]), B, Hd, Hd, ACT_GELU,
                                               static_cast<uint16_t*>(h2), Hd, s)); }
          } else {
            { PROF(DELS_KCLASS_HEAD_GEMM); DELS_CUDA(run(g1, s)); }
            { PROF(DELS_KCLASS_HEAD_MISC); DELS_CUDA(launch_splitk_finish(mpart, g1.a.total_splits, B, Hd, nullptr, ACT_GELU, nullptr, 0,
                                           static_cast<uint16_t*>(h1), Hd, s)); }
            if (head->n_layers == 2) {
              { PROF(DELS_KCLASS_HEAD_GEMM); DELS_CUDA(run(g2, s)); }
              { PROF(DELS_KCLASS_HEAD_MISC); DELS_CUDA(launch_splitk_finish(mpart, g2.a.total_splits, B, Hd, nullptr, ACT_GELU, nullptr, 0,
                                             static_cast<uint16_t*>(h2), Hd, s)); }
            }
          }
          gv.a.j = j;
          gv.a.sample = sm.on;
          gv.a.seed = sm.seed;
          gv.a.step = sm.step;
          gv.a.alpha = aw(j);
          gv.a.beta = bw(j);
          { PROF(DELS_KCLASS_VOCAB_COMBINE); DELS_CUDA(run(gv, s)); }
          MergeArgs m = mb;
          m.count = gv.grid;
          m.j = j;
          if (j == n - 1) m.table = nullptr;
          { PROF(DELS_KCLASS_MERGE); DELS_CUDA(launch_draft_merge(m, s)); }
        }
      } else {
        const int nch = std::max(1, std::min(L.partial_ld, (V + 255) / 256));
        for (int j = 1; j < n; ++j) {
          { PROF(DELS_KCLASS_HEAD_MISC); DELS_CUDA(launch_gemv_f32(static_cast<const float*>(u), K1, static_cast<const float*>(head->w[0]), B, Hd,
                                    K1, ACT_GELU, static_cast<float*>(h1), Hd, s)); }
          if (head->n_layers == 2)
            { PROF(DELS_KCLASS_HEAD_MISC); DELS_CUDA(launch_gemv_f32(static_cast<const float*>(h1), Hd, static_cast<const float*>(head->w[1]), B,
                                      Hd, Hd, ACT_GELU, static_cast<float*>(h2), Hd, s)); }
          { PROF(DELS_KCLASS_VOCAB_COMBINE); DELS_CUDA(launch_vocab_combine_f32(static_cast<const float*>(feat), Hd,
                                             static_cast<const float*>(head->w_vocab),
                                             static_cast<const uint8_t*>(long_logits) +
                                                 (size_t)j * V * (logit_dtype == DELS_F32 ? 4 : 2),
                                             logit_dtype == DELS_F32, (long long)n * V, log_prior, aw(j), bw(j), B, V,
                                             partials, L.partial_ld, nch, status, s, &sm, j)); }
          MergeArgs m = mb;
          m.count = nch;
          m.j = j;
          if (j == n - 1) m.table = nullptr;
          { PROF(DELS_KCLASS_MERGE); DELS_CUDA(launch_draft_merge(m, s)); }
        }
      }
      return DELS_OK;
    }
    case DELS_HEAD_XFMR: {
      const int D = head->d_model, F = head->d_hidden, P = head->max_pos, NH = head->n_heads;
      uint16_t* ex = at<uint16_t>(workspace, L.ex);
      float* t = at<float>(workspace, L.t);
      uint16_t* ab = at<uint16_t>(workspace, L.ab);
      float* q = at<float>(workspace, L.q);
      float* kc = at<float>(workspace, L.kc);
      float* vc = at<float>(workspace, L.vc);
      float* xpart = at<float>(workspace, L.xpart);
      float* xpqkv = at<float>(workspace, L.xpqkv);
      const uint16_t* wq = static_cast<const uint16_t*>(head->w[1]);
      const uint16_t* wqkv = wq;
      const size_t dd = (size_t)D * D;
      if (static_cast<const uint16_t*>(head->w[2]) != wq + dd || static_cast<const uint16_t*>(head->w[3]) != wq + 2 * dd) {
        uint16_t* packed = at<uint16_t>(workspace, L.wqkv);
        for (int k = 0; k < 3; ++k)
          DELS_CUDA(cudaMemcpyAsync(packed + k * dd, head->w[1 + k], dd * 2, cudaMemcpyDeviceToDevice, s));
        wqkv = packed;
      }
      uint16_t* ob = at<uint16_t>(workspace, L.ob);
      float* uu = at<float>(workspace, L.uu);
      uint16_t* anb = at<uint16_t>(workspace, L.anb);
      uint16_t* fb = at<uint16_t>(workspace, L.fb);
      float* y = at<float>(workspace, L.y);
      uint16_t* feat = at<uint16_t>(workspace, L.feat);
      mb.D = D;
      mb.dest = ex;
      mb.smp.src_r = feat;
      r = draft_position0(long_logits, logit_dtype, B, n, V, partials, L.partial_ld, status, mb, sms, s);
      if (r != DELS_OK || n == 1) return r;
      constexpr int T = kXfmrTerms;
      RowBlocks gqkv, go, g1, g2;
      Gemm gv;
      bool ok = plan_store_rows(gqkv, T * B, 3 * D, ab, wqkv, D, L.xs_qkv, xpqkv, status, sms) &&
                plan_store_rows(go, T * B, D, ob, head->w[4], D, L.xs_o, xpart, status, sms) &&
                plan_store_rows(g1, T * B, F, anb, head->w[5], D, L.xs_1, xpart, status, sms) &&
                plan_store_rows(g2, T * B, D, fb, head->w[6], F, L.xs_2, xpart, status, sms) &&
                plan_combine(gv, B, V, n, feat, D, head->w_vocab, long_logits, logit_dtype, log_prior, alpha, beta,
                             partials, L.partial_ld, status, sms, true);
      if (!ok) return DELS_ERR_CUDA;
      const int Sqkv = gqkv.g[0].a.total_splits;
      const int So = go.g[0].a.total_splits, S1 = g1.g[0].a.total_splits, S2 = g2.g[0].a.total_splits;
      const uint16_t* pos = static_cast<const uint16_t*>(head->w[0]);
      for (int j = 1; j < n; ++j) {
        const int p = j - 1;   // position of the newest drafted token x_{j-1}
        { PROF(DELS_KCLASS_HEAD_MISC); DELS_CUDA(launch_xfmr_embed(ex, pos, p, B, D, t, ab, s, T)); }
        { PROF(DELS_KCLASS_HEAD_GEMM); DELS_CUDA(run_rows(gqkv, s)); }
        {
          // q, and the k / v cache rows of position p, from the stacked partials
          SplitkJobs3 jq{};
          jq.j[0] = SplitkJob{xpqkv, Sqkv, 0, q, (long long)D};
          jq.j[1] = SplitkJob{xpqkv, Sqkv, D, kc + (size_t)p * D, (long long)P * D};
          jq.j[2] = SplitkJob{xpqkv, Sqkv, 2 * D, vc + (size_t)p * D, (long long)P * D};
          PROF(DELS_KCLASS_HEAD_MISC);
          DELS_CUDA(launch_splitk_finish3(jq, 3, B, D, 3 * D, T, s));
        }
        { PROF(DELS_KCLASS_HEAD_MISC); DELS_CUDA(launch_attention(q, kc, vc, B, D, NH, p + 1, P, ob, s, T)); }
        { PROF(DELS_KCLASS_HEAD_GEMM); DELS_CUDA(run_rows(go, s)); }
        { PROF(DELS_KCLASS_HEAD_MISC); DELS_CUDA(launch_finish_rmsnorm(xpart, So, T, B, D, t, uu, anb, T, s)); }
        { PROF(DELS_KCLASS_HEAD_GEMM); DELS_CUDA(run_rows(g1, s)); }
        { PROF(DELS_KCLASS_HEAD_MISC); DELS_CUDA(launch_splitk_finish(xpart, S1, B, F, nullptr, ACT_GELU, nullptr, 0, fb, F, s, T, T)); }
        { PROF(DELS_KCLASS_HEAD_GEMM); DELS_CUDA(run_rows(g2, s)); }
        { PROF(DELS_KCLASS_HEAD_MISC); DELS_CUDA(launch_finish_rmsnorm(xpart, S2, T, B, D, uu, y, feat, 1, s)); }
        gv.a.j = j;
          gv.a.sample = sm.on;
          gv.a.seed = sm.seed;
          gv.a.step = sm.step;
        gv.a.alpha = aw(j);
        gv.a.beta = bw(j);
        { PROF(DELS_KCLASS_VOCAB_COMBINE); DELS_CUDA(run(gv, s)); }
        MergeArgs m = mb;
        m.count = gv.grid;
        m.j = j;
        if (j == n - 1) m.table = nullptr;
        { PROF(DELS_KCLASS_MERGE); DELS_CUDA(launch_draft_merge(m, s)); }
      }
      return DELS_OK;
    }
    case DELS_HEAD_MARKOV: {
      const int R = head->d_rank;
      void* feat = at<void>(workspace, L.mk);
      mb.D = R;
      mb.dest = feat;
      mb.smp.src_r = feat;
      r = draft_position0(long_logits, logit_dtype, B, n, V, partials, L.partial_ld, status, mb, sms, s);
      if (r != DELS_OK || n == 1) return r;
      Gemm gv;
      if (bf && !plan_combine(gv, B, V, n, feat, R, head->w_vocab, long_logits, logit_dtype, log_prior, alpha, beta,
                              partials, L.partial_ld, status, sms, true))
        return DELS_ERR_CUDA;
      const int nch = std::max(1, std::min(L.partial_ld, (V + 255) / 256));
      for (int j = 1; j < n; ++j) {
        int count;
        if (bf) {
          gv.a.j = j;
          gv.a.sample = sm.on;
          gv.a.seed = sm.seed;
          gv.a.step = sm.step;
          gv.a.alpha = aw(j);
          gv.a.beta = bw(j);
          { PROF(DELS_KCLASS_VOCAB_COMBINE); DELS_CUDA(run(gv, s)); }
          count = gv.grid;
        } else {
          { PROF(DELS_KCLASS_VOCAB_COMBINE); DELS_CUDA(launch_vocab_combine_f32(static_cast<const float*>(feat), R,
                                             static_cast<const float*>(head->w_vocab),
                                             static_cast<const uint8_t*>(long_logits) +
                                                 (size_t)j * V * (logit_dtype == DELS_F32 ? 4 : 2),
                                             logit_dtype == DELS_F32, (long long)n * V, log_prior, aw(j), bw(j), B, V,
                                             partials, L.partial_ld, nch, status, s, &sm, j)); }
          count = nch;
        }
        MergeArgs m = mb;
        m.count = count;
        m.j = j;
        if (j == n - 1) m.table = nullptr;
        { PROF(DELS_KCLASS_MERGE); DELS_CUDA(launch_draft_merge(m, s)); }
      }
      return DELS_OK;
    }
    default:
      return DELS_ERR_UNSUPPORTED;
  }
}

}  // namespace
}  // namespace dels

extern "C" {

int dels_draft_block(const dels_local_head* head, const void* long_logits, dels_dtype logit_dtype,
                     const float* log_prior, float alpha, float beta, int B, int n, int V, int32_t* out_tokens,
                     float* out_logprob, float* out_top2_gap, void* workspace, size_t workspace_bytes,
                     dels_stream_t stream) {
  return draft_block_impl(head, long_logits, logit_dtype, log_prior, alpha, beta, nullptr, nullptr, B, n, V,
                          out_tokens, out_logprob, out_top2_gap, workspace, workspace_bytes, stream);
}

size_t dels_draft_state_bytes(const dels_local_head* head, int B, int n) {
  if (!head || B < 0 || n < 1) return 0;
  const size_t es = head->wdtype == DELS_BF16 ? 2 : 4;
  return round_up((size_t)B * n * 4, 256) + (size_t)B * n * (size_t)head->d_rank * es;
}

int dels_draft_block_sampled(const dels_local_head* head, const void* long_logits, dels_dtype logit_dtype,
                             const float* log_prior, const float* alpha, const float* beta, int B, int n, int V,
                             uint64_t seed, uint64_t step, int32_t* out_tokens, float* out_logprob,
                             float* out_key_gap, void* draft_state, size_t state_bytes, void* workspace,
                             size_t workspace_bytes, dels_stream_t stream) {
  if (!head || !alpha || !beta || !out_logprob) return DELS_ERR_NULL_POINTER;
  if (n < 1 || n > 32 || B < 0) return DELS_ERR_BAD_SHAPE;
  if (!sample_counter_ok(B, step)) return DELS_ERR_BAD_SHAPE;
  for (int j = 0; j < n; ++j)
    if (!std::isfinite(alpha[j]) || !std::isfinite(beta[j])) return DELS_ERR_BAD_SHAPE;
  const size_t es = head->wdtype == DELS_BF16 ? 2 : 4;
  if (((size_t)head->d_rank * es) % 16 != 0) return DELS_ERR_UNSUPPORTED;
  if (draft_state) {
    if (state_bytes < dels_draft_state_bytes(head, B, n)) return DELS_ERR_WORKSPACE;
    if (!aligned16(draft_state)) return DELS_ERR_ALIGNMENT;
  }
  SampleArgs sm{};
  sm.on = 1;
  sm.seed = seed;
  sm.step = step;
  sm.out_lse = static_cast<float*>(draft_state);
  sm.state_r = draft_state ? static_cast<uint8_t*>(draft_state) + round_up((size_t)B * n * 4, 256) : nullptr;
  return draft_block_impl(head, long_logits, logit_dtype, log_prior, 0.f, 0.f, alpha, beta, B, n, V, out_tokens,
                          out_logprob, out_key_gap, workspace, workspace_bytes, stream, &sm);
}

namespace {

struct VerifySampledLayout {
  RowsPlan t;                 // target-row records
  int r_nchunks, r_chunk_cols;
  size_t t_rec, acc, lse_t, rg, ls, r_rec, total;
};

VerifySampledLayout verify_sampled_layout(const dels_local_head* head, int B, int n, int V, dels_dtype tdt, int sms) {
  VerifySampledLayout L{};
  const int es_t = tdt == DELS_F32 ? 4 : 2;
  const bool vec = (V % 8) == 0;
  const int rows = B * (n + 1);
  L.t = plan_rows(std::max(rows, 1), V, es_t, sms, vec, 1 << 20);
  L.r_nchunks = std::max(1, std::min((V + 2047) / 2048, (4 * sms + std::max(B, 1) - 1) / std::max(B, 1)));
  L.r_chunk_cols = (int)round_up((size_t)((V + L.r_nchunks - 1) / L.r_nchunks), 8);
  L.r_nchunks = (V + L.r_chunk_cols - 1) / L.r_chunk_cols;
  const size_t es_w = head->wdtype == DELS_BF16 ? 2 : 4;
  size_t off = kHeaderBytes;
  L.t_rec = off;
  off = round_up(off + (size_t)rows * L.t.nchunks * 16, 256);
  L.acc = off;
  off = round_up(off + (size_t)B * 4, 256);
  L.lse_t = off;
  off = round_up(off + (size_t)B * 4, 256);
  L.rg = off;
  off = round_up(off + (size_t)B * head->d_rank * es_w, 256);
  L.ls = off;
  off = round_up(off + (size_t)B * V * 4, 256);
  L.r_rec = off;
  off = round_up(off + (size_t)B * L.r_nchunks * 32, 256);
  L.total = off;
  return L;
}

}  // namespace

size_t dels_verify_sampled_workspace_bytes(const dels_local_head* head, int B, int n, int V, dels_dtype target_dtype) {
  if (!head || B < 0 || n < 1 || n > kMaxSampledBlock || V < 1) return 0;
  if (target_dtype != DELS_F32 && target_dtype != DELS_BF16) return 0;
  const int sms = device_sm_count();
  if (sms <= 0) return 0;
  return verify_sampled_layout(head, B, n, V, target_dtype, sms).total;
}

int dels_verify_block_sampled(const dels_local_head* head, const int32_t* draft_tokens, const float* draft_logprob,
                              const void* draft_state, const void* long_logits, dels_dtype logit_dtype,
                              const float* log_prior, const float* alpha, const float* beta,
                              const void* target_logits, dels_dtype target_dtype, int B, int n, int V, uint64_t seed,
                              uint64_t step, int32_t* out_accept_len, int32_t* out_bonus, float* out_bonus_gap,
                              void* workspace, size_t workspace_bytes, dels_stream_t stream) {
  if (!head || !alpha || !beta) return DELS_ERR_NULL_POINTER;
  if ((logit_dtype != DELS_F32 && logit_dtype != DELS_BF16) || (target_dtype != DELS_F32 && target_dtype != DELS_BF16))
    return DELS_ERR_BAD_DTYPE;
  if (B < 0 || n < 1 || n > kMaxSampledBlock || V < 1) return DELS_ERR_BAD_SHAPE;
  if ((long long)B * (n + 1) > INT32_MAX) return DELS_ERR_BAD_SHAPE;
  if (!sample_counter_ok(B, step)) return DELS_ERR_BAD_SHAPE;
  const bool bf = head->wdtype == DELS_BF16;
  if (bf && B > kMaxBatchTile) return DELS_ERR_BAD_SHAPE;
  for (int j = 0; j < n; ++j)
    if (!std::isfinite(alpha[j]) || !std::isfinite(beta[j])) return DELS_ERR_BAD_SHAPE;
  if (!workspace) return DELS_ERR_WORKSPACE;
  if (B == 0) return DELS_OK;
  if (!draft_tokens || !draft_logprob || !draft_state || !long_logits || !target_logits || !out_accept_len ||
      !out_bonus || !head->w_vocab)
    return DELS_ERR_NULL_POINTER;
  const size_t es_w = bf ? 2 : 4;
  if (((size_t)head->d_rank * es_w) % 16 != 0) return DELS_ERR_UNSUPPORTED;
  if (!aligned16(workspace) || !aligned16(draft_state) || !aligned16(target_logits) || !aligned16(long_logits))
    return DELS_ERR_ALIGNMENT;
  const int sms = device_sm_count();
  if (sms <= 0) return DELS_ERR_CUDA;
  const VerifySampledLayout L = verify_sampled_layout(head, B, n, V, target_dtype, sms);
  if (workspace_bytes < L.total) return DELS_ERR_WORKSPACE;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int* status = at<int>(workspace, 0);
  // 1. records of the target rows (their LSEs)
  RowsArgs t{};
  t.longp = target_logits;
  t.rows = B * (n + 1);
  t.V = V;
  t.ld_long = V;
  t.chunk_cols = L.t.chunk_cols;
  t.nchunks = L.t.nchunks;
  t.rows_per_cta = 1;
  t.partials = at<void>(workspace, L.t_rec);
  t.partial_ld = L.t.nchunks;
  t.status = status;
  const int es_t = target_dtype == DELS_F32 ? 4 : 2;
  const bool vec = (V % 8) == 0;
  { PROF(DELS_KCLASS_VERIFY); DELS_CUDA(launch_combine_rows(t, target_dtype, vec, false, s)); }
  // 2. the acceptance tests and the rejected position's input
  VerifySampledArgs a{};
  a.B = B;
  a.n = n;
  a.V = V;
  a.draft = draft_tokens;
  a.draft_lp = draft_logprob;
  a.state_lse = static_cast<const float*>(draft_state);
  a.state_r = static_cast<const uint8_t*>(draft_state) + round_up((size_t)B * n * 4, 256);
  a.R = head->d_rank;
  a.r_bytes = (int)es_w;
  a.target = target_logits;
  a.target_f32 = target_dtype == DELS_F32;
  a.longp = long_logits;
  a.long_f32 = logit_dtype == DELS_F32;
  a.prior = log_prior;
  for (int j = 0; j < n; ++j) {
    a.alpha[j] = alpha[j];
    a.beta[j] = beta[j];
  }
  a.seed = seed;
  a.step = step;
  a.t_records = t.partials;
  a.t_nchunks = L.t.nchunks;
  a.t_ld = L.t.nchunks;
  a.acc = at<int>(workspace, L.acc);
  a.lse_t = at<float>(workspace, L.lse_t);
  a.rg = at<void>(workspace, L.rg);
  a.ls = at<float>(workspace, L.ls);
  a.r_records = at<void>(workspace, L.r_rec);
  a.r_nchunks = L.r_nchunks;
  a.r_chunk_cols = L.r_chunk_cols;
  a.out_accept = out_accept_len;
  a.out_bonus = out_bonus;
  a.out_bonus_gap = out_bonus_gap;
  a.status = status;
  { PROF(DELS_KCLASS_VERIFY); DELS_CUDA(launch_verify_accept(a, s)); }
  // 3. l_S of the rejected positions: W_vocab r (rows with no head input are zero)
  if (bf) {
    Gemm g;
    if (!plan_store(g, B, V, a.rg, head->w_vocab, head->d_rank, nullptr, nullptr, 0, 128, 1, 0, ACT_NONE,
                    at<float>(workspace, L.ls), nullptr, 0, status, sms))
      return DELS_ERR_CUDA;
    { PROF(DELS_KCLASS_VERIFY); DELS_CUDA(run(g, s)); }
  } else {
    { PROF(DELS_KCLASS_VERIFY);
      DELS_CUDA(launch_gemv_f32(static_cast<const float*>(a.rg), head->d_rank,
                                static_cast<const float*>(head->w_vocab), B, V, head->d_rank, ACT_NONE,
                                at<float>(workspace, L.ls), V, s)); }
  }
  // 4. the bonus draw: the residual at the rejection, or p_n after n acceptances
  { PROF(DELS_KCLASS_VERIFY); DELS_CUDA(launch_residual_rows(a, s)); }
  { PROF(DELS_KCLASS_VERIFY); DELS_CUDA(launch_residual_merge(a, s)); }
  return DELS_OK;
}

int dels_draft_block_weighted(const dels_local_head* head, const void* long_logits, dels_dtype logit_dtype,
                              const float* log_prior, const float* alpha, const float* beta, int B, int n, int V,
                              int32_t* out_tokens, float* out_logprob, float* out_top2_gap, void* workspace,
                              size_t workspace_bytes, dels_stream_t stream) {
  if (!alpha || !beta) return DELS_ERR_NULL_POINTER;
  if (n < 1 || n > 32) return DELS_ERR_BAD_SHAPE;
  for (int j = 0; j < n; ++j)
    if (!std::isfinite(alpha[j]) || !std::isfinite(beta[j])) return DELS_ERR_BAD_SHAPE;
  return draft_block_impl(head, long_logits, logit_dtype, log_prior, 0.f, 0.f, alpha, beta, B, n, V, out_tokens,
                          out_logprob, out_top2_gap, workspace, workspace_bytes, stream);
}

}  // extern "C"