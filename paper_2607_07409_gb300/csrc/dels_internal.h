// Internal declarations shared by the library's translation units (host side
// launchers and the parameter blocks their kernels take).
#pragma once

#include <cstddef>
#include <cstdint>
#include <utility>
#include <cuda_runtime.h>
#include <cuda.h>

#include "../../include/dels.h"

namespace dels {

constexpr int kHeaderBytes = 256;          // workspace: status word + padding
constexpr int kRowsThreads = 256;          // row-reduction kernels
constexpr int kMaxBatchTile = 128;         // tcgen05 M: batch rows per tile
constexpr uint64_t kWaitBudgetNs = 2000000000ull;   // bounded device waits: 2 s

struct RowAcc;

// Launch with programmatic stream serialization: the kernel may begin while
// its predecessor on the stream is still running; it waits for it with
// griddepcontrol.wait before touching the predecessor's outputs.
// As launch_pdl, with thread-block clusters of `cluster_x` CTAs along x
// (1: no cluster attribute).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl_cluster(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                               int cluster_x, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  int na = 1;
  if (cluster_x > 1) {
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = (unsigned)cluster_x;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    na = 2;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args&&... args) {
  return launch_pdl_cluster(kernel, grid, block, smem, s, 1, std::forward<Args>(args)...);
}

// ---- row reductions (combine / verify / draft position 0) -------------------
constexpr int kMaxVerifyBlock = 1024;    // greedy verification: n <= 1024 draft positions

struct RowsArgs {
  const void* longp;
  const void* shortp;
  const float* prior;
  float alpha, beta;
  int rows, V;
  long long ld_long, ld_short;   // row pitch in elements
  int chunk_cols;                // columns per chunk (multiple of 8)
  int nchunks;                   // chunks per row
  int rows_per_cta;              // R
  void* partials;                // [rows][partial_ld] 16-byte records
  int partial_ld;
  int* counters;                 // combine: one ticket per row group
  int* counters_b;               // verify: per request
  int32_t* out_token;
  float* out_lp;
  float* out_gap;
  // verify
  const int32_t* draft;
  int n;                         // draft positions (verify)
  int32_t* out_accept;
  int32_t* out_bonus;
  int* status;
};

struct RowsPlan {
  int nchunks, chunk_cols, rows_per_cta, grid;
};

// Chunks per row for the row kernels. slots_per_sm > 0 (resident CTAs per
// SM): when every row group fits in one wave, as many chunks as that wave
// holds; otherwise about 16 CTAs per SM.
RowsPlan plan_rows(int rows, int V, int bytes_per_col, int num_sms, bool vec, int max_chunks,
                  bool multi_row = false, int slots_per_sm = 0);
// Resident CTAs per SM of the combine (verify = false) or verification row
// kernel for this dtype (0 if the query fails).
int rows_slots_per_sm(bool verify, dels_dtype dt);
cudaError_t launch_combine_rows(const RowsArgs& a, dels_dtype dt, bool vec, bool finalize, cudaStream_t s);
cudaError_t launch_verify_rows(const RowsArgs& a, dels_dtype dt, bool vec, cudaStream_t s);

// Workspace layout of dels_combine_argmax (shared with the no-allocation
// entry point, which clears the header and the tickets itself).
struct CombineLayout {
  bool vec;
  RowsPlan p;
  size_t tickets_off, partials_off, total;
};
CombineLayout combine_layout(int rows, int V, dels_dtype dtype, int sms);

// ---- draft merge + gather of the next local-head input ----------------------
// Temperature-1 drafting (on = 0: temperature 0). The uniforms of (request
// b, position j, stream, vocabulary index) come from Philox4x32-10 keyed by
// the seed, with the step in the counter.
struct SampleArgs {
  int on;
  unsigned long long seed, step;
  float* out_lse;                // [B, n] LSE of the fused row, or null
  void* state_r;                 // [B][n][R] kept vocabulary-projection inputs, or null
  const void* src_r;             // [B][R] the current position's input
  int R, r_bytes;                // elements per row and bytes per element
};

// Records of Gumbel-max keys over logit rows (temperature 1).
struct SampleRowsArgs {
  const void* src;               // row r starts at src + r * ld (elements)
  long long ld;
  int rows, rows_per_request, j0;
  int V, chunk_cols, nchunks, vec;
  unsigned long long seed, step;
  int stream;
  void* partials;                // [rows][partial_ld] RowAcc
  int partial_ld;
};
cudaError_t launch_sample_rows(const SampleRowsArgs& a, bool f32, cudaStream_t s);
// The Gumbel transform of Philox words, element-wise (test hook).
cudaError_t launch_selftest_gumbel(const uint32_t* bits, float* g, long long n, int sms, cudaStream_t s);

// Verification of a temperature-1 block by lossless speculative sampling.
constexpr int kMaxSampledBlock = 32;
// Temperature-1 counters: the step fills one 32-bit Philox counter word and
// the request 16 bits of another.
inline bool sample_counter_ok(int B, unsigned long long step) { return step < (1ull << 32) && B <= (1 << 16); }
struct VerifySampledArgs {
  int B, n, V;
  const int32_t* draft;          // [B, n]
  const float* draft_lp;         // [B, n] log q_j(x_j)
  const float* state_lse;        // [B, n] LSE of the fused rows
  const void* state_r;           // [B][n][R] vocabulary-projection inputs (j >= 1)
  int R, r_bytes;
  const void* target;            // [B, n+1, V]
  int target_f32;
  const void* longp;             // [B, n, V]
  int long_f32;
  const float* prior;            // [V] or null
  float alpha[kMaxSampledBlock], beta[kMaxSampledBlock];
  unsigned long long seed, step;
  const void* t_records;         // [B * (n+1)][t_ld] RowAcc of the target rows
  int t_nchunks, t_ld;
  int* acc;                      // [B] accepted length
  float* lse_t;                  // [B] LSE of target row acc[b]
  void* rg;                      // [B][R] the rejected position's input (zeros at j = 0 and n)
  const float* ls;               // [B][V] W_vocab rg
  void* r_records;               // [B][r_nchunks][2] RowAcc: residual keys, then target keys
  int r_nchunks, r_chunk_cols;
  int32_t* out_accept;
  int32_t* out_bonus;
  float* out_bonus_gap;          // or null
  int* status;
};
cudaError_t launch_verify_accept(const VerifySampledArgs& a, cudaStream_t s);
cudaError_t launch_residual_rows(const VerifySampledArgs& a, cudaStream_t s);
cudaError_t launch_residual_merge(const VerifySampledArgs& a, cudaStream_t s);

struct MergeArgs {
  const void* partials;          // [B][partial_ld] RowAcc
  int partial_ld, count;
  int B, n, j;
  int32_t* tokens;               // [B, n]
  float* out_lp;                 // [B, n]
  float* out_gap;                // [B, n] or null
  int* status;
  // gather: dest[b, k*D:(k+1)*D] = table[token(b, j-k)] or 0 for k < window
  const void* table;             // [V, D] (bf16 or f32) or null
  int table_f32;
  int D, window;
  void* dest;                    // [B, window*D] same dtype as table
  // optional per-row zeroing (recurrent state at the start of a block)
  float* zero_f32;               // [B, zero_len]
  uint16_t* zero_bf16;           // [B, zero_len]
  int zero_len;
  SampleArgs smp;
};
cudaError_t launch_draft_merge(const MergeArgs& a, cudaStream_t s);

// ---- tcgen05 GEMM (batched skinny products and the vocab projection) --------
enum EpiKind { EPI_STORE = 0, EPI_COMBINE = 1 };
enum ActKind { ACT_NONE = 0, ACT_SILU = 1, ACT_GELU = 2 };

struct TcGemmArgs {
  int B;                         // real batch rows (<= 128)
  int O;                         // rows of W (outputs)
  int n_tile;                    // N per tile (multiple of 16, <= 256)
  int num_o_tiles;
  int seg_chunks[2];             // K chunks of 64 per segment
  int seg_splits[2];             // K splits per segment (0 splits: unused segment)
  int total_splits;
  int epi;
  int a_resident;                // A (activations) loaded once per CTA
  int b_chunks;                  // K chunks per pipeline stage: 2 (the weights' as one 3-D box); 0 or 1: one
  int stages;
  int max_items_per_cta;         // EPI_COMBINE: sizes the per-CTA prior slice in smem
  int a_box_rows;                // activation rows per TMA box (the map's box height)
  int a_copies;                  // copies of the activation rows stacked in the 128-row tile
  // EPI_STORE
  int act;
  float* out_f32;                // [split][B][ldo] (or final when total_splits == 1)
  long long out_split_stride;
  int ldo;
  uint16_t* out_bf16;            // [B][ldo_bf16] activation output (total_splits == 1)
  int ldo_bf16;
  int out_bmajor;                // f32 output as [split][o][ldb] (batch index fastest): each warp
  int ldb;                       // store instruction then writes one contiguous 128-byte line
  // EPI_COMBINE
  const float* prior;
  float alpha, beta;
  int V;
  int j;                         // block position: coordinate into the long-logit map
  int long_f32;
  int l_box_cols, l_box_rows, l_boxes;   // long-logit tile = l_boxes boxes
  void* partials;                // [B][partial_ld] RowAcc
  int partial_ld;
  int* status;
  int debug_skip_producer;       // test hook: producer never fills (exercises the bounded waits)
  // EPI_COMBINE at temperature 1: Gumbel-max keys (Philox4x32-10 of (seed, step))
  int sample;
  unsigned long long seed, step;
  // EPI_STORE, optional: the K splits of one output tile run on the CTAs of
  // one thread-block cluster (cluster_k CTAs, split = rank in the cluster);
  // the others send their accumulators to rank 0 through distributed shared
  // memory, and rank 0 sums, applies the activation and stores. 1: off.
  int cluster_k;
};

// One launch of k_tc_gemm runs one GEMM on `grid` CTAs, or two independent
// GEMMs side by side ("grouped"): CTAs [0, grid) run the first, CTAs
// [grid, grid + grid2) the second (single K segment, its own A/B maps).
struct TcGemmGroup {
  const TcGemmArgs* a;           // null: no second GEMM
  const CUtensorMap* mA;
  const CUtensorMap* mB;
  int grid;
};
// Shared memory of the f32-row store transpose (8 epilogue warps x 32 x 33 floats).
constexpr int kStoreTransposeBytes = 8 * 32 * 33 * 4;
cudaError_t launch_tc_gemm(const TcGemmArgs& a, const CUtensorMap* mA0, const CUtensorMap* mB0,
                           const CUtensorMap* mA1, const CUtensorMap* mB1, const CUtensorMap* mL, int grid,
                           size_t smem_bytes, cudaStream_t s, const TcGemmGroup* second = nullptr);
size_t tc_gemm_smem_bytes(const TcGemmArgs& a);

// ---- persistent per-block drafting kernel (GRU head, bf16) --------------------
struct PersistGruArgs {
  int B, n, V, D, H, R;
  int stages;                    // pipeline stages shared by the three GEMM phases
  TcGemmArgs gru, rank, vocab;   // the tensor-core phases of one position
  const uint16_t* emb;           // E_tgt [V, D]
  const void* longp;             // [B, n, V]
  int long_f32;
  uint16_t* eg;                  // [B, D] gathered embeddings
  float* h;                      // [H, B] GRU state (batch index fastest)
  uint16_t* hb;                  // [B, H] its bf16 copy
  float* gpart;                  // [S0 + S1][3H][B] gate-product partials (batch fastest)
  uint16_t* r;                   // [B, R] low-rank state
  void* partials;                // [B][partial_ld] RowAcc
  int partial_ld;
  int pos0_chunks, pos0_chunk_cols;
  int32_t* tokens;
  float* out_lp;
  float* out_gap;
  int* status;
  unsigned* grid_bar;            // grid-barrier counter (workspace header)
  int* abort_global;             // set by a CTA whose bounded wait expired
};
size_t draft_gru_smem_bytes(const PersistGruArgs& P);
cudaError_t launch_draft_gru(const PersistGruArgs& P, const CUtensorMap* maps, int grid, size_t smem,
                             cudaStream_t s);

// ---- products of h_j + vocabulary projection, one cooperative launch ----------
struct ProdVocabArgs {
  TcGemmArgs rank;               // W_rank h, K split over the CTAs of a cluster (cluster_k)
  TcGemmArgs hh;                 // split-K partials of W_hh h (for the next gates launch)
  TcGemmArgs vocab;              // EPI_COMBINE, activations r (resident)
  int rank_ctas, hh_ctas;        // CTAs [0, rank_ctas) rank splits, then hh_ctas recurrent CTAs
  int stages;                    // ring stages shared by the two phases
  unsigned* r_ready;             // rank tiles finished since the start of the block
  unsigned r_target;             // the vocabulary phase waits until *r_ready >= r_target
  uint16_t* r;                   // [B, R] bf16 = SiLU(sum of the rank partials)
  int R;
};
size_t prod_vocab_smem_bytes(const ProdVocabArgs& P);
cudaError_t launch_prod_vocab(const ProdVocabArgs& P, const CUtensorMap* maps, int grid, size_t smem,
                              cudaStream_t s);

// ---- small head kernels -------------------------------------------------------
cudaError_t launch_gru_gates(const float* part, int S0, int S1, int B, int H, float* h, uint16_t* h_bf16,
                             cudaStream_t s);
// GRU step with a precomputed input table G = E W_ih^T [V, 3H] (f32), fused
// with the merge of the previous position: x = the merged argmax of request
// b's `count` records [B][partial_ld] (written to tokens/lp/gap at column
// jprev), gi = G[x], gh = sum of S recurrent partials [S][B][3H] (S = 0:
// gh = 0, the step from h = 0).
struct GatesTableArgs {
  const void* partials;
  int partial_ld, count;
  int32_t* tokens;               // [B, n]
  float* out_lp;                 // [B, n]
  float* out_gap;                // [B, n] or null
  int n, jprev;
  const float* G;                // [V, 3H]
  int V;
  const float* part;             // [S][B][3H]
  int S, B, H;
  float* h;                      // [B, H]
  uint16_t* h_bf16;              // [B, H]
  int* status;
  SampleArgs smp;
};
cudaError_t launch_gru_gates_table(const GatesTableArgs& a, cudaStream_t s);
// bf16 activations of the head products are written as `terms` bf16 terms:
// 1 = rounded to bf16; 3 = the exact three-term expansion hi + mid + lo in
// rows [0, B), [B, 2B), [2B, 3B) of a [3B, ld] buffer (a product over the 3B
// rows then writes partials [S][3B][O], summed back by in_terms = 3).
cudaError_t launch_splitk_finish(const float* part, int S, int B, int O, const float* residual, int act,
                                 float* out_f32, int ld_f32, uint16_t* out_bf16, int ld_bf16, cudaStream_t s,
                                 int in_terms = 1, int out_terms = 1);
cudaError_t launch_rmsnorm_bf16(const float* x, int B, int D, int ld, uint16_t* out, cudaStream_t s, int terms = 1);
// Up to three split-K reductions (float32 outputs, own row pitches) in one
// launch: job k sums columns col0 .. col0 + O - 1 of partials
// [S][in_terms * B][ldp].
struct SplitkJob {
  const float* part;
  int S;
  int col0;
  float* out;          // row b at out + b * ld
  long long ld;
};
struct SplitkJobs3 {
  SplitkJob j[3];
};
cudaError_t launch_splitk_finish3(const SplitkJobs3& jobs, int njobs, int B, int O, int ldp, int in_terms,
                                  cudaStream_t s);
// Split-K reduction + residual (out_f32) and RMSNorm of each row as `terms`
// bf16 terms (norm_bf16, row pitch D); a cluster of kNormCluster CTAs per row.
constexpr int kNormCluster = 8;
cudaError_t launch_finish_rmsnorm(const float* part, int S, int in_terms, int B, int D, const float* residual,
                                  float* out_f32, uint16_t* norm_bf16, int terms, cudaStream_t s);
cudaError_t launch_xfmr_embed(const uint16_t* e_rows, const uint16_t* pos_table, int pos, int B, int D,
                              float* t_out, uint16_t* a_bf16, cudaStream_t s, int terms = 1);
cudaError_t launch_attention(const float* q, const float* kcache, const float* vcache, int B, int D, int nh,
                             int npos, int cache_ld_pos, uint16_t* o_bf16, cudaStream_t s, int terms = 1);
cudaError_t launch_gemv_f32(const float* X, int ldx, const float* W, int B, int O, int K, int act, float* Y,
                            int ldy, cudaStream_t s);
// bf16 weights and activations, bf16 output after the activation, B <= kGemvBf16MaxRows.
constexpr int kGemvBf16MaxRows = 4;
// the X rows are staged in (at most 48 KB of) shared memory
inline bool gemv_bf16_ok(int B, int K) {
  return B >= 1 && B <= kGemvBf16MaxRows && K % 8 == 0 && (long long)B * K * 2 <= 48 * 1024;
}
cudaError_t launch_gemv_bf16(const uint16_t* X, int ldx, const uint16_t* W, int B, int O, int K, int act,
                             uint16_t* Y, int ldy, cudaStream_t s);
cudaError_t launch_vocab_combine_f32(const float* feat, int K, const float* Wv, const void* longp, int long_f32,
                                     long long ld_long, const float* prior, float alpha, float beta, int B,
                                     int V, void* partials, int partial_ld, int nchunks, int* status,
                                     cudaStream_t s,
                                     const SampleArgs* smp = nullptr, int j = 0);

// ---- host utilities ---------------------------------------------------------
// Host-side checks of dels_combine_argmax's input and output pointers (NULL,
// 16-byte alignment), shared with the no-allocation variant so that both
// reject the same calls before anything is enqueued.
int combine_check_inputs(const void* long_logits, const void* short_logits, const float* log_prior,
                         const int32_t* out_token);
int device_sm_count();
int device_max_smem_optin();
// Raises `kernel`'s dynamic shared-memory limit on the current device to at
// least `bytes`, once per kernel, device and size (safe from several host
// threads; the attribute is per device).
cudaError_t ensure_dynamic_smem(const void* kernel, size_t bytes);
bool encode_tmap_2d(CUtensorMap* m, const void* base, CUtensorMapDataType dt, int elem_bytes, uint64_t inner,
                    uint64_t outer, uint64_t row_pitch_bytes, uint32_t box_inner, uint32_t box_outer,
                    CUtensorMapSwizzle swz);
bool encode_tmap_3d(CUtensorMap* m, const void* base, CUtensorMapDataType dt, int elem_bytes, uint64_t d0,
                    uint64_t d1, uint64_t d2, uint64_t pitch1_bytes, uint64_t pitch2_bytes, uint32_t b0,
                    uint32_t b1, uint32_t b2, CUtensorMapSwizzle swz);

// ---- unigram prior estimation (Appendix A) -----------------------------------
constexpr int kPriorMaxPartials = 1024;            // CTAs of the two-level count sum
constexpr int kPriorHistBuckets = 3776;            // count buckets of the hot-set choice
constexpr long long kPriorHotMinN = 1ll << 24;     // shorter ranges: slice histograms only
constexpr long long kPriorChunk = 1ll << 36;       // positions per launch (per-thread tallies stay < 2^32)

// Positions [0, n) of tokens / mask; [head, head + nvec) takes the vector
// path (tokens + head 16-byte aligned, mask + head 4-byte aligned, nvec a
// multiple of 512).
struct PriorRange {
  const int32_t* tokens;
  const uint8_t* mask;        // nonzero = loss-masked
  long long n;
  long long head;
  long long nvec;
};

struct PriorSliceArgs {
  PriorRange range;
  int V;
  int slices;                       // P
  int slice;                        // ids per slice (bins per CTA)
  unsigned long long* counts;       // [V], accumulated
  unsigned long long* tally;        // [2] or null
  int* status;
};

struct PriorSelectArgs {
  const unsigned long long* counts;   // [V]
  int V;
  int K;                              // hot slots
  int nent;                           // remap words: ceil(V / 15)
  unsigned* hist;                     // [kPriorHistBuckets], zero on entry and on exit
  uint32_t* entries;                  // [nent]
  int32_t* stage;                     // [nent * 15] hot ids per CTA, before placement
  unsigned* cta_total;                // [CTAs] hot ids per CTA
  int32_t* slot_id;                   // [K]
  unsigned* n_hot;
};

struct PriorHotArgs {
  PriorRange range;
  int V;
  int K;
  int nent;
  int ctas;
  const uint32_t* entries;
  const int32_t* slot_id;
  const unsigned* n_hot;
  unsigned* partials;                 // [ctas][(K + 1) / 2] words of two 16-bit bins
  unsigned long long* counts;
  unsigned long long* tally;
  int* status;
};

struct PriorLogArgs {
  const unsigned long long* counts;   // [V]
  int V;
  double lambda;
  unsigned long long* partials;       // [kPriorMaxPartials]
  unsigned* ticket;
  unsigned long long* total;          // sum_v counts[v] (written by k_prior_total, or the tally)
  const unsigned long long* tally;    // [2] copied to tally_out when both are set
  float* out;                         // [V] log prior
  unsigned long long* counts_out;     // [V] or null
  unsigned long long* tally_out;      // [2] or null
};

// How a count call runs for (V, N) on this device.
struct PriorPlan {
  bool ok;
  int slices, slice;          // slice histograms: P slices of `slice` ids
  size_t slice_smem;
  bool use_hot;               // hot ids on chip
  int nent, K;                // remap words, hot slots
  size_t hot_smem;
  int ctas;                   // CTAs of the hot pass (one per SM)
  int select_ctas;            // CTAs of the hot-set choice
  long long prefix;           // positions counted by the slices before the hot set is chosen
};

PriorPlan plan_prior(int V, long long N, int sms);
cudaError_t launch_prior_slices(const PriorSliceArgs& a, size_t smem, int max_members, int sms, cudaStream_t s);
cudaError_t launch_prior_select(const PriorSelectArgs& a, int ctas, cudaStream_t s);
cudaError_t launch_prior_hot(const PriorHotArgs& a, size_t smem, cudaStream_t s);
cudaError_t launch_prior_total(const PriorLogArgs& a, int sms, cudaStream_t s);
cudaError_t launch_prior_log(const PriorLogArgs& a, int sms, cudaStream_t s);

}  // namespace dels
