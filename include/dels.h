/*
 * dels.h — C ABI of the DeLS-Spec per-block drafting hot path on GB300 (sm_103a).
 *
 * DeLS-Spec ("Decoupled Long-Short Contexts for Parallel Speculative
 * Drafting") keeps a block-parallel drafter (DFlash) fixed as the
 * long-context expert, adds a small autoregressive local head over the tokens
 * already drafted in the block as the short-context expert, and fuses the
 * two with a unigram prior correction (Section 4.3):
 *
 *     l(x) = l_L(x | y) + alpha * l_S(x | z) - beta * l_P(x)
 *
 * Each block position is decoded from softmax(l) and fed back to the local
 * head; the finished block is verified by the target model (Algorithm 1).
 * This library runs that loop as hand-written CUDA kernels at temperature 0
 * (Decode = argmax, lowest vocabulary index on exact ties; greedy
 * verification) and at temperature 1 (Decode = a Gumbel-max draw; lossless
 * speculative-sampling verification), and estimates the unigram prior from a
 * corpus on the device (Appendix A).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Pointers marked [device] are CUDA device pointers owned by the caller;
 *   tensors are contiguous, row-major, the vocabulary dimension innermost,
 *   and 16-byte aligned. Pointers marked [host] are ordinary host memory.
 * - Calls are asynchronous on the given stream (a cudaStream_t; NULL is the
 *   legacy default stream) and never synchronise, except dels_read_status.
 * - The library allocates no memory and keeps no state between calls, with
 *   one exception: dels_combine_argmax_noalloc keeps a fixed scratch array per
 *   device and caches its address (see there). Every other
 *   call takes a caller-owned device workspace of at least the size its
 *   *_workspace_bytes function returns for the same arguments on the current
 *   device. A workspace must be zero-filled once before its first use (for
 *   example with cudaMemset); every call leaves it ready for the next call.
 *   Calls that share a workspace must be ordered on one stream. Calls with
 *   distinct workspaces may be issued from several host threads at once
 *   (except the profiler switches, and dels_combine_argmax_noalloc, whose
 *   calls share one scratch per device).
 * - Return value: DELS_OK (0) or a negative DELS_ERR_* code detected on the
 *   host, in which case nothing was enqueued. Errors detected on the device
 *   (non-finite logits, an out-of-range token, a timed-out wait) are OR-ed
 *   into a status word inside the workspace; read and clear it with
 *   dels_read_status.
 * - dtype codes: DELS_F32 (IEEE float32) or DELS_BF16 (bfloat16 bit pattern).
 */
#ifndef DELS_H_
#define DELS_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Binary-compatible with cudaStream_t (struct CUstream_st*). */
typedef struct CUstream_st* dels_stream_t;

/* ---- status codes ------------------------------------------------------ */
enum {
  DELS_OK = 0,
  /* detected on the host; nothing was enqueued */
  DELS_ERR_NULL_POINTER = -1,      /* a required pointer is NULL */
  DELS_ERR_BAD_SHAPE = -2,         /* a size is out of the supported range */
  DELS_ERR_BAD_DTYPE = -3,         /* unknown or unsupported dtype code */
  DELS_ERR_ALIGNMENT = -4,         /* a pointer or row pitch is not 16-byte aligned */
  DELS_ERR_WORKSPACE = -5,         /* workspace NULL or smaller than required */
  DELS_ERR_UNSUPPORTED = -6,       /* head kind / dims this build does not run */
  DELS_ERR_CUDA = -7,              /* a CUDA runtime or driver call failed */
  DELS_ERR_TOO_LARGE = -8,         /* problem needs more than the fixed no-allocation scratch */
  /* detected on the device; bits of the workspace status word */
  DELS_STATUS_NONFINITE = 1,       /* NaN or +inf logit, or a row that is all -inf */
  DELS_STATUS_TIMEOUT = 2,         /* a bounded device-side wait expired */
  DELS_STATUS_BAD_TOKEN = 4        /* a draft or loss-masked corpus token outside [0, V) */
};

typedef enum { DELS_F32 = 0, DELS_BF16 = 1 } dels_dtype;

typedef enum {
  DELS_HEAD_GRU = 0,    /* Appendix A RNN head (the paper's default)      */
  DELS_HEAD_MLP = 1,    /* window MLP over the last `window` drafted tokens */
  DELS_HEAD_XFMR = 2,   /* 1-layer causal transformer over the block prefix */
  DELS_HEAD_MARKOV = 3  /* Appendix A Markov head                        */
} dels_head_kind;

/*
 * Local head (short-context expert) weights. All matrices are [device],
 * row-major [out, in] like a Linear layer, dtype `wdtype` (bf16 heads run the
 * matrix products on tcgen05 tensor cores; f32 heads on CUDA cores). V is the
 * vocabulary size of the call. Weight slots by kind:
 *
 * DELS_HEAD_GRU  (Appendix A): emb = E_tgt [V, d_model];
 *     w[0] = W_ih [3*d_hidden, d_model], gate rows ordered (r, z, n);
 *     w[1] = W_hh [3*d_hidden, d_hidden]; w[2] = W_rank [d_rank, d_hidden];
 *     w_vocab = W_vocab [V, d_rank].
 *     h_j = GRU(E_tgt[x_{j-1}], h_{j-1}) bias-free (PyTorch gate form),
 *     h_0 = 0; r_j = SiLU(W_rank h_j); l_S = W_vocab r_j.
 *     Optional, bf16 heads only: w[3] = G [V, 3*d_hidden] float32, the input
 *     table G = E_tgt W_ih^T written by dels_gru_build_input_table. When set,
 *     the input product W_ih E_tgt[x] of every step is read as row x of G
 *     instead of being recomputed (same value up to float32 summation order);
 *     w[0] is then not read by dels_draft_block.
 * DELS_HEAD_MLP: emb = E [V, d_model]; w[0] = W_1 [d_hidden, window*d_model];
 *     w[1] = W_2 [d_hidden, d_hidden] when n_layers == 2; w_vocab [V, d_hidden];
 *     d_rank must equal d_hidden. u = [E x_{j-1}; ...; E x_{j-window}] with
 *     zero blocks before the block start; h = GELU(W_1 u) (then GELU(W_2 h)).
 * DELS_HEAD_XFMR: emb = E [V, d_model]; w[0] = P [max_pos, d_model] position
 *     table; w[1..4] = W_q, W_k, W_v, W_o [d_model, d_model];
 *     w[5] = W_1 [d_hidden, d_model]; w[6] = W_2 [d_model, d_hidden];
 *     w_vocab [V, d_model]; d_rank must equal d_model. Pre-RMSNorm block
 *     (eps 1e-6, unit gain), n_heads causal heads, GELU FFN, final RMSNorm.
 * DELS_HEAD_MARKOV (Appendix A): emb = E_M [V, d_rank]; w_vocab = W_M [V, d_rank];
 *     l_S = W_M E_M[x_{j-1}].
 *
 * Activations that feed a bf16 product are rounded to bf16 (round to nearest
 * even); accumulation and the recurrent GRU state are float32. Exception: the
 * transformer head's own products (W_q, W_k, W_v, W_o, W_1, W_2) take their
 * activations at float32 precision, passed to the tensor cores as the exact
 * three-term bf16 expansion hi + mid + lo of each value; its feature is
 * rounded to bf16 for W_vocab like the other heads'.
 */
typedef struct {
  dels_head_kind kind;
  dels_dtype wdtype;
  int d_model;
  int d_hidden;
  int d_rank;
  int window;
  int n_layers;
  int n_heads;
  int max_pos;
  const void* emb;
  const void* w[8];
  const void* w_vocab;
} dels_local_head;

/* ---- self test of the bounded waits ------------------------------------- */

/*
 * Every wait inside the library's kernels (on an mbarrier, a flag or another
 * CTA) has a time limit; when it runs out the kernel stops waiting, frees
 * what it holds, returns, and sets DELS_STATUS_TIMEOUT in the status word.
 * This launches one small tensor-core product whose producer never issues a
 * load, so each wait expires (after 0.1 s) and the status word reports
 * DELS_STATUS_TIMEOUT; the context stays usable. (A test hook; the paper has
 * no counterpart.) `workspace` [device] >= dels_selftest_timeout_bytes(),
 * zero-filled, 16-byte aligned; read the status with dels_read_status.
 */
size_t dels_selftest_timeout_bytes(void);
int dels_selftest_timeout(void* workspace, size_t workspace_bytes, dels_stream_t stream);

/* ---- self test of the Gumbel transform ---------------------------------- */

/*
 * Writes g[i] = the device's Gumbel variate of the 32-bit Philox output word
 * bits[i]: u = (floor(bits / 2^9) + 1/2) / 2^23, g = -ln(-ln u), computed as
 * every temperature-1 kernel of the library computes it (a test hook for
 * its error against the exact transform; the paper has no counterpart).
 * `bits` [device, n uint32] and `g` [device, n float32], caller-owned.
 * Asynchronous on `stream`. Returns DELS_OK, DELS_ERR_BAD_SHAPE for n < 0,
 * DELS_ERR_NULL_POINTER for a missing pointer with n > 0, or DELS_ERR_CUDA.
 */
int dels_selftest_gumbel(const uint32_t* bits, float* g, long long n, dels_stream_t stream);

/* ---- GRU input table (head preparation, once per set of weights) -------- */

/*
 * The GRU's input product depends on the previous token only:
 * W_ih E_tgt[x] = (E_tgt W_ih^T)[x] (Appendix A). Precomputing the table
 * G = E_tgt W_ih^T [V, 3*d_hidden] float32 once per head trades HBM capacity
 * (V * 3 * d_hidden * 4 bytes, 1.87 GB for V = 151936, d_hidden = 1024) for
 * the W_ih stream of every drafted position (3*d_hidden*d_model*2 bytes).
 * (The paper computes the product directly; this is an implementation
 * choice with the same result up to float32 summation order.)
 *
 * dels_gru_input_table_bytes: bytes of G for this head and V; 0 if the head
 * is not a bf16 GRU head.
 * dels_gru_build_input_table: writes G into `table` [device], caller-owned,
 * >= dels_gru_input_table_bytes bytes, 16-byte aligned. Reads head->emb and
 * head->w[0] (bf16). `workspace` [device] >= 256 bytes, zero-filled, holds
 * the device status word (read with dels_read_status). Asynchronous on
 * `stream`; bf16 products with float32 accumulation on tensor cores.
 * Returns DELS_OK or a negative host-detected error (nothing enqueued).
 */
size_t dels_gru_input_table_bytes(const dels_local_head* head, int V);
int dels_gru_build_input_table(const dels_local_head* head, int V, float* table, size_t table_bytes,
                               void* workspace, size_t workspace_bytes, dels_stream_t stream);

/* ---- per-block drafting (Algorithm 1, temperature 0) --------------------- */

/* Workspace bytes for dels_draft_block with these arguments on the current
 * device; 0 if the arguments are not supported. */
size_t dels_draft_workspace_bytes(const dels_local_head* head, int B, int n, int V);

/*
 * Drafts one block of n tokens for each of B independent requests
 * (Algorithm 1; fusion of Section 4.3):
 *   x_0 = argmax_v l_L[b,0,v]                          (no head, no prior)
 *   for j = 1..n-1:  l_S = head(x_{0:j-1});
 *                    x_j = argmax_v l_L[b,j,v] + alpha*l_S[v] - beta*l_P[v]
 * long_logits  [device] [B, n, V] of logit_dtype (DFlash logits l_L).
 * log_prior    [device] [V] float32 log unigram prior l_P (finite).
 * out_tokens   [device] [B, n] int32 drafted tokens.
 * out_logprob  [device] [B, n] float32 log softmax of the fused row at x_j.
 * out_top2_gap [device] [B, n] float32 top-1 minus top-2 fused value; may be NULL.
 * Limits: 1 <= B <= 128, 1 <= n <= 32, 8 <= V < 2^31, V % 8 == 0; bf16 heads
 * need d_model, d_hidden, d_rank multiples of 16 (d_rank <= 4096); the
 * transformer head needs n <= max_pos, d_model % n_heads == 0, d_model <=
 * 32768 and a head width d_model / n_heads <= 8192 (DELS_ERR_UNSUPPORTED
 * otherwise).
 * B == 0 is a no-op.
 */
int dels_draft_block(const dels_local_head* head, const void* long_logits, dels_dtype logit_dtype,
                     const float* log_prior, float alpha, float beta, int B, int n, int V,
                     int32_t* out_tokens, float* out_logprob, float* out_top2_gap, void* workspace,
                     size_t workspace_bytes, dels_stream_t stream);

/*
 * dels_draft_block with position-dependent fusion weights: position j >= 1
 * uses l = l_L + alpha[j] l_S - beta[j] l_P (the learned per-position weights
 * reported in Appendix C). alpha, beta: [host] float arrays of n entries
 * (entry 0 is not used: position 0 has no head and no prior term), finite;
 * read during the call. Everything else as dels_draft_block (same workspace).
 */
int dels_draft_block_weighted(const dels_local_head* head, const void* long_logits, dels_dtype logit_dtype,
                              const float* log_prior, const float* alpha, const float* beta, int B, int n, int V,
                              int32_t* out_tokens, float* out_logprob, float* out_top2_gap, void* workspace,
                              size_t workspace_bytes, dels_stream_t stream);

/* ---- fused combine + argmax over independent rows ---------------------- */

size_t dels_combine_workspace_bytes(int rows, int V, dels_dtype dtype);

/*
 * For each of `rows` independent rows: l = l_L + alpha*l_S - beta*l_P
 * (Section 4.3), then x = argmax l (lowest index on ties),
 * logprob = l[x] - logsumexp(l), gap = l[x] - max_{v != x} l[v]
 * (+inf when V == 1). One pass over the inputs; no [rows, V] intermediate
 * is written.
 * long_logits, short_logits [device] [rows, V] of `dtype`; short_logits may
 * be NULL (then the alpha term is absent). log_prior [device] [V] float32,
 * may be NULL (then the beta term is absent).
 * out_token [device] [rows] int32; out_logprob [device] [rows] float32 (may
 * be NULL); out_top2_gap [device] [rows] float32 (may be NULL).
 * Limits: 0 <= rows < 2^31, 1 <= V < 2^31. Any V works; V % 8 == 0 (bf16) or
 * V % 4 == 0 (f32) takes the 128-bit vector path.
 */
int dels_combine_argmax(const void* long_logits, const void* short_logits, dels_dtype dtype,
                        const float* log_prior, float alpha, float beta, int rows, int V,
                        int32_t* out_token, float* out_logprob, float* out_top2_gap, void* workspace,
                        size_t workspace_bytes, dels_stream_t stream);

/*
 * dels_combine_argmax for callers that cannot allocate device memory.
 *
 * Same operation, arguments and outputs as dels_combine_argmax, minus the
 * workspace. (The paper has no counterpart; this is a deployment variant.)
 * It is meant for callers that own only the buffers they pass in and out —
 * a plugin inside a host framework whose allocator it cannot reach, or a
 * latency-critical loop where an allocation could stall the device — and so
 * cannot provide a workspace.
 *
 * Scratch: a fixed 4 MiB array compiled into the library; every GPU that
 * loads the library holds it until the process exits. A call whose scratch
 * need (dels_combine_workspace_bytes for the same rows, V, dtype) exceeds
 * 4 MiB returns DELS_ERR_TOO_LARGE and enqueues nothing; at V = 151936 that
 * is reached only beyond roughly 200,000 rows.
 * Set-up: the first call on a device, with that device current, looks up
 * the scratch's device address (cudaGetSymbolAddress) and caches it for the
 * rest of the process; make that first call before any stream capture. The
 * cached address does not survive cudaDeviceReset: after a reset of the
 * device, do not call this entry point again in the same process.
 * The call allocates nothing (no cudaMalloc, cudaFree or allocating library
 * routine). It clears the part of the scratch that must start at zero with
 * cudaMemsetAsync on `stream`. All calls on a device share the one scratch,
 * which keeps the last call's contents: calls that overlap on the GPU (on
 * different streams without ordering) race and give wrong results.
 * Device-detected errors cannot be read back through a status word here:
 * a non-finite row shows up as token -1 and logprob NaN in the outputs.
 */
int dels_combine_argmax_noalloc(const void* long_logits, const void* short_logits, dels_dtype dtype,
                                const float* log_prior, float alpha, float beta, int rows, int V,
                                int32_t* out_token, float* out_logprob, float* out_top2_gap,
                                dels_stream_t stream);

/* ---- temperature 1 (Algorithm 1 with Decode = a draw from the softmax) --- */

/*
 * Random numbers. Every uniform is drawn from Philox4x32-10 (Salmon et al.,
 * "Parallel random numbers: as easy as 1, 2, 3", SC 2011) under the key
 * (seed mod 2^32, seed div 2^32) with the counter (v / 4, step, b + 2^16 j +
 * 2^24 stream, 0) for vocabulary index v, block position j, request b and
 * stream (0 drafting, 1 acceptance tests, 2 residual / bonus draws); output
 * word v mod 4 (a 32-bit value h) gives u = (floor(h / 2^9) + 1/2) / 2^23.
 * Draws use the Gumbel-max rule: x = argmax_v (l_v + g_v), g = -log(-log u),
 * evaluated in float32 within 4e-6 of the exact transform for every u
 * (dels_selftest_gumbel exposes the device's g).
 * Give each block its own `step`; step >= 2^32 or B >= 2^16 returns
 * DELS_ERR_BAD_SHAPE.
 *
 * dels_draft_block_sampled: as dels_draft_block_weighted, but every position
 * is drawn: x_0 ~ softmax(l_L^(0)), x_j ~ softmax(l^(j)).
 *   out_logprob  [device] [B, n] float32 log softmax(l^(j))[x_j] (required: the
 *                verification's q_j(x_j));
 *   out_key_gap  [device] [B, n] float32 key gap k[x_j] - max_{v != x_j} k[v], or NULL;
 *   draft_state  [device] >= dels_draft_state_bytes(head, B, n), 16-byte aligned,
 *                or NULL: what dels_verify_block_sampled needs to rebuild a
 *                rejected position's draft distribution (the LSE of every
 *                fused row and the vocabulary-projection input of every
 *                position j >= 1); contents private to the library.
 *   alpha, beta  [host] [n] float32 per-position weights (entry 0 unused).
 * Requires d_rank * (2 for bf16 heads, 4 for float32 heads) to be a multiple of 16.
 */
size_t dels_draft_state_bytes(const dels_local_head* head, int B, int n);
int dels_draft_block_sampled(const dels_local_head* head, const void* long_logits, dels_dtype logit_dtype,
                             const float* log_prior, const float* alpha, const float* beta, int B, int n, int V,
                             uint64_t seed, uint64_t step, int32_t* out_tokens, float* out_logprob,
                             float* out_key_gap, void* draft_state, size_t state_bytes, void* workspace,
                             size_t workspace_bytes, dels_stream_t stream);

/*
 * Verification of a temperature-1 block by lossless speculative sampling
 * (accept with probability min(1, p/q), resample the residual), so that the
 * emitted tokens follow the target model's distribution:
 * for j = 0..n-1, x_j is accepted when u_j < p_j(x_j) / q_j(x_j), with p_j =
 * softmax(target row j), q_j the distribution x_j was drawn from
 * (exp(draft_logprob)), u_j the acceptance uniform of (b, j) (stream 1,
 * v = 0). At the first rejection a the bonus token is drawn from
 * max(0, p_a - q_a) (normalised) and after n acceptances from p_n, both by
 * the Gumbel-max rule with the residual stream (2) at position a (or n).
 * q_a is rebuilt from draft_state: l = l_L[b, a] + alpha[a] W_vocab r_a -
 * beta[a] l_P (l_L[b, 0] at a = 0) and its LSE.
 *   head, long_logits, log_prior, alpha, beta, seed, step, B, n, V: those of
 *        the dels_draft_block_sampled call that produced the block;
 *   draft_tokens [device] [B, n] int32, draft_logprob [device] [B, n] float32,
 *   draft_state [device]: that call's outputs;
 *   target_logits [device] [B, n+1, V] of target_dtype;
 *   out_accept_len [device] [B] int32 (0..n), out_bonus [device] [B] int32,
 *   out_bonus_gap [device] [B] float32 key gap of the bonus draw, or NULL.
 * Limits: 1 <= n <= 32; B <= 128 for bf16 heads.
 */
size_t dels_verify_sampled_workspace_bytes(const dels_local_head* head, int B, int n, int V, dels_dtype target_dtype);
int dels_verify_block_sampled(const dels_local_head* head, const int32_t* draft_tokens, const float* draft_logprob,
                              const void* draft_state, const void* long_logits, dels_dtype logit_dtype,
                              const float* log_prior, const float* alpha, const float* beta,
                              const void* target_logits, dels_dtype target_dtype, int B, int n, int V, uint64_t seed,
                              uint64_t step, int32_t* out_accept_len, int32_t* out_bonus, float* out_bonus_gap,
                              void* workspace, size_t workspace_bytes, dels_stream_t stream);

/* ---- greedy verification (Algorithm 1, last two steps) ------------------ */

size_t dels_verify_workspace_bytes(int B, int n, int V, dels_dtype dtype);

/*
 * Greedy verification of drafted blocks against the target's logits.
 * draft_tokens  [device] [B, n] int32 x_0..x_{n-1}.
 * target_logits [device] [B, n+1, V] of `dtype`: row j is the target's
 *               distribution for draft position j; row n is the bonus row.
 * t_j = argmax_v target[b,j,v] (lowest index on ties);
 * out_accept_len [device] [B] int32: a = number of leading j with x_j == t_j (0..n);
 * out_bonus      [device] [B] int32: t_a (the token the target adds);
 * out_target_argmax [device] [B, n+1] int32 t_j, may be NULL.
 * Limits: 0 <= B, 1 <= n <= 1024, 1 <= V < 2^31.
 */
int dels_verify_block(const int32_t* draft_tokens, const void* target_logits, dels_dtype dtype, int B, int n,
                      int V, int32_t* out_accept_len, int32_t* out_bonus, int32_t* out_target_argmax,
                      void* workspace, size_t workspace_bytes, dels_stream_t stream);

/* ---- helpers ------------------------------------------------------------ */

/*
 * Reads the device status word of `workspace` into *out_status (an OR of
 * DELS_STATUS_* bits, 0 when every call since the last read succeeded) and
 * clears it. Synchronises `stream`.
 */
int dels_read_status(void* workspace, dels_stream_t stream, int32_t* out_status);

/*
 * Unigram log prior of Appendix A on the host:
 *   l_P(v) = log( (counts[v] + lambda) / sum_u (counts[u] + lambda) ), in float64,
 * stored as float32. counts [host] [V] int64 >= 0; lambda > 0 (the paper uses 1);
 * out_log_prior [host] [V] float32.
 */
int dels_prior_from_counts(const int64_t* counts, int V, double lambda, float* out_log_prior);

/* ---- unigram prior estimation on the device (Appendix A) ----------------- */

/*
 * The prior the fusion subtracts is estimated once from the training corpus:
 * c(v) counts the corpus positions that carry loss (assistant-response
 * tokens) and hold token v; p0(v) = (c(v) + lambda) / sum_u (c(u) + lambda)
 * with lambda = 1 by default; l_P(v) = log p0(v).
 *
 * Corpus layout: tokens [device] [N] int32 ids (4-byte aligned; any offset
 * into a larger corpus is accepted, 16-byte alignment is fastest) and
 * loss_mask [device] [N] uint8, one byte per position, nonzero = the position
 * carries loss. Counts are uint64. A loss-masked position whose id lies
 * outside [0, V) is not counted: it is tallied separately and sets
 * DELS_STATUS_BAD_TOKEN in the workspace status word.
 */
size_t dels_prior_workspace_bytes(int V, int64_t N);

/*
 * Adds one corpus piece's loss-masked token counts to `counts`:
 *   counts[v] += #{ t < N : loss_mask[t] != 0 and tokens[t] == v }.
 * counts [device] [V] uint64, accumulated (zero it before the first piece);
 * tally  [device] [2] uint64 or NULL, accumulated: tally[0] += positions
 *        counted, tally[1] += loss-masked positions with an id outside [0, V).
 * workspace [device] >= dels_prior_workspace_bytes(V, N) (a workspace sized
 * for the longest piece serves every piece).
 * Large vocabularies count long pieces in two steps: the first positions
 * exactly, then the rest with the ids that are most frequent in `counts` so
 * far held on chip; the result is the exact count either way.
 * Limits: N >= 0 (N = 0 enqueues nothing), 1 <= V < 2^31.
 */
int dels_prior_count(const int32_t* tokens, const uint8_t* loss_mask, int64_t N, int V, uint64_t* counts,
                     uint64_t* tally, void* workspace, size_t workspace_bytes, dels_stream_t stream);

/*
 * l_P from counts on the device: the sum of the counts, then
 *   out_log_prior[v] = log(counts[v] + lambda) - log(sum_u counts[u] + V * lambda)
 * evaluated in float64 and stored as float32 (within one float32 rounding of
 * the exact value). counts [device] [V] uint64; out_log_prior [device] [V]
 * float32; lambda > 0 and finite; workspace >= dels_prior_workspace_bytes(V, 0).
 */
int dels_prior_log(const uint64_t* counts, int V, double lambda, float* out_log_prior, void* workspace,
                   size_t workspace_bytes, dels_stream_t stream);

/*
 * Both steps for a corpus held in device memory: zeroes counts kept in the
 * workspace, counts, and writes l_P. out_counts [device] [V] uint64 and
 * out_tally [device] [2] uint64 (as for dels_prior_count) are optional copies.
 * workspace >= dels_prior_workspace_bytes(V, N).
 */
int dels_prior_estimate(const int32_t* tokens, const uint8_t* loss_mask, int64_t N, int V, double lambda,
                        float* out_log_prior, uint64_t* out_counts, uint64_t* out_tally, void* workspace,
                        size_t workspace_bytes, dels_stream_t stream);

/* ---- instrumentation (not part of the method) ---------------------------- */

/* Kernel classes timed by the optional per-kernel profiler. */
enum {
  DELS_KCLASS_VOCAB_COMBINE = 0, /* tcgen05 vocabulary projection fused with the combine */
  DELS_KCLASS_HEAD_GEMM = 1,     /* tcgen05 local-head products                          */
  DELS_KCLASS_HEAD_MISC = 2,     /* head gates / norms / attention / f32 head kernels     */
  DELS_KCLASS_MERGE = 3,         /* per-position merge + next-input gather                */
  DELS_KCLASS_POS0 = 4,          /* position-0 row reduction                              */
  DELS_KCLASS_VERIFY = 5,        /* verification                                          */
  DELS_KCLASS_COMBINE = 6,       /* dels_combine_argmax                                   */
  DELS_KCLASS_DRAFT_BLOCK = 7,   /* persistent per-block drafting kernel (whole block)    */
  DELS_KCLASS_PRIOR = 8,         /* unigram prior estimation (count, sum, log)            */
  DELS_KCLASS_COUNT = 9
};

/*
 * Per-kernel timing for performance analysis. While enabled, every kernel the
 * library launches is bracketed by CUDA events recorded on the launching
 * stream (the events are created by the library and reused). dels_profile_read
 * waits for the recorded events and returns, for one kernel class, the number
 * of launches and their summed device time in milliseconds since the last
 * reset. Process-wide; not thread-safe against concurrent library calls.
 */
int dels_profile_enable(int on);
int dels_profile_reset(void);
int dels_profile_read(int kernel_class, int* out_launches, double* out_total_ms);

/* Human-readable name of a status or error code. */
const char* dels_status_string(int code);

/* Library ABI version (major * 10000 + minor * 100 + patch). */
int dels_version(void);

#ifdef __cplusplus
}
#endif

#endif /* DELS_H_ */
