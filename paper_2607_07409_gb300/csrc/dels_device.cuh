// Device-side building blocks for the DeLS-Spec drafting kernels (sm_103a).
//
// * RowAcc: one-pass state of a fused-logit row: running maximum (which is
//   also the top-1 value), its lowest index, the runner-up value, and the
//   sum of exp(l - max) rescaled online (Milakov & Gimelshein's online
//   normaliser). Log-softmax of the argmax is -log(sum); the top-2 gap is
//   max - second. This is the temperature-0 Decode of Algorithm 1.
// * Thin inline-PTX wrappers for mbarrier, TMA (cp.async.bulk.tensor),
//   tcgen05 (alloc / mma / commit / ld) and the async-proxy fences.
//   Every mbarrier wait is bounded by a global-timer deadline; on expiry the
//   CTA-wide abort flag is raised and the caller unwinds without hanging.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>
#include <cuda.h>

#include "dels_internal.h"

namespace dels {

// ----------------------------------------------------------------------------
// status word
// ----------------------------------------------------------------------------
__device__ __forceinline__ void raise_status(int* status, int code) {
  if (status) atomicOr(status, code);
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
  return t;
}

// ----------------------------------------------------------------------------
// bf16 <-> f32 (bit level; the 16 stored bits are the top half of an f32)
// ----------------------------------------------------------------------------
__device__ __forceinline__ float bf16lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__device__ __forceinline__ uint16_t f32_to_bf16_rne(float f) {
  uint32_t u = __float_as_uint(f);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

// ----------------------------------------------------------------------------
// RowAcc: top-1 / top-2 / online log-sum-exp of one row
// ----------------------------------------------------------------------------
struct RowAcc {
  float m;       // running max == top-1 value
  float s;       // sum exp(l - m)
  float second;  // runner-up value (equal to m on an exact tie)
  int idx;       // lowest index attaining m
};
static_assert(sizeof(RowAcc) == 16, "RowAcc is one 16-byte record");

__device__ __forceinline__ RowAcc rowacc_init() {
  RowAcc a;
  a.m = -INFINITY; a.s = 0.f; a.second = -INFINITY; a.idx = 0x7FFFFFFF;
  return a;
}

// Top-2 update for one element, visited in increasing index order within a
// thread (so a strict '>' keeps the lowest index on ties).
__device__ __forceinline__ void top2_push(float x, int v, float& best, float& second, int& idx) {
  const bool gt = x > best;
  second = gt ? best : fmaxf(second, x);
  idx = gt ? v : idx;
  best = gt ? x : best;
}

// Online-normaliser update for a chunk of K values whose top-2 has already
// been pushed (so `best` is the new running max); `m` is the old max.
template <int K>
__device__ __forceinline__ void lse_chunk(const float (&x)[K], float best, float& m, float& s) {
  if (best == -INFINITY) return;               // chunk and history all -inf
  s *= __expf(m - best);                       // m == -inf -> 0 (s was 0)
  m = best;
  float acc = 0.f;
#pragma unroll
  for (int i = 0; i < K; ++i) acc += __expf(x[i] - best);   // -inf -> 0; NaN/+inf -> NaN
  s += acc;
}

// Hardware base-2 exponential (PTX ex2.approx, flush-to-zero); -inf -> 0.
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

constexpr float kLog2e = 1.4426950408889634f;

// lse_chunk with the exponent pre-scaled to base 2: one FFMA + one ex2 per
// element (exp(x - best) = 2^(x*log2e - best*log2e)). The running sum is
// rescaled only when the maximum moved (rare after the first chunks).
template <int K>
__device__ __forceinline__ void lse_chunk_ex2(const float (&x)[K], float best, float& m, float& s) {
  if (best == -INFINITY) return;
  const float nb = -best * kLog2e;
  if (best != m) {
    s *= ex2_approx(fmaf(m, kLog2e, nb));
    m = best;
  }
  float acc = 0.f;
#pragma unroll
  for (int i = 0; i < K; ++i) acc += ex2_approx(fmaf(x[i], kLog2e, nb));
  s += acc;
}

// Merge two partial states (any index order). Ties on the value go to the
// lower index; the runner-up becomes the larger of the loser's top-1 and the
// winner's runner-up.
__device__ __forceinline__ RowAcc rowacc_merge(const RowAcc& a, const RowAcc& b) {
  const bool b_wins = (b.m > a.m) || (b.m == a.m && b.idx < a.idx);
  const RowAcc& w = b_wins ? b : a;
  const RowAcc& l = b_wins ? a : b;
  RowAcc r;
  r.m = w.m;
  r.idx = w.idx;
  r.second = fmaxf(w.second, l.m);
  if (r.m == -INFINITY) {
    r.s = (a.s != a.s || b.s != b.s) ? NAN : 0.f;
  } else {
    const float sa = (a.m == -INFINITY) ? (a.s != a.s ? NAN : 0.f) : a.s * __expf(a.m - r.m);
    const float sb = (b.m == -INFINITY) ? (b.s != b.s ? NAN : 0.f) : b.s * __expf(b.m - r.m);
    r.s = sa + sb;
  }
  return r;
}

__device__ __forceinline__ RowAcc rowacc_shfl_down(const RowAcc& a, int delta) {
  RowAcc r;
  r.m = __shfl_down_sync(0xFFFFFFFFu, a.m, delta);
  r.s = __shfl_down_sync(0xFFFFFFFFu, a.s, delta);
  r.second = __shfl_down_sync(0xFFFFFFFFu, a.second, delta);
  r.idx = __shfl_down_sync(0xFFFFFFFFu, a.idx, delta);
  return r;
}

// Warp-level merge in a fixed tree order; lane 0 holds the result.
__device__ __forceinline__ RowAcc rowacc_warp_reduce(RowAcc a) {
#pragma unroll
  for (int d = 16; d > 0; d >>= 1) a = rowacc_merge(a, rowacc_shfl_down(a, d));
  return a;
}

// A finished row is valid when it had at least one finite entry and no
// NaN / +inf (either of which turns s into NaN).
__device__ __forceinline__ bool rowacc_valid(const RowAcc& a) {
  return a.m > -INFINITY && a.m < INFINITY && a.s == a.s && a.s > 0.5f && a.s < INFINITY;
}

// A published RowAcc record (16 bytes), read past L1: records are written by
// other CTAs of the same or an earlier grid.
__device__ __forceinline__ RowAcc ld_rowacc_cg(const void* base, long long i) {
  const float4 v = __ldcg(reinterpret_cast<const float4*>(base) + i);
  RowAcc r;
  r.m = v.x; r.s = v.y; r.second = v.z; r.idx = __float_as_int(v.w);
  return r;
}

// Greedy decode of one fully merged row: token = argmax, logprob of the token
// = -log(sum exp(l - max)), top-2 gap. A row with no finite value flags the
// status word and yields token -1.
__device__ __forceinline__ void write_decode(const RowAcc& r, long long out_i, int32_t* tok, float* lp, float* gap,
                                             int* status) {
  const bool ok = rowacc_valid(r);
  if (!ok) raise_status(status, DELS_STATUS_NONFINITE);
  tok[out_i] = ok ? r.idx : -1;
  if (lp) lp[out_i] = ok ? -logf(r.s) : NAN;
  if (gap) gap[out_i] = ok ? (r.m - r.second) : NAN;
}

// ----------------------------------------------------------------------------
// bf16 activations of the heads' products, block sums
// ----------------------------------------------------------------------------
__device__ __forceinline__ float bf16_to_f(uint16_t u) { return __uint_as_float((uint32_t)u << 16); }

// Stores v for a bf16 product. terms = 1: v rounded to bf16 (nearest even)
// at row b of an [B, ld] buffer. terms = 3: the three-term expansion
// v = hi + mid + lo, each term the bf16 rounding of what the terms before it
// left (every difference is exact in float32, and the three terms hold all
// 24 significand bits of v), at rows b, B + b and 2B + b of a [3B, ld]
// buffer; a bf16 product over the three rows, accumulated in float32, then
// equals the product of the float32 activation.
__device__ __forceinline__ void store_bf16_terms(uint16_t* out, int terms, int B, int b, long long ld, long long o,
                                                 float v) {
  const uint16_t hi = f32_to_bf16_rne(v);
  out[(long long)b * ld + o] = hi;
  if (terms == 3) {
    const float r1 = v - bf16_to_f(hi);
    const uint16_t mid = f32_to_bf16_rne(r1);
    const float r2 = r1 - bf16_to_f(mid);
    out[(long long)(B + b) * ld + o] = mid;
    out[(long long)(2 * B + b) * ld + o] = f32_to_bf16_rne(r2);
  }
}

// Sum of v over the CTA (every thread gets the result).
__device__ __forceinline__ float block_sum(float v) {
  __shared__ float red[32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int d = 16; d > 0; d >>= 1) v += __shfl_down_sync(0xFFFFFFFFu, v, d);
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  const int nw = (blockDim.x + 31) >> 5;
  v = (threadIdx.x < nw) ? red[threadIdx.x] : 0.f;
  if (warp == 0) {
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) v += __shfl_down_sync(0xFFFFFFFFu, v, d);
    if (lane == 0) red[0] = v;
  }
  __syncthreads();
  return red[0];
}

// ----------------------------------------------------------------------------
// temperature 1: Gumbel-max draws with Philox4x32-10 uniforms
// ----------------------------------------------------------------------------
// Philox4x32-10 (Salmon, Moraes, Dror and Shaw, "Parallel random numbers: as
// easy as 1, 2, 3", SC 2011): ten rounds of two 32 x 32 -> 64-bit products on
// a counter of four 32-bit words, the key bumped by two Weyl constants
// between rounds.
constexpr uint32_t kPhiloxM0 = 0xD2511F53u, kPhiloxM1 = 0xCD9E8D57u;
constexpr uint32_t kPhiloxW0 = 0x9E3779B9u, kPhiloxW1 = 0xBB67AE85u;
enum { kStreamDraft = 0, kStreamAccept = 1, kStreamResidual = 2 };

__device__ __forceinline__ void philox4x32_10(uint32_t (&x)[4], uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint32_t hi0 = __umulhi(kPhiloxM0, x[0]), lo0 = kPhiloxM0 * x[0];
    const uint32_t hi1 = __umulhi(kPhiloxM1, x[2]), lo1 = kPhiloxM1 * x[2];
    x[0] = hi1 ^ x[1] ^ k0;
    x[1] = lo1;
    x[2] = hi0 ^ x[3] ^ k1;
    x[3] = lo0;
    k0 += kPhiloxW0;
    k1 += kPhiloxW1;
  }
}

// A 32-bit output word h gives u = (floor(h / 2^9) + 1/2) / 2^23, exact in
// float32: with k = floor(h / 2^9), the float 1 + k 2^-23 (k as the mantissa)
// minus (1 - 2^-24) is (2k + 1) 2^-24, which a float holds exactly.
__device__ __forceinline__ float uniform_from_bits(uint32_t h) {
  return __uint_as_float(0x3F800000u | (h >> 9)) - 0.999999940395355224609375f;
}

// E = -ln u for the uniforms above (u = (2k + 1) 2^-24), an exponential
// variate, without the general logarithm's range handling:
//  * u >= 7/8: with d = 1 - u (exact: Sterbenz), -ln(1 - d) is the series
//    d + d^2/2 + ... + d^8/8, truncated with a relative error below
//    d^8/9 / (1 - d) < 7e-9 for d <= 1/8 (Horner form, float32);
//  * u < 7/8: -ln 2 * log2 u through the hardware base-2 logarithm
//    (lg2.approx: absolute error about 2^-22 in log2 u, so a relative error
//    below 2^-22 / |log2(7/8)| = 1.3e-6 here).
// Relative error of E within ~1.5e-6 (checked exhaustively over all 2^23
// uniforms against the float64 logarithm by the test suite).
__device__ __forceinline__ float neg_log_uniform(float u) {
  const float d = 1.0f - u;
  float p = fmaf(d, 0.125f, 0.142857142857142857f);
  p = fmaf(d, p, 0.166666666666666667f);
  p = fmaf(d, p, 0.2f);
  p = fmaf(d, p, 0.25f);
  p = fmaf(d, p, 0.333333333333333333f);
  p = fmaf(d, p, 0.5f);
  p = fmaf(d, p, 1.0f);
  const float near_one = d * p;
  const float elsewhere = -0.693147180559945309f * __log2f(u);
  return d <= 0.125f ? near_one : elsewhere;
}

// Standard Gumbel variate g = -ln E = -ln(-ln u): E as above (its relative
// error is what g's absolute error inherits), the outer logarithm through
// the fast log. |g - g_exact| stays within a few 1e-6.
__device__ __forceinline__ float gumbel_from_bits(uint32_t h) { return -__logf(neg_log_uniform(uniform_from_bits(h))); }

// Key (seed mod 2^32, seed div 2^32), counter (c, step, b + 2^16 j + 2^24
// stream, 0): the 4 uniforms of vocabulary indices 4c .. 4c + 3, one per
// output word. step < 2^32, b < 2^16, j < 2^8 (checked by the entry points).
__device__ __forceinline__ void philox_block(uint64_t seed, uint64_t step, int b, int j, int stream, long long c,
                                             uint32_t (&x)[4]) {
  x[0] = (uint32_t)c;
  x[1] = (uint32_t)step;
  x[2] = (uint32_t)b | ((uint32_t)j << 16) | ((uint32_t)stream << 24);
  x[3] = 0u;
  philox4x32_10(x, (uint32_t)seed, (uint32_t)(seed >> 32));
}

// The Gumbel variates of vocabulary indices 8 c8 .. 8 c8 + 7 (two blocks).
__device__ __forceinline__ void gumbel8(uint64_t seed, uint64_t step, int b, int j, int stream, long long c8,
                                        float (&g)[8]) {
  uint32_t x[4], y[4];
  philox_block(seed, step, b, j, stream, 2 * c8, x);
  philox_block(seed, step, b, j, stream, 2 * c8 + 1, y);
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    g[k] = gumbel_from_bits(x[k]);
    g[4 + k] = gumbel_from_bits(y[k]);
  }
}

__device__ __forceinline__ uint32_t philox_word_at(uint64_t seed, uint64_t step, int b, int j, int stream,
                                                   long long v) {
  uint32_t x[4];
  philox_block(seed, step, b, j, stream, v >> 2, x);
  const int w = (int)(v & 3);
  return w == 0 ? x[0] : w == 1 ? x[1] : w == 2 ? x[2] : x[3];
}

__device__ __forceinline__ float gumbel_at(uint64_t seed, uint64_t step, int b, int j, int stream, long long v) {
  return gumbel_from_bits(philox_word_at(seed, step, b, j, stream, v));
}

__device__ __forceinline__ float uniform_at(uint64_t seed, uint64_t step, int b, int j, int stream, long long v) {
  return uniform_from_bits(philox_word_at(seed, step, b, j, stream, v));
}

// A record of temperature-1 drafting holds the largest key k = l + g, its
// index and the runner-up key, and s = sum_v exp(l_v - k_max): the key max
// is at least l_v + g_v, and g > -2.82 for these uniforms, so no term
// exceeds e^2.82. LSE(l) = k_max + log s and log softmax(l)[x] = -g_x - log s.
__device__ __forceinline__ bool rowacc_valid_sampled(const RowAcc& a) {
  return a.m > -INFINITY && a.m < INFINITY && a.s == a.s && a.s > 0.f && a.s < INFINITY;
}

__device__ __forceinline__ void write_decode_sampled(const RowAcc& r, long long out_i, int32_t* tok, float* lp,
                                                     float* gap, float* lse, int* status, float g_idx) {
  const bool ok = rowacc_valid_sampled(r);
  if (!ok) raise_status(status, DELS_STATUS_NONFINITE);
  tok[out_i] = ok ? r.idx : -1;
  const float ls = logf(r.s);
  if (lp) lp[out_i] = ok ? -g_idx - ls : NAN;
  if (gap) gap[out_i] = ok ? (r.m - r.second) : NAN;
  if (lse) lse[out_i] = ok ? r.m + ls : NAN;
}

// Decode of a merged record of position j for request b at either temperature;
// returns the token (-1 for an invalid row).
__device__ __forceinline__ int decode_record(const RowAcc& x, const SampleArgs& smp, int b, int n, int j,
                                             int32_t* tok, float* lp, float* gap, int* status) {
  const long long o = (long long)b * n + j;
  if (!smp.on) {
    write_decode(x, o, tok, lp, gap, status);
    return rowacc_valid(x) ? x.idx : -1;
  }
  const bool ok = rowacc_valid_sampled(x);
  const float gx = ok ? gumbel_at(smp.seed, smp.step, b, j, kStreamDraft, x.idx) : 0.f;
  write_decode_sampled(x, o, tok, lp, gap, smp.out_lse, status, gx);
  return ok ? x.idx : -1;
}

// Temperature-1 drafting keeps the vocabulary-projection input of every
// position j >= 1 for the verification's residual row: row b of `src_r`
// ([B][R] elements of r_bytes) goes to state_r[b][j]. Called by one CTA per
// request with all its threads.
__device__ __forceinline__ void keep_draft_input(const SampleArgs& smp, int b, int n, int j) {
  if (!smp.on || !smp.state_r || j < 1) return;
  const int vecs = smp.R * smp.r_bytes / 16;   // R * r_bytes is a multiple of 16
  const uint4* src = reinterpret_cast<const uint4*>(static_cast<const uint8_t*>(smp.src_r) +
                                                    (long long)b * smp.R * smp.r_bytes);
  uint4* dst = reinterpret_cast<uint4*>(static_cast<uint8_t*>(smp.state_r) +
                                        ((long long)b * n + j) * smp.R * smp.r_bytes);
  for (int i = threadIdx.x; i < vecs; i += blockDim.x) dst[i] = __ldcg(src + i);
}

// Argmax-only update (verification): value and lowest index.
__device__ __forceinline__ void argmax_push(float x, int v, float& best, int& idx, bool& nan_seen) {
  const bool gt = x > best;
  idx = gt ? v : idx;
  best = gt ? x : best;
  nan_seen |= (x != x);
}

// ----------------------------------------------------------------------------
// shared-memory address helpers
// ----------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ----------------------------------------------------------------------------
// mbarrier
// ----------------------------------------------------------------------------
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbarrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}

// Adds `bytes` to the barrier's expected transaction count without arriving.
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait: returns false (and raises the CTA abort flag) if the barrier
// phase has not completed by `deadline_ns`, or if another role of the CTA
// already aborted.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, uint64_t deadline_ns,
                                          volatile int* abort_flag) {
  uint32_t polls = 0;
  while (!mbar_try_wait(bar, parity)) {
    if ((++polls & 63u) == 0u) {
      if (*abort_flag) return false;
      if (globaltimer_ns() > deadline_ns) {
        *abort_flag = 1;
        return false;
      }
    }
  }
  return true;
}

// ----------------------------------------------------------------------------
// programmatic dependent launch: a kernel launched with the programmatic
// stream-serialization attribute may start before its predecessor finishes;
// it must call pdl_wait() before touching anything the predecessor writes.
// Both are no-ops for a normally launched kernel.
// ----------------------------------------------------------------------------
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Orders this thread's generic-proxy global writes before later async-proxy
// (TMA) accesses of the same memory, and vice versa.
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

__device__ __forceinline__ void st_release_gpu(unsigned* p, unsigned v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ unsigned ld_acquire_gpu(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// ----------------------------------------------------------------------------
// TMA (tiled tensor copies global -> shared, completion on an mbarrier)
// ----------------------------------------------------------------------------
__device__ __forceinline__ void tma_prefetch_desc(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar, int x, int y,
                                            uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%3, %4}], [%2], %5;" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y), "l"(policy)
      : "memory");
}

__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, uint64_t* bar, int x, int y,
                                            int z, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%3, %4, %5}], [%2], %6;" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y), "r"(z), "l"(policy)
      : "memory");
}

// Release/acquire fence at GPU scope (lighter than the sequentially
// consistent fence of __threadfence()).
__device__ __forceinline__ void fence_acq_rel_gpu() { asm volatile("fence.acq_rel.gpu;" ::: "memory"); }

// ---------------------------------------------------------------------------
// thread-block clusters: barrier and distributed shared memory

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// Full cluster barrier (every thread of every CTA of the cluster), with
// release/acquire ordering of the shared-memory writes before it.
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Address of the same shared-memory offset in CTA `rank` of this cluster.
__device__ __forceinline__ uint32_t cluster_map(uint32_t local_smem_addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(local_smem_addr), "r"(rank));
  return r;
}
// Arrive (release at cluster scope) on an mbarrier of another CTA of the
// cluster, addressed through cluster_map: the arriving thread's earlier
// writes to that CTA's shared memory are visible to whoever completes a wait
// on the barrier's phase.
__device__ __forceinline__ void mbar_arrive_remote(uint32_t cluster_bar_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_bar_addr) : "memory");
}
// Bounded wait with acquire at cluster scope (pairs with mbar_arrive_remote).
__device__ __forceinline__ bool mbar_wait_cluster(uint64_t* bar, uint32_t parity, uint64_t deadline_ns,
                                                  volatile int* abort_flag) {
  uint32_t polls = 0;
  for (;;) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    if (ok) return true;
    if ((++polls & 63u) == 0u) {
      if (*abort_flag) return false;
      if (globaltimer_ns() > deadline_ns) {
        *abort_flag = 1;
        return false;
      }
    }
  }
}
__device__ __forceinline__ void st_cluster_f32(uint32_t addr, float v) {
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(addr), "f"(v) : "memory");
}
__device__ __forceinline__ void st_cluster_v4(uint32_t addr, float a, float b, float c, float d) {
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(a), "f"(b), "f"(c), "f"(d)
               : "memory");
}

// L2 eviction-priority policies for the cache hints above.
__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t l2_policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t l2_policy_evict_normal() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// ----------------------------------------------------------------------------
// tcgen05 (5th-generation tensor cores, tensor memory)
// ----------------------------------------------------------------------------
__device__ __forceinline__ void tmem_alloc(uint32_t* smem_dst, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(smem_dst)),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, kind::f16 (bf16 inputs, f32 accumulate).
__device__ __forceinline__ void tc_mma_f16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                           uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive once on `bar` when all previously issued tcgen05 ops of this thread complete.
__device__ __forceinline__ void tc_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   smem_u32(bar))
               : "memory");
}

// 32 lanes x 32 consecutive 32-bit columns: thread i of the warp receives
// row (lane base + i), columns [col, col + 32).
__device__ __forceinline__ void tmem_ld_32x32b_x32(uint32_t taddr, float (&r)[32]) {
  uint32_t* u = reinterpret_cast<uint32_t*>(r);
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(u[0]), "=r"(u[1]), "=r"(u[2]), "=r"(u[3]), "=r"(u[4]), "=r"(u[5]), "=r"(u[6]), "=r"(u[7]),
        "=r"(u[8]), "=r"(u[9]), "=r"(u[10]), "=r"(u[11]), "=r"(u[12]), "=r"(u[13]), "=r"(u[14]), "=r"(u[15]),
        "=r"(u[16]), "=r"(u[17]), "=r"(u[18]), "=r"(u[19]), "=r"(u[20]), "=r"(u[21]), "=r"(u[22]), "=r"(u[23]),
        "=r"(u[24]), "=r"(u[25]), "=r"(u[26]), "=r"(u[27]), "=r"(u[28]), "=r"(u[29]), "=r"(u[30]), "=r"(u[31])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld_32x32b_x8(uint32_t taddr, float (&r)[8]) {
  uint32_t* u = reinterpret_cast<uint32_t*>(r);
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
               : "=r"(u[0]), "=r"(u[1]), "=r"(u[2]), "=r"(u[3]), "=r"(u[4]), "=r"(u[5]), "=r"(u[6]), "=r"(u[7])
               : "r"(taddr));
}
__device__ __forceinline__ void tmem_st_32x32b_x8(uint32_t taddr, const float (&r)[8]) {
  const uint32_t* u = reinterpret_cast<const uint32_t*>(r);
  asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"r"(taddr), "r"(u[0]),
               "r"(u[1]), "r"(u[2]), "r"(u[3]), "r"(u[4]), "r"(u[5]), "r"(u[6]), "r"(u[7])
               : "memory");
}
__device__ __forceinline__ void tmem_st_wait() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_ld_wait() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Shared-memory matrix descriptor for a K-major bf16 operand stored in the
// 128-byte-swizzled layout that TMA writes with CU_TENSOR_MAP_SWIZZLE_128B:
// rows of 64 elements (128 B), 8-row groups 1024 B apart. `addr` must lie in
// a 1024-byte-aligned buffer; stepping K by 16 elements adds 32 B to it.
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t addr) {
  uint64_t d = 0;
  d |= (uint64_t)((addr & 0x3FFFFu) >> 4);          // start address
  d |= (uint64_t)(16u >> 4) << 16;                   // leading byte offset (unused for SW128 K-major)
  d |= (uint64_t)(1024u >> 4) << 32;                 // stride byte offset: 8 rows x 128 B
  d |= (uint64_t)1 << 46;                            // descriptor version (fixed 0b001)
  d |= (uint64_t)2 << 61;                            // swizzle: 128 B
  return d;
}

// Instruction descriptor, kind::f16: bf16 A and B, f32 accumulator, both
// operands K-major, shape M x N.
__host__ __device__ __forceinline__ uint32_t idesc_bf16_f32(int M, int N) {
  return (1u << 4)                      // D format: f32
         | (1u << 7)                    // A format: bf16
         | (1u << 10)                   // B format: bf16
         | ((uint32_t)(N >> 3) << 17)   // N / 8
         | ((uint32_t)(M >> 4) << 24);  // M / 16
}

// Named barrier among a subset of warps (id 1..15, an immediate so that the
// compiler reserves it).
template <int ID>
__device__ __forceinline__ void named_bar_sync(int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"n"(ID), "r"(nthreads) : "memory");
}

}  // namespace dels
