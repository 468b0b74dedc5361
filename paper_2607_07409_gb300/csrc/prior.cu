// Unigram prior estimation on the device (Appendix A, "Unigram Prior
// Estimation"): c(v) counts the corpus positions whose loss mask is set and
// whose token is v; p0(v) = (c(v) + lambda) / sum_u (c(u) + lambda) and the
// prior logit is l_P(v) = log p0(v).
//
// Counting is a streaming pass over the corpus (4 bytes of id + 1 byte of
// mask per position) that HBM bandwidth should bound. Global atomics cannot
// keep up: token frequencies are Zipf-like, and the adds to the most frequent
// id (about 13% of positions) serialise at one L2 address. So the counts are
// kept per CTA in shared memory, which holds 227 KB: about 57K 32-bit bins,
// a third of a 152K vocabulary. Two pieces:
//
// * Slice histograms (k_prior_slices): the vocabulary is cut into P slices
//   that each fit; P groups of CTAs read the same positions, each group
//   counting one slice. Used alone when P = 1 (small vocabularies) or when
//   the range is short.
// * Hot ids on chip (large vocabularies, long corpora): a short prefix is
//   counted exactly by the slices; the ids with the largest counts so far
//   become the hot set, at most K of them (k_prior_hist, k_prior_mark,
//   k_prior_place: a count histogram, presence bits, slot numbers). A remap
//   word covers 15 ids: 15 presence bits and the 17-bit slot number of the
//   first hot one. The main pass (k_prior_hot) counts hot ids in 16-bit
//   shared-memory bins, two to a word (about 95K of them), which hand 2^15
//   to the global count each time they reach it; the few cold ids go to the
//   global counts directly. The per-CTA bins are summed at the end
//   (k_prior_hot_reduce). Every position is counted exactly once whichever
//   ids are hot; the hot set only decides the speed.
//
// The log step is a map over V after a two-level sum of the counts.
#include <algorithm>

#include "dels_device.cuh"

namespace dels {

namespace {

constexpr int kThreads = 1024;               // smem-bound kernels: one CTA per SM
constexpr int kWarps = kThreads / 32;
constexpr int kMapThreads = 256;             // the V-sized maps (sum, log)
constexpr int kWarpSpan = 512;               // positions a warp takes per vector step
constexpr int kSelectBuckets = kPriorHistBuckets;   // count buckets of the hot-set choice (32 x 118)
constexpr int kIdsPerWord = 15;              // remap word: 15 presence bits + a 17-bit slot number
constexpr unsigned kFlush = 0x8000u;         // a 16-bit hot bin hands this to the global count
constexpr int kLogTable = 256;               // log(c + lambda) tabulated for counts below this

struct Tally {   // per thread; a thread sees far fewer than 2^32 positions per launch
  unsigned in = 0, out = 0;
};

__device__ __forceinline__ unsigned long long warp_sum_u64(unsigned long long x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

__device__ __forceinline__ int int4_at(const int4& v, int k) {
  return k == 0 ? v.x : k == 1 ? v.y : k == 2 ? v.z : v.w;
}

// id / 15 for any 32-bit id: multiply by ceil(2^35 / 15) and keep bits 35 and up
__device__ __forceinline__ unsigned div15(unsigned id) { return __umulhi(id, 0x88888889u) >> 3; }

// byte k of w, zero-extended (k a compile-time constant after unrolling)
__device__ __forceinline__ uint32_t mask_byte(uint32_t w, int k) { return __byte_perm(w, 0u, 0x4440u | (unsigned)k); }

// Adds the block's tallies to the global pair (one atomic per CTA) and raises
// DELS_STATUS_BAD_TOKEN when a loss-masked id was out of range.
__device__ void flush_tally(Tally t, unsigned long long* tally, int* status, unsigned long long* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const unsigned long long tin = warp_sum_u64(t.in);
  const unsigned long long tout = warp_sum_u64(t.out);
  if (lane == 0) {
    red[2 * warp] = tin;
    red[2 * warp + 1] = tout;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long si = 0, so = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
      si += red[2 * w];
      so += red[2 * w + 1];
    }
    if (tally) {
      if (si) atomicAdd(tally, si);
      if (so) atomicAdd(tally + 1, so);
    }
    if (so) raise_status(status, DELS_STATUS_BAD_TOKEN);
  }
}

// Calls f(id, mask_byte, uniform) for every position of the range [0, r.n)
// that falls to this worker: vector steps of 512 positions go to warps
// (worker, worker + nworkers, ...), with all 32 lanes converged (uniform =
// true); the scalar head and tail go to single threads (uniform = false).
// STREAM: evict-first loads for data read once; otherwise L2-cached loads
// (the slice groups read each position P times).
template <bool STREAM, class F>
__device__ __forceinline__ void visit(const PriorRange& r, long long worker, long long nworkers, F&& f) {
  const int lane = threadIdx.x & 31;
  const long long steps = r.nvec / kWarpSpan;
  const int4* tv = reinterpret_cast<const int4*>(r.tokens + r.head);
  const uint32_t* mv = reinterpret_cast<const uint32_t*>(r.mask + r.head);
  for (long long st = worker; st < steps; st += nworkers) {
    const long long w0 = st * (kWarpSpan / 4) + lane;   // units of 4 positions
    int4 t[4];
    uint32_t m[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) t[k] = STREAM ? __ldcs(tv + w0 + 32 * k) : __ldcg(tv + w0 + 32 * k);
#pragma unroll
    for (int k = 0; k < 4; ++k) m[k] = STREAM ? __ldcs(mv + w0 + 32 * k) : __ldcg(mv + w0 + 32 * k);
#pragma unroll
    for (int q = 0; q < 16; ++q) f(int4_at(t[q >> 2], q & 3), mask_byte(m[q >> 2], q & 3), true);
  }
  const long long rest = r.n - r.nvec;
  for (long long j = worker * 32 + lane; j < rest; j += nworkers * 32) {
    const long long i = j < r.head ? j : j + r.nvec;
    f(r.tokens[i], (uint32_t)r.mask[i], false);
  }
}

// Slice histograms. CTA b counts slice b % P of the vocabulary over the
// positions its group member index b / P takes; the bins are added to the
// 64-bit counts at the end (coalesced atomics). Group 0 keeps the tallies.
__global__ void __launch_bounds__(kThreads) k_prior_slices(PriorSliceArgs a) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  unsigned* bins = reinterpret_cast<unsigned*>(smem_raw);
  __shared__ unsigned long long red[2 * kWarps];
  const int P = a.slices;
  const int g = blockIdx.x % P;
  const long long member = blockIdx.x / P, members = gridDim.x / P;
  const int lo = g * a.slice;
  const int nb = max(0, min(a.slice, a.V - lo));
  for (int b = threadIdx.x; b < nb; b += kThreads) bins[b] = 0u;
  __syncthreads();
  pdl_wait();
  Tally t;
  visit<false>(a.range, member * kWarps + (threadIdx.x >> 5), members * kWarps, [&](int id, uint32_t m, bool) {
    const bool masked = m != 0u;
    const bool in_range = (unsigned)id < (unsigned)a.V;
    t.in += (masked && in_range) ? 1u : 0u;
    t.out += (masked && !in_range) ? 1u : 0u;
    const unsigned u = (unsigned)(id - lo);   // < nb only for in-range ids of the slice
    if (masked && u < (unsigned)nb) atomicAdd(bins + u, 1u);
  });
  if (g != 0) t = Tally{};
  __syncthreads();
  for (int b = threadIdx.x; b < nb; b += kThreads) {
    const unsigned c = bins[b];
    if (c) atomicAdd(a.counts + lo + b, (unsigned long long)c);
  }
  flush_tally(t, a.tally, a.status, red);
}

// Count buckets of the hot-set choice: exact below 2048, then 32 buckets per
// power of two (monotone in c; 3744 buckets cover every 64-bit count).
__device__ __forceinline__ int count_bucket(unsigned long long c) {
  if (c < 2048ull) return (int)c;
  const int lg = 63 - __clzll((long long)c);
  return 2048 + (lg - 11) * 32 + (int)((c >> (lg - 5)) & 31ull);
}

__device__ __forceinline__ unsigned long long bucket_low(int b) {
  if (b < 2048) return (unsigned long long)b;
  if (b >= 2048 + 53 * 32) return ~0ull;   // past the last 64-bit bucket
  const int lg = (b - 2048) / 32 + 11, sub = (b - 2048) % 32;
  return (1ull << lg) | ((unsigned long long)sub << (lg - 5));
}

// Step 1 of the hot-set choice: the histogram of count buckets, into the
// global hist (zero on entry; k_prior_place clears it again). Most ids have
// tiny counts, so buckets 0..7 are counted per thread instead of with
// shared-memory atomics on a handful of addresses.
__global__ void __launch_bounds__(kThreads) k_prior_hist(PriorSelectArgs a) {
  __shared__ unsigned h[kSelectBuckets];
  const int lane = threadIdx.x & 31;
  for (int i = threadIdx.x; i < kSelectBuckets; i += kThreads) h[i] = 0u;
  __syncthreads();
  pdl_wait();
  constexpr int U = 4, kSmall = 8;
  unsigned small[kSmall];
#pragma unroll
  for (int j = 0; j < kSmall; ++j) small[j] = 0u;
  const int stride = gridDim.x * kThreads;
  for (int v0 = blockIdx.x * kThreads + threadIdx.x; v0 < a.V; v0 += U * stride) {
    unsigned long long c[U];
#pragma unroll
    for (int k = 0; k < U; ++k) {
      const int v = v0 + k * stride;
      c[k] = v < a.V ? __ldcg(a.counts + v) : ~0ull;
    }
#pragma unroll
    for (int k = 0; k < U; ++k) {
      if (v0 + k * stride >= a.V) continue;
      if (c[k] < (unsigned long long)kSmall) {
#pragma unroll
        for (int j = 0; j < kSmall; ++j) small[j] += c[k] == (unsigned long long)j ? 1u : 0u;
      } else {
        atomicAdd(h + count_bucket(c[k]), 1u);
      }
    }
  }
#pragma unroll
  for (int j = 0; j < kSmall; ++j) {
    unsigned x = small[j];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    if (lane == 0 && x) atomicAdd(h + j, x);
  }
  __syncthreads();
  for (int i = threadIdx.x; i < kSelectBuckets; i += kThreads)
    if (h[i]) atomicAdd(a.hist + i, h[i]);
}

// The smallest bucket boundary T >= 1 with #{v : c(v) >= T} <= K, from a
// shared-memory copy of the histogram (run by warp 0).
__device__ unsigned long long hot_threshold(const unsigned* hist, int K) {
  const int lane = threadIdx.x & 31;
  constexpr int per = kSelectBuckets / 32;
  unsigned s = 0;
  for (int i = 0; i < per; ++i) s += hist[lane * per + i];
  unsigned S = s;   // #{bucket >= per * lane}
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned y = __shfl_down_sync(0xffffffffu, S, o);
    if (lane + o < 32) S += y;
  }
  unsigned S_next = __shfl_down_sync(0xffffffffu, S, 1);
  if (lane == 31) S_next = 0u;
  int t = 0;
  if (S > (unsigned)K && S_next <= (unsigned)K) {
    // the crossing lies in this lane's buckets
    unsigned above = S_next;
    for (int i = per - 1; i >= 0; --i) {
      const unsigned h = hist[lane * per + i];
      if (above + h > (unsigned)K) {
        t = lane * per + i + 1;
        break;
      }
      above += h;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) t = max(t, __shfl_xor_sync(0xffffffffu, t, o));
  return bucket_low(max(t, 1));
}

// Step 2: presence bits. CTA c owns remap words [c * per, (c + 1) * per);
// hot ids get slot numbers counted from the CTA's first word (the CTA's own
// base is added by k_prior_place), and are listed in stage[15 * first word ..].
__global__ void __launch_bounds__(kThreads) k_prior_mark(PriorSelectArgs a) {
  __shared__ unsigned hs[kSelectBuckets];
  __shared__ unsigned wsum[kWarps];
  __shared__ unsigned wbase[kWarps];
  __shared__ unsigned long long thr;
  __shared__ unsigned run_base;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  pdl_wait();
  for (int i = threadIdx.x; i < kSelectBuckets; i += kThreads) hs[i] = __ldcg(a.hist + i);
  __syncthreads();
  if (warp == 0) {
    const unsigned long long T = hot_threshold(hs, a.K);
    if (lane == 0) {
      thr = T;
      run_base = 0u;
    }
  }
  __syncthreads();
  const unsigned long long T = thr;
  const int per = (a.nent + gridDim.x - 1) / gridDim.x;
  const int w_begin = min(a.nent, (int)blockIdx.x * per), w_end = min(a.nent, w_begin + per);
  int32_t* stage = a.stage + (long long)w_begin * kIdsPerWord;
  for (int w0 = w_begin; w0 < w_end; w0 += kThreads) {
    const int w = w0 + threadIdx.x;
    unsigned bits = 0;
    if (w < w_end) {
      unsigned long long c[kIdsPerWord];
#pragma unroll
      for (int j = 0; j < kIdsPerWord; ++j) {
        const int v = w * kIdsPerWord + j;
        c[j] = v < a.V ? __ldcg(a.counts + v) : 0ull;
      }
#pragma unroll
      for (int j = 0; j < kIdsPerWord; ++j)
        if (c[j] >= T) bits |= 1u << j;
    }
    const unsigned cnt = __popc(bits);
    unsigned incl = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    if (warp == 0) {
      const unsigned x0 = wsum[lane];
      unsigned x = x0;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const unsigned y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
      }
      wbase[lane] = x - x0;
    }
    __syncthreads();
    unsigned base = run_base + wbase[warp] + incl - cnt;   // local slot of this word's first hot id
    if (w < w_end) {
      a.entries[w] = bits | (base << kIdsPerWord);
      for (unsigned b = bits; b; b &= b - 1u) stage[base++] = w * kIdsPerWord + (__ffs(b) - 1);
    }
    __syncthreads();
    if (threadIdx.x == kThreads - 1) run_base = base;
    __syncthreads();
  }
  if (threadIdx.x == 0) a.cta_total[blockIdx.x] = run_base;
}

// Step 3: each CTA adds its base (the hot ids of the CTAs before it) to its
// remap words and moves its staged ids to slot_id. A word whose slots would
// not all fit in K (never, when the histogram is right) is left with no hot
// ids, so its ids are counted as cold. CTA 0 clears the histogram.
__global__ void __launch_bounds__(kMapThreads) k_prior_place(PriorSelectArgs a) {
  __shared__ unsigned base_s, total_s;
  pdl_wait();
  if (threadIdx.x < 32) {
    const int lane = threadIdx.x;
    unsigned before = 0, total = 0;
    for (int c = lane; c < (int)gridDim.x; c += 32) {
      const unsigned x = __ldcg(a.cta_total + c);
      total += x;
      if (c < (int)blockIdx.x) before += x;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      before += __shfl_xor_sync(0xffffffffu, before, o);
      total += __shfl_xor_sync(0xffffffffu, total, o);
    }
    if (lane == 0) {
      base_s = before;
      total_s = total;
    }
  }
  __syncthreads();
  const unsigned base = base_s;
  const int per = (a.nent + gridDim.x - 1) / gridDim.x;
  const int w_begin = min(a.nent, (int)blockIdx.x * per), w_end = min(a.nent, w_begin + per);
  for (int w = w_begin + threadIdx.x; w < w_end; w += kMapThreads) {
    const uint32_t e = __ldcg(a.entries + w);
    const unsigned bits = e & ((1u << kIdsPerWord) - 1u);
    const unsigned slot0 = base + (e >> kIdsPerWord);
    a.entries[w] = slot0 + __popc(bits) <= (unsigned)a.K ? (bits | (slot0 << kIdsPerWord)) : 0u;
  }
  const unsigned mine = __ldcg(a.cta_total + blockIdx.x);
  const int32_t* stage = a.stage + (long long)w_begin * kIdsPerWord;
  for (unsigned i = threadIdx.x; i < mine; i += kMapThreads)
    if (base + i < (unsigned)a.K) a.slot_id[base + i] = __ldcg(stage + i);
  if (blockIdx.x == 0) {
    if (threadIdx.x == 0) *a.n_hot = min(total_s, (unsigned)a.K);
    for (int i = threadIdx.x; i < kSelectBuckets; i += kMapThreads) a.hist[i] = 0u;
  }
}

// Main pass over a long range: loss-masked hot ids are counted in 16-bit
// shared-memory bins (two per word; a bin that reaches 2^15 hands 2^15 to the
// global count, so it never carries into its neighbour), the others go to the
// global counts directly. Writes the CTA's bin words to partials.
__global__ void __launch_bounds__(kThreads, 1) k_prior_hot(PriorHotArgs a) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  uint32_t* ent = reinterpret_cast<uint32_t*>(smem_raw);
  unsigned* words = ent + a.nent;
  __shared__ unsigned long long red[2 * kWarps];
  const int kw = (a.K + 1) / 2;
  pdl_wait();
  for (int i = threadIdx.x; i < a.nent; i += kThreads) ent[i] = __ldcg(a.entries + i);
  for (int i = threadIdx.x; i < kw; i += kThreads) words[i] = 0u;
  __syncthreads();
  const int lane = threadIdx.x & 31;
  Tally t;
  // one loss-masked in-range id
  auto count_one = [&](int id) {
    const unsigned q = div15((unsigned)id);
    const uint32_t e = ent[q];
    const uint32_t bit = 1u << ((unsigned)id - q * kIdsPerWord);
    const uint32_t slot = (e >> kIdsPerWord) + __popc(e & (bit - 1u));
    if ((e & bit) != 0u && slot < (uint32_t)a.K) {
      const unsigned sh = (slot & 1u) << 4;
      const unsigned old = atomicAdd(words + (slot >> 1), 1u << sh);
      if (((old >> sh) & 0xFFFFu) == kFlush - 1u) {
        atomicSub(words + (slot >> 1), kFlush << sh);
        atomicAdd(a.counts + id, (unsigned long long)kFlush);
      }
    } else {
      atomicAdd(a.counts + id, 1ull);
    }
  };
  const PriorRange& r = a.range;
  const long long worker = (long long)blockIdx.x * kWarps + (threadIdx.x >> 5);
  const long long nworkers = (long long)gridDim.x * kWarps;
  const long long steps = r.nvec / kWarpSpan;
  const int4* tv = reinterpret_cast<const int4*>(r.tokens + r.head);
  const uint32_t* mv = reinterpret_cast<const uint32_t*>(r.mask + r.head);
  for (long long st = worker; st < steps; st += nworkers) {
    const long long w0 = st * (kWarpSpan / 4) + lane;
    int4 tk[4];
    uint32_t mk[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) tk[k] = __ldcs(tv + w0 + 32 * k);
#pragma unroll
    for (int k = 0; k < 4; ++k) mk[k] = __ldcs(mv + w0 + 32 * k);
#pragma unroll
    for (int q = 0; q < 16; ++q) {
      const int id = int4_at(tk[q >> 2], q & 3);
      const bool masked = mask_byte(mk[q >> 2], q & 3) != 0u;
      const bool in_range = (unsigned)id < (unsigned)a.V;
      t.in += (masked && in_range) ? 1u : 0u;
      t.out += (masked && !in_range) ? 1u : 0u;
      if (masked && in_range) count_one(id);
    }
  }
  const long long rest = r.n - r.nvec;
  for (long long j = worker * 32 + lane; j < rest; j += nworkers * 32) {
    const long long i = j < r.head ? j : j + r.nvec;
    const int id = r.tokens[i];
    if (!r.mask[i]) continue;
    if ((unsigned)id >= (unsigned)a.V) {
      ++t.out;
      continue;
    }
    ++t.in;
    count_one(id);
  }
  __syncthreads();
  unsigned* out = a.partials + (long long)blockIdx.x * kw;
  for (int i = threadIdx.x; i < kw; i += kThreads) out[i] = words[i];
  flush_tally(t, a.tally, a.status, red);
}

// counts[slot_id[s]] += the sum over CTAs of bin s (the 16-bit halves of the
// partial words), for the n_hot slots.
__global__ void __launch_bounds__(kMapThreads) k_prior_hot_reduce(PriorHotArgs a) {
  pdl_wait();
  const unsigned n_hot = min(__ldcg(a.n_hot), (unsigned)a.K);
  const long long kw = (a.K + 1) / 2;
  for (long long w = (long long)blockIdx.x * kMapThreads + threadIdx.x; 2 * w < n_hot;
       w += (long long)gridDim.x * kMapThreads) {
    unsigned long long lo = 0, hi = 0;
    constexpr int U = 8;
    for (int c0 = 0; c0 < a.ctas; c0 += U) {
      unsigned x[U];
#pragma unroll
      for (int k = 0; k < U; ++k) x[k] = c0 + k < a.ctas ? __ldcg(a.partials + (long long)(c0 + k) * kw + w) : 0u;
#pragma unroll
      for (int k = 0; k < U; ++k) {
        lo += x[k] & 0xFFFFu;
        hi += x[k] >> 16;
      }
    }
    if (lo) a.counts[__ldcg(a.slot_id + 2 * w)] += lo;
    if (hi && 2 * w + 1 < n_hot) a.counts[__ldcg(a.slot_id + 2 * w + 1)] += hi;
  }
}

// sum_v counts[v] in two levels: one partial per CTA, then the last CTA to
// finish (ticket) adds the partials, stores the total and re-arms the ticket.
__global__ void __launch_bounds__(kMapThreads) k_prior_total(PriorLogArgs a) {
  __shared__ unsigned long long red[kMapThreads / 32];
  __shared__ bool last;
  pdl_wait();
  unsigned long long s = 0;
  for (long long v = (long long)blockIdx.x * kMapThreads + threadIdx.x; v < a.V;
       v += (long long)gridDim.x * kMapThreads)
    s += __ldcg(a.counts + v);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  s = warp_sum_u64(s);
  if (lane == 0) red[warp] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long b = 0;
    for (int w = 0; w < kMapThreads / 32; ++w) b += red[w];
    a.partials[blockIdx.x] = b;
    __threadfence();
    last = atomicAdd(a.ticket, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!last || threadIdx.x != 0) return;
  __threadfence();
  unsigned long long t = 0;
  for (int b = 0; b < (int)gridDim.x; ++b) t += __ldcg(a.partials + b);
  *a.total = t;
  *a.ticket = 0u;
}

// l_P(v) = log(c(v) + lambda) - log(sum_u c(u) + V lambda), in float64,
// stored as float32; log(c + lambda) of the small counts (most ids) comes
// from a per-CTA table. Optionally copies the counts and the tally out (the
// one-call estimate keeps both in its workspace).
__global__ void __launch_bounds__(kMapThreads) k_prior_log(PriorLogArgs a) {
  __shared__ double tab[kLogTable];
  __shared__ double log_s_sh;
  const double lam = a.lambda;
  for (int i = threadIdx.x; i < kLogTable; i += kMapThreads) tab[i] = log((double)i + lam);
  pdl_wait();
  if (threadIdx.x == 0) log_s_sh = log((double)__ldcg(a.total) + (double)a.V * lam);
  __syncthreads();
  const double log_s = log_s_sh;
  const long long stride = (long long)gridDim.x * kMapThreads;
  for (long long v = (long long)blockIdx.x * kMapThreads + threadIdx.x; v < a.V; v += stride) {
    const unsigned long long c = __ldcg(a.counts + v);
    const double lc = c < (unsigned long long)kLogTable ? tab[c] : log((double)c + lam);
    a.out[v] = (float)(lc - log_s);
    if (a.counts_out) a.counts_out[v] = c;
  }
  if (a.tally_out && blockIdx.x == 0 && threadIdx.x < 2) a.tally_out[threadIdx.x] = __ldcg(a.tally + threadIdx.x);
}

// CTAs per SM that one k_prior_slices launch can keep resident
int slices_per_sm(size_t smem) {
  if (ensure_dynamic_smem(reinterpret_cast<const void*>(k_prior_slices), smem) != cudaSuccess) return 0;
  int v = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, k_prior_slices, kThreads, smem) != cudaSuccess) return 0;
  return v;
}

}  // namespace

PriorPlan plan_prior(int V, long long N, int sms) {
  PriorPlan p{};
  const int smem = device_max_smem_optin();
  if (smem <= 0 || sms <= 0 || V < 1) return p;
  // slices: the bins take all but a little of the shared memory
  const int bins_max = (smem - 2048) / 4;
  p.slices = (V + bins_max - 1) / bins_max;
  p.slice = (V + p.slices - 1) / p.slices;
  p.slice_smem = (size_t)p.slice * 4;
  // hot ids: the remap and as many 16-bit bins as fit beside it (slot
  // numbers have 17 bits in a remap word)
  p.nent = (V + kIdsPerWord - 1) / kIdsPerWord;
  const long long hot_bytes = (long long)smem - 2048 - (long long)p.nent * 4;
  p.K = hot_bytes > 0 ? (int)std::min<long long>(hot_bytes / 2 / 64 * 64, (1 << 17) - 64) : 0;
  p.hot_smem = (size_t)p.nent * 4 + (size_t)(p.K + 1) / 2 * 4;
  p.ctas = sms;
  p.select_ctas = std::min(sms, kPriorMaxPartials);
  // a CTA of the hot-set choice numbers its hot ids locally in the 17-bit field
  const long long words_per_cta = (p.nent + p.select_ctas - 1) / p.select_ctas;
  p.use_hot = p.slices > 1 && p.K >= 4096 && N >= kPriorHotMinN && words_per_cta * kIdsPerWord < (1 << 17);
  if (p.use_hot) p.prefix = std::min<long long>(N, std::max<long long>(kPriorHotMinN / 4, N / 64));
  p.ok = true;
  return p;
}

cudaError_t launch_prior_slices(const PriorSliceArgs& a, size_t smem, int max_members, int sms, cudaStream_t s) {
  const int per_sm = slices_per_sm(smem);
  if (per_sm < 1 || per_sm * sms < a.slices) return cudaErrorInvalidConfiguration;
  const int members = std::max(1, std::min(per_sm * sms / a.slices, max_members));
  return launch_pdl(k_prior_slices, dim3((unsigned)(members * a.slices)), dim3(kThreads), smem, s, a);
}

cudaError_t launch_prior_select(const PriorSelectArgs& a, int ctas, cudaStream_t s) {
  cudaError_t e = launch_pdl(k_prior_hist, dim3((unsigned)ctas), dim3(kThreads), 0, s, a);
  if (e != cudaSuccess) return e;
  e = launch_pdl(k_prior_mark, dim3((unsigned)ctas), dim3(kThreads), 0, s, a);
  if (e != cudaSuccess) return e;
  return launch_pdl(k_prior_place, dim3((unsigned)ctas), dim3(kMapThreads), 0, s, a);
}

cudaError_t launch_prior_hot(const PriorHotArgs& a, size_t smem, cudaStream_t s) {
  cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void*>(k_prior_hot), smem);
  if (e != cudaSuccess) return e;
  e = launch_pdl(k_prior_hot, dim3((unsigned)a.ctas), dim3(kThreads), smem, s, a);
  if (e != cudaSuccess) return e;
  const int kw = (a.K + 1) / 2;
  const int blocks = std::max(1, std::min(a.ctas * 4, (kw + kMapThreads - 1) / kMapThreads));
  return launch_pdl(k_prior_hot_reduce, dim3((unsigned)blocks), dim3(kMapThreads), 0, s, a);
}

cudaError_t launch_prior_total(const PriorLogArgs& a, int sms, cudaStream_t s) {
  long long blocks = ((long long)a.V + 4 * kMapThreads - 1) / (4 * kMapThreads);
  blocks = std::max<long long>(1, std::min<long long>(blocks, std::min(sms, kPriorMaxPartials)));
  return launch_pdl(k_prior_total, dim3((unsigned)blocks), dim3(kMapThreads), 0, s, a);
}

cudaError_t launch_prior_log(const PriorLogArgs& a, int sms, cudaStream_t s) {
  long long blocks = ((long long)a.V + 4 * kMapThreads - 1) / (4 * kMapThreads);
  blocks = std::max<long long>(1, std::min<long long>(blocks, (long long)sms));
  return launch_pdl(k_prior_log, dim3((unsigned)blocks), dim3(kMapThreads), 0, s, a);
}

}  // namespace dels
