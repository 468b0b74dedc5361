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
//   the range is short, and for the steps below.
// * Hot/cold (large vocabularies, long corpora): a short prefix is counted
//   exactly by the slices; the K ids with the largest counts so far become
//   the hot set (k_prior_select), addressed through a 16-ids-per-word remap
//   (16 presence bits + the number of hot ids before the word). The main pass
//   (k_prior_hot) counts hot ids in shared memory and appends the others to
//   a per-CTA cold buffer; the per-CTA hot bins are then summed
//   (k_prior_hot_reduce) and the cold buffer is counted by the slices.
//   Every position is counted exactly once whichever ids are hot; the hot
//   set only decides the speed.
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
constexpr int kSelectBuckets = 3776;         // count buckets of the hot-set choice (32 x 118)

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
// 64-bit counts at the end (coalesced atomics). Source: the corpus range
// (COLD = false; group 0 keeps the tallies) or the per-CTA cold buffers of
// k_prior_hot (COLD = true; every entry is an in-range id).
template <bool COLD>
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
  if (!COLD) {
    // every group sees every position; group 0's tallies are the ones kept
    visit<false>(a.range, member * kWarps + (threadIdx.x >> 5), members * kWarps,
                 [&](int id, uint32_t m, bool) {
                   const bool masked = m != 0u;
                   const bool in_range = (unsigned)id < (unsigned)a.V;
                   t.in += (masked && in_range) ? 1u : 0u;
                   t.out += (masked && !in_range) ? 1u : 0u;
                   const unsigned u = (unsigned)(id - lo);   // < nb only for in-range ids of the slice
                   if (masked && u < (unsigned)nb) atomicAdd(bins + u, 1u);
                 });
    if (g != 0) t = Tally{};
  } else {
    // regions start 16-byte aligned (cold_cap is a multiple of 4 entries)
    for (long long rgn = member; rgn < a.cold_regions; rgn += members) {
      const long long len = min((long long)__ldcg(a.cold_len + rgn), a.cold_cap);
      const int32_t* buf = a.cold_buf + rgn * a.cold_cap;
      const int4* b4 = reinterpret_cast<const int4*>(buf);
      const long long n4 = len / 4;
      constexpr int U = 4;
      for (long long i0 = threadIdx.x; i0 < n4; i0 += U * kThreads) {
        int4 v[U];
#pragma unroll
        for (int k = 0; k < U; ++k) {
          const long long i = i0 + (long long)k * kThreads;
          v[k] = i < n4 ? __ldcg(b4 + i) : make_int4(-1, -1, -1, -1);
        }
#pragma unroll
        for (int k = 0; k < U; ++k)
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            const unsigned u = (unsigned)(int4_at(v[k], c) - lo);
            if (u < (unsigned)nb) atomicAdd(bins + u, 1u);
          }
      }
      for (long long i = n4 * 4 + threadIdx.x; i < len; i += kThreads) {
        const unsigned u = (unsigned)(__ldcg(buf + i) - lo);
        if (u < (unsigned)nb) atomicAdd(bins + u, 1u);
      }
    }
  }
  __syncthreads();
  for (int b = threadIdx.x; b < nb; b += kThreads) {
    const unsigned c = bins[b];
    if (c) atomicAdd(a.counts + lo + b, (unsigned long long)c);
  }
  if (!COLD) flush_tally(t, a.tally, a.status, red);
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

// The hot set: the ids whose count so far is at least T, for the smallest
// bucket boundary T >= 1 that keeps the set within K slots (so it never
// exceeds K), as the remap entries[e] = presence bits of ids 16e..16e+15 in
// the low half and the number of hot ids before id 16e in the high half,
// plus slot_id[s] = the id of hot slot s. One CTA; the counts are read once
// into a byte copy min(c, 255) in shared memory, which decides presence when
// T <= 255 (otherwise the counts are read again).
__global__ void __launch_bounds__(kThreads) k_prior_select(PriorSelectArgs a) {
  extern __shared__ __align__(16) unsigned char c8[];   // [nent * 16] when a.cache_bytes
  __shared__ unsigned hist[kSelectBuckets];
  __shared__ unsigned wsum[kWarps];
  __shared__ unsigned wbase[kWarps];
  __shared__ unsigned thr_bucket;
  __shared__ unsigned run_base;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int i = threadIdx.x; i < kSelectBuckets; i += kThreads) hist[i] = 0u;
  if (a.cache_bytes)
    for (int i = a.V + threadIdx.x; i < a.nent * 16; i += kThreads) c8[i] = 0;
  if (threadIdx.x == 0) run_base = 0u;
  __syncthreads();
  pdl_wait();
  // most ids have tiny counts: buckets 0..7 are counted per thread (no
  // shared-memory atomics on a handful of addresses), the rest in smem
  constexpr int U = 8, kSmall = 8;
  unsigned small[kSmall];
#pragma unroll
  for (int j = 0; j < kSmall; ++j) small[j] = 0u;
  for (int v0 = threadIdx.x; v0 < a.V; v0 += U * kThreads) {
    unsigned long long c[U];
#pragma unroll
    for (int k = 0; k < U; ++k) {
      const int v = v0 + k * kThreads;
      c[k] = v < a.V ? __ldcg(a.counts + v) : ~0ull;
    }
#pragma unroll
    for (int k = 0; k < U; ++k) {
      const int v = v0 + k * kThreads;
      if (v < a.V) {
        if (c[k] < (unsigned long long)kSmall) {
#pragma unroll
          for (int j = 0; j < kSmall; ++j) small[j] += c[k] == (unsigned long long)j ? 1u : 0u;
        } else {
          atomicAdd(hist + count_bucket(c[k]), 1u);
        }
        if (a.cache_bytes) c8[v] = (unsigned char)min(c[k], 255ull);
      }
    }
  }
#pragma unroll
  for (int j = 0; j < kSmall; ++j) {
    unsigned x = small[j];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    if (lane == 0 && x) atomicAdd(hist + j, x);
  }
  __syncthreads();
  if (warp == 0) {
    // lane L holds buckets [per L, per L + per); S = #{c : bucket >= per L}
    constexpr int per = kSelectBuckets / 32;
    unsigned s = 0;
    for (int i = 0; i < per; ++i) s += hist[lane * per + i];
    unsigned S = s;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned y = __shfl_down_sync(0xffffffffu, S, o);
      if (lane + o < 32) S += y;
    }
    unsigned S_next = __shfl_down_sync(0xffffffffu, S, 1);
    if (lane == 31) S_next = 0u;
    int t = 0;
    if (S > (unsigned)a.K && S_next <= (unsigned)a.K) {
      // the crossing lies in this lane's range: smallest t with #{bucket >= t} <= K
      unsigned above = S_next;
      for (int b = lane * per + per - 1; b >= lane * per; --b) {
        if (above + hist[b] > (unsigned)a.K) {
          t = b + 1;
          break;
        }
        above += hist[b];
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t = max(t, __shfl_xor_sync(0xffffffffu, t, o));
    if (lane == 0) thr_bucket = (unsigned)max(t, 1);
  }
  __syncthreads();
  const unsigned long long T = bucket_low((int)thr_bucket);
  const bool from_cache = a.cache_bytes && T <= 255ull;
  // rounds of kThreads entries; thread i takes entry r * kThreads + i
  for (int e0 = 0; e0 < a.nent; e0 += kThreads) {
    const int e = e0 + threadIdx.x;
    unsigned bits = 0;
    if (e < a.nent) {
      if (from_cache) {
        const uint4 q = *reinterpret_cast<const uint4*>(c8 + (size_t)e * 16);
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int j = 0; j < 16; ++j)
          if (((w[j >> 2] >> (8 * (j & 3))) & 0xFFu) >= (uint32_t)T) bits |= 1u << j;
      } else {
        unsigned long long c[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const int v = e * 16 + j;
          c[j] = v < a.V ? __ldcg(a.counts + v) : 0ull;
        }
#pragma unroll
        for (int j = 0; j < 16; ++j)
          if (c[j] >= T) bits |= 1u << j;
      }
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
      const unsigned w0 = wsum[lane];
      unsigned w = w0;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const unsigned y = __shfl_up_sync(0xffffffffu, w, o);
        if (lane >= o) w += y;
      }
      wbase[lane] = w - w0;
    }
    __syncthreads();
    unsigned base = run_base + wbase[warp] + incl - cnt;
    if (e < a.nent) {
      a.entries[e] = bits | (base << 16);
      while (bits) {
        const int j = __ffs(bits) - 1;
        bits &= bits - 1u;
        if (base < (unsigned)a.K) a.slot_id[base] = e * 16 + j;
        ++base;
      }
    }
    __syncthreads();
    if (threadIdx.x == kThreads - 1) run_base = base;
    __syncthreads();
  }
  if (threadIdx.x == 0) *a.n_hot = min(run_base, (unsigned)a.K);
}

// Main pass over a long range: loss-masked hot ids are counted in shared
// memory, other in-range ids are appended to this CTA's cold buffer (past
// its capacity they go to the global counts directly). Writes the CTA's hot
// bins to partials[blockIdx.x][0..K) and its cold length.
__global__ void __launch_bounds__(kThreads, 1) k_prior_hot(PriorHotArgs a) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  uint32_t* ent = reinterpret_cast<uint32_t*>(smem_raw);
  unsigned* bins = ent + a.nent;
  __shared__ unsigned long long red[2 * kWarps];
  __shared__ unsigned cursor;
  pdl_wait();
  for (int i = threadIdx.x; i < a.nent; i += kThreads) ent[i] = __ldcg(a.entries + i);
  for (int i = threadIdx.x; i < a.K; i += kThreads) bins[i] = 0u;
  if (threadIdx.x == 0) cursor = 0u;
  __syncthreads();
  const int lane = threadIdx.x & 31;
  int32_t* cold = a.cold_buf + (long long)blockIdx.x * a.cold_cap;
  const unsigned cap = (unsigned)a.cold_cap;
  Tally t;
  auto put_cold = [&](unsigned slot, int id) {
    if (slot < cap) cold[slot] = id;
    else atomicAdd(a.counts + id, 1ull);
  };
  // true: hot (counted here); false: a loss-masked in-range id that is cold
  auto count_hot = [&](int id) -> bool {
    const uint32_t e = ent[id >> 4];
    const uint32_t bit = 1u << (id & 15);
    const uint32_t slot = (e >> 16) + __popc(e & (bit - 1u));
    if ((e & bit) && slot < (uint32_t)a.K) {
      atomicAdd(bins + slot, 1u);
      return true;
    }
    return false;
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
    uint32_t cold_bits = 0;
#pragma unroll
    for (int q = 0; q < 16; ++q) {
      // straight-line and predicated: no branch per position
      const int id = int4_at(tk[q >> 2], q & 3);
      const bool masked = mask_byte(mk[q >> 2], q & 3) != 0u;
      const bool in_range = (unsigned)id < (unsigned)a.V;
      const bool valid = masked && in_range;
      t.in += valid ? 1u : 0u;
      t.out += (masked && !in_range) ? 1u : 0u;
      uint32_t e = 0;
      if (valid) e = ent[id >> 4];
      const uint32_t bit = 1u << (id & 15);
      const uint32_t slot = (e >> 16) + __popc(e & (bit - 1u));
      const bool hot = (e & bit) != 0u && slot < (uint32_t)a.K;
      if (hot) atomicAdd(bins + slot, 1u);
      cold_bits |= (valid && !hot) ? (1u << q) : 0u;
    }
    // one cursor add per warp step: lanes take consecutive runs of the cold buffer
    const unsigned n = __popc(cold_bits);
    unsigned incl = n;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    const unsigned total = __shfl_sync(0xffffffffu, incl, 31);
    if (total) {
      unsigned base = 0;
      if (lane == 31) base = atomicAdd(&cursor, total);
      base = __shfl_sync(0xffffffffu, base, 31) + incl - n;
#pragma unroll
      for (int q = 0; q < 16; ++q)
        if ((cold_bits >> q) & 1u) put_cold(base++, int4_at(tk[q >> 2], q & 3));
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
    if (!count_hot(id)) put_cold(atomicAdd(&cursor, 1u), id);
  }
  __syncthreads();
  unsigned* out = a.partials + (long long)blockIdx.x * a.K;
  for (int i = threadIdx.x; i < a.K; i += kThreads) out[i] = bins[i];
  if (threadIdx.x == 0) a.cold_len[blockIdx.x] = min(cursor, cap);
  flush_tally(t, a.tally, a.status, red);
}

// counts[slot_id[s]] += sum over CTAs of partials[cta][s], for the n_hot slots.
__global__ void __launch_bounds__(kMapThreads) k_prior_hot_reduce(PriorHotArgs a) {
  pdl_wait();
  const unsigned n_hot = min(__ldcg(a.n_hot), (unsigned)a.K);
  for (long long s = (long long)blockIdx.x * kMapThreads + threadIdx.x; s < n_hot;
       s += (long long)gridDim.x * kMapThreads) {
    unsigned long long sum = 0;
    for (int c = 0; c < a.ctas; ++c) sum += __ldcg(a.partials + (long long)c * a.K + s);
    if (sum) {
      const int id = __ldcg(a.slot_id + s);
      a.counts[id] += sum;
    }
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
// stored as float32. Optionally copies the counts and the tally out (the
// one-call estimate keeps both in its workspace).
__global__ void __launch_bounds__(kMapThreads) k_prior_log(PriorLogArgs a) {
  pdl_wait();
  const double lam = a.lambda;
  const double log_s = log((double)__ldcg(a.total) + (double)a.V * lam);
  const long long stride = (long long)gridDim.x * kMapThreads;
  for (long long v = (long long)blockIdx.x * kMapThreads + threadIdx.x; v < a.V; v += stride) {
    const unsigned long long c = __ldcg(a.counts + v);
    a.out[v] = (float)(log((double)c + lam) - log_s);
    if (a.counts_out) a.counts_out[v] = c;
  }
  if (a.tally_out && blockIdx.x == 0 && threadIdx.x < 2) a.tally_out[threadIdx.x] = __ldcg(a.tally + threadIdx.x);
}

int max_smem_optin() {
  static int v = -1;
  if (v < 0) {
    int dev = 0, x = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&x, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
      x = 0;
    v = x;
  }
  return v;
}

// CTAs per SM that one k_prior_slices launch can keep resident
int slices_per_sm(size_t smem) {
  static size_t set_for[2] = {0, 0};
  int per_sm = 0;
  for (int c = 0; c < 2; ++c) {
    void (*k)(PriorSliceArgs) = c ? k_prior_slices<true> : k_prior_slices<false>;
    if (set_for[c] < smem) {
      if (cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess) return 0;
      set_for[c] = smem;
    }
    int v = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, k, kThreads, smem) != cudaSuccess) return 0;
    per_sm = c ? std::min(per_sm, v) : v;
  }
  return per_sm;
}

}  // namespace

PriorPlan plan_prior(int V, long long N, int sms) {
  PriorPlan p{};
  const int smem = max_smem_optin();
  if (smem <= 0 || sms <= 0 || V < 1) return p;
  // slices: the bins take all but a little of the shared memory
  const int bins_max = (smem - 2048) / 4;
  p.slices = (V + bins_max - 1) / bins_max;
  p.slice = (V + p.slices - 1) / p.slices;
  p.slice_smem = (size_t)p.slice * 4;
  // hot/cold: the remap and as many hot bins as fit beside it (slot numbers
  // live in the 16-bit high half of a remap entry)
  p.nent = (V + 15) / 16;
  const long long hot_bytes = (long long)smem - 2048 - (long long)p.nent * 4;
  p.K = hot_bytes > 0 ? (int)std::min<long long>(hot_bytes / 4 / 32 * 32, 65504) : 0;
  p.hot_smem = (size_t)(p.nent + p.K) * 4;
  const size_t cache = (size_t)p.nent * 16;
  p.select_cache = cache + 8192 + 16 * 1024 <= (size_t)smem ? cache : 0;   // beside the static hist
  p.ctas = sms;
  p.use_hot = p.slices > 1 && p.K >= 4096 && N >= kPriorHotMinN;
  if (p.use_hot) {
    p.prefix = std::min<long long>(N, std::max<long long>(kPriorHotMinN / 4, N / 64));
    const long long main_n = std::min<long long>(N - p.prefix, kPriorChunk);
    p.cold_cap = (std::max<long long>(4096, (main_n / 8 + sms - 1) / sms) + 127) / 128 * 128;
  }
  p.ok = true;
  return p;
}

cudaError_t launch_prior_slices(const PriorSliceArgs& a, bool cold, size_t smem, int max_members, int sms,
                                cudaStream_t s) {
  const int per_sm = slices_per_sm(smem);
  if (per_sm < 1 || per_sm * sms < a.slices) return cudaErrorInvalidConfiguration;
  const int members = std::max(1, std::min(per_sm * sms / a.slices, max_members));
  const dim3 grid((unsigned)(members * a.slices));
  return cold ? launch_pdl(k_prior_slices<true>, grid, dim3(kThreads), smem, s, a)
              : launch_pdl(k_prior_slices<false>, grid, dim3(kThreads), smem, s, a);
}

cudaError_t launch_prior_select(const PriorSelectArgs& a, cudaStream_t s) {
  static size_t set_for = 0;
  const size_t smem = a.cache_bytes;
  if (set_for < smem) {
    cudaError_t e = cudaFuncSetAttribute(k_prior_select, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    set_for = smem;
  }
  return launch_pdl(k_prior_select, dim3(1), dim3(kThreads), smem, s, a);
}

cudaError_t launch_prior_hot(const PriorHotArgs& a, size_t smem, cudaStream_t s) {
  static size_t set_for = 0;
  if (set_for < smem) {
    cudaError_t e = cudaFuncSetAttribute(k_prior_hot, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    set_for = smem;
  }
  cudaError_t e = launch_pdl(k_prior_hot, dim3((unsigned)a.ctas), dim3(kThreads), smem, s, a);
  if (e != cudaSuccess) return e;
  const int blocks = std::max(1, std::min(a.ctas * 4, (a.K + kMapThreads - 1) / kMapThreads));
  return launch_pdl(k_prior_hot_reduce, dim3((unsigned)blocks), dim3(kMapThreads), 0, s, a);
}

cudaError_t launch_prior_total(const PriorLogArgs& a, int sms, cudaStream_t s) {
  long long blocks = ((long long)a.V + 4 * kMapThreads - 1) / (4 * kMapThreads);
  blocks = std::max<long long>(1, std::min<long long>(blocks, std::min(sms, kPriorMaxPartials)));
  return launch_pdl(k_prior_total, dim3((unsigned)blocks), dim3(kMapThreads), 0, s, a);
}

cudaError_t launch_prior_log(const PriorLogArgs& a, int sms, cudaStream_t s) {
  long long blocks = ((long long)a.V + kMapThreads - 1) / kMapThreads;
  blocks = std::max<long long>(1, std::min<long long>(blocks, (long long)sms * 4));
  return launch_pdl(k_prior_log, dim3((unsigned)blocks), dim3(kMapThreads), 0, s, a);
}

}  // namespace dels
