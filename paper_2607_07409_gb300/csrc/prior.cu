// Unigram prior estimation on the device (Appendix A, "Unigram Prior
// Estimation"): c(v) counts the corpus positions whose loss mask is set and
// whose token is v; p0(v) = (c(v) + lambda) / sum_u (c(u) + lambda) and the
// prior logit is l_P(v) = log p0(v).
//
// The count is one streaming pass over the corpus (4 bytes of id + 1 byte of
// mask per position), bound by HBM bandwidth: each warp takes 512 positions
// per step with coalesced 16-byte id loads and 4-byte mask loads, and adds
// each loss-masked id into a 64-bit count with a fire-and-forget global
// atomic. The V counts (1.2 MB at V = 151936) stay resident in L2, where the
// atomics resolve; at HBM speed the corpus delivers about one position per
// 240 SM cycles, far below the L2 atomic rate, even for the most frequent id.
// The log step is a map over V after a two-level sum of the counts.
#include <algorithm>

#include "dels_device.cuh"

namespace dels {

namespace {

constexpr int kPriorThreads = 256;
constexpr int kWarpSpan = 512;   // positions a warp takes per step: 4 x (32 lanes x 4 ids)

__device__ __forceinline__ void count_one(int id, uint32_t m, int V, unsigned long long* counts,
                                          unsigned long long& n_in, unsigned long long& n_out) {
  if (m) {
    if ((unsigned)id < (unsigned)V) {
      atomicAdd(counts + id, 1ull);
      ++n_in;
    } else {
      ++n_out;
    }
  }
}

__device__ __forceinline__ void count_word(int4 t, uint32_t m, int V, unsigned long long* counts,
                                           unsigned long long& n_in, unsigned long long& n_out) {
  count_one(t.x, m & 0xFFu, V, counts, n_in, n_out);
  count_one(t.y, (m >> 8) & 0xFFu, V, counts, n_in, n_out);
  count_one(t.z, (m >> 16) & 0xFFu, V, counts, n_in, n_out);
  count_one(t.w, m >> 24, V, counts, n_in, n_out);
}

__device__ __forceinline__ unsigned long long warp_sum_u64(unsigned long long x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

// Sums x over the block into smem slot 0 of `red` (kPriorThreads / 32 entries);
// the result is valid in thread 0.
__device__ __forceinline__ unsigned long long block_sum_u64(unsigned long long x, unsigned long long* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  x = warp_sum_u64(x);
  if (lane == 0) red[warp] = x;
  __syncthreads();
  unsigned long long s = 0;
  if (threadIdx.x == 0)
    for (int w = 0; w < kPriorThreads / 32; ++w) s += red[w];
  return s;
}

// One pass over positions [0, N). Positions [head, head + nvec) go through
// the vector path (nvec a multiple of kWarpSpan, tokens + head 16-byte
// aligned, mask + head 4-byte aligned); the few others go one by one.
__global__ void __launch_bounds__(kPriorThreads) k_prior_count(PriorCountArgs a) {
  __shared__ unsigned long long red[2][kPriorThreads / 32];
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const long long gwarp = ((long long)blockIdx.x * kPriorThreads + threadIdx.x) >> 5;
  const long long nwarps = (long long)gridDim.x * (kPriorThreads / 32);
  unsigned long long n_in = 0, n_out = 0;

  const long long steps = a.nvec / kWarpSpan;
  const int4* tv = reinterpret_cast<const int4*>(a.tokens + a.head);
  const uint32_t* mv = reinterpret_cast<const uint32_t*>(a.mask + a.head);
  for (long long st = gwarp; st < steps; st += nwarps) {
    // 4 coalesced 512-byte id loads and 4 coalesced 128-byte mask loads per warp
    const long long w0 = st * (kWarpSpan / 4) + lane;   // index in units of 4 positions
    int4 t[4];
    uint32_t m[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) t[k] = __ldcs(tv + w0 + 32 * k);
#pragma unroll
    for (int k = 0; k < 4; ++k) m[k] = __ldcs(mv + w0 + 32 * k);
#pragma unroll
    for (int k = 0; k < 4; ++k) count_word(t[k], m[k], a.V, a.counts, n_in, n_out);
  }

  // the head (< 4 positions) and the tail (< kWarpSpan positions, or all of
  // them when the pointers do not allow the vector path)
  const long long rest = a.N - a.nvec;
  const long long tid = (long long)blockIdx.x * kPriorThreads + threadIdx.x;
  const long long nthr = (long long)gridDim.x * kPriorThreads;
  for (long long j = tid; j < rest; j += nthr) {
    const long long i = j < a.head ? j : j + a.nvec;
    count_one(a.tokens[i], a.mask[i], a.V, a.counts, n_in, n_out);
  }

  const int warp = threadIdx.x >> 5;
  n_in = warp_sum_u64(n_in);
  n_out = warp_sum_u64(n_out);
  if (lane == 0) {
    red[0][warp] = n_in;
    red[1][warp] = n_out;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long si = 0, so = 0;
    for (int w = 0; w < kPriorThreads / 32; ++w) {
      si += red[0][w];
      so += red[1][w];
    }
    if (a.tally) {
      if (si) atomicAdd(a.tally, si);
      if (so) atomicAdd(a.tally + 1, so);
    }
    if (so) raise_status(a.status, DELS_STATUS_BAD_TOKEN);
  }
}

// sum_v counts[v] in two levels: one partial per CTA, then the last CTA to
// finish (ticket) adds the partials, stores the total and re-arms the ticket.
__global__ void __launch_bounds__(kPriorThreads) k_prior_total(PriorLogArgs a) {
  __shared__ unsigned long long red[kPriorThreads / 32];
  __shared__ bool last;
  pdl_wait();
  unsigned long long s = 0;
  for (long long v = (long long)blockIdx.x * kPriorThreads + threadIdx.x; v < a.V;
       v += (long long)gridDim.x * kPriorThreads)
    s += __ldcg(a.counts + v);
  s = block_sum_u64(s, red);
  if (threadIdx.x == 0) {
    a.partials[blockIdx.x] = s;
    __threadfence();
    last = atomicAdd(a.ticket, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!last) return;
  __threadfence();
  unsigned long long t = 0;
  for (int b = threadIdx.x; b < (int)gridDim.x; b += kPriorThreads) t += __ldcg(a.partials + b);
  __syncthreads();
  t = block_sum_u64(t, red);
  if (threadIdx.x == 0) {
    *a.total = t;
    *a.ticket = 0u;
  }
}

// l_P(v) = log(c(v) + lambda) - log(sum_u c(u) + V lambda), in float64,
// stored as float32. Optionally copies the counts and the tally out (the
// one-call estimate keeps both in its workspace).
__global__ void __launch_bounds__(kPriorThreads) k_prior_log(PriorLogArgs a) {
  pdl_wait();
  const double lam = a.lambda;
  const double log_s = log((double)__ldcg(a.total) + (double)a.V * lam);
  const long long stride = (long long)gridDim.x * kPriorThreads;
  for (long long v = (long long)blockIdx.x * kPriorThreads + threadIdx.x; v < a.V; v += stride) {
    const unsigned long long c = __ldcg(a.counts + v);
    a.out[v] = (float)(log((double)c + lam) - log_s);
    if (a.counts_out) a.counts_out[v] = c;
  }
  if (a.tally_out && blockIdx.x == 0 && threadIdx.x < 2) a.tally_out[threadIdx.x] = __ldcg(a.tally + threadIdx.x);
}

}  // namespace

cudaError_t launch_prior_count(const PriorCountArgs& a, int sms, cudaStream_t s) {
  const long long steps = a.nvec / kWarpSpan;
  long long blocks = (steps + (kPriorThreads / 32) - 1) / (kPriorThreads / 32);
  const long long tail_blocks = (a.N - a.nvec + kPriorThreads - 1) / kPriorThreads;
  blocks = std::max(blocks, tail_blocks);
  // a grid-stride pass: every CTA resident at once, so none is left for a second wave
  static int per_sm = 0;
  if (per_sm == 0) {
    int v = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, k_prior_count, kPriorThreads, 0) != cudaSuccess || v < 1)
      v = 1;
    per_sm = v;
  }
  blocks = std::min<long long>(blocks, (long long)sms * per_sm);
  blocks = std::max<long long>(blocks, 1);
  return launch_pdl(k_prior_count, dim3((unsigned)blocks), dim3(kPriorThreads), 0, s, a);
}

cudaError_t launch_prior_total(const PriorLogArgs& a, int sms, cudaStream_t s) {
  long long blocks = ((long long)a.V + 4 * kPriorThreads - 1) / (4 * kPriorThreads);
  blocks = std::max<long long>(1, std::min<long long>(blocks, std::min(sms, kPriorMaxPartials)));
  return launch_pdl(k_prior_total, dim3((unsigned)blocks), dim3(kPriorThreads), 0, s, a);
}

cudaError_t launch_prior_log(const PriorLogArgs& a, int sms, cudaStream_t s) {
  long long blocks = ((long long)a.V + kPriorThreads - 1) / kPriorThreads;
  blocks = std::max<long long>(1, std::min<long long>(blocks, (long long)sms * 4));
  return launch_pdl(k_prior_log, dim3((unsigned)blocks), dim3(kPriorThreads), 0, s, a);
}

}  // namespace dels
