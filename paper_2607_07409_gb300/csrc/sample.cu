// Temperature-1 kernels outside the tensor-core engine (Algorithm 1 with
// Decode = a draw from the softmax; verification by lossless speculative
// sampling):
//
// * k_sample_rows — per-(row, column chunk) records of the Gumbel-max keys
//   k = l + g of a logit row (position 0 of the drafting loop draws x_0 from
//   softmax(l_L^(0))).
// * k_verify_accept, k_residual_rows, k_residual_merge — speculative sampling
//   (Leviathan et al. 2023; Chen et al. 2023): x_j is accepted when
//   u_j < p_j(x_j) / q_j(x_j); at the first rejection a the bonus token is
//   drawn from max(0, p_a - q_a) (normalised), and after n acceptances from
//   p_n. q_a is rebuilt from the drafting's kept state: the fused row
//   l_L + alpha_a W_vocab r_a - beta_a l_P and its LSE.
#include <algorithm>

#include "dels_device.cuh"

namespace dels {

namespace {

constexpr int kSampleThreads = 256;

template <typename T>
__device__ __forceinline__ void load8(const T* row, long long c0, long long c1, bool vec, float (&x)[8]);

template <>
__device__ __forceinline__ void load8<uint16_t>(const uint16_t* row, long long c0, long long c1, bool vec,
                                                float (&x)[8]) {
  if (vec && c0 + 8 <= c1) {
    const uint4 w = __ldcs(reinterpret_cast<const uint4*>(row + c0));
    x[0] = bf16lo(w.x); x[1] = bf16hi(w.x); x[2] = bf16lo(w.y); x[3] = bf16hi(w.y);
    x[4] = bf16lo(w.z); x[5] = bf16hi(w.z); x[6] = bf16lo(w.w); x[7] = bf16hi(w.w);
  } else {
#pragma unroll
    for (int i = 0; i < 8; ++i) x[i] = c0 + i < c1 ? __uint_as_float((uint32_t)row[c0 + i] << 16) : -INFINITY;
  }
}

template <>
__device__ __forceinline__ void load8<float>(const float* row, long long c0, long long c1, bool vec, float (&x)[8]) {
  if (vec && c0 + 8 <= c1) {
    const float4 p = __ldcs(reinterpret_cast<const float4*>(row + c0));
    const float4 q = __ldcs(reinterpret_cast<const float4*>(row + c0 + 4));
    x[0] = p.x; x[1] = p.y; x[2] = p.z; x[3] = p.w;
    x[4] = q.x; x[5] = q.y; x[6] = q.z; x[7] = q.w;
  } else {
#pragma unroll
    for (int i = 0; i < 8; ++i) x[i] = c0 + i < c1 ? row[c0 + i] : -INFINITY;
  }
}

// Block-wide merge of the threads' records; thread 0 gets the result.
__device__ __forceinline__ RowAcc block_merge(RowAcc x, RowAcc* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  x = rowacc_warp_reduce(x);
  if (lane == 0) red[warp] = x;
  __syncthreads();
  if (warp == 0) {
    x = lane < (int)(blockDim.x >> 5) ? red[lane] : rowacc_init();
    x = rowacc_warp_reduce(x);
  }
  return x;
}

// Records of the keys k_v = l_v + g_v of rows [0, rows): row r is
// src + r * ld; its request index (for the variates) is r / rows_per_request
// and its position j0 + r % rows_per_request. CTA = (row, chunk of
// chunk_cols columns, a multiple of 8). Each thread visits its 8-column
// groups in increasing order (lowest index on exact key ties).
template <typename T>
__global__ void __launch_bounds__(kSampleThreads) k_sample_rows(SampleRowsArgs a) {
  __shared__ RowAcc red[kSampleThreads / 32];
  pdl_wait();
  const int chunk = blockIdx.x % a.nchunks;
  const long long row = blockIdx.x / a.nchunks;
  const int b = (int)(row / a.rows_per_request);
  const int j = a.j0 + (int)(row % a.rows_per_request);
  const T* src = static_cast<const T*>(a.src) + row * a.ld;
  const long long c0 = (long long)chunk * a.chunk_cols;
  const long long c1 = min((long long)a.V, c0 + a.chunk_cols);
  float best = -INFINITY, second = -INFINITY, m = -INFINITY, s = 0.f;
  int idx = 0x7FFFFFFF;
  for (long long c = c0 + 8 * (long long)threadIdx.x; c < c1; c += 8 * kSampleThreads) {
    float x[8], g[8];
    load8<T>(src, c, c1, a.vec != 0, x);
    gumbel8(a.seed, a.step, b, j, a.stream, c >> 3, g);
#pragma unroll
    for (int i = 0; i < 8; ++i) top2_push(x[i] + g[i], (int)(c + i), best, second, idx);
    lse_chunk_ex2<8>(x, best, m, s);
  }
  RowAcc r;
  r.m = best;
  r.s = s;
  r.second = second;
  r.idx = idx;
  // lse_chunk_ex2 keeps s relative to the running key max: r.m == best
  r = block_merge(r, red);
  if (threadIdx.x == 0)
    reinterpret_cast<float4*>(a.partials)[row * a.partial_ld + chunk] =
        make_float4(r.m, r.s, r.second, __int_as_float(r.idx));
}

template <typename T>
__device__ __forceinline__ float ld_logit(const void* p, long long i) {
  if constexpr (sizeof(T) == 4) return __ldg(static_cast<const float*>(p) + i);
  else return __uint_as_float((uint32_t)__ldg(static_cast<const uint16_t*>(p) + i) << 16);
}

__device__ __forceinline__ float ld_logit_any(const void* p, int f32, long long i) {
  return f32 ? ld_logit<float>(p, i) : ld_logit<uint16_t>(p, i);
}

// One CTA per request: the LSE of each target row from its records, then the
// acceptance tests in order, then the gather of the rejected position's
// vocabulary-projection input.
__global__ void __launch_bounds__(256) k_verify_accept(VerifySampledArgs a) {
  __shared__ float lse_s[kMaxSampledBlock + 1];
  __shared__ int acc_s;
  pdl_wait();
  const int b = blockIdx.x;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  for (int j = warp; j <= a.n; j += nw) {
    RowAcc x = rowacc_init();
    const long long row = (long long)b * (a.n + 1) + j;
    for (int k = lane; k < a.t_nchunks; k += 32) x = rowacc_merge(x, ld_rowacc_cg(a.t_records, row * a.t_ld + k));
    x = rowacc_warp_reduce(x);
    if (lane == 0) {
      const bool ok = rowacc_valid(x);
      if (!ok) raise_status(a.status, DELS_STATUS_NONFINITE);
      lse_s[j] = ok ? x.m + logf(x.s) : NAN;
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int acc = a.n;
    for (int j = 0; j < a.n; ++j) {
      const int x = a.draft[(long long)b * a.n + j];
      if (x < 0 || x >= a.V) {
        raise_status(a.status, DELS_STATUS_BAD_TOKEN);
        acc = j;
        break;
      }
      const float t = ld_logit_any(a.target, a.target_f32, ((long long)b * (a.n + 1) + j) * a.V + x);
      const float ratio = expf((t - lse_s[j]) - a.draft_lp[(long long)b * a.n + j]);
      const float u = uniform_at(a.seed, a.step, b, j, kStreamAccept, 0);
      if (!(u < ratio)) {
        acc = j;
        break;
      }
    }
    acc_s = acc;
    a.acc[b] = acc;
    a.out_accept[b] = acc;
    a.lse_t[b] = lse_s[acc];
  }
  __syncthreads();
  const int acc = acc_s;
  const int vecs = a.R * a.r_bytes / 16;
  uint4* dst = reinterpret_cast<uint4*>(static_cast<uint8_t*>(a.rg) + (long long)b * a.R * a.r_bytes);
  if (acc >= 1 && acc < a.n && a.state_r) {
    const uint4* src = reinterpret_cast<const uint4*>(static_cast<const uint8_t*>(a.state_r) +
                                                      ((long long)b * a.n + acc) * a.R * a.r_bytes);
    for (int i = threadIdx.x; i < vecs; i += blockDim.x) dst[i] = __ldcg(src + i);
  } else {
    for (int i = threadIdx.x; i < vecs; i += blockDim.x) dst[i] = make_uint4(0, 0, 0, 0);
  }
}

// Records of the bonus draw of request b over one chunk of the vocabulary:
// residual keys log(max(0, p_a - q_a)) + g (a < n) and target keys t + g
// (used after n acceptances, or when every residual weight rounded to zero).
__global__ void __launch_bounds__(kSampleThreads) k_residual_rows(VerifySampledArgs a) {
  __shared__ RowAcc red[kSampleThreads / 32];
  pdl_wait();
  const int b = blockIdx.x / a.r_nchunks, chunk = blockIdx.x % a.r_nchunks;
  const int acc = __ldcg(a.acc + b);
  const float lse_t = __ldcg(a.lse_t + b);
  const long long trow = ((long long)b * (a.n + 1) + acc) * a.V;
  const bool resid = acc < a.n;
  const long long lrow = ((long long)b * a.n + (resid ? acc : 0)) * a.V;
  const float lse_q = resid ? a.state_lse[(long long)b * a.n + acc] : 0.f;
  const bool head = resid && acc >= 1;
  const float al = head ? a.alpha[acc] : 0.f, nbe = head ? -a.beta[acc] : 0.f;
  const float* ls = a.ls + (long long)b * a.V;
  const long long c0 = (long long)chunk * a.r_chunk_cols;
  const long long c1 = min((long long)a.V, c0 + a.r_chunk_cols);
  float rb = -INFINITY, rs = -INFINITY, pb = -INFINITY, ps = -INFINITY;
  int ri = 0x7FFFFFFF, pi = 0x7FFFFFFF;
  for (long long c = c0 + 8 * (long long)threadIdx.x; c < c1; c += 8 * kSampleThreads) {
    float g[8];
    gumbel8(a.seed, a.step, b, acc, kStreamResidual, c >> 3, g);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const long long v = c + i;
      if (v >= c1) break;
      const float t = ld_logit_any(a.target, a.target_f32, trow + v);
      top2_push(t + g[i], (int)v, pb, ps, pi);
      if (resid) {
        float l = ld_logit_any(a.longp, a.long_f32, lrow + v);
        if (head) l = fmaf(nbe, a.prior ? __ldg(a.prior + v) : 0.f, fmaf(al, __ldcg(ls + v), l));
        const float w = __expf(t - lse_t) - __expf(l - lse_q);
        top2_push(w > 0.f ? __logf(w) + g[i] : -INFINITY, (int)v, rb, rs, ri);
      }
    }
  }
  RowAcc r;
  r.m = rb; r.s = 1.f; r.second = rs; r.idx = ri;
  RowAcc p;
  p.m = pb; p.s = 1.f; p.second = ps; p.idx = pi;
  r = block_merge(r, red);
  __syncthreads();
  p = block_merge(p, red);
  if (threadIdx.x == 0) {
    float4* out = reinterpret_cast<float4*>(a.r_records) + ((long long)b * a.r_nchunks + chunk) * 2;
    out[0] = make_float4(r.m, r.s, r.second, __int_as_float(r.idx));
    out[1] = make_float4(p.m, p.s, p.second, __int_as_float(p.idx));
  }
}

// One CTA per request: the bonus token from the merged records.
__global__ void __launch_bounds__(256) k_residual_merge(VerifySampledArgs a) {
  __shared__ RowAcc red[8];
  pdl_wait();
  const int b = blockIdx.x;
  RowAcc r = rowacc_init(), p = rowacc_init();
  for (int k = threadIdx.x; k < a.r_nchunks; k += blockDim.x) {
    r = rowacc_merge(r, ld_rowacc_cg(a.r_records, ((long long)b * a.r_nchunks + k) * 2));
    p = rowacc_merge(p, ld_rowacc_cg(a.r_records, ((long long)b * a.r_nchunks + k) * 2 + 1));
  }
  r = block_merge(r, red);
  __syncthreads();
  p = block_merge(p, red);
  if (threadIdx.x == 0) {
    const int acc = __ldcg(a.acc + b);
    const bool use_r = acc < a.n && r.m > -INFINITY;
    const RowAcc& x = use_r ? r : p;
    const bool ok = x.m > -INFINITY && x.m < INFINITY;
    if (!ok) raise_status(a.status, DELS_STATUS_NONFINITE);
    a.out_bonus[b] = ok ? x.idx : -1;
    if (a.out_bonus_gap) a.out_bonus_gap[b] = ok ? x.m - x.second : NAN;
  }
}

__global__ void __launch_bounds__(256) k_selftest_gumbel(const uint32_t* __restrict__ bits, float* __restrict__ g,
                                                        long long n) {
  const long long stride = (long long)gridDim.x * blockDim.x;
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride)
    g[i] = gumbel_from_bits(bits[i]);
}

}  // namespace

cudaError_t launch_selftest_gumbel(const uint32_t* bits, float* g, long long n, int sms, cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  const long long blocks = std::min<long long>((n + 255) / 256, (long long)sms * 8);
  k_selftest_gumbel<<<(unsigned)blocks, 256, 0, s>>>(bits, g, n);
  return cudaGetLastError();
}

cudaError_t launch_verify_accept(const VerifySampledArgs& a, cudaStream_t s) {
  return launch_pdl(k_verify_accept, dim3((unsigned)a.B), dim3(256), 0, s, a);
}

cudaError_t launch_residual_rows(const VerifySampledArgs& a, cudaStream_t s) {
  return launch_pdl(k_residual_rows, dim3((unsigned)(a.B * a.r_nchunks)), dim3(kSampleThreads), 0, s, a);
}

cudaError_t launch_residual_merge(const VerifySampledArgs& a, cudaStream_t s) {
  return launch_pdl(k_residual_merge, dim3((unsigned)a.B), dim3(256), 0, s, a);
}

cudaError_t launch_sample_rows(const SampleRowsArgs& a, bool f32, cudaStream_t s) {
  const long long grid = (long long)a.rows * a.nchunks;
  if (grid == 0) return cudaSuccess;
  return f32 ? launch_pdl(k_sample_rows<float>, dim3((unsigned)grid), dim3(kSampleThreads), 0, s, a)
             : launch_pdl(k_sample_rows<uint16_t>, dim3((unsigned)grid), dim3(kSampleThreads), 0, s, a);
}

}  // namespace dels
