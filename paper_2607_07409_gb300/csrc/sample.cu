// Temperature-1 kernels outside the tensor-core engine (Algorithm 1 with
// Decode = a draw from the softmax; verification by lossless speculative
// sampling):
//
// * k_sample_rows — per-(row, column chunk) records of the Gumbel-max keys
//   k = l + g of a logit row (position 0 of the drafting loop draws x_0 from
//   softmax(l_L^(0)); the verification draws the bonus token from p_n).
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

}  // namespace

cudaError_t launch_sample_rows(const SampleRowsArgs& a, bool f32, cudaStream_t s) {
  const long long grid = (long long)a.rows * a.nchunks;
  if (grid == 0) return cudaSuccess;
  return f32 ? launch_pdl(k_sample_rows<float>, dim3((unsigned)grid), dim3(kSampleThreads), 0, s, a)
             : launch_pdl(k_sample_rows<uint16_t>, dim3((unsigned)grid), dim3(kSampleThreads), 0, s, a);
}

}  // namespace dels
