// Row reductions over the vocabulary: the fused combine + argmax (Section 4.3
// fusion, temperature-0 Decode of Algorithm 1), greedy verification against
// target logits (Algorithm 1, verification step), and the per-position merge
// of the drafting loop (which also gathers the next local-head input).
//
// These are pure HBM streams: every kernel reads each logit once with 128-bit
// loads (streaming cache hint) and keeps its per-row state in registers; a
// row split over several CTAs is finished by the last CTA to arrive (atomic
// ticket, reset by that CTA), so no [rows, V] intermediate is ever written.
#include <algorithm>
#include <climits>

#include <cuda_bf16.h>

#include "dels_device.cuh"

namespace dels {

namespace {

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
__device__ __forceinline__ float load1(const uint16_t* p) { return __uint_as_float((uint32_t)__ldcs(p) << 16); }

// 8 values from raw 16-byte words: one word of 8 bf16, or two words of 4 f32.
template <typename T, int W>
__device__ __forceinline__ void unpack8(const uint4 (&w)[W], float (&x)[8]);
template <>
__device__ __forceinline__ void unpack8<uint16_t, 1>(const uint4 (&w)[1], float (&x)[8]) {
  x[0] = bf16lo(w[0].x); x[1] = bf16hi(w[0].x); x[2] = bf16lo(w[0].y); x[3] = bf16hi(w[0].y);
  x[4] = bf16lo(w[0].z); x[5] = bf16hi(w[0].z); x[6] = bf16lo(w[0].w); x[7] = bf16hi(w[0].w);
}
template <>
__device__ __forceinline__ void unpack8<float, 2>(const uint4 (&w)[2], float (&x)[8]) {
  x[0] = __uint_as_float(w[0].x); x[1] = __uint_as_float(w[0].y); x[2] = __uint_as_float(w[0].z);
  x[3] = __uint_as_float(w[0].w); x[4] = __uint_as_float(w[1].x); x[5] = __uint_as_float(w[1].y);
  x[6] = __uint_as_float(w[1].z); x[7] = __uint_as_float(w[1].w);
}

// Maximum of the 8 bf16 values of a 16-byte vector, NaN ignored
// (flagged in `nan`): packed bf16 maxima, then the two halves.
__device__ __forceinline__ float vec_max_bf16(const uint4& w, bool& nan) {
  const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162*>(&w.x);
  const __nv_bfloat162 b = *reinterpret_cast<const __nv_bfloat162*>(&w.y);
  const __nv_bfloat162 c = *reinterpret_cast<const __nv_bfloat162*>(&w.z);
  const __nv_bfloat162 d = *reinterpret_cast<const __nv_bfloat162*>(&w.w);
  const __nv_bfloat162 m = __hmax2(__hmax2(a, b), __hmax2(c, d));
  const __nv_bfloat162 mn = __hmax2_nan(__hmax2_nan(a, b), __hmax2_nan(c, d));
  const float lo = __low2float(m), hi = __high2float(m);
  const float nlo = __low2float(mn), nhi = __high2float(mn);
  nan = (nlo != nlo) | (nhi != nhi);
  return fmaxf(lo, hi);
}
template <typename T>
__device__ __forceinline__ float vec_max(const uint4& w, bool& nan);
template <>
__device__ __forceinline__ float vec_max<uint16_t>(const uint4& w, bool& nan) { return vec_max_bf16(w, nan); }
__device__ __forceinline__ void load_vec(const uint16_t* p, float (&x)[8]) { load8(p, x); }

__device__ __forceinline__ float load1(const float* p) { return __ldcs(p); }

__device__ __forceinline__ void st_rowacc(void* base, long long i, const RowAcc& r) {
  reinterpret_cast<float4*>(base)[i] = make_float4(r.m, r.s, r.second, __int_as_float(r.idx));
}


// Per-thread running state of one row.
struct RowState {
  float best, second, m, s;
  int idx;
  __device__ __forceinline__ void init() {
    best = -INFINITY; second = -INFINITY; m = -INFINITY; s = 0.f; idx = INT_MAX;
  }
  // An element at or below the runner-up changes neither the top-1 nor the
  // top-2, so the element-wise top-2 update runs only for groups whose
  // maximum exceeds the runner-up (rare once the row's head is seen).
  template <int K>
  __device__ __forceinline__ void push(const float (&f)[K], int c) {
    float vm = f[0];
#pragma unroll
    for (int i = 1; i < K; ++i) vm = fmaxf(vm, f[i]);
    if (vm > second) {
#pragma unroll
      for (int i = 0; i < K; ++i) top2_push(f[i], c + i, best, second, idx);
    }
    lse_chunk_ex2<K>(f, best, m, s);
  }
  __device__ __forceinline__ RowAcc acc() const {
    RowAcc r;
    r.m = best; r.s = s; r.second = second; r.idx = idx;
    return r;
  }
};

// Merge each row's RowAcc across the CTA; the results are valid in warp 0.
template <int R>
__device__ __forceinline__ void block_reduce_rows(const RowAcc (&acc)[R], RowAcc (&out)[R]) {
  __shared__ RowAcc red[kRowsThreads / 32][R];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int r = 0; r < R; ++r) {
    RowAcc x = rowacc_warp_reduce(acc[r]);
    if (lane == 0) red[warp][r] = x;
  }
  __syncthreads();
  if (warp == 0) {
#pragma unroll
    for (int r = 0; r < R; ++r) {
      RowAcc x = lane < kRowsThreads / 32 ? red[lane][r] : rowacc_init();
      out[r] = rowacc_warp_reduce(x);
    }
  }
}

// ----------------------------------------------------------------------------
// fused combine: l = l_L + alpha l_S - beta l_P, then top-1/top-2/LSE per row
// ----------------------------------------------------------------------------
template <typename T, int R, bool VEC, bool SH, bool PR, bool FINAL>
__global__ void __launch_bounds__(kRowsThreads, sizeof(T) == 2 ? 4 : 2) k_combine_rows(RowsArgs a) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const int chunk = blockIdx.x % a.nchunks;
  const int group = blockIdx.x / a.nchunks;
  const int r0 = group * R;
  const int nr = min(R, a.rows - r0);
  const int c0 = chunk * a.chunk_cols;
  const int c1 = min(a.V, c0 + a.chunk_cols);
  const T* L = static_cast<const T*>(a.longp) + (long long)r0 * a.ld_long;
  const T* S = SH ? static_cast<const T*>(a.shortp) + (long long)r0 * a.ld_short : nullptr;
  const float alpha = a.alpha, nbeta = -a.beta;

  RowState st[R];
#pragma unroll
  for (int r = 0; r < R; ++r) st[r].init();

  if constexpr (VEC) {
    // Raw 16-byte words stay in registers until used: U groups of 8 values
    // per row in flight (one row per CTA). U = 4 for both types: deeper
    // unrolling of bf16 rows (8 loads) costs registers, and with two CTAs
    // per SM instead of four the issue-heavy bf16 update stalls (measured
    // 172 us against 126 us for 1024 rows of 151936).
    constexpr int WPV = sizeof(T) == 2 ? 1 : 2;            // 16-byte words per 8 values
    constexpr int U = (R == 1) ? 4 : (R == 2 ? 2 : 1);
    const int step = kRowsThreads * 8;
    for (int cb = c0 + threadIdx.x * 8; cb < c1; cb += step * U) {
      uint4 lw[U][R][WPV];
      uint4 sw[U][R][WPV];
      // f32: the prior goes out with the logits; bf16: it is read where it
      // is used (fewer registers: four CTAs per SM)
      constexpr bool kPriorEarly = sizeof(T) == 4;
      float4 pw[kPriorEarly ? U : 1][2];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int c = cb + u * step;
        if (c < c1) {
          if constexpr (PR && kPriorEarly) {
            pw[u][0] = __ldg(reinterpret_cast<const float4*>(a.prior + c));
            pw[u][1] = __ldg(reinterpret_cast<const float4*>(a.prior + c) + 1);
          }
#pragma unroll
          for (int r = 0; r < R; ++r) {
            if (r < nr) {
#pragma unroll
              for (int k = 0; k < WPV; ++k) {
                lw[u][r][k] = __ldcs(reinterpret_cast<const uint4*>(L + (long long)r * a.ld_long + c) + k);
                if constexpr (SH) sw[u][r][k] = __ldcs(reinterpret_cast<const uint4*>(S + (long long)r * a.ld_short + c) + k);
              }
            }
          }
        }
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int c = cb + u * step;
        if (c < c1) {
          float pv[8];
          if constexpr (PR) {
            float4 p0, p1;
            if constexpr (kPriorEarly) {
              p0 = pw[u][0];
              p1 = pw[u][1];
            } else {
              p0 = __ldg(reinterpret_cast<const float4*>(a.prior + c));
              p1 = __ldg(reinterpret_cast<const float4*>(a.prior + c) + 1);
            }
            pv[0] = p0.x; pv[1] = p0.y; pv[2] = p0.z; pv[3] = p0.w;
            pv[4] = p1.x; pv[5] = p1.y; pv[6] = p1.z; pv[7] = p1.w;
          }
#pragma unroll
          for (int r = 0; r < R; ++r) {
            if (r < nr) {
              float lv[8], sv[8];
              unpack8<T, WPV>(lw[u][r], lv);
              if constexpr (SH) unpack8<T, WPV>(sw[u][r], sv);
              float f[8];
#pragma unroll
              for (int i = 0; i < 8; ++i) {
                float x = lv[i];
                if constexpr (SH) x = fmaf(alpha, sv[i], x);
                if constexpr (PR) x = fmaf(nbeta, pv[i], x);
                f[i] = x;
              }
              st[r].template push<8>(f, c);
            }
          }
        }
      }
    }
  } else {
    for (int c = c0 + threadIdx.x; c < c1; c += kRowsThreads) {
      const float p = PR ? __ldg(a.prior + c) : 0.f;
#pragma unroll
      for (int r = 0; r < R; ++r) {
        if (r < nr) {
          float x = load1(L + (long long)r * a.ld_long + c);
          if constexpr (SH) x = fmaf(alpha, load1(S + (long long)r * a.ld_short + c), x);
          if constexpr (PR) x = fmaf(nbeta, p, x);
          float f[1] = {x};
          st[r].template push<1>(f, c);
        }
      }
    }
  }

  RowAcc acc[R], res[R];
#pragma unroll
  for (int r = 0; r < R; ++r) acc[r] = st[r].acc();
  block_reduce_rows<R>(acc, res);

  __shared__ int s_last;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (a.nchunks == 1 && FINAL) {
    if (threadIdx.x == 0) {
      for (int r = 0; r < nr; ++r) write_decode(res[r], r0 + r, a.out_token, a.out_lp, a.out_gap, a.status);
    }
    return;
  }
  if (threadIdx.x == 0) {
    for (int r = 0; r < nr; ++r) st_rowacc(a.partials, (long long)(r0 + r) * a.partial_ld + chunk, res[r]);
  }
  if (!FINAL) return;
  if (threadIdx.x == 0) {
    __threadfence();
    const int ticket = atomicAdd(&a.counters[group], 1);
    s_last = (ticket == a.nchunks - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (warp < nr) {
    const long long row = r0 + warp;
    RowAcc x = rowacc_init();
    for (int k = lane; k < a.nchunks; k += 32) x = rowacc_merge(x, ld_rowacc_cg(a.partials, row * a.partial_ld + k));
    x = rowacc_warp_reduce(x);
    if (lane == 0) write_decode(x, row, a.out_token, a.out_lp, a.out_gap, a.status);
  }
  if (threadIdx.x == 0) a.counters[group] = 0;
}

// ----------------------------------------------------------------------------
// verification: t_j = argmax target[b, j, :]; accept = leading matches; bonus
// ----------------------------------------------------------------------------
struct ArgAcc {
  float best;
  int idx;
  int nan;
};

__device__ __forceinline__ ArgAcc argacc_merge(const ArgAcc& a, const ArgAcc& b) {
  const bool b_wins = (b.best > a.best) || (b.best == a.best && b.idx < a.idx);
  ArgAcc r = b_wins ? b : a;
  r.nan = a.nan | b.nan;
  return r;
}
__device__ __forceinline__ ArgAcc argacc_shfl_down(const ArgAcc& a, int d) {
  ArgAcc r;
  r.best = __shfl_down_sync(0xFFFFFFFFu, a.best, d);
  r.idx = __shfl_down_sync(0xFFFFFFFFu, a.idx, d);
  r.nan = __shfl_down_sync(0xFFFFFFFFu, a.nan, d);
  return r;
}
__device__ __forceinline__ ArgAcc argacc_warp_reduce(ArgAcc a) {
#pragma unroll
  for (int d = 16; d > 0; d >>= 1) a = argacc_merge(a, argacc_shfl_down(a, d));
  return a;
}

template <typename T, bool VEC>
__global__ void __launch_bounds__(kRowsThreads) k_verify_rows(RowsArgs a) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const int chunk = blockIdx.x % a.nchunks;
  const int row = blockIdx.x / a.nchunks;        // b * (n + 1) + j
  const int c0 = chunk * a.chunk_cols;
  const int c1 = min(a.V, c0 + a.chunk_cols);
  const T* L = static_cast<const T*>(a.longp) + (long long)row * a.ld_long;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;

  float best = -INFINITY;
  int idx = INT_MAX;
  bool nan_seen = false;
  if constexpr (VEC && sizeof(T) == 2) {
    // bf16, vector by vector: the maximum of each 16-byte vector (packed max
    // instructions), a strict '>' against the running best (the first vector
    // holding the thread's maximum wins), and at the end the first element of
    // that vector equal to the maximum: the same lowest-index argmax as an
    // element-by-element scan, at a fraction of the instructions.
    constexpr int U = 4;   // 16-byte loads in flight per thread (8: 2.7% slower, same box)
    constexpr int E = 16 / sizeof(T);
    const int step = kRowsThreads * E;
    int bvec = -1;
    for (int cb = c0 + threadIdx.x * E; cb < c1; cb += step * U) {
      uint4 w[U];
#pragma unroll
      for (int u = 0; u < U; ++u)
        if (cb + u * step < c1) w[u] = __ldcs(reinterpret_cast<const uint4*>(L + cb + u * step));
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int c = cb + u * step;
        if (c < c1) {
          bool nan_v;
          const float mv = vec_max<T>(w[u], nan_v);
          nan_seen |= nan_v;
          if (mv > best) {
            best = mv;
            bvec = c;
          }
        }
      }
    }
    if (bvec >= 0) {
      float x[E];
      load_vec(L + bvec, x);
#pragma unroll
      for (int i = E - 1; i >= 0; --i)
        if (x[i] == best) idx = bvec + i;
    }
  } else if constexpr (VEC) {
    // f32: element by element (measured faster than the vector form here)
    constexpr int U = 4;
    const int step = kRowsThreads * 8;
    for (int cb = c0 + threadIdx.x * 8; cb < c1; cb += step * U) {
      float lv[U][8];
#pragma unroll
      for (int u = 0; u < U; ++u)
        if (cb + u * step < c1) load8(L + cb + u * step, lv[u]);
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int c = cb + u * step;
        if (c < c1) {
#pragma unroll
          for (int i = 0; i < 8; ++i) argmax_push(lv[u][i], c + i, best, idx, nan_seen);
        }
      }
    }
  } else {
    for (int c = c0 + threadIdx.x; c < c1; c += kRowsThreads) argmax_push(load1(L + c), c, best, idx, nan_seen);
  }

  __shared__ ArgAcc red[kRowsThreads / 32];
  __shared__ int s_last;
  __shared__ int s_targ[kMaxVerifyBlock + 1];
  ArgAcc x{best, idx, nan_seen ? 1 : 0};
  x = argacc_warp_reduce(x);
  if (lane == 0) red[warp] = x;
  __syncthreads();
  // One ticket per request over its (n + 1) rows x nchunks records: the last
  // CTA to publish merges every row of the request and takes the accept
  // length and the bonus token.
  const int n = a.n;
  const int b = row / (n + 1);
  if (warp == 0) {
    x = lane < kRowsThreads / 32 ? red[lane] : ArgAcc{-INFINITY, INT_MAX, 0};
    x = argacc_warp_reduce(x);
    if (lane == 0) {
      reinterpret_cast<float4*>(a.partials)[(long long)row * a.partial_ld + chunk] =
          make_float4(x.best, __int_as_float(x.idx), __int_as_float(x.nan), 0.f);
      __threadfence();
      s_last = (atomicAdd(&a.counters_b[b], 1) == (n + 1) * a.nchunks - 1);
    }
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const long long row0 = (long long)b * (n + 1);
  for (int j = warp; j <= n; j += kRowsThreads / 32) {
    ArgAcc y{-INFINITY, INT_MAX, 0};
    for (int k = lane; k < a.nchunks; k += 32) {
      const float4 v = __ldcg(reinterpret_cast<const float4*>(a.partials) + (row0 + j) * a.partial_ld + k);
      y = argacc_merge(y, ArgAcc{v.x, __float_as_int(v.y), __float_as_int(v.z)});
    }
    y = argacc_warp_reduce(y);
    if (lane == 0) {
      if (y.nan) raise_status(a.status, DELS_STATUS_NONFINITE);
      const int t = (y.idx == INT_MAX) ? 0 : y.idx;   // an all -inf row: first index
      s_targ[j] = t;
      if (a.out_token) a.out_token[row0 + j] = t;
    }
  }
  __syncthreads();
  if (threadIdx.x != 0) return;
  int acc = 0;
  bool bad = false;
  for (; acc < n; ++acc) {
    const int xd = a.draft[(long long)b * n + acc];
    bad |= (xd < 0 || xd >= a.V);
    if (xd != s_targ[acc]) break;
  }
  for (int k = acc; k < n && !bad; ++k) {
    const int xd = a.draft[(long long)b * n + k];
    bad |= (xd < 0 || xd >= a.V);
  }
  if (bad) raise_status(a.status, DELS_STATUS_BAD_TOKEN);
  a.out_accept[b] = acc;
  a.out_bonus[b] = s_targ[acc];
  a.counters_b[b] = 0;
}

// ----------------------------------------------------------------------------
// drafting: merge the per-CTA partials of position j, emit x_j, and gather the
// local head's next input rows
// ----------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_draft_merge(MergeArgs a) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x;
  if (a.zero_len > 0) {
    for (int i = threadIdx.x; i < a.zero_len; i += blockDim.x) {
      if (a.zero_f32) a.zero_f32[(long long)b * a.zero_len + i] = 0.f;
      if (a.zero_bf16) a.zero_bf16[(long long)b * a.zero_len + i] = 0;
    }
  }
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  __shared__ RowAcc red[8];
  __shared__ int s_tok;
  RowAcc x = rowacc_init();
  for (int k = threadIdx.x; k < a.count; k += blockDim.x)
    x = rowacc_merge(x, ld_rowacc_cg(a.partials, (long long)b * a.partial_ld + k));
  x = rowacc_warp_reduce(x);
  if (lane == 0) red[warp] = x;
  // temperature 1: keep this position's vocabulary-projection input before
  // the gather below may overwrite it (the Markov head gathers into it)
  keep_draft_input(a.smp, b, a.n, a.j);
  __syncthreads();
  if (warp == 0) {
    x = lane < (int)(blockDim.x >> 5) ? red[lane] : rowacc_init();
    x = rowacc_warp_reduce(x);
    if (lane == 0) s_tok = decode_record(x, a.smp, b, a.n, a.j, a.tokens, a.out_lp, a.out_gap, a.status);
  }
  __syncthreads();
  if (a.table == nullptr) return;
  const int es = a.table_f32 ? 4 : 2;
  const int vec_per_row = a.D * es / 16;                 // D * es is a multiple of 16
  for (int k = 0; k < a.window; ++k) {
    const int jj = a.j - k;
    int tok = -1;
    if (k == 0) tok = s_tok;
    else if (jj >= 0) tok = a.tokens[(long long)b * a.n + jj];
    uint4* dst = reinterpret_cast<uint4*>(static_cast<uint8_t*>(a.dest) +
                                          ((long long)b * a.window + k) * (long long)a.D * es);
    if (tok < 0) {
      for (int i = threadIdx.x; i < vec_per_row; i += blockDim.x) dst[i] = make_uint4(0, 0, 0, 0);
    } else {
      const uint4* src = reinterpret_cast<const uint4*>(static_cast<const uint8_t*>(a.table) +
                                                        (long long)tok * a.D * es);
      for (int i = threadIdx.x; i < vec_per_row; i += blockDim.x) dst[i] = __ldg(src + i);
    }
  }
}

template <typename T, int R, bool VEC, bool SH, bool PR>
cudaError_t launch_combine_t(const RowsArgs& a, bool finalize, cudaStream_t s) {
  const int groups = (a.rows + R - 1) / R;
  const long long grid = (long long)groups * a.nchunks;
  if (grid == 0) return cudaSuccess;
  if (finalize)
    return launch_pdl(k_combine_rows<T, R, VEC, SH, PR, true>, dim3((unsigned)grid), dim3(kRowsThreads), 0, s, a);
  return launch_pdl(k_combine_rows<T, R, VEC, SH, PR, false>, dim3((unsigned)grid), dim3(kRowsThreads), 0, s, a);
}

template <typename T, int R, bool VEC>
cudaError_t dispatch_sp(const RowsArgs& a, bool finalize, cudaStream_t s) {
  const bool sh = a.shortp != nullptr, pr = a.prior != nullptr;
  if (sh && pr) return launch_combine_t<T, R, VEC, true, true>(a, finalize, s);
  if (sh) return launch_combine_t<T, R, VEC, true, false>(a, finalize, s);
  if (pr) return launch_combine_t<T, R, VEC, false, true>(a, finalize, s);
  return launch_combine_t<T, R, VEC, false, false>(a, finalize, s);
}

template <typename T>
cudaError_t dispatch_rv(const RowsArgs& a, bool vec, bool finalize, cudaStream_t s) {
  if (a.rows_per_cta == 4) {
    return vec ? dispatch_sp<T, 4, true>(a, finalize, s) : dispatch_sp<T, 4, false>(a, finalize, s);
  }
  if (a.rows_per_cta == 2 && vec) return dispatch_sp<T, 2, true>(a, finalize, s);
  return vec ? dispatch_sp<T, 1, true>(a, finalize, s) : dispatch_sp<T, 1, false>(a, finalize, s);
}

}  // namespace

RowsPlan plan_rows(int rows, int V, int bytes_per_col, int num_sms, bool vec, int max_chunks, bool multi_row,
                   int slots_per_sm) {
  RowsPlan p{};
  const long long slots = (long long)slots_per_sm * num_sms;
  // Rows per CTA (the prior read once for all of them): four for very many
  // short rows; two for bf16 combines whose rows do not fit in one wave of
  // resident CTAs (measured: 1024 rows of 151936, 141 -> 133 us; 1024 rows of
  // 32000, 53 -> 39 us; no gain for f32 rows or for fewer rows).
  p.rows_per_cta = 1;
  if (multi_row && vec && rows >= 64LL * num_sms) p.rows_per_cta = 4;
  else if (multi_row && vec && bytes_per_col <= 4 && slots > 0 && rows > slots) p.rows_per_cta = 2;
  const long long groups0 = ((long long)rows + p.rows_per_cta - 1) / p.rows_per_cta;
  int nchunks = 1;
  if (slots > 0 && groups0 > 0 && groups0 <= slots) {
    // every row group fits in one wave of resident CTAs: split the rows into
    // as many chunks as that wave holds (a second, partial wave would cost a
    // whole CTA lifetime for a few CTAs), down to 2048 columns (one 8-value
    // group per thread), so that small calls take one round trip per CTA
    nchunks = (int)std::min<long long>(slots / groups0, std::max(1, V / 2048));
  } else {
    const long long target_items = 16LL * num_sms;
    if (groups0 > 0 && groups0 < target_items) nchunks = (int)((target_items + groups0 - 1) / groups0);
    const int min_cols = std::max(2048, 32768 / std::max(1, bytes_per_col));
    nchunks = std::min(nchunks, std::max(1, V / min_cols));
  }
  nchunks = std::max(1, std::min(nchunks, max_chunks));
  int chunk_cols = (V + nchunks - 1) / nchunks;
  chunk_cols = (chunk_cols + 7) / 8 * 8;
  nchunks = (V + chunk_cols - 1) / chunk_cols;
  p.nchunks = std::max(1, nchunks);
  p.chunk_cols = std::max(8, chunk_cols);
  p.grid = (int)std::min<long long>(groups0 * p.nchunks, INT_MAX);
  return p;
}

int rows_slots_per_sm(bool verify, dels_dtype dt) {
  // resident CTAs per SM of the main instantiation (all four combine
  // variants use the same registers to within a few), queried once
  static int cache[4] = {-1, -1, -1, -1};
  const int k = (verify ? 2 : 0) + (dt == DELS_F32 ? 1 : 0);
  if (cache[k] < 0) {
    int n = 0;
    cudaError_t e;
    if (verify)
      e = dt == DELS_F32 ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_verify_rows<float, true>, kRowsThreads, 0)
                         : cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_verify_rows<uint16_t, true>, kRowsThreads, 0);
    else
      e = dt == DELS_F32
              ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_combine_rows<float, 1, true, true, true, true>,
                                                              kRowsThreads, 0)
              : cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_combine_rows<uint16_t, 1, true, true, true, true>,
                                                              kRowsThreads, 0);
    cache[k] = (e == cudaSuccess && n > 0) ? n : 0;
  }
  return cache[k];
}

cudaError_t launch_combine_rows(const RowsArgs& a, dels_dtype dt, bool vec, bool finalize, cudaStream_t s) {
  if (dt == DELS_BF16) return dispatch_rv<uint16_t>(a, vec, finalize, s);
  return dispatch_rv<float>(a, vec, finalize, s);
}

cudaError_t launch_verify_rows(const RowsArgs& a, dels_dtype dt, bool vec, cudaStream_t s) {
  const long long grid = (long long)a.rows * a.nchunks;
  if (grid == 0) return cudaSuccess;
  const dim3 g((unsigned)grid), blk(kRowsThreads);
  if (dt == DELS_BF16)
    return vec ? launch_pdl(k_verify_rows<uint16_t, true>, g, blk, 0, s, a)
               : launch_pdl(k_verify_rows<uint16_t, false>, g, blk, 0, s, a);
  return vec ? launch_pdl(k_verify_rows<float, true>, g, blk, 0, s, a)
             : launch_pdl(k_verify_rows<float, false>, g, blk, 0, s, a);
}

cudaError_t launch_draft_merge(const MergeArgs& a, cudaStream_t s) {
  if (a.B == 0) return cudaSuccess;
  return launch_pdl(k_draft_merge, dim3(a.B), dim3(256), 0, s, a);
}

}  // namespace dels
