// Element-wise and small reduction kernels of the local heads (Appendix A
// GRU head; the window-MLP and transformer heads of the synthetic
// workloads), plus the float32 CUDA-core path used when the head's weights
// are float32. The large matrix products of bf16 heads run in tc_gemm.cu.
#include <climits>

#include <algorithm>

#include "dels_device.cuh"

namespace dels {

namespace {

__device__ __forceinline__ float sigmoidf_(float x) { return 1.f / (1.f + __expf(-x)); }

__device__ __forceinline__ float act_f(int act, float x) {
  if (act == ACT_SILU) return x / (1.f + __expf(-x));
  if (act == ACT_GELU) return 0.5f * x * (1.f + erff(x * 0.70710678118654752f));
  return x;
}

// GRU gates (PyTorch bias-free form; gate rows r, z, n):
//   gi = sum of the S0 input-product partials, gh = sum of the S1 recurrent ones
//   r = sigmoid(gi_r + gh_r), z = sigmoid(gi_z + gh_z)
//   c = tanh(gi_n + r * gh_n), h' = (1 - z) * c + z * h
__global__ void k_gru_gates(const float* __restrict__ part, int S0, int S1, int B, int H, float* __restrict__ h,
                            uint16_t* __restrict__ h_bf16) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const long long total = (long long)B * H;
  const long long split_stride = (long long)B * 3 * H;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const int b = (int)(e / H), i = (int)(e % H);
    const long long base = (long long)b * 3 * H + i;
    float gir = 0.f, giz = 0.f, gin = 0.f, ghr = 0.f, ghz = 0.f, ghn = 0.f;
    for (int s = 0; s < S0; ++s) {
      const float* p = part + s * split_stride + base;
      gir += p[0]; giz += p[H]; gin += p[2 * H];
    }
    for (int s = S0; s < S0 + S1; ++s) {
      const float* p = part + s * split_stride + base;
      ghr += p[0]; ghz += p[H]; ghn += p[2 * H];
    }
    const float r = sigmoidf_(gir + ghr);
    const float z = sigmoidf_(giz + ghz);
    const float c = tanhf(gin + r * ghn);
    const float hp = h[e];
    const float hn = (1.f - z) * c + z * hp;
    h[e] = hn;
    h_bf16[e] = f32_to_bf16_rne(hn);
  }
}

// The same GRU step with the input product read from a precomputed table:
// gi = W_ih E[x] = G[x] with G = E W_ih^T [V, 3H] (row x holds the r, z, n
// gate inputs of token x). The CTA first merges request b's per-CTA records
// of the previous position into x (every CTA of the row does this; the
// first also writes the decoded token, logprob and gap), so the merge costs
// no launch of its own. gh is the sum of S recurrent partials [S][B][3H];
// S = 0 means gh = 0 (the step from h = 0). A row that decoded to no token
// (non-finite logits, already flagged) takes gi = 0.
constexpr int kGatesThreads = 256;

__device__ __forceinline__ float ld_cg_f32(const float* p) {
  float v;
  asm volatile("ld.global.cg.f32 %0, [%1];" : "=f"(v) : "l"(p));
  return v;
}

__global__ void __launch_bounds__(kGatesThreads) k_gru_gates_table(GatesTableArgs a) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int H = a.H;
  // This thread's hidden unit (one per thread: the launch covers H with
  // gridDim.y CTAs of kGatesThreads).
  const int i = blockIdx.y * kGatesThreads + threadIdx.x;
  const bool live = i < H;
  // Loads that do not depend on the token are issued first (volatile, so
  // they stay ahead of the merge); their sums come after it.
  constexpr int kMaxS = 8;
  float q[kMaxS][3];
  float hp = 0.f;
  const int S = min(a.S, kMaxS);
  if (live) {
    const long long split_stride = (long long)a.B * 3 * H;
    const float* base = a.part + (long long)b * 3 * H + i;
#pragma unroll
    for (int sp = 0; sp < kMaxS; ++sp) {
      if (sp < S) {
        q[sp][0] = ld_cg_f32(base + sp * split_stride);
        q[sp][1] = ld_cg_f32(base + sp * split_stride + H);
        q[sp][2] = ld_cg_f32(base + sp * split_stride + 2 * H);
      }
    }
    if (S > 0) hp = ld_cg_f32(a.h + (long long)b * H + i);
  }
  // merge of request b's records: warp 0 alone, every record load in flight at once
  __shared__ int s_tok;
  if (warp == 0) {
    RowAcc x = rowacc_init();
    const float4* rec = reinterpret_cast<const float4*>(a.partials) + (long long)b * a.partial_ld;
    for (int k0 = 0; k0 < a.count; k0 += 8 * 32) {
      float4 v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int k = k0 + u * 32 + lane;
        v[u] = k < a.count ? __ldcg(rec + k) : make_float4(-INFINITY, 0.f, -INFINITY, __int_as_float(INT_MAX));
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        RowAcc y;
        y.m = v[u].x; y.s = v[u].y; y.second = v[u].z; y.idx = __float_as_int(v[u].w);
        x = rowacc_merge(x, y);
      }
    }
    x = rowacc_warp_reduce(x);
    if (lane == 0) {
      if (!a.smp.on) {
        s_tok = rowacc_valid(x) ? x.idx : -1;
        if (blockIdx.y == 0) write_decode(x, (long long)b * a.n + a.jprev, a.tokens, a.out_lp, a.out_gap, a.status);
      } else if (blockIdx.y == 0) {
        s_tok = decode_record(x, a.smp, b, a.n, a.jprev, a.tokens, a.out_lp, a.out_gap, a.status);
      } else {
        s_tok = rowacc_valid_sampled(x) ? x.idx : -1;
      }
    }
  }
  // temperature 1: keep r_{jprev} (not yet overwritten: the next products launch follows this one)
  if (blockIdx.y == 0) keep_draft_input(a.smp, b, a.n, a.jprev);
  __syncthreads();
  if (!live) return;
  const int tok = s_tok;
  float gir = 0.f, giz = 0.f, gin = 0.f;
  if (tok >= 0 && tok < a.V) {
    const float* g = a.G + (long long)tok * 3 * H + i;
    gir = __ldg(g);
    giz = __ldg(g + H);
    gin = __ldg(g + 2 * H);
  }
  float ghr = 0.f, ghz = 0.f, ghn = 0.f;
#pragma unroll
  for (int sp = 0; sp < kMaxS; ++sp) {
    if (sp < S) {
      ghr += q[sp][0];
      ghz += q[sp][1];
      ghn += q[sp][2];
    }
  }
  const float r = sigmoidf_(gir + ghr);
  const float z = sigmoidf_(giz + ghz);
  const float c = tanhf(gin + r * ghn);
  const float hn = (1.f - z) * c + z * hp;
  const long long e = (long long)b * H + i;
  a.h[e] = hn;
  a.h_bf16[e] = f32_to_bf16_rne(hn);
}

// sum_s sum_t part[s * split_stride + t * total + e] over S splits and
// in_terms terms (terms last to first within a split), eight loads in flight
// before they are added in that order.
__device__ __forceinline__ float splitk_sum(const float* __restrict__ part, int S, int in_terms, long long total,
                                           long long e) {
  const long long split_stride = total * in_terms;
  const int n = S * in_terms;
  float acc = 0.f;
  int s = 0, t = in_terms - 1;
  for (int k0 = 0; k0 < n; k0 += 8) {
    float v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      v[k] = k0 + k < n ? part[s * split_stride + t * total + e] : 0.f;
      if (--t < 0) {
        t = in_terms - 1;
        ++s;
      }
    }
#pragma unroll
    for (int k = 0; k < 8; ++k)
      if (k0 + k < n) acc += v[k];
  }
  return acc;
}

// out[b, o] = act(sum_s sum_t part[s, t*B + b, o] (+ residual[b, o])):
// partials [S][in_terms*B][O] (in_terms = 3 when the product's input rows were
// a three-term expansion), the residual dense [B, O]; the f32 output has its
// own row pitch, the bf16 output is written as out_terms terms (see
// store_bf16_terms).
__global__ void k_splitk_finish(const float* __restrict__ part, int S, int B, int O,
                                const float* __restrict__ residual, int act, float* __restrict__ out_f32, int ld_f32,
                                uint16_t* __restrict__ out_bf16, int ld_bf16, int in_terms, int out_terms) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const long long total = (long long)B * O;
  const long long split_stride = total * in_terms;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const int b = (int)(e / O), o = (int)(e % O);
    float acc = 0.f;
    if (in_terms == 1) {
      // eight partial loads in flight before they are added in split order
      for (int s0 = 0; s0 < S; s0 += 8) {
        float v[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) v[k] = s0 + k < S ? part[(s0 + k) * split_stride + e] : 0.f;
#pragma unroll
        for (int k = 0; k < 8; ++k)
          if (s0 + k < S) acc += v[k];
      }
    } else {
      acc = splitk_sum(part, S, in_terms, total, e);
    }
    if (residual) acc += residual[e];
    acc = act_f(act, acc);
    if (out_f32) out_f32[(long long)b * ld_f32 + o] = acc;
    if (out_bf16) store_bf16_terms(out_bf16, out_terms, B, b, ld_bf16, o, acc);
  }
}

// Up to three split-K reductions in one launch (blockIdx.y = job): the same
// sum as k_splitk_finish with in_terms-term partials of row pitch ldp (job k
// reads columns col0 .. col0 + O - 1), no residual, no activation, float32
// output with its own row pitch (the transformer head's q, k and v of the
// newest position, from the partials of their stacked product).
__global__ void k_splitk_finish3(SplitkJobs3 jobs, int B, int O, int ldp, int in_terms) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const SplitkJob& jb = jobs.j[blockIdx.y];
  const long long total = (long long)B * O;
  const long long term_stride = (long long)B * ldp;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const int b = (int)(e / O), o = (int)(e % O);
    jb.out[(long long)b * jb.ld + o] =
        splitk_sum(jb.part, jb.S, in_terms, term_stride, (long long)b * ldp + jb.col0 + o);
  }
}

// out = RMSNorm(x) = x / sqrt(mean(x^2) + 1e-6) as `terms` bf16 terms (rows
// of pitch ld, see store_bf16_terms); one CTA per row.
__global__ void k_rmsnorm_bf16(const float* __restrict__ x, int D, int ld, uint16_t* __restrict__ out, int terms,
                               int B) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const float* row = x + (long long)blockIdx.x * ld;
  float ss = 0.f;
  for (int i = threadIdx.x; i < D; i += blockDim.x) ss += row[i] * row[i];
  ss = block_sum(ss);
  const float inv = rsqrtf(ss / (float)D + 1e-6f);
  for (int i = threadIdx.x; i < D; i += blockDim.x) store_bf16_terms(out, terms, B, blockIdx.x, ld, i, row[i] * inv);
}

// Split-K reduction + residual followed by RMSNorm, for one row per
// thread-block cluster of kNormCluster CTAs: each CTA reduces a slice of the
// row (as k_splitk_finish: sum over splits, terms last to first, then the
// residual), writes the float32 sum, and adds its slice's sum of squares into
// every CTA of the cluster (distributed shared memory, between two cluster
// barriers: all CTAs running, all sums written); each CTA then normalises its
// slice and writes it as `terms` bf16 terms.
__global__ void k_finish_rmsnorm(const float* __restrict__ part, int S, int in_terms, int B, int D,
                                 const float* __restrict__ residual, float* __restrict__ out_f32,
                                 uint16_t* __restrict__ norm_bf16, int terms) {
  __shared__ float ssq[kNormCluster];
  __shared__ float red[32];
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const uint32_t rank = cluster_ctarank();
  const int b = blockIdx.x / kNormCluster;
  const int per = (D + kNormCluster - 1) / kNormCluster;
  const int o0 = (int)rank * per, o1 = min(D, o0 + per);
  const long long total = (long long)B * D;
  constexpr int kMaxPer = 4;     // row elements per thread (D <= kNormCluster * 4 * blockDim.x)
  float v[kMaxPer];
  float ss = 0.f;
#pragma unroll
  for (int k = 0; k < kMaxPer; ++k) {
    const int o = o0 + (int)threadIdx.x + k * (int)blockDim.x;
    v[k] = 0.f;
    if (o < o1) {
      const long long e = (long long)b * D + o;
      float acc = splitk_sum(part, S, in_terms, total, e);
      if (residual) acc += residual[e];
      out_f32[e] = acc;
      v[k] = acc;
      ss += acc * acc;
    }
  }
  // slice sum of squares (block), then into slot `rank` of every CTA of the cluster
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int d = 16; d > 0; d >>= 1) ss += __shfl_down_sync(0xFFFFFFFFu, ss, d);
  if (lane == 0) red[warp] = ss;
  __syncthreads();
  if (warp == 0) {
    const int nw = (blockDim.x + 31) >> 5;
    ss = lane < nw ? red[lane] : 0.f;
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) ss += __shfl_down_sync(0xFFFFFFFFu, ss, d);
    ss = __shfl_sync(0xFFFFFFFFu, ss, 0);
  }
  // every CTA of the cluster is running before its shared memory is written
  cluster_sync_all();
  if (warp == 0 && lane < kNormCluster) st_cluster_f32(cluster_map(smem_u32(&ssq[rank]), (uint32_t)lane), ss);
  cluster_sync_all();
  float tot = 0.f;
#pragma unroll
  for (int r = 0; r < kNormCluster; ++r) tot += ssq[r];
  const float inv = rsqrtf(tot / (float)D + 1e-6f);
#pragma unroll
  for (int k = 0; k < kMaxPer; ++k) {
    const int o = o0 + (int)threadIdx.x + k * (int)blockDim.x;
    if (o < o1) store_bf16_terms(norm_bf16, terms, B, b, D, o, v[k] * inv);
  }
}

// t = E[x] + P[pos] (float32), a = RMSNorm(t) as `terms` bf16 terms; one CTA
// per row.
__global__ void k_xfmr_embed(const uint16_t* __restrict__ e_rows, const uint16_t* __restrict__ pos_table, int pos,
                             int D, float* __restrict__ t_out, uint16_t* __restrict__ a_bf16, int terms, int B) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const long long off = (long long)blockIdx.x * D;
  const int nv = D / 8;   // 8-value vectors (D is a multiple of 16)
  const uint4* e4 = reinterpret_cast<const uint4*>(e_rows + off);
  const uint4* p4 = reinterpret_cast<const uint4*>(pos_table + (long long)pos * D);
  float4* t4 = reinterpret_cast<float4*>(t_out + off);
  float ss = 0.f;
  for (int v = threadIdx.x; v < nv; v += blockDim.x) {
    const uint4 e = e4[v], pp = __ldg(p4 + v);
    const float4 a = make_float4(bf16lo(e.x) + bf16lo(pp.x), bf16hi(e.x) + bf16hi(pp.x),
                                 bf16lo(e.y) + bf16lo(pp.y), bf16hi(e.y) + bf16hi(pp.y));
    const float4 c = make_float4(bf16lo(e.z) + bf16lo(pp.z), bf16hi(e.z) + bf16hi(pp.z),
                                 bf16lo(e.w) + bf16lo(pp.w), bf16hi(e.w) + bf16hi(pp.w));
    t4[2 * v] = a;
    t4[2 * v + 1] = c;
    ss += a.x * a.x + a.y * a.y + a.z * a.z + a.w * a.w + c.x * c.x + c.y * c.y + c.z * c.z + c.w * c.w;
  }
  ss = block_sum(ss);   // also orders this CTA's t writes before the reads below
  const float inv = rsqrtf(ss / (float)D + 1e-6f);
  for (int v = threadIdx.x; v < nv; v += blockDim.x) {
    const float4 a = t4[2 * v], c = t4[2 * v + 1];
    const float t8[8] = {a.x, a.y, a.z, a.w, c.x, c.y, c.z, c.w};
#pragma unroll
    for (int i = 0; i < 8; ++i) store_bf16_terms(a_bf16, terms, B, blockIdx.x, D, 8 * v + i, t8[i] * inv);
  }
}

// Causal attention of the newest position over positions 0..npos-1 of the
// block: one CTA per (row, head); o = softmax(q k^T / sqrt(dh)) v, stored as
// `terms` bf16 terms. q is staged in shared memory; one warp per position
// computes a score with four loads of the key in flight; each output element
// sums over the positions four values at a time.
__global__ void k_attention(const float* __restrict__ q, const float* __restrict__ kc, const float* __restrict__ vc,
                            int D, int nh, int npos, int cache_ld_pos, uint16_t* __restrict__ o_bf16, int terms,
                            int B) {
  extern __shared__ float sq[];   // dh
  __shared__ float w[64];
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x / nh, hd = blockIdx.x % nh;
  const int dh = D / nh;
  const float scale = rsqrtf((float)dh);
  for (int i = threadIdx.x; i < dh; i += blockDim.x) sq[i] = q[(long long)b * D + hd * dh + i];
  __syncthreads();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  for (int p = warp; p < npos; p += nw) {
    const float* kv = kc + ((long long)b * cache_ld_pos + p) * D + hd * dh;
    float d[4] = {0.f, 0.f, 0.f, 0.f};
    for (int i0 = lane; i0 < dh; i0 += 128) {
      float k4[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) k4[u] = i0 + 32 * u < dh ? kv[i0 + 32 * u] : 0.f;
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (i0 + 32 * u < dh) d[u] = fmaf(sq[i0 + 32 * u], k4[u], d[u]);
    }
    float dd = (d[0] + d[1]) + (d[2] + d[3]);
#pragma unroll
    for (int k = 16; k > 0; k >>= 1) dd += __shfl_down_sync(0xFFFFFFFFu, dd, k);
    if (lane == 0) w[p] = dd * scale;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float m = -INFINITY;
    for (int p = 0; p < npos; ++p) m = fmaxf(m, w[p]);
    float s = 0.f;
    for (int p = 0; p < npos; ++p) { w[p] = __expf(w[p] - m); s += w[p]; }
    for (int p = 0; p < npos; ++p) w[p] /= s;
  }
  __syncthreads();
  const long long row0 = (long long)b * cache_ld_pos * D + hd * dh;
  for (int i = threadIdx.x; i < dh; i += blockDim.x) {
    float o[4] = {0.f, 0.f, 0.f, 0.f};
    int p = 0;
    for (; p + 4 <= npos; p += 4) {
      float v4[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) v4[u] = vc[row0 + (long long)(p + u) * D + i];
#pragma unroll
      for (int u = 0; u < 4; ++u) o[u] = fmaf(w[p + u], v4[u], o[u]);
    }
    for (; p < npos; ++p) o[0] = fmaf(w[p], vc[row0 + (long long)p * D + i], o[0]);
    store_bf16_terms(o_bf16, terms, B, b, D, hd * dh + i, (o[0] + o[1]) + (o[2] + o[3]));
  }
}

// bf16 skinny product on CUDA cores for a few rows, with the activation and
// the bf16 rounding of the output fused: Y[b, o] = bf16(act(sum_k X[b, k]
// W[o, k])) for B <= BMAX, float32 accumulation. One warp per output row o;
// each lane keeps up to 16 weight loads of 16 bytes (8 values) in flight, the
// first ones issued before waiting for the predecessor (the weights are not
// its output); the X rows are staged in shared memory once per CTA. K is a
// multiple of 8 and the rows are 16-byte aligned.
template <int BMAX>
__global__ void k_gemv_bf16(const uint16_t* __restrict__ X, int ldx, const uint16_t* __restrict__ W, int B, int O,
                            int K, int act, uint16_t* __restrict__ Y, int ldy) {
  extern __shared__ __align__(16) uint16_t sx[];   // [B][K]
  constexpr int U = 16;   // weight vectors per lane in flight
  if (threadIdx.x == 0) pdl_trigger();
  const int lane = threadIdx.x & 31;
  const int o = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const bool live = o < O;
  const int nv = K / 8;
  const uint4* w = reinterpret_cast<const uint4*>(W + (long long)(live ? o : 0) * K);
  uint4 wv[U];
#pragma unroll
  for (int u = 0; u < U; ++u) {
    const int v = lane + u * 32;
    wv[u] = (live && v < nv) ? __ldg(w + v) : make_uint4(0, 0, 0, 0);
  }
  pdl_wait();
  uint4* sx4 = reinterpret_cast<uint4*>(sx);
  for (int i = threadIdx.x; i < B * nv; i += blockDim.x) {
    const int b = i / nv, v = i - b * nv;
    sx4[i] = __ldg(reinterpret_cast<const uint4*>(X + (long long)b * ldx) + v);
  }
  __syncthreads();
  if (!live) return;
  float acc[BMAX];
#pragma unroll
  for (int i = 0; i < BMAX; ++i) acc[i] = 0.f;
  for (int v0 = 0; v0 < nv; v0 += 32 * U) {
    if (v0 > 0) {
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int v = v0 + lane + u * 32;
        wv[u] = v < nv ? __ldg(w + v) : make_uint4(0, 0, 0, 0);
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int v = v0 + lane + u * 32;
      if (v >= nv) continue;
      const float w8[8] = {bf16lo(wv[u].x), bf16hi(wv[u].x), bf16lo(wv[u].y), bf16hi(wv[u].y),
                           bf16lo(wv[u].z), bf16hi(wv[u].z), bf16lo(wv[u].w), bf16hi(wv[u].w)};
#pragma unroll
      for (int i = 0; i < BMAX; ++i) {
        if (i < B) {
          const uint4 xv = sx4[i * nv + v];
          acc[i] = fmaf(w8[0], bf16lo(xv.x), acc[i]);
          acc[i] = fmaf(w8[1], bf16hi(xv.x), acc[i]);
          acc[i] = fmaf(w8[2], bf16lo(xv.y), acc[i]);
          acc[i] = fmaf(w8[3], bf16hi(xv.y), acc[i]);
          acc[i] = fmaf(w8[4], bf16lo(xv.z), acc[i]);
          acc[i] = fmaf(w8[5], bf16hi(xv.z), acc[i]);
          acc[i] = fmaf(w8[6], bf16lo(xv.w), acc[i]);
          acc[i] = fmaf(w8[7], bf16hi(xv.w), acc[i]);
        }
      }
    }
  }
#pragma unroll
  for (int i = 0; i < BMAX; ++i) {
    float v = acc[i];
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) v += __shfl_down_sync(0xFFFFFFFFu, v, d);
    if (lane == 0 && i < B) Y[(long long)i * ldy + o] = f32_to_bf16_rne(act_f(act, v));
  }
}

// float32 skinny product on CUDA cores: Y[b, o] = act(sum_k X[b, k] W[o, k]);
// one warp per output row o, lanes stride over k, all batch rows at once.
template <int BMAX>
__global__ void k_gemv_f32(const float* __restrict__ X, int ldx, const float* __restrict__ W, int B, int O, int K,
                           int act, float* __restrict__ Y, int ldy) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int o = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (o >= O) return;
  const float* w = W + (long long)o * K;
  for (int b0 = 0; b0 < B; b0 += BMAX) {
    float acc[BMAX];
#pragma unroll
    for (int i = 0; i < BMAX; ++i) acc[i] = 0.f;
    for (int k = lane; k < K; k += 32) {
      const float wk = w[k];
#pragma unroll
      for (int i = 0; i < BMAX; ++i)
        if (b0 + i < B) acc[i] = fmaf(wk, X[(long long)(b0 + i) * ldx + k], acc[i]);
    }
#pragma unroll
    for (int i = 0; i < BMAX; ++i) {
      float v = acc[i];
#pragma unroll
      for (int d = 16; d > 0; d >>= 1) v += __shfl_down_sync(0xFFFFFFFFu, v, d);
      if (lane == 0 && b0 + i < B) Y[(long long)(b0 + i) * ldy + o] = act_f(act, v);
    }
  }
}

// float32 vocabulary projection fused with the combine: CTA (chunk, b)
// computes l_S[v] = W_vocab[v] . feat[b] for its vocabulary chunk (one warp
// per row v), fuses l = l_L + alpha l_S - beta l_P and reduces to one RowAcc.
__global__ void __launch_bounds__(256) k_vocab_combine_f32(const float* __restrict__ feat, int K,
                                                           const float* __restrict__ Wv, const void* longp,
                                                           int long_f32, long long ld_long,
                                                           const float* __restrict__ prior, float alpha, float beta,
                                                           int V, void* partials, int partial_ld, int nchunks,
                                                           int* status, SampleArgs smp, int j) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const int chunk = blockIdx.x % nchunks, b = blockIdx.x / nchunks;
  const int per = (V + nchunks - 1) / nchunks;
  const int v0 = chunk * per, v1 = min(V, v0 + per);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  const float* fb = feat + (long long)b * K;
  float best = -INFINITY, second = -INFINITY, m = -INFINITY, s = 0.f;
  int idx = INT_MAX;
  for (int v = v0 + warp; v < v1; v += nw) {
    const float* w = Wv + (long long)v * K;
    float d = 0.f;
    for (int k = lane; k < K; k += 32) d = fmaf(w[k], fb[k], d);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) d += __shfl_xor_sync(0xFFFFFFFFu, d, o);
    const float l = long_f32 ? static_cast<const float*>(longp)[(long long)b * ld_long + v]
                             : bf16_to_f(static_cast<const uint16_t*>(longp)[(long long)b * ld_long + v]);
    float f[1] = {fmaf(-beta, prior[v], fmaf(alpha, d, l))};
    // temperature 1: the top-2 over the keys f + g (see write_decode_sampled)
    const float key = smp.on ? f[0] + gumbel_at(smp.seed, smp.step, b, j, kStreamDraft, v) : f[0];
    top2_push(key, v, best, second, idx);
    lse_chunk<1>(f, best, m, s);
  }
  RowAcc r;
  r.m = best; r.s = s; r.second = second; r.idx = idx;
  // lanes of a warp hold identical states; merge across warps
  __shared__ RowAcc red[32];
  if (lane == 0) red[warp] = r;
  __syncthreads();
  if (warp == 0) {
    RowAcc x = lane < nw ? red[lane] : rowacc_init();
    x = rowacc_warp_reduce(x);
    if (lane == 0)
      reinterpret_cast<float4*>(partials)[(long long)b * partial_ld + chunk] =
          make_float4(x.m, x.s, x.second, __int_as_float(x.idx));
  }
  (void)status;
}

inline int grid_for(long long total, int threads) {
  long long g = (total + threads - 1) / threads;
  return (int)std::min<long long>(std::max<long long>(g, 1), 65535LL * 16);
}

}  // namespace

cudaError_t launch_gru_gates(const float* part, int S0, int S1, int B, int H, float* h, uint16_t* h_bf16,
                             cudaStream_t s) {
  return launch_pdl(k_gru_gates, dim3(grid_for((long long)B * H, 256)), dim3(256), 0, s, part, S0, S1, B, H, h, h_bf16);
}

cudaError_t launch_gru_gates_table(const GatesTableArgs& a, cudaStream_t s) {
  const int chunks = (a.H + kGatesThreads - 1) / kGatesThreads;   // one hidden unit per thread
  if (chunks > 65535 || a.S > 8) return cudaErrorInvalidValue;
  return launch_pdl(k_gru_gates_table, dim3(a.B, chunks), dim3(kGatesThreads), 0, s, a);
}

cudaError_t launch_splitk_finish(const float* part, int S, int B, int O, const float* residual, int act,
                                 float* out_f32, int ld_f32, uint16_t* out_bf16, int ld_bf16, cudaStream_t s,
                                 int in_terms, int out_terms) {
  return launch_pdl(k_splitk_finish, dim3(grid_for((long long)B * O, 256)), dim3(256), 0, s, part, S, B, O, residual,
                    act, out_f32, ld_f32, out_bf16, ld_bf16, in_terms, out_terms);
}

cudaError_t launch_splitk_finish3(const SplitkJobs3& jobs, int njobs, int B, int O, int ldp, int in_terms,
                                  cudaStream_t s) {
  if (njobs < 1 || njobs > 3) return cudaErrorInvalidValue;
  return launch_pdl(k_splitk_finish3, dim3(grid_for((long long)B * O, 256), njobs), dim3(256), 0, s, jobs, B, O, ldp,
                    in_terms);
}

cudaError_t launch_finish_rmsnorm(const float* part, int S, int in_terms, int B, int D, const float* residual,
                                  float* out_f32, uint16_t* norm_bf16, int terms, cudaStream_t s) {
  const int per = (D + kNormCluster - 1) / kNormCluster;
  const int threads = std::min(1024, (per + 31) / 32 * 32);
  if ((long long)threads * 4 < per) return cudaErrorInvalidValue;   // kMaxPer elements per thread
  return launch_pdl_cluster(k_finish_rmsnorm, dim3(B * kNormCluster), dim3(threads), 0, s, kNormCluster, part, S,
                            in_terms, B, D, residual, out_f32, norm_bf16, terms);
}

cudaError_t launch_rmsnorm_bf16(const float* x, int B, int D, int ld, uint16_t* out, cudaStream_t s, int terms) {
  return launch_pdl(k_rmsnorm_bf16, dim3(B), dim3(256), 0, s, x, D, ld, out, terms, B);
}

cudaError_t launch_xfmr_embed(const uint16_t* e_rows, const uint16_t* pos_table, int pos, int B, int D,
                              float* t_out, uint16_t* a_bf16, cudaStream_t s, int terms) {
  if (D % 8 != 0) return cudaErrorInvalidValue;
  return launch_pdl(k_xfmr_embed, dim3(B), dim3(256), 0, s, e_rows, pos_table, pos, D, t_out, a_bf16, terms, B);
}

cudaError_t launch_attention(const float* q, const float* kcache, const float* vcache, int B, int D, int nh,
                             int npos, int cache_ld_pos, uint16_t* o_bf16, cudaStream_t s, int terms) {
  if (npos < 1 || npos > 64) return cudaErrorInvalidValue;
  const int dh = D / nh;
  return launch_pdl(k_attention, dim3(B * nh), dim3(256), (size_t)dh * 4, s, q, kcache, vcache, D, nh, npos,
                    cache_ld_pos, o_bf16, terms, B);
}

cudaError_t launch_gemv_bf16(const uint16_t* X, int ldx, const uint16_t* W, int B, int O, int K, int act,
                             uint16_t* Y, int ldy, cudaStream_t s) {
  if (!gemv_bf16_ok(B, K)) return cudaErrorInvalidValue;
  const int warps = 4;
  return launch_pdl(k_gemv_bf16<kGemvBf16MaxRows>, dim3((O + warps - 1) / warps), dim3(warps * 32),
                    (size_t)B * K * 2, s, X, ldx, W, B, O, K, act, Y, ldy);
}

cudaError_t launch_gemv_f32(const float* X, int ldx, const float* W, int B, int O, int K, int act, float* Y, int ldy,
                            cudaStream_t s) {
  const int warps = 8;
  return launch_pdl(k_gemv_f32<8>, dim3((O + warps - 1) / warps), dim3(warps * 32), 0, s, X, ldx, W, B, O, K, act, Y,
                    ldy);
}

cudaError_t launch_vocab_combine_f32(const float* feat, int K, const float* Wv, const void* longp, int long_f32,
                                     long long ld_long, const float* prior, float alpha, float beta, int B, int V,
                                     void* partials, int partial_ld, int nchunks, int* status, cudaStream_t s,
                                     const SampleArgs* smp, int j) {
  const SampleArgs sm = smp ? *smp : SampleArgs{};
  return launch_pdl(k_vocab_combine_f32, dim3(B * nchunks), dim3(256), 0, s, feat, K, Wv, longp, long_f32, ld_long,
                    prior, alpha, beta, V, partials, partial_ld, nchunks, status, sm, j);
}

}  // namespace dels
