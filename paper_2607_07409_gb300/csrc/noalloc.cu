// dels_combine_argmax_noalloc: the fused combine + argmax for callers that
// cannot allocate device memory. Some callers only own the buffers they pass
// in and out — for example a plugin running inside a host framework whose
// allocator it cannot reach, or a latency-critical loop where an allocation
// could synchronise the device — so they cannot provide the workspace that
// dels_combine_argmax asks for. This entry point uses a fixed scratch area
// compiled into the library instead.
//
// The scratch is a file-scope __device__ array: every GPU that loads the
// library holds it until the process exits. Host code cannot use the array's
// name as a device address (in host code it is only a stand-in symbol), so
// the first call on each device looks the address up with
// cudaGetSymbolAddress while that device is current and caches it. The cache
// assumes the device is not reset while the process runs: after
// cudaDeviceReset the cached address is stale and the entry point must not
// be called again in that process.
#include <mutex>

#include "dels_internal.h"

namespace dels {

namespace {

constexpr size_t kNoAllocScratchBytes = 4u << 20;   // 4 MiB per device

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
void* g_noalloc_addr[kMaxDevices] = {nullptr};

// Device address of the scratch for the current device (set up once per device).
int noalloc_scratch(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return DELS_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return DELS_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (g_noalloc_addr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return DELS_ERR_CUDA;
    g_noalloc_addr[dev] = p;
  }
  *out = g_noalloc_addr[dev];
  return DELS_OK;
}

}  // namespace
}  // namespace dels

using namespace dels;

extern "C" int dels_combine_argmax_noalloc(const void* long_logits, const void* short_logits, dels_dtype dtype,
                                           const float* log_prior, float alpha, float beta, int rows, int V,
                                           int32_t* out_token, float* out_logprob, float* out_top2_gap,
                                           dels_stream_t stream) {
  if (dtype != DELS_F32 && dtype != DELS_BF16) return DELS_ERR_BAD_DTYPE;
  if (rows < 0 || V < 1) return DELS_ERR_BAD_SHAPE;
  if (rows == 0) return DELS_OK;
  // every host-side check of dels_combine_argmax runs before the scratch is
  // touched, so a rejected call enqueues nothing (not even the clearing)
  const int chk = combine_check_inputs(long_logits, short_logits, log_prior, out_token);
  if (chk != DELS_OK) return chk;
  const size_t need = dels_combine_workspace_bytes(rows, V, dtype);
  if (need == 0) return DELS_ERR_CUDA;
  if (need > kNoAllocScratchBytes) return DELS_ERR_TOO_LARGE;
  void* scratch = nullptr;
  int r = noalloc_scratch(&scratch);
  if (r != DELS_OK) return r;
  // The status word and the per-row-group tickets must start at zero; the
  // scratch keeps whatever the previous call left, so clear that prefix.
  const CombineLayout L = combine_layout(rows, V, dtype, device_sm_count());
  const size_t zero_bytes = L.partials_off;   // the header and the tickets
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(scratch, 0, zero_bytes, s) != cudaSuccess) return DELS_ERR_CUDA;
  return dels_combine_argmax(long_logits, short_logits, dtype, log_prior, alpha, beta, rows, V, out_token,
                             out_logprob, out_top2_gap, scratch, kNoAllocScratchBytes, stream);
}
