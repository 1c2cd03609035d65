// dc_noalloc.cu -- full-cache decode attention for callers that cannot
// allocate device memory: the split-K partial results live in a fixed,
// file-scope device array instead of buffers allocated by the library.
//
// Which callers cannot allocate: runtimes that reserve all device memory up
// front and forbid further allocation (fixed-footprint serving processes),
// and latency-critical paths where an implicit device synchronisation from
// cudaMalloc/cudaFree is not acceptable. None of the handle-based calls fit
// them, because dc_cache_create allocates.
//
// The scratch array is reserved on a device when this library's device code
// is loaded there, and stays reserved until the process exits. Under lazy
// module loading (CUDA's default) that happens at the first call on the
// device, inside cudaGetSymbolAddress below: a caller that reserves the rest
// of device memory must make its first call before doing so.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdio>
#include <mutex>
#include <string>

#include "../../include/distillcache.h"
#include "dc_common.cuh"
#include "dc_kernels.h"

namespace {

// Split-K partials: per (row, split, head) the running max and denominator
// (4 floats) and the unnormalised output (head_dim floats).
constexpr size_t kScratchBytes = (size_t)16 << 20;  // 16 MiB
static __device__ __align__(256) float g_noalloc_scratch[kScratchBytes / sizeof(float)];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
float* g_scratch_ptr[kMaxDevices] = {};
int g_num_sms[kMaxDevices] = {};

thread_local std::string g_noalloc_error;

dc_status noalloc_fail(dc_status s, const std::string& msg) {
  g_noalloc_error = msg;
  return s;
}

}  // namespace

extern "C" const char* dc_noalloc_last_error(void) { return g_noalloc_error.c_str(); }

extern "C" dc_status dc_attend_noalloc(const void* q, const void* k, const void* v, int rows, int n,
                                       int head_dim, int group, float* out, void* stream) {
  if (!q || !k || !v || !out) return noalloc_fail(DC_ERR_INVALID_ARG, "NULL pointer");
  if (head_dim != 64 && head_dim != 128) return noalloc_fail(DC_ERR_INVALID_ARG, "head_dim must be 64 or 128");
  if (group != 1 && group != 2 && group != 4 && group != 8)
    return noalloc_fail(DC_ERR_INVALID_ARG, "group must be 1, 2, 4 or 8");
  if (rows < 1 || rows > 65535 || n < 1) return noalloc_fail(DC_ERR_INVALID_ARG, "need 1 <= rows <= 65535 and n >= 1");
  if (((uintptr_t)k | (uintptr_t)v) & 15) return noalloc_fail(DC_ERR_INVALID_ARG, "k and v must be 16-byte aligned");
  // one split's partials for every row must fit the scratch array
  const size_t per_split = (size_t)rows * group * (head_dim + 4) * sizeof(float);
  if (per_split > kScratchBytes) {
    char buf[192];
    std::snprintf(buf, sizeof buf,
                  "rows * group * (head_dim + 4) * 4 = %zu bytes exceeds the %zu-byte scratch of the no-allocation path",
                  per_split, kScratchBytes);
    return noalloc_fail(DC_ERR_CAPACITY, buf);
  }
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return noalloc_fail(DC_ERR_CUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return noalloc_fail(DC_ERR_INVALID_ARG, "device ordinal out of range");
  float* scratch = nullptr;
  int num_sms = 0;
  {
    // set-up, once per device, with that device current
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_scratch_ptr[dev]) {
      void* ptr = nullptr;
      e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
      if (e != cudaSuccess)
        return noalloc_fail(DC_ERR_CUDA, std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
      int sms = 0;
      e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
      if (e != cudaSuccess)
        return noalloc_fail(DC_ERR_CUDA, std::string("cudaDeviceGetAttribute: ") + cudaGetErrorString(e));
      g_scratch_ptr[dev] = static_cast<float*>(ptr);
      g_num_sms[dev] = sms;
    }
    scratch = g_scratch_ptr[dev];
    num_sms = g_num_sms[dev];
  }
  // split plan: enough CTAs to fill the GPU, bounded by the scratch array
  int want = (int)((8ll * num_sms + rows - 1) / rows);
  want = want < 1 ? 1 : (want > 64 ? 64 : want);
  const int max_tiles = (n + 127) / 128;
  if (want > max_tiles) want = max_tiles;
  const int fit = (int)(kScratchBytes / per_split);
  if (want > fit) want = fit;
  int chunk = (n + want - 1) / want;
  chunk = (chunk + 127) / 128 * 128;
  const int nsplit = (n + chunk - 1) / chunk;

  dc::Dev p{};
  p.R = rows;
  p.cap = n;
  p.stride = n;
  p.d = head_dim;
  p.G = group;
  p.qh = group;  // q and out are [rows][group][head_dim]
  p.kvh = 1;
  p.K = const_cast<__nv_bfloat16*>(static_cast<const __nv_bfloat16*>(k));
  p.V = const_cast<__nv_bfloat16*>(static_cast<const __nv_bfloat16*>(v));
  p.smax = nsplit;
  p.part = scratch;
  p.opart = scratch + (size_t)rows * nsplit * group * 4;
  p.c = (float)(1.4426950408889634 / std::sqrt((double)head_dim));
  if (!dc::launch_full_decode(p, n, nsplit, chunk, q, out, static_cast<cudaStream_t>(stream)))
    return noalloc_fail(DC_ERR_INVALID_ARG, "unsupported head_dim / group");
  e = cudaGetLastError();
  if (e != cudaSuccess) return noalloc_fail(DC_ERR_CUDA, std::string("launch: ") + cudaGetErrorString(e));
  return DC_OK;
}
