// dc_selftest.cu -- a check of the bounded waits every kernel of the library
// relies on: a wait that can never be satisfied must give up after its time
// limit, record where, and let the kernel return with an error status, so that
// a lost peer or a lost arrival ends as DC_ERR_DEVICE on the host with the
// CUDA context intact instead of a hung GPU.
#include <cuda_runtime.h>

#include <string>

#include "../../include/distillcache.h"
#include "dc_common.cuh"
#include "dc_sm100.cuh"

namespace dc {
namespace {

using namespace sm100;

// One thread waits on a flag in global memory that nothing sets, then on an
// mbarrier that nothing arrives on, each for limit_ns. out[0]: bit 0 the flag
// wait gave up, bit 1 the mbarrier wait gave up; out[1..4] the first timeout's
// record (claim, site, block, waited value); out[5], out[6]: elapsed ns of the
// two waits (low 32 bits each, in microseconds).
__global__ void wait_selftest_kernel(const unsigned* never_set, unsigned* out, unsigned long long limit_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x != 0) return;
  volatile int* ab = &abort;
  unsigned* dbg = out + 1;
  const uint64_t t0 = globaltimer_ns();
  const bool f = flag_wait(never_set, 1u, ab, dbg, 901u, 0u, limit_ns);
  const uint64_t t1 = globaltimer_ns();
  *ab = 0;
  const bool m = mbar_wait(&bar, 0u, ab, dbg, 902u, 0u, limit_ns);
  const uint64_t t2 = globaltimer_ns();
  out[0] = (f ? 0u : 1u) | (m ? 0u : 2u);
  out[5] = (unsigned)((t1 - t0) / 1000u);
  out[6] = (unsigned)((t2 - t1) / 1000u);
}

// The index check of debug builds (DC_INB): thread 0 writes buf[i] for an i
// one past the checked limit `lim`; the check must fail, raise the status bit,
// record site 903 and skip the write. buf holds lim + 1 elements, so even a
// check that let the write through would stay inside the allocation.
__global__ void bounds_selftest_kernel(unsigned* buf, int lim, unsigned* status, unsigned* dbg) {
  if (threadIdx.x != 0) return;
  Dev p{};
  p.status = status;
  p.dbg = dbg;
  const int i = lim;
  if (DC_INB(p, i, lim, 903)) buf[i] = 0xBADu;
  (void)p;
}

thread_local std::string g_selftest_error;

}  // namespace
}  // namespace dc

extern "C" dc_status dc_debug_bounds_selftest(unsigned* result, void* stream) {
  using namespace dc;
  if (!result) {
    g_selftest_error = "NULL pointer";
    return DC_ERR_INVALID_ARG;
  }
#ifndef DC_DEBUG_BOUNDS
  (void)stream;
  g_selftest_error = "not a debug build (DC_DEBUG_BOUNDS): the index checks are compiled out";
  return DC_ERR_STATE;
#else
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  constexpr int kLim = 64;
  unsigned* d = nullptr;  // [0, kLim] the buffer, then the status word and dbg[8]
  cudaError_t e = cudaMalloc(&d, (kLim + 1 + 1 + 8) * sizeof(unsigned));
  if (e == cudaSuccess) e = cudaMemsetAsync(d, 0, (kLim + 1 + 1 + 8) * sizeof(unsigned), s);
  if (e == cudaSuccess) {
    bounds_selftest_kernel<<<1, 32, 0, s>>>(d, kLim, d + kLim + 1, d + kLim + 2);
    e = cudaGetLastError();
  }
  unsigned h[kLim + 1 + 1 + 8] = {};
  if (e == cudaSuccess) e = cudaMemcpyAsync(h, d, sizeof h, cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (d) cudaFree(d);
  if (e != cudaSuccess) {
    g_selftest_error = cudaGetErrorString(e);
    return DC_ERR_CUDA;
  }
  const unsigned* dbg = h + kLim + 2;
  result[0] = h[kLim + 1];                // status word
  result[1] = dbg[5];                     // site of the first failed check
  result[2] = dbg[6];                     // its index
  result[3] = dbg[7];                     // its limit
  result[4] = h[kLim] == 0u ? 1u : 0u;    // the write was skipped
  return DC_OK;
#endif
}

extern "C" const char* dc_selftest_last_error(void) { return dc::g_selftest_error.c_str(); }

extern "C" dc_status dc_wait_selftest(unsigned long long limit_ns, unsigned* result, void* stream) {
  using namespace dc;
  if (!result) {
    g_selftest_error = "NULL pointer";
    return DC_ERR_INVALID_ARG;
  }
  if (limit_ns < 1000000ull || limit_ns > 1000000000ull) {
    g_selftest_error = "limit_ns must be within [1 ms, 1 s]";
    return DC_ERR_INVALID_ARG;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  unsigned* d = nullptr;  // [0] the flag nothing sets, [1..7] the results
  cudaError_t e = cudaMalloc(&d, 8 * sizeof(unsigned));
  if (e == cudaSuccess) e = cudaMemsetAsync(d, 0, 8 * sizeof(unsigned), s);
  if (e == cudaSuccess) {
    wait_selftest_kernel<<<1, 32, 0, s>>>(d, d + 1, limit_ns);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) e = cudaMemcpyAsync(result, d + 1, 7 * sizeof(unsigned), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (d) cudaFree(d);
  if (e != cudaSuccess) {
    g_selftest_error = cudaGetErrorString(e);
    return DC_ERR_CUDA;
  }
  return DC_OK;
}
