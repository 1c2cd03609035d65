// dc_train.cu -- the training-side kernels of App. C: the exact log-partition
// function of the Plackett-Luce distribution over size-B subsets, and
// Gumbel-top-B sampling with the log-probability of the sampled subset.
//
// log Z(s, B, tau) = log sum over subsets a of [L], |a| = B, of
// exp(sum_{i in a} s_i / tau): the log of the elementary symmetric polynomial
// e_B of x_i = exp(s_i / tau). With E_i[k] = e_k(x_1..x_i), adding item i
// gives E_i[k] = E_{i-1}[k] + x_i E_{i-1}[k-1] (E[0] = 1): L sequential steps,
// each an independent update of k = 1..B -- O(L B) work in O(B) memory, one
// CTA per row with the B + 1 terms in shared memory, kept in log space
// (logaddexp), fp32.
//
// Gumbel-top-B: perturbed scores s_i / tau + g_i (g_i ~ Gumbel(0, 1), given by
// the caller), the B largest kept (ties: lower index), their indices written
// in ascending order; log pi(a) = sum_{i in a} s_i / tau - log Z.
#include <cuda_runtime.h>

#include <cmath>
#include <string>

#include "../../include/distillcache.h"
#include "dc_common.cuh"
#include "dc_select.cuh"

namespace dc {
namespace {

constexpr int kLzThreads = 1024;
constexpr int kTopThreads = 512;

__device__ __forceinline__ float lg2(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// log2(2^a + 2^b) with the hardware base-2 exponential and logarithm.
__device__ __forceinline__ float log2_add_exp2(float a, float b) {
  const float m = fmaxf(a, b);
  if (m == -INFINITY) return -INFINITY;
  return m + lg2(1.f + ex2(fminf(a, b) - m));
}

// One CTA per row, kLzThreads threads (each owns the terms k = tid, tid +
// kLzThreads, ...), E = log2 e_k in shared memory, double-buffered ([2][B + 1]).
__global__ void __launch_bounds__(kLzThreads) pl_logz_kernel(const float* __restrict__ scores, int L, int B,
                                                             float tau, float* __restrict__ out) {
  extern __shared__ float E[];
  constexpr float kLog2e = 1.4426950408889634f, kLn2 = 0.6931471805599453f;
  const int row = blockIdx.x;
  const float* s = scores + (size_t)row * L;
  float* cur = E;
  float* nxt = E + (B + 1);
  for (int k = threadIdx.x; k <= B; k += blockDim.x) cur[k] = k == 0 ? 0.f : -INFINITY;
  __syncthreads();
  const int lane = threadIdx.x % kWarp;
  for (int i0 = 0; i0 < L; i0 += kWarp) {
    // the next 32 items' s_i / tau in log2 units, one per lane, broadcast
    // per step by shuffle (off the step's dependency chain)
    const float yl = i0 + lane < L ? __fmul_rn(__fdiv_rn(s[i0 + lane], tau), kLog2e) : 0.f;
    const int cnt = min(kWarp, L - i0);
    for (int j = 0; j < cnt; ++j) {
      const float y = __shfl_sync(0xffffffffu, yl, j);
      const int i = i0 + j;
      // after item i (0-based) only E[0..i+1] can be finite
      const int kmax = min(B, i + 1);
      for (int k = threadIdx.x; k <= B; k += blockDim.x)
        nxt[k] = (k == 0 || k > kmax) ? cur[k] : log2_add_exp2(cur[k], y + cur[k - 1]);
      __syncthreads();
      float* t = cur;
      cur = nxt;
      nxt = t;
    }
  }
  if (threadIdx.x == 0) out[row] = cur[B] * kLn2;
}

// One CTA per row: top-B of the perturbed scores by (value desc, index asc),
// indices ascending into idx[row][0..B), and sum_{i in a} s_i / tau.
__global__ void __launch_bounds__(kTopThreads) gumbel_topb_kernel(const float* __restrict__ scores,
                                                                  const float* __restrict__ gumbel, int L,
                                                                  int B, float tau, int* __restrict__ idx,
                                                                  float* __restrict__ logp,
                                                                  const float* __restrict__ logz) {
  __shared__ int hist[256];
  __shared__ int sh[4];
  __shared__ int wsum[kTopThreads / kWarp];
  __shared__ unsigned long long best[kTopThreads / kWarp];
  __shared__ int best_slot[kTopThreads / kWarp];
  __shared__ double dsum[kTopThreads / kWarp];
  const SelectScratch scr{hist, sh, wsum, best, best_slot};
  auto sync = [] { __syncthreads(); };
  const int row = blockIdx.x, tid = threadIdx.x;
  const float* s = scores + (size_t)row * L;
  const float* g = gumbel + (size_t)row * L;
  auto key = [&](int i) { return score_key(__fadd_rn(__fdiv_rn(s[i], tau), g[i])); };
  auto all = [](int) { return true; };
  int gt = 0;
  const uint32_t T = team_radix_select<kTopThreads>(L, B, key, all, tid, scr, &gt, sync);
  const int need_eq = B - gt;  // ties at T kept by lowest index
  int eq_local = 0;
  for (int i = tid; i < L; i += kTopThreads) eq_local += (key(i) == T);
  int eq_total;
  (void)team_exclusive_scan<kTopThreads>(eq_local, tid, scr.wsum, &eq_total, sync);
  uint32_t P = 0;  // ties kept when ~index >= P
  if (eq_total > need_eq) {
    auto ikey = [](int i) { return ~(uint32_t)i; };
    auto tied = [&](int i) { return key(i) == T; };
    int gt2 = 0;
    P = team_radix_select<kTopThreads>(L, need_eq, ikey, tied, tid, scr, &gt2, sync);
  }
  auto keep = [&](int i) {
    const uint32_t k = key(i);
    return k > T || (k == T && ~(uint32_t)i >= P);
  };
  int base = 0;
  double part = 0.0;
  for (int c0 = 0; c0 < L; c0 += kTopThreads) {
    const int i = c0 + tid;
    const int f = (i < L && keep(i)) ? 1 : 0;
    int tot;
    const int rank = team_exclusive_scan<kTopThreads>(f, tid, scr.wsum, &tot, sync);
    if (f) {
      idx[(size_t)row * B + base + rank] = i;
      part += (double)__fdiv_rn(s[i], tau);
    }
    base += tot;
  }
  if (logp) {
    // sum_{i in a} s_i / tau in double, fixed reduction order
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) part += __shfl_xor_sync(0xffffffffu, part, off);
    if (tid % kWarp == 0) dsum[tid / kWarp] = part;
    __syncthreads();
    if (tid == 0) {
      double t = 0.0;
      for (int w = 0; w < kTopThreads / kWarp; ++w) t += dsum[w];
      logp[row] = (float)(t - (double)logz[row]);
    }
  }
}

thread_local std::string g_train_error;

dc_status train_fail(dc_status s, const char* msg) {
  g_train_error = msg;
  return s;
}

}  // namespace
}  // namespace dc

extern "C" const char* dc_train_last_error(void) { return dc::g_train_error.c_str(); }

extern "C" dc_status dc_pl_log_partition(const float* scores, int rows, int L, int B, float tau, float* out,
                                         void* stream) {
  using namespace dc;
  if (!scores || !out) return train_fail(DC_ERR_INVALID_ARG, "NULL pointer");
  if (rows < 1 || rows > 65535 || L < 1 || B < 1 || B > L || !(tau > 0.f))
    return train_fail(DC_ERR_INVALID_ARG, "need 1 <= rows <= 65535, 1 <= B <= L and tau > 0");
  const size_t smem = 2 * (size_t)(B + 1) * sizeof(float);
  if (smem > 200 * 1024) return train_fail(DC_ERR_INVALID_ARG, "B too large (at most 25599)");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(pl_logz_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return train_fail(DC_ERR_CUDA, cudaGetErrorString(e));
  }
  const int threads = B + 1 < kLzThreads ? (B + 1 + 31) / 32 * 32 : kLzThreads;
  pl_logz_kernel<<<rows, threads, smem, s>>>(scores, L, B, tau, out);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return train_fail(DC_ERR_CUDA, cudaGetErrorString(e));
  return DC_OK;
}

extern "C" dc_status dc_gumbel_top_b(const float* scores, const float* gumbel, int rows, int L, int B, float tau,
                                     int* idx, float* logp, float* logz_scratch, void* stream) {
  using namespace dc;
  if (!scores || !gumbel || !idx || (logp && !logz_scratch)) return train_fail(DC_ERR_INVALID_ARG, "NULL pointer");
  if (rows < 1 || rows > 65535 || L < 1 || B < 1 || B > L || !(tau > 0.f))
    return train_fail(DC_ERR_INVALID_ARG, "need 1 <= rows <= 65535, 1 <= B <= L and tau > 0");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (logp) {
    dc_status st = dc_pl_log_partition(scores, rows, L, B, tau, logz_scratch, stream);
    if (st != DC_OK) return st;
  }
  gumbel_topb_kernel<<<rows, kTopThreads, 0, s>>>(scores, gumbel, L, B, tau, idx, logp, logz_scratch);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return train_fail(DC_ERR_CUDA, cudaGetErrorString(e));
  return DC_OK;
}
