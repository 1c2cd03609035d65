// dc_train.cu -- the training-side kernels of App. C: the exact log-partition
// function of the Plackett-Luce distribution over size-B subsets, and
// Gumbel-top-B sampling with the log-probability of the sampled subset.
//
// log Z(s, B, tau) = log sum over subsets a of [L], |a| = B, of
// exp(sum_{i in a} s_i / tau): the log of the elementary symmetric polynomial
// e_B of x_i = exp(s_i / tau). With E_i[k] = e_k(x_1..x_i), adding item i
// gives E_i[k] = E_{i-1}[k] + x_i E_{i-1}[k-1] (E[0] = 1). Items are added in
// chunks of 31: the generating polynomial prod_i (1 + x_i t) of a chunk has
// coefficients c_m = e_m(chunk), and E_{i+31}[k] = sum_m E_i[k-m] c_m (the
// product of the two polynomials). One warp builds a chunk's c_m by the
// item-by-item recurrence (lane m holds c_m); the CTA then convolves, one
// barrier per chunk instead of per item. O(L B) work in O(B) memory, one CTA
// per row, in log space (log-sum-exp), fp32.
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

constexpr int kChunk = 31;        // items per chunk: c_0..c_31 in one warp's lanes
constexpr int kChunkBatch = 64;   // chunks whose polynomials are built per pass

// One CTA per row, up to kLzThreads threads (each owns the terms k = 1 + tid,
// 1 + tid + blockDim, ...; e_0 = 1 never changes, so B = 1024 takes one term
// per thread). Shared memory: E = log2 e_k, double-buffered ([2][B + 1]), then
// the polynomials of a batch of chunks ([kChunkBatch][32], log2 c_m).
__global__ void __launch_bounds__(kLzThreads) pl_logz_kernel(const float* __restrict__ scores, int L, int B,
                                                             float tau, float* __restrict__ out) {
  extern __shared__ float E[];
  constexpr float kLog2e = 1.4426950408889634f, kLn2 = 0.6931471805599453f;
  const int row = blockIdx.x, tid = threadIdx.x, lane = tid % kWarp, warp = tid / kWarp;
  const int nwarps = blockDim.x / kWarp;
  const float* s = scores + (size_t)row * L;
  float* cur = E;
  float* nxt = E + (B + 1);
  float* C = E + 2 * (B + 1);
  for (int k = tid; k <= B; k += blockDim.x) cur[k] = nxt[k] = k == 0 ? 0.f : -INFINITY;
  const int nchunks = (L + kChunk - 1) / kChunk;
  for (int c0 = 0; c0 < nchunks; c0 += kChunkBatch) {
    const int cb = min(kChunkBatch, nchunks - c0);
    // each warp: the polynomials of its chunks, item by item (lane m: c_m;
    // all lanes read c_{m-1} before any writes, through the shuffle)
    for (int ci = warp; ci < cb; ci += nwarps) {
      const int i0 = (c0 + ci) * kChunk, cnt = min(kChunk, L - i0);
      // the chunk's s_i / tau in log2 units, one per lane
      const float yl = lane < cnt ? __fmul_rn(__fdiv_rn(s[i0 + lane], tau), kLog2e) : 0.f;
      float e = lane == 0 ? 0.f : -INFINITY;
      for (int j = 0; j < cnt; ++j) {
        const float y = __shfl_sync(0xffffffffu, yl, j);
        const float below = __shfl_up_sync(0xffffffffu, e, 1);
        if (lane >= 1 && lane <= j + 1) e = log2_add_exp2(e, y + below);
      }
      C[ci * kWarp + lane] = e;
    }
    __syncthreads();
    // E <- E * c, chunk by chunk: E'[k] = log2 sum_m 2^(E[k-m] + c_m)
    for (int ci = 0; ci < cb; ++ci) {
      const float* c = C + ci * kWarp;
      const int cnt = min(kChunk, L - (c0 + ci) * kChunk);
      for (int k = 1 + tid; k <= B; k += blockDim.x) {
        const int mmax = min(k, cnt);
        // the terms in registers: shared memory is read once
        float t[kChunk + 1];
        float mx = -INFINITY;
#pragma unroll
        for (int m = 0; m <= kChunk; ++m) {
          t[m] = m <= mmax ? cur[k - m] + c[m] : -INFINITY;
          mx = fmaxf(mx, t[m]);
        }
        float acc = 0.f;
#pragma unroll
        for (int m = 0; m <= kChunk; ++m) acc += ex2(t[m] - mx);
        nxt[k] = mx == -INFINITY ? -INFINITY : mx + lg2(acc);
      }
      __syncthreads();
      float* t = cur;
      cur = nxt;
      nxt = t;
    }
  }
  if (tid == 0) out[row] = cur[B] * kLn2;
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
  const size_t smem = (2 * (size_t)(B + 1) + kChunkBatch * kWarp) * sizeof(float);
  if (2 * (size_t)(B + 1) * sizeof(float) > 200 * 1024) return train_fail(DC_ERR_INVALID_ARG, "B too large (at most 25599)");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(pl_logz_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return train_fail(DC_ERR_CUDA, cudaGetErrorString(e));
  }
  const int threads = B < kLzThreads ? (B + 31) / 32 * 32 : kLzThreads;
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
