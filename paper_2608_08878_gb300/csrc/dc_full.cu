// dc_full.cu -- full-cache decode attention (the comparator of the paper's
// latency table, "Full" row): split-K flash-decode of the G query heads of each
// row over all n cached tokens, with no append, no features and no eviction.
#include "dc_common.cuh"
#include "dc_kernels.h"

namespace dc {

constexpr int kFullTile = 128;

template <int D>
__device__ __forceinline__ void full_load_tile(__nv_bfloat16 (*dst)[D + 8], const __nv_bfloat16* src,
                                               int rows) {
  constexpr int VPR = D / 8;
  for (int e = threadIdx.x; e < rows * VPR; e += blockDim.x) {
    int rr = e / VPR, cc = e % VPR;
    *reinterpret_cast<uint4*>(&dst[rr][cc * 8]) =
        __ldg(reinterpret_cast<const uint4*>(src) + (size_t)rr * VPR + cc);
  }
}

// grid (nsplit, R), block kFullTile. Writes per-split (m, l) to part and the
// unnormalised output sum 2^((s-m)c) v to opart.
template <int D, int G>
__global__ void __launch_bounds__(kFullTile) full_split_kernel(Dev p, int n, int chunk,
                                                               const __nv_bfloat16* __restrict__ q) {
  __shared__ float qs[G][D];
  __shared__ __align__(16) __nv_bfloat16 kt[kFullTile][D + 8];
  __shared__ float pt[kFullTile][G];
  __shared__ float red[kFullTile / kWarp][G];
  __shared__ float mnew[G], scale[G];
  const int r = blockIdx.y, sp = blockIdx.x, tid = threadIdx.x;
  const int c0 = sp * chunk, c1 = min(n, c0 + chunk);
  const int qo = ((r / p.kvh) * p.qh + (r % p.kvh) * G) * D;
  for (int e = tid; e < G * D; e += blockDim.x) qs[e / D][e % D] = __bfloat162float(q[qo + e]);
  constexpr int NOUT = G * D;
  constexpr int OPT = NOUT >= kFullTile ? NOUT / kFullTile : 1;
  const int o0 = tid * OPT;
  const bool owns = o0 < NOUT;
  const int oh = owns ? o0 / D : 0, oc = owns ? o0 % D : 0;
  float oacc[OPT];
#pragma unroll
  for (int e = 0; e < OPT; ++e) oacc[e] = 0.f;
  float M[G], L[G];  // running max / denominator (kept identical in all threads)
#pragma unroll
  for (int h = 0; h < G; ++h) { M[h] = -INFINITY; L[h] = 0.f; }
  const float c = p.c;
  const int lane = tid % kWarp, wid = tid / kWarp;
  for (int base = c0; base < c1; base += kFullTile) {
    const int rows = min(kFullTile, c1 - base);
    __syncthreads();
    full_load_tile<D>(kt, p.K + ((size_t)r * p.stride + base) * D, rows);
    __syncthreads();
    float s[G];
#pragma unroll
    for (int h = 0; h < G; ++h) s[h] = -INFINITY;
    if (tid < rows) {
#pragma unroll
      for (int h = 0; h < G; ++h) s[h] = 0.f;
      for (int c8 = 0; c8 < D / 8; ++c8) {
        uint4 u = *reinterpret_cast<const uint4*>(&kt[tid][c8 * 8]);
        float kf[8] = {bf16lo(u.x), bf16hi(u.x), bf16lo(u.y), bf16hi(u.y),
                       bf16lo(u.z), bf16hi(u.z), bf16lo(u.w), bf16hi(u.w)};
#pragma unroll
        for (int e = 0; e < 8; ++e)
#pragma unroll
          for (int h = 0; h < G; ++h) s[h] = fmaf(qs[h][c8 * 8 + e], kf[e], s[h]);
      }
    }
    // tile max per head
#pragma unroll
    for (int h = 0; h < G; ++h) {
      float x = s[h];
      for (int off = 16; off > 0; off >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, off));
      if (lane == 0) red[wid][h] = x;
    }
    __syncthreads();
    if (tid < G) {
      float x = -INFINITY;
      for (int wv = 0; wv < kFullTile / kWarp; ++wv) x = fmaxf(x, red[wv][tid]);
      const float mn = fmaxf(M[tid], x);
      mnew[tid] = mn;
      scale[tid] = (M[tid] == -INFINITY) ? 0.f : ex2((M[tid] - mn) * c);
    }
    __syncthreads();
#pragma unroll
    for (int h = 0; h < G; ++h) {
      const float pe = (tid < rows) ? ex2((s[h] - mnew[h]) * c) : 0.f;
      pt[tid][h] = pe;
    }
    // denominators: block sum of the tile's weights
#pragma unroll
    for (int h = 0; h < G; ++h) {
      float x = pt[tid][h];
      for (int off = 16; off > 0; off >>= 1) x += __shfl_xor_sync(0xffffffffu, x, off);
      if (lane == 0) red[wid][h] = x;
    }
    __syncthreads();
#pragma unroll
    for (int h = 0; h < G; ++h) {
      float t = 0.f;
      for (int wv = 0; wv < kFullTile / kWarp; ++wv) t += red[wv][h];
      L[h] = L[h] * scale[h] + t;
      M[h] = mnew[h];
    }
    // V tile reuses the key buffer
    __syncthreads();
    full_load_tile<D>(kt, p.V + ((size_t)r * p.stride + base) * D, rows);
    __syncthreads();
    if (owns) {
      const float f = scale[oh];
#pragma unroll
      for (int e = 0; e < OPT; ++e) oacc[e] *= f;
      for (int i = 0; i < rows; ++i) {
        const float pi = pt[i][oh];
#pragma unroll
        for (int e = 0; e < OPT; ++e) oacc[e] = fmaf(pi, __bfloat162float(kt[i][oc + e]), oacc[e]);
      }
    }
  }
  if (owns) {
    float* op = p.opart + (((size_t)r * p.smax + sp) * G) * D + o0;
#pragma unroll
    for (int e = 0; e < OPT; ++e) op[e] = oacc[e];
  }
  if (tid < G) {
    float* pp = p.part + (((size_t)r * p.smax + sp) * G + tid) * 4;
    pp[0] = M[tid]; pp[1] = L[tid]; pp[2] = 0.f; pp[3] = 0.f;
  }
}

// grid (R), block G*D (<= 1024): out = sum_j 2^((m_j-M)c) o_j / sum_j 2^((m_j-M)c) l_j.
template <int D, int G>
__global__ void full_combine_kernel(Dev p, int nsplit, float* __restrict__ out) {
  const int r = blockIdx.x;
  const int qo = ((r / p.kvh) * p.qh + (r % p.kvh) * G) * D;
  for (int e = threadIdx.x; e < G * D; e += blockDim.x) {
    const int h = e / D;
    float M = -INFINITY;
    for (int sp = 0; sp < nsplit; ++sp) M = fmaxf(M, p.part[(((size_t)r * p.smax + sp) * G + h) * 4]);
    float num = 0.f, den = 0.f;
    for (int sp = 0; sp < nsplit; ++sp) {
      const float* pp = p.part + (((size_t)r * p.smax + sp) * G + h) * 4;
      if (pp[0] == -INFINITY) continue;
      const float f = ex2((pp[0] - M) * p.c);
      den += pp[1] * f;
      num += p.opart[(((size_t)r * p.smax + sp) * G) * D + e] * f;
    }
    out[qo + e] = num / den;
  }
}

template <int D, int G>
static void full_t(const Dev& p, int n, int nsplit, int chunk, const void* q, float* out,
                   cudaStream_t s) {
  dim3 grid(nsplit, p.R);
  full_split_kernel<D, G><<<grid, kFullTile, 0, s>>>(p, n, chunk, (const __nv_bfloat16*)q);
  full_combine_kernel<D, G><<<p.R, G * D < 1024 ? G * D : 1024, 0, s>>>(p, nsplit, out);
}

bool launch_full_decode(const Dev& p, int n, int nsplit, int chunk, const void* q, float* out,
                        cudaStream_t s) {
#define DC_CASE(D_, G_) \
  if (p.d == D_ && p.G == G_) { full_t<D_, G_>(p, n, nsplit, chunk, q, out, s); return true; }
  DC_CASE(64, 1) DC_CASE(64, 2) DC_CASE(64, 4) DC_CASE(64, 8)
  DC_CASE(128, 1) DC_CASE(128, 2) DC_CASE(128, 4) DC_CASE(128, 8)
#undef DC_CASE
  return false;
}

}  // namespace dc
