// dc_evict.cu -- argtop_B and prune (Algorithm 1) for every row: an exact
// radix select of the B-th ranked token followed by hole-fill compaction.
//
// Ranking: score descending, then position ascending (Sec. 3.1.2: inference
// keeps the top-B tokens deterministically). Scores become order-preserving
// 32-bit keys; four 8-bit MSB-first histogram passes find the threshold key T
// with #(key > T) < B <= #(key >= T). When keys equal to T are more than the
// places left, a second select over their positions keeps the lowest ones.
//
// Compaction: slots [0, B) must end up holding the survivors. Evicted slots
// below B are holes; survivors at slots >= B are movers; #holes == #movers.
// The k-th mover (ascending slot) moves into the k-th hole (ascending slot)
// with its key, value, position and window state. Survivors below B stay put.
#include "dc_common.cuh"
#include "dc_kernels.h"

namespace dc {

constexpr int kEvictThreads = 1024;

// Exclusive prefix sum over the CTA of one int per thread; returns the prefix
// and writes the CTA total to *total (all threads).
__device__ __forceinline__ int block_exclusive_scan(int v, int* wsum, int* total) {
  const int lane = threadIdx.x % kWarp, wid = threadIdx.x / kWarp, nw = blockDim.x / kWarp;
  int x = v;
#pragma unroll
  for (int off = 1; off < kWarp; off <<= 1) {
    int y = __shfl_up_sync(0xffffffffu, x, off);
    if (lane >= off) x += y;
  }
  if (lane == kWarp - 1) wsum[wid] = x;
  __syncthreads();
  if (wid == 0) {
    int s = lane < nw ? wsum[lane] : 0;
#pragma unroll
    for (int off = 1; off < kWarp; off <<= 1) {
      int y = __shfl_up_sync(0xffffffffu, s, off);
      if (lane >= off) s += y;
    }
    if (lane < nw) wsum[lane] = s;  // inclusive warp prefix
  }
  __syncthreads();
  const int before = (wid > 0 ? wsum[wid - 1] : 0) + x - v;
  *total = wsum[nw - 1];
  __syncthreads();
  return before;
}

// MSB-first radix select over the keys produced by `keyf(i)` for i in [0, n)
// restricted to `pred(i)`: returns the key T of the need-th largest element
// and leaves in *gt the number of elements with key > T.
template <class KeyF, class Pred>
__device__ uint32_t radix_select(int n, int need, KeyF keyf, Pred pred, int* hist, int* shared_out,
                                 int* gt) {
  uint32_t prefix = 0, mask = 0;
  int above = 0;
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int b = threadIdx.x; b < 256; b += blockDim.x) hist[b] = 0;
    __syncthreads();
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
      if (!pred(i)) continue;
      const uint32_t k = keyf(i);
      if ((k & mask) == prefix) atomicAdd(&hist[(k >> shift) & 255u], 1);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int cum = 0, dgt = 0;
      for (int b = 255; b >= 0; --b) {
        if (above + cum + hist[b] >= need) { dgt = b; break; }
        cum += hist[b];
      }
      shared_out[0] = dgt;
      shared_out[1] = above + cum;
    }
    __syncthreads();
    prefix |= (uint32_t)shared_out[0] << shift;
    mask |= 255u << shift;
    above = shared_out[1];
    __syncthreads();
  }
  *gt = above;
  return prefix;
}

// grid (R), block kEvictThreads.
__global__ void __launch_bounds__(kEvictThreads) evict_kernel(Dev p, int n, int B) {
  __shared__ int hist[256];
  __shared__ int sh[2];
  __shared__ int wsum[kEvictThreads / kWarp];
  const int r = blockIdx.x;
  const size_t base = (size_t)r * p.cap;
  const float* sc = p.score + base;
  const int* ps = p.pos + base;
  auto key = [&](int i) { return score_key(sc[i]); };
  auto all = [](int) { return true; };
  int gt = 0;
  const uint32_t T = radix_select(n, B, key, all, hist, sh, &gt);
  const int need_eq = B - gt;  // tokens with key == T to keep (>= 1)
  // Count keys equal to T.
  int eq_local = 0;
  for (int i = threadIdx.x; i < n; i += blockDim.x) eq_local += (key(i) == T);
  int eq_total;
  (void)block_exclusive_scan(eq_local, wsum, &eq_total);
  uint32_t P = 0;  // keep ties with ~pos >= P (lowest positions)
  if (eq_total > need_eq) {
    auto pkey = [&](int i) { return ~(uint32_t)ps[i]; };
    auto tied = [&](int i) { return key(i) == T; };
    int gt2 = 0;
    P = radix_select(n, need_eq, pkey, tied, hist, sh, &gt2);
  }
  auto keep = [&](int i) {
    const uint32_t k = key(i);
    return k > T || (k == T && ~(uint32_t)ps[i] >= P);
  };
  // Holes: evicted slots below B, in ascending order.
  int* holes = p.holes + base;
  int nh = 0;
  for (int c0 = 0; c0 < B; c0 += blockDim.x) {
    const int i = c0 + threadIdx.x;
    const int f = (i < B && !keep(i)) ? 1 : 0;
    int tot;
    const int rank = block_exclusive_scan(f, wsum, &tot);
    if (f) holes[nh + rank] = i;
    nh += tot;
  }
  __syncthreads();
  // Movers: survivors at slots >= B, in ascending order, fill the holes.
  const int VPR = p.d / 8;
  int nm = 0;
  for (int c0 = B; c0 < n; c0 += blockDim.x) {
    const int i = c0 + threadIdx.x;
    const int f = (i < n && keep(i)) ? 1 : 0;
    int tot;
    const int rank = block_exclusive_scan(f, wsum, &tot);
    if (f && nm + rank < nh) {
      const int dst = holes[nm + rank];
      const size_t s = base + i, t = base + dst;
      const uint4* ks = reinterpret_cast<const uint4*>(p.K) + s * VPR;
      const uint4* vs = reinterpret_cast<const uint4*>(p.V) + s * VPR;
      uint4* kd = reinterpret_cast<uint4*>(p.K) + t * VPR;
      uint4* vd = reinterpret_cast<uint4*>(p.V) + t * VPR;
      for (int e = 0; e < VPR; ++e) { kd[e] = ks[e]; vd[e] = vs[e]; }
      p.pos[t] = p.pos[s];
      p.S[t] = p.S[s];
      p.Z[t] = p.Z[s];
      p.score[t] = p.score[s];
      if (p.acc) p.acc[t] = p.acc[s];
      if (p.keep_features)
        for (int e = 0; e < 5; ++e) p.feat[t * 5 + e] = p.feat[s * 5 + e];
    }
    nm += tot;
  }
  if (threadIdx.x == 0 && nm != nh) atomicOr(p.status, kStatusBadShape);
}

void launch_evict(const Dev& p, int n, int B, cudaStream_t s) {
  evict_kernel<<<p.R, kEvictThreads, 0, s>>>(p, n, B);
}

}  // namespace dc
