// dc_evict.cu -- argtop_B and prune (Algorithm 1) of every row as its own
// kernel (dc_evict): one CTA per row runs the team selection and compaction of
// dc_select.cuh.
#include "dc_common.cuh"
#include "dc_kernels.h"
#include "dc_select.cuh"

namespace dc {

// One CTA of 1024 threads per row. The row's order keys are computed once
// into shared memory (16-byte score loads, all of a thread's loads in flight
// together), so that the select's passes (radix digits, ties, the hole and
// mover lists) read shared memory instead of waiting on HBM in every pass;
// then each warp copies four slots at a time. Rows longer than kSmemKeys keep
// reading their keys from the score array.
constexpr int kEvictThreads = 1024;
constexpr int kSmemKeys = 48 * 1024;  // 192 KB of keys

// grid (R), block kEvictThreads, dynamic shared memory: the keys of up to
// min(n, kSmemKeys) tokens (none when the launcher passes n > kSmemKeys).
__global__ void __launch_bounds__(kEvictThreads) evict_kernel(Dev p, int n, int B, int smem_keys) {
  extern __shared__ uint32_t skeys[];
  __shared__ int hist[256];
  __shared__ int sh[4];
  __shared__ int wsum[kEvictThreads / kWarp];
  __shared__ unsigned long long best[kEvictThreads / kWarp];
  __shared__ int best_slot[kEvictThreads / kWarp];
  const SelectScratch scr{hist, sh, wsum, best, best_slot};
  auto sync = [] { __syncthreads(); };
  const int r = blockIdx.x, tid = threadIdx.x;
  int nr = n, Br = B;
  if (p.rowlen) {
    // per-row lengths and budgets (B > 0 overrides every row's budget)
    nr = p.rowlen[r];
    Br = B > 0 ? B : p.rowbudget[r];
  }
  const int keep = nr < Br ? nr : Br;
  if (keep < nr) {
    const float* score = p.score + (size_t)r * p.stride;
    if (nr <= smem_keys) {
      // the row's scores start 16-byte aligned (the stride is a multiple of
      // 128 slots): four keys per 16-byte load, up to eight loads per thread
      // issued before their keys are stored
      const int n4 = nr >> 2;
      const float4* s4 = reinterpret_cast<const float4*>(score);
      for (int c0 = 0; c0 < n4; c0 += 8 * kEvictThreads) {
        float4 v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int e = c0 + u * kEvictThreads + tid;
          if (e < n4) v[u] = s4[e];
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int e = c0 + u * kEvictThreads + tid;
          if (e < n4)
            *reinterpret_cast<uint4*>(skeys + 4 * e) =
                make_uint4(score_key(v[u].x), score_key(v[u].y), score_key(v[u].z), score_key(v[u].w));
        }
      }
      for (int i = 4 * n4 + tid; i < nr; i += kEvictThreads) skeys[i] = score_key(score[i]);
      sync();
      team_select_compact_k<kEvictThreads, true>(p, r, nr, keep, [&](int i) { return skeys[i]; }, tid, scr, sync);
    } else {
      team_select_compact_k<kEvictThreads, true>(p, r, nr, keep, [&](int i) { return score_key(score[i]); }, tid,
                                                 scr, sync);
    }
  }
  if (p.rowlen && tid == 0) p.rowlen[r] = keep;
}

void launch_evict(const Dev& p, int n, int B, cudaStream_t s) {
  static bool attr = false;
  if (!attr) {
    if (cudaFuncSetAttribute(evict_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             kSmemKeys * (int)sizeof(uint32_t)) != cudaSuccess)
      return;  // the launch below then fails and the caller reports the error
    attr = true;
  }
  const int smem_keys = n <= kSmemKeys ? n : 0;
  evict_kernel<<<p.R, kEvictThreads, (size_t)smem_keys * sizeof(uint32_t), s>>>(p, n, B, smem_keys);
}

}  // namespace dc
