// dc_evict.cu -- argtop_B and prune (Algorithm 1) of every row as its own
// kernel (dc_evict): one CTA per row runs the team selection and compaction of
// dc_select.cuh.
#include "dc_common.cuh"
#include "dc_kernels.h"
#include "dc_select.cuh"

namespace dc {

constexpr int kEvictThreads = 1024;

// grid (R), block kEvictThreads: the whole CTA selects and compacts one row.
__global__ void __launch_bounds__(kEvictThreads) evict_kernel(Dev p, int n, int B) {
  __shared__ int hist[256];
  __shared__ int sh[4];
  __shared__ int wsum[kEvictThreads / kWarp];
  __shared__ unsigned long long best[kEvictThreads / kWarp];
  __shared__ int best_slot[kEvictThreads / kWarp];
  const SelectScratch scr{hist, sh, wsum, best, best_slot};
  auto sync = [] { __syncthreads(); };
  const int r = blockIdx.x;
  if (p.rowlen) {
    // per-row lengths and budgets (B > 0 overrides every row's budget)
    const int nr = p.rowlen[r], Br = B > 0 ? B : p.rowbudget[r];
    const int keep = nr < Br ? nr : Br;
    if (keep < nr)
      team_select_compact<kEvictThreads>(p, r, nr, keep, p.score + (size_t)r * p.stride, threadIdx.x, scr, sync);
    if (threadIdx.x == 0) p.rowlen[r] = keep;
    return;
  }
  team_select_compact<kEvictThreads>(p, r, n, B, p.score + (size_t)r * p.stride, threadIdx.x, scr, sync);
}

void launch_evict(const Dev& p, int n, int B, cudaStream_t s) {
  evict_kernel<<<p.R, kEvictThreads, 0, s>>>(p, n, B);
}

}  // namespace dc
