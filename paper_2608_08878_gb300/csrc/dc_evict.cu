// dc_evict.cu -- argtop_B and prune (Algorithm 1) of every row as kernels of
// their own (dc_evict, and dc_step's many-eviction steps): a select kernel,
// one CTA per row, ranks the row and lists its holes and movers; a move
// kernel, spread over the whole GPU, copies the movers into the holes.
#include "dc_common.cuh"
#include "dc_kernels.h"
#include "dc_select.cuh"

namespace dc {

// Select: one CTA of 1024 threads per row. The row's order keys are computed
// once into shared memory (16-byte score loads, all of a thread's loads in
// flight together), so that the select's passes (radix digits, ties, the hole
// and mover lists) read shared memory instead of waiting on HBM in every
// pass. Rows longer than kSmemKeys keep reading their keys from the scores.
constexpr int kEvictThreads = 1024;
constexpr int kSmemKeys = 48 * 1024;  // 192 KB of keys
// Move: 256 threads (8 warps) per block, 32 moves per warp, blocks laid out
// as (move chunk, row) so that every SM holds many rows' moves at once.
constexpr int kMoveThreads = 256;

// grid (R), block kEvictThreads, dynamic shared memory: the keys of up to
// min(n, kSmemKeys) tokens (none when the launcher passes n > kSmemKeys).
// One eviction is moved here; several are listed for evict_move_kernel.
__global__ void __launch_bounds__(kEvictThreads) evict_select_kernel(Dev p, int n, int B, int smem_keys) {
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
  if (tid == 0) {
    p.nmoves[2 * (size_t)r] = 0;  // no moves unless the lists below say so
    p.nmoves[2 * (size_t)r + 1] = 0;
  }
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

// grid (ceil(max moves / kMoveThreads), R), block kMoveThreads: warp w of block
// x moves entries [x * 256 + 32 w, + 32) of row y's lists.
__global__ void __launch_bounds__(kMoveThreads) evict_move_kernel(Dev p) {
  const int r = blockIdx.y;
  const int nmv = p.nmoves[2 * (size_t)r], nh = p.nmoves[2 * (size_t)r + 1];
  const int k0 = blockIdx.x * kMoveThreads + (threadIdx.x / kWarp) * kWarp;
  if (k0 >= nmv) return;
  const size_t base = (size_t)r * p.stride;
  warp_move_batch(p, base, p.holes + base, p.holes + base + nh, k0, nmv, threadIdx.x % kWarp);
}

// A row moves at most min(B, n - B) slots; with per-row budgets (B <= 0) at
// most n / 2.
static int max_moves(int n, int B) { return B > 0 ? (B < n - B ? B : n - B) : n / 2; }

int evict_kernel_count(int n, int B) { return max_moves(n, B) > 0 ? 2 : 1; }

void launch_evict(const Dev& p, int n, int B, cudaStream_t s) {
  static bool attr = false;
  if (!attr) {
    if (cudaFuncSetAttribute(evict_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             kSmemKeys * (int)sizeof(uint32_t)) != cudaSuccess)
      return;  // the launch below then fails and the caller reports the error
    attr = true;
  }
  const int smem_keys = n <= kSmemKeys ? n : 0;
  evict_select_kernel<<<p.R, kEvictThreads, (size_t)smem_keys * sizeof(uint32_t), s>>>(p, n, B, smem_keys);
  const int mm = max_moves(n, B);
  if (mm > 0) {
    const dim3 grid((unsigned)((mm + kMoveThreads - 1) / kMoveThreads), (unsigned)p.R);
    evict_move_kernel<<<grid, kMoveThreads, 0, s>>>(p);
  }
}

}  // namespace dc
