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
// flight together), so that the select's passes read shared memory instead
// of waiting on HBM in every pass. Rows longer than kSmemKeys keep reading
// their keys from the scores.
constexpr int kEvictThreads = 1024;
constexpr int kSmemKeys = 44 * 1024;  // 176 KB of keys (dynamic shared memory)
// Equal-width key bins of the first select pass, and the keys of the
// threshold bin listed for the exact passes (more than kCandCap keys in one
// bin, as with many equal scores, take the radix passes over the whole row).
constexpr int kBins = 2 * kEvictThreads;
constexpr int kCandCap = 8192;
// Move: 256 threads (8 warps) per block, 32 moves per warp, blocks laid out
// as (move chunk, row) so that every SM holds many rows' moves at once.
constexpr int kMoveThreads = 256;

// Top-B select of a row with several evictions, keys in shared memory, in
// five passes over the keys instead of the eight of the radix select: (1) the
// keys' minimum and maximum, taken while they are loaded (the caller's);
// (2) a histogram of kBins equal-width bins over [min, max], and the bin
// that holds the B-th largest key; (3) that bin's keys listed; the threshold
// key T and, among keys equal to T, the position cut P radix-selected over
// the list alone; (4, 5) the hole and mover lists. Exact: every key of a
// higher bin is larger than every key of the threshold bin, and keys equal
// to T all share its bin, so T, P and the lists are those of the radix
// select over the whole row.
template <class Sync>
__device__ void select_lists_binned(const Dev& p, int r, int n, int B, const uint32_t* skeys, uint32_t kmin,
                                    uint32_t kmax, int* hist, int* cand, int tid, const SelectScratch& s,
                                    Sync sync) {
  constexpr int NT = kEvictThreads;
  const int lane = tid % kWarp;
  const unsigned lt = (1u << lane) - 1u;
  const uint32_t span = kmax - kmin;
  const int bits = span ? 32 - __clz(span) : 0;
  const int shift = bits > 11 ? bits - 11 : 0;  // (key - kmin) >> shift < kBins
  auto bin = [&](int i) { return (skeys[i] - kmin) >> shift; };
  for (int b = tid; b < kBins; b += NT) hist[b] = 0;
  if (tid == 0) s.sh[2] = 0;
  sync();
  // pass 2: histogram; a warp whose keys share one bin (equal scores) adds once
#pragma unroll 4
  for (int i0 = 0; i0 < n; i0 += NT) {
    const int i = i0 + tid;
    const bool v = i < n;
    const uint32_t b = v ? bin(i) : 0u;
    const uint32_t b0 = __shfl_sync(0xffffffffu, b, 0);
    const unsigned vm = __ballot_sync(0xffffffffu, v);
    if (__all_sync(0xffffffffu, !v || b == b0)) {
      if (lane == 0 && vm) atomicAdd(&hist[b0], __popc(vm));
    } else if (v) {
      atomicAdd(&hist[b], 1);
    }
  }
  sync();
  // the threshold bin: thread t holds bins kBins-1-2t and kBins-2-2t, so that
  // an exclusive scan over the threads counts the keys of higher bins
  const int hi = kBins - 1 - 2 * tid, lo = hi - 1;
  const int chi = hist[hi], clo = hist[lo];
  int tot;
  const int before = team_exclusive_scan<NT>(chi + clo, tid, s.wsum, &tot, sync);
  if (before < B && B <= before + chi + clo) {
    s.sh[0] = before + chi >= B ? hi : lo;
    s.sh[1] = before + chi >= B ? before : before + chi;
  }
  sync();
  const uint32_t dsel = (uint32_t)s.sh[0];
  const int above = s.sh[1], m = hist[dsel];
  if (m > kCandCap) {
    team_select_compact_k<NT, true>(p, r, n, B, [&](int i) { return skeys[i]; }, tid, s, sync);
    return;
  }
  // pass 3: the threshold bin's keys, listed in any order
  for (int i0 = 0; i0 < n; i0 += NT) {
    const int i = i0 + tid;
    const bool f = i < n && bin(i) == dsel;
    const unsigned fm = __ballot_sync(0xffffffffu, f);
    if (fm) {
      int c0 = 0;
      if (lane == 0) c0 = atomicAdd(&s.sh[2], __popc(fm));
      c0 = __shfl_sync(0xffffffffu, c0, 0);
      if (f && DC_INB(p, c0 + __popc(fm & lt), m, 205)) cand[c0 + __popc(fm & lt)] = i;
    }
  }
  sync();
  auto ck = [&](int j) { return skeys[cand[j]]; };
  auto all = [](int) { return true; };
  int gtc = 0;
  const uint32_t T = team_radix_select_wide<NT>(m, B - above, ck, all, tid, s, &gtc, sync);
  const int need_eq = B - above - gtc;
  int eq_local = 0;
  for (int j = tid; j < m; j += NT) eq_local += ck(j) == T;
  int eq_total;
  (void)team_exclusive_scan<NT>(eq_local, tid, s.wsum, &eq_total, sync);
  const int* ps = p.pos + (size_t)r * p.stride;
  uint32_t P = 0;  // ties kept when ~pos >= P (the lowest positions)
  if (eq_total > need_eq) {
    int gt2 = 0;
    P = team_radix_select_wide<NT>(m, need_eq, [&](int j) { return ~(uint32_t)ps[cand[j]]; },
                                   [&](int j) { return ck(j) == T; }, tid, s, &gt2, sync);
  }
  auto keep = [&](int i) {
    const uint32_t k = skeys[i];
    return k > T || (k == T && ~(uint32_t)ps[i] >= P);
  };
  team_move_lists<NT>(p, r, n, B, keep, tid, s, sync);
}

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
  __shared__ int bins[kBins];
  __shared__ int cand[kCandCap];
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
      // issued before their keys are stored; the keys' range on the way
      uint32_t kmin = 0xFFFFFFFFu, kmax = 0u;
      auto put = [&](float x) {
        const uint32_t k = score_key(x);
        kmin = k < kmin ? k : kmin;
        kmax = k > kmax ? k : kmax;
        return k;
      };
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
            *reinterpret_cast<uint4*>(skeys + 4 * e) = make_uint4(put(v[u].x), put(v[u].y), put(v[u].z), put(v[u].w));
        }
      }
      for (int i = 4 * n4 + tid; i < nr; i += kEvictThreads) skeys[i] = put(score[i]);
      kmin = __reduce_min_sync(0xffffffffu, kmin);
      kmax = __reduce_max_sync(0xffffffffu, kmax);
      if (tid % kWarp == 0) best[tid / kWarp] = ((unsigned long long)kmax << 32) | kmin;
      sync();
      for (int w = 0; w < kEvictThreads / kWarp; ++w) {
        const unsigned long long x = best[w];
        const uint32_t wmin = (uint32_t)(x & 0xFFFFFFFFull), wmax = (uint32_t)(x >> 32);
        kmin = wmin < kmin ? wmin : kmin;
        kmax = wmax > kmax ? wmax : kmax;
      }
      sync();
      if (nr > keep + 1)
        select_lists_binned(p, r, nr, keep, skeys, kmin, kmax, bins, cand, tid, scr, sync);
      else
        team_select_compact_k<kEvictThreads, true>(p, r, nr, keep, [&](int i) { return skeys[i]; }, tid, scr,
                                                   sync);
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
