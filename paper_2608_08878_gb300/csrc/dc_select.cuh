// dc_select.cuh -- argtop_B and prune of one row (Algorithm 1), run by a team
// of NT threads of one CTA (the whole CTA in the evict kernel, the epilogue
// warps in the fused kernel).
//
// Ranking: score descending, then position ascending (Sec. 3.1.2: inference
// keeps the top-B tokens deterministically). Scores become order-preserving
// 32-bit keys (score_key). One eviction (n == B + 1, the steady state) is an
// argmin over (score key, -position). Otherwise four 8-bit
// MSB-first histogram passes find the threshold key T with
// #(key > T) < B <= #(key >= T); when keys equal to T outnumber the places
// left, a second select over their positions keeps the lowest ones.
//
// Compaction: slots [0, B) end up holding the survivors. Evicted slots below B
// are holes, survivors at slots >= B are movers, and #holes == #movers; the
// k-th mover (ascending slot) moves into the k-th hole (ascending slot) with
// its key, value, position and window state. Survivors below B stay put.
#pragma once

#include "dc_common.cuh"

namespace dc {

struct SelectScratch {
  int* hist;   // [256]
  int* sh;     // [4]
  int* wsum;   // [NT / 32]
  unsigned long long* best;  // [NT / 32] argmin keys
  int* best_slot;            // [NT / 32]
};

// Exclusive prefix sum over the team of one int per thread; returns the
// prefix and writes the team total to *total (all threads).
template <int NT, class Sync>
__device__ __forceinline__ int team_exclusive_scan(int v, int tid, int* wsum, int* total, Sync sync) {
  constexpr int NW = NT / kWarp;
  const int lane = tid % kWarp, wid = tid / kWarp;
  int x = v;
#pragma unroll
  for (int off = 1; off < kWarp; off <<= 1) {
    int y = __shfl_up_sync(0xffffffffu, x, off);
    if (lane >= off) x += y;
  }
  if (lane == kWarp - 1) wsum[wid] = x;
  sync();
  if (wid == 0) {
    int s = lane < NW ? wsum[lane] : 0;
#pragma unroll
    for (int off = 1; off < kWarp; off <<= 1) {
      int y = __shfl_up_sync(0xffffffffu, s, off);
      if (lane >= off) s += y;
    }
    if (lane < NW) wsum[lane] = s;
  }
  sync();
  const int before = (wid > 0 ? wsum[wid - 1] : 0) + x - v;
  *total = wsum[NW - 1];
  sync();
  return before;
}

// MSB-first radix select over keyf(i), i in [0, n) with pred(i): the key of
// the need-th largest element; *gt gets the count of larger keys.
template <int NT, class KeyF, class Pred, class Sync>
__device__ uint32_t team_radix_select(int n, int need, KeyF keyf, Pred pred, int tid,
                                      const SelectScratch& s, int* gt, Sync sync) {
  uint32_t prefix = 0, mask = 0;
  int above = 0;
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int b = tid; b < 256; b += NT) s.hist[b] = 0;
    sync();
    for (int i = tid; i < n; i += NT) {
      if (!pred(i)) continue;
      const uint32_t k = keyf(i);
      if ((k & mask) == prefix) atomicAdd(&s.hist[(k >> shift) & 255u], 1);
    }
    sync();
    if (tid == 0) {
      int cum = 0, dgt = 0;
      for (int b = 255; b >= 0; --b) {
        if (above + cum + s.hist[b] >= need) { dgt = b; break; }
        cum += s.hist[b];
      }
      s.sh[0] = dgt;
      s.sh[1] = above + cum;
    }
    sync();
    prefix |= (uint32_t)s.sh[0] << shift;
    mask |= 255u << shift;
    above = s.sh[1];
    sync();
  }
  *gt = above;
  return prefix;
}

// Copies slot `src` of a row to slot `dst` (K, V, position, window state and
// the per-token extras), using `nl` cooperating lanes starting at lane `l`.
__device__ __forceinline__ void move_slot(const Dev& p, size_t src, size_t dst, int l, int nl) {
  const int VPR = p.d / 8;
  const uint4* ks = reinterpret_cast<const uint4*>(p.K) + src * VPR;
  const uint4* vs = reinterpret_cast<const uint4*>(p.V) + src * VPR;
  uint4* kd = reinterpret_cast<uint4*>(p.K) + dst * VPR;
  uint4* vd = reinterpret_cast<uint4*>(p.V) + dst * VPR;
  for (int e = l; e < 2 * VPR; e += nl) {
    if (e < VPR) kd[e] = ks[e];
    else vd[e - VPR] = vs[e - VPR];
  }
  if (l == 0) {
    p.pos[dst] = p.pos[src];
    p.vnorm[dst] = p.vnorm[src];
    p.SZ[dst] = p.SZ[src];
    p.score[dst] = p.score[src];
    if (p.acc) p.acc[dst] = p.acc[src];
    if (p.keep_features)
      for (int e = 0; e < 5; ++e) p.feat[dst * 5 + e] = p.feat[src * 5 + e];
  }
}

// Keeps the top B of the row's n tokens (scores from `score`, length n) and
// compacts them into slots [0, B). Requires 1 <= B < n. All NT threads of the
// team call it.
template <int NT, class Sync>
__device__ void team_select_compact(const Dev& p, int r, int n, int B, const float* score, int tid,
                                    const SelectScratch& s, Sync sync) {
  const size_t base = (size_t)r * p.stride;
  const int* ps = p.pos + base;
  auto key = [&](int i) { return score_key(score[i]); };
  if (n == B + 1) {
    // One eviction: the lowest-ranked token (smallest score key; among equal
    // keys the highest position). Positions are read only to break ties.
    uint32_t bk = 0xFFFFFFFFu;
    int bs = -1;
    for (int i = tid; i < n; i += NT) {
      const uint32_t k = key(i);
      if (k < bk || (k == bk && bs >= 0 && ps[i] > ps[bs])) { bk = k; bs = i; }
    }
    auto better = [&](uint32_t ka, int sa, uint32_t kb, int sb) {  // (kb, sb) ranks lower?
      if (sb < 0) return false;
      if (sa < 0) return true;
      return kb < ka || (kb == ka && ps[sb] > ps[sa]);
    };
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const uint32_t ok = __shfl_xor_sync(0xffffffffu, bk, off);
      const int os = __shfl_xor_sync(0xffffffffu, bs, off);
      if (better(bk, bs, ok, os)) { bk = ok; bs = os; }
    }
    const int lane = tid % kWarp, wid = tid / kWarp;
    if (lane == 0) { s.best[wid] = bk; s.best_slot[wid] = bs; }
    sync();
    uint32_t fk = (uint32_t)s.best[0];
    int e = s.best_slot[0];
    for (int w = 1; w < NT / kWarp; ++w)
      if (better(fk, e, (uint32_t)s.best[w], s.best_slot[w])) { fk = (uint32_t)s.best[w]; e = s.best_slot[w]; }
    // slot B (the last) is the only candidate mover; it fills the hole at e
    if (e >= 0 && e < B && tid < kWarp) move_slot(p, base + B, base + e, tid, kWarp);
    sync();
    return;
  }
  int gt = 0;
  auto all = [](int) { return true; };
  const uint32_t T = team_radix_select<NT>(n, B, key, all, tid, s, &gt, sync);
  const int need_eq = B - gt;
  int eq_local = 0;
  for (int i = tid; i < n; i += NT) eq_local += (key(i) == T);
  int eq_total;
  (void)team_exclusive_scan<NT>(eq_local, tid, s.wsum, &eq_total, sync);
  uint32_t P = 0;  // ties kept when ~pos >= P (the lowest positions)
  if (eq_total > need_eq) {
    auto pkey = [&](int i) { return ~(uint32_t)ps[i]; };
    auto tied = [&](int i) { return key(i) == T; };
    int gt2 = 0;
    P = team_radix_select<NT>(n, need_eq, pkey, tied, tid, s, &gt2, sync);
  }
  auto keep = [&](int i) {
    const uint32_t k = key(i);
    return k > T || (k == T && ~(uint32_t)ps[i] >= P);
  };
  int* holes = p.holes + base;
  int nh = 0;
  for (int c0 = 0; c0 < B; c0 += NT) {
    const int i = c0 + tid;
    const int f = (i < B && !keep(i)) ? 1 : 0;
    int tot;
    const int rank = team_exclusive_scan<NT>(f, tid, s.wsum, &tot, sync);
    if (f) holes[nh + rank] = i;
    nh += tot;
  }
  sync();
  int nm = 0;
  for (int c0 = B; c0 < n; c0 += NT) {
    const int i = c0 + tid;
    const int f = (i < n && keep(i)) ? 1 : 0;
    int tot;
    const int rank = team_exclusive_scan<NT>(f, tid, s.wsum, &tot, sync);
    if (f && nm + rank < nh) move_slot(p, base + i, base + holes[nm + rank], 0, 1);
    nm += tot;
  }
  if (tid == 0 && nm != nh) atomicOr(p.status, kStatusBadShape);
  sync();
}

}  // namespace dc
