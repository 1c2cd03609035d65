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

// team_radix_select for large teams over keys in shared memory (the eviction
// kernel): the lanes of a warp that share a histogram bin add to it once, and
// one warp finds the digit with a prefix sum over its lanes instead of one
// thread walking the 256 bins. Needs whole warps (every lane of every team
// warp calls it) and 1 <= need <= the number of elements with pred. (The
// fused kernel keeps the plain form: this one needs more registers.)
template <int NT, class KeyF, class Pred, class Sync>
__device__ uint32_t team_radix_select_wide(int n, int need, KeyF keyf, Pred pred, int tid,
                                      const SelectScratch& s, int* gt, Sync sync) {
  uint32_t prefix = 0, mask = 0;
  int above = 0;
  const int lane = tid % kWarp;
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int b = tid; b < 256; b += NT) s.hist[b] = 0;
    sync();
    // histogram of the next digit among the keys that match the prefix; the
    // lanes of a warp that share a bin add to it once (scores cluster in a
    // few bins, where one atomic per lane would serialise)
    for (int i0 = 0; i0 < n; i0 += NT) {
      const int i = i0 + tid;
      unsigned bin = 256u;
      if (i < n && pred(i)) {
        const uint32_t k = keyf(i);
        if ((k & mask) == prefix) bin = (k >> shift) & 255u;
      }
      const unsigned peers = __match_any_sync(0xffffffffu, bin);
      if (bin < 256u && lane == __ffs(peers) - 1) atomicAdd(&s.hist[bin], __popc(peers));
    }
    sync();
    if (tid < kWarp) {
      // the digit: the highest bin where the count of larger-or-equal keys
      // reaches `need`. Lane L holds bins 255 - 8L - j (j = 0..7, descending);
      // a prefix sum over the lanes finds the lane, the lane finds the bin.
      int c[8], tot = 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        c[j] = s.hist[255 - 8 * lane - j];
        tot += c[j];
      }
      int inc = tot;
#pragma unroll
      for (int off = 1; off < kWarp; off <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, inc, off);
        if (lane >= off) inc += y;
      }
      const unsigned hit = __ballot_sync(0xffffffffu, above + inc >= need);
      const int all = __shfl_sync(0xffffffffu, inc, kWarp - 1);
      if (hit == 0u) {
        if (lane == 0) {  // fewer keys than `need` (not reached for valid arguments)
          s.sh[0] = 0;
          s.sh[1] = above + all;
        }
      } else if (lane == __ffs(hit) - 1) {
        int cum = above + inc - tot, dgt = 255 - 8 * lane - 7;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if (cum + c[j] >= need) {
            dgt = 255 - 8 * lane - j;
            break;
          }
          cum += c[j];
        }
        s.sh[0] = dgt;
        s.sh[1] = cum;
      }
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

// One slot's contents held by a warp: lane l keeps 16-byte chunk l of the
// slot's [K | V] row (d / 4 chunks) and per-token field l: 0 position, 1 |v|,
// 2 window sums, 3 score, 4 cumulative alpha, 5..9 features. Every lane loads
// before any stores, so a move costs one memory round trip.
struct SlotCopy {
  uint4 kv;
  uint4 f;
};

__device__ __forceinline__ SlotCopy slot_load(const Dev& p, size_t src, int lane) {
  SlotCopy c{};
  const int VPR = p.d / 8;
  if (lane < VPR) c.kv = reinterpret_cast<const uint4*>(p.K)[src * VPR + lane];
  else if (lane < 2 * VPR) c.kv = reinterpret_cast<const uint4*>(p.V)[src * VPR + lane - VPR];
  if (lane == 0) c.f.x = (unsigned)p.pos[src];
  else if (lane == 1) c.f.x = __float_as_uint(p.vnorm[src]);
  else if (lane == 2) c.f = *reinterpret_cast<const uint4*>(p.SZ + src);
  else if (lane == 3) c.f.x = __float_as_uint(p.score[src]);
  else if (lane == 4 && p.acc) c.f.x = __float_as_uint(p.acc[src]);
  else if (lane >= 5 && lane < 10 && p.keep_features) c.f.x = __float_as_uint(p.feat[src * 5 + lane - 5]);
  return c;
}

// slot_load in two parts, for a caller that loads a slot early, while the
// slot's score, cumulative alpha and features may still be written:
// slot_load_settled takes K, V, position, |v|, window sums (and the score when
// `score_late` is false); slot_load_late takes the rest.
__device__ __forceinline__ void slot_load_settled(const Dev& p, size_t src, int lane, bool score_late, SlotCopy& c) {
  const int VPR = p.d / 8;
  if (lane < VPR) c.kv = reinterpret_cast<const uint4*>(p.K)[src * VPR + lane];
  else if (lane < 2 * VPR) c.kv = reinterpret_cast<const uint4*>(p.V)[src * VPR + lane - VPR];
  if (lane == 0) c.f.x = (unsigned)p.pos[src];
  else if (lane == 1) c.f.x = __float_as_uint(p.vnorm[src]);
  else if (lane == 2) c.f = *reinterpret_cast<const uint4*>(p.SZ + src);
  else if (lane == 3 && !score_late) c.f.x = __float_as_uint(p.score[src]);
}

__device__ __forceinline__ void slot_load_late(const Dev& p, size_t src, int lane, bool score_late, SlotCopy& c) {
  if (lane == 3 && score_late) c.f.x = __float_as_uint(p.score[src]);
  else if (lane == 4 && p.acc) c.f.x = __float_as_uint(p.acc[src]);
  else if (lane >= 5 && lane < 10 && p.keep_features) c.f.x = __float_as_uint(p.feat[src * 5 + lane - 5]);
}

__device__ __forceinline__ void slot_store(const Dev& p, size_t dst, int lane, const SlotCopy& c) {
  const int VPR = p.d / 8;
  if (lane < VPR) reinterpret_cast<uint4*>(p.K)[dst * VPR + lane] = c.kv;
  else if (lane < 2 * VPR) reinterpret_cast<uint4*>(p.V)[dst * VPR + lane - VPR] = c.kv;
  if (lane == 0) p.pos[dst] = (int)c.f.x;
  else if (lane == 1) p.vnorm[dst] = __uint_as_float(c.f.x);
  else if (lane == 2) *reinterpret_cast<uint4*>(p.SZ + dst) = c.f;
  else if (lane == 3) p.score[dst] = __uint_as_float(c.f.x);
  else if (lane == 4 && p.acc) p.acc[dst] = __uint_as_float(c.f.x);
  else if (lane >= 5 && lane < 10 && p.keep_features) p.feat[dst * 5 + lane - 5] = __uint_as_float(c.f.x);
}

// Copies slot `src` of a row to slot `dst` with one thread (loads first).
__device__ __forceinline__ void move_slot_1(const Dev& p, size_t src, size_t dst) {
  const int VPR = p.d / 8;
  const int ps = p.pos[src];
  const float vn = p.vnorm[src];
  const float4 sz = p.SZ[src];
  const float scr = p.score[src];
  const float ac = p.acc ? p.acc[src] : 0.f;
  const uint4* ks = reinterpret_cast<const uint4*>(p.K) + src * VPR;
  const uint4* vs = reinterpret_cast<const uint4*>(p.V) + src * VPR;
  uint4* kd = reinterpret_cast<uint4*>(p.K) + dst * VPR;
  uint4* vd = reinterpret_cast<uint4*>(p.V) + dst * VPR;
  for (int e = 0; e < VPR; e += 4) {
    const uint4 k0 = ks[e], k1 = ks[e + 1], k2 = ks[e + 2], k3 = ks[e + 3];
    const uint4 v0 = vs[e], v1 = vs[e + 1], v2 = vs[e + 2], v3 = vs[e + 3];
    kd[e] = k0; kd[e + 1] = k1; kd[e + 2] = k2; kd[e + 3] = k3;
    vd[e] = v0; vd[e + 1] = v1; vd[e + 2] = v2; vd[e + 3] = v3;
  }
  p.pos[dst] = ps;
  p.vnorm[dst] = vn;
  p.SZ[dst] = sz;
  p.score[dst] = scr;
  if (p.acc) p.acc[dst] = ac;
  if (p.keep_features)
    for (int e = 0; e < 5; ++e) p.feat[dst * 5 + e] = p.feat[src * 5 + e];
}

// K/V rows a warp of the list-based compaction loads before it stores them.
constexpr int kMoveUnroll = 8;

// One warp moves entries [k0, min(k0 + 32, nmv)) of a row's move lists: the
// k-th mover (slot movers[k] >= B) fills the k-th hole (slot holes[k] < B).
// Sources are at or above B and destinations below it, so all moves of a row
// are independent. Lane l copies the per-token fields of move k0 + l (uniform
// code, one slot per lane); then the warp copies the K and V rows, each lane
// one 16-byte chunk, kMoveUnroll rows' loads in flight before their stores.
__device__ __forceinline__ void warp_move_batch(const Dev& p, size_t base, const int* holes, const int* movers,
                                                int k0, int nmv, int lane) {
  const int VPR = p.d / 8;                 // 16-byte chunks per K (or V) row
  const int rows_per = kWarp / (2 * VPR);  // slots copied per warp instruction
  const int sub = lane / (2 * VPR), chunk = lane % (2 * VPR);
  const int k = k0 + lane;
  const bool live = k < nmv;
  int src = live ? movers[k] : 0, dst = live ? holes[k] : 0;
  if (live && !(DC_INB(p, src, p.stride, 203) && DC_INB(p, dst, p.stride, 204))) src = dst = -1;
  if (live && src >= 0) {
    const size_t fs = base + src, fd = base + dst;
    const int ps_ = p.pos[fs];
    const float vn = p.vnorm[fs];
    const float4 sz = p.SZ[fs];
    const float sc = p.score[fs];
    const float ac = p.acc ? p.acc[fs] : 0.f;
    p.pos[fd] = ps_;
    p.vnorm[fd] = vn;
    p.SZ[fd] = sz;
    p.score[fd] = sc;
    if (p.acc) p.acc[fd] = ac;
    if (p.keep_features)
      for (int e = 0; e < 5; ++e) p.feat[fd * 5 + e] = p.feat[fs * 5 + e];
  }
  const int cnt = nmv - k0 < kWarp ? nmv - k0 : kWarp;
  const uint4* gk = reinterpret_cast<const uint4*>(chunk < VPR ? p.K : p.V);
  uint4* gkw = reinterpret_cast<uint4*>(chunk < VPR ? p.K : p.V);
  const int c = chunk < VPR ? chunk : chunk - VPR;
  for (int j0 = 0; j0 < cnt; j0 += kMoveUnroll * rows_per) {
    uint4 v[kMoveUnroll];
    int d_[kMoveUnroll];
#pragma unroll
    for (int u = 0; u < kMoveUnroll; ++u) {
      const int j = j0 + u * rows_per + sub;
      const int sj = __shfl_sync(0xffffffffu, src, j & (kWarp - 1));
      d_[u] = __shfl_sync(0xffffffffu, dst, j & (kWarp - 1));
      if (j >= cnt || sj < 0) d_[u] = -1;
      if (d_[u] >= 0) v[u] = gk[(base + sj) * VPR + c];
    }
#pragma unroll
    for (int u = 0; u < kMoveUnroll; ++u)
      if (d_[u] >= 0) gkw[(base + d_[u]) * VPR + c] = v[u];
  }
}

// Hole and mover lists of a row in ascending slot order, for keep(i) = "slot
// i survives": holes (evicted slots below B) in p.holes[row][0, nh), movers
// (survivors at or above B) in p.holes[row][nh, nh + nm) (the row's scratch
// has n >= nh + nm entries), the counts in p.nmoves[row]. Each warp takes a
// contiguous run of 32-slot groups: it counts its flags with ballots, the
// warps' counts are prefix-summed once, and a second walk writes the indices.
// The moves themselves are evict_move_kernel's (warp_move_batch).
template <int NT, class Keep, class Sync>
__device__ void team_move_lists(const Dev& p, int r, int n, int B, Keep keep, int tid, const SelectScratch& s,
                                Sync sync) {
  const size_t base = (size_t)r * p.stride;
  int* holes = p.holes + base;
  constexpr int NW = NT / kWarp;
  const int lane = tid % kWarp, wid = tid / kWarp;
  const int ng = (n + kWarp - 1) / kWarp;
  const int g0 = (int)((long long)ng * wid / NW), g1 = (int)((long long)ng * (wid + 1) / NW);
  int ch = 0, cm = 0;
  for (int gi = g0; gi < g1; ++gi) {
    const int i = gi * kWarp + lane;
    const bool kp = i < n && keep(i);
    ch += __popc(__ballot_sync(0xffffffffu, i < B && !kp));
    cm += __popc(__ballot_sync(0xffffffffu, i >= B && kp));
  }
  if (lane == 0) s.best[wid] = ((unsigned long long)(unsigned)cm << 32) | (unsigned)ch;
  sync();
  int hb = 0, mb = 0, nh = 0, nm = 0;
  for (int w = 0; w < NW; ++w) {
    const unsigned long long v = s.best[w];
    const int vh = (int)(unsigned)(v & 0xFFFFFFFFull), vm = (int)(unsigned)(v >> 32);
    if (w < wid) {
      hb += vh;
      mb += vm;
    }
    nh += vh;
    nm += vm;
  }
  int* movers = holes + nh;
  const unsigned lt = (1u << lane) - 1u;
  for (int gi = g0; gi < g1; ++gi) {
    const int i = gi * kWarp + lane;
    const bool kp = i < n && keep(i);
    const bool fh = i < B && !kp, fm = i >= B && kp;
    const unsigned bh = __ballot_sync(0xffffffffu, fh), bm = __ballot_sync(0xffffffffu, fm);
    if (fh && DC_INB(p, hb + __popc(bh & lt), B, 201)) holes[hb + __popc(bh & lt)] = i;
    if (fm && DC_INB(p, nh + mb + __popc(bm & lt), p.stride, 202)) movers[mb + __popc(bm & lt)] = i;
    hb += __popc(bh);
    mb += __popc(bm);
  }
  if (tid == 0 && nm != nh) atomicOr(p.status, kStatusBadShape);
  sync();
  if (tid == 0) {
    p.nmoves[2 * (size_t)r] = nm < nh ? nm : nh;
    p.nmoves[2 * (size_t)r + 1] = nh;
  }
  sync();
}

// Keeps the top B of the row's n tokens (order keys keyf(i), i < n) and
// compacts them into slots [0, B). Requires 1 <= B < n. All NT threads of the
// team call it. Two compactions: WARP_MOVES (the eviction kernel, many moves):
// team_move_lists, the moves left to a kernel of their own
// (evict_move_kernel); otherwise (the fused kernel's epilogue, where
// registers are scarce) chunks of NT candidate slots are ranked with a team
// scan and each mover thread copies its slot.
template <int NT, bool WARP_MOVES, class KeyF, class Sync>
__device__ void team_select_compact_k(const Dev& p, int r, int n, int B, KeyF key, int tid,
                                      const SelectScratch& s, Sync sync) {
  const size_t base = (size_t)r * p.stride;
  const int* ps = p.pos + base;
  if (n == B + 1) {
    // One eviction: the lowest-ranked token (smallest score key; among equal
    // keys the highest position). Positions are read only to break ties.
    // Slot B (the last) is the only candidate mover: load it meanwhile.
    SlotCopy mv{};
    if (tid < kWarp) mv = slot_load(p, base + B, tid);
    uint32_t bk = 0xFFFFFFFFu;
    int bs = -1;
    for (int i = tid; i < n; i += NT) {
      const uint32_t k = key(i);
      if (bs < 0 || k < bk || (k == bk && ps[i] > ps[bs])) { bk = k; bs = i; }
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
    // slot B fills the hole at e
    if (e >= 0 && e < B && tid < kWarp) slot_store(p, base + e, tid, mv);
    sync();
    return;
  }
  int gt = 0;
  auto all = [](int) { return true; };
  auto radix = [&](int nn, int need, auto kf, auto pr, int* g) {
    if constexpr (WARP_MOVES) return team_radix_select_wide<NT>(nn, need, kf, pr, tid, s, g, sync);
    else return team_radix_select<NT>(nn, need, kf, pr, tid, s, g, sync);
  };
  const uint32_t T = radix(n, B, key, all, &gt);
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
    P = radix(n, need_eq, pkey, tied, &gt2);
  }
  auto keep = [&](int i) {
    const uint32_t k = key(i);
    return k > T || (k == T && ~(uint32_t)ps[i] >= P);
  };
  if constexpr (!WARP_MOVES) {
    int* holes = p.holes + base;
    int nh = 0;
    for (int c0 = 0; c0 < B; c0 += NT) {
      const int i = c0 + tid;
      const int f = (i < B && !keep(i)) ? 1 : 0;
      int tot;
      const int rank = team_exclusive_scan<NT>(f, tid, s.wsum, &tot, sync);
      if (f && DC_INB(p, nh + rank, B, 201)) holes[nh + rank] = i;
      nh += tot;
    }
    sync();
    int nm = 0;
    for (int c0 = B; c0 < n; c0 += NT) {
      const int i = c0 + tid;
      const int f = (i < n && keep(i)) ? 1 : 0;
      int tot;
      const int rank = team_exclusive_scan<NT>(f, tid, s.wsum, &tot, sync);
      if (f && nm + rank < nh && DC_INB(p, holes[nm + rank], B, 204)) move_slot_1(p, base + i, base + holes[nm + rank]);
      nm += tot;
    }
    if (tid == 0 && nm != nh) atomicOr(p.status, kStatusBadShape);
    sync();
  } else {
    team_move_lists<NT>(p, r, n, B, keep, tid, s, sync);
  }
}

// team_select_compact_k over a score array (shared or global memory), with
// the per-thread compaction.
template <int NT, class Sync>
__device__ void team_select_compact(const Dev& p, int r, int n, int B, const float* score, int tid,
                                    const SelectScratch& s, Sync sync) {
  team_select_compact_k<NT, false>(p, r, n, B, [&](int i) { return score_key(score[i]); }, tid, s, sync);
}

// The same selection as team_select_compact without moving anything: writes
// the compaction's (hole, mover) pairs to moves[1 + 2k], moves[2 + 2k] and
// their count to moves[0] (for sequences whose rows all move alike). `holes`
// is scratch of n ints. Requires 1 <= B; B >= n gives no moves.
template <int NT, class Sync>
__device__ void team_select_moves(const float* score, const int* ps, int n, int B, int* holes, int* moves,
                                  int tid, const SelectScratch& s, Sync sync) {
  if (B >= n) {
    if (tid == 0) moves[0] = 0;
    sync();
    return;
  }
  auto key = [&](int i) { return score_key(score[i]); };
  if (n == B + 1) {
    uint32_t bk = 0xFFFFFFFFu;
    int bs = -1;
    for (int i = tid; i < n; i += NT) {
      const uint32_t k = key(i);
      if (bs < 0 || k < bk || (k == bk && ps[i] > ps[bs])) { bk = k; bs = i; }
    }
    auto better = [&](uint32_t ka, int sa, uint32_t kb, int sb) {
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
    if (tid == 0) {
      uint32_t fk = (uint32_t)s.best[0];
      int e = s.best_slot[0];
      for (int w = 1; w < NT / kWarp; ++w)
        if (better(fk, e, (uint32_t)s.best[w], s.best_slot[w])) { fk = (uint32_t)s.best[w]; e = s.best_slot[w]; }
      if (e >= 0 && e < B) {
        moves[0] = 1;
        moves[1] = e;
        moves[2] = B;
      } else {
        moves[0] = 0;
      }
    }
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
  uint32_t P = 0;
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
    if (f && nm + rank < nh) {
      moves[1 + 2 * (nm + rank)] = holes[nm + rank];
      moves[2 + 2 * (nm + rank)] = i;
    }
    nm += tot;
  }
  if (tid == 0) moves[0] = nm < nh ? nm : nh;
  sync();
}

}  // namespace dc
