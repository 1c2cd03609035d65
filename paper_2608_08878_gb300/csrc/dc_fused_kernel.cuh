// dc_fused_kernel.cuh -- the fused kernel template and its launcher, shared by
// the translation units that instantiate its variants (dc_fused.cu: per-row
// selection with the policy; dc_fused_modes.cu: heuristic scorers and per-row
// budgets; dc_fused_glob.cu: global token mode and the full-cache comparator),
// so that they compile in parallel. Everything here has internal linkage.
#pragma once
// The fused engine: one persistent kernel streams every row's
// keys and values from HBM exactly once per decode step and does the whole
// step of Algorithm 1 for that row: attention (with the exact row softmax
// statistics), the five token features of Sec. 3.1.1, the policy MLP of
// Sec. 3.1.2 / App. D, and (dc_step) the top-B select and compaction.
//
// One CTA per SM (or per row, or two per row: rows of 12 tiles or more are
// split in halves when there are at most half as many rows as SMs); the CTAs
// take rows, half rows (also for a partly filled last wave) or, on short rows,
// row pairs (PAIR) from a shared queue as they become free. A row's ragged
// last tile is loaded in boxes of 16 tokens.
// Warp roles (352 threads):
//   warp 0     producer: takes the next row, writes its query tile (current,
//              previous and departing queries) and streams K then V tiles of
//              128 tokens with TMA (128-byte swizzle) through a 4-stage ring,
//              K tiles with their tokens' positions and window sums;
//   warp 1     MMA issuer (one lane): tcgen05.mma, accumulators in TMEM:
//                S  = K Q^T        [128 tokens x 16]  per K tile
//                O^T += V^T P^T    [d x 16]           per V tile (P = weights,
//                                  bf16 high and low parts in separate columns)
//   warp 10    policy-layer MMA issuer (one lane):
//                Z  = A W^T        [128 tokens x 128] per V tile
//   warps 2-9  epilogue: two warpgroups; warpgroup w takes the tiles whose
//              global index is w mod 2, one token (TMEM lane) per thread:
//                K pass: online softmax statistics, window-sum update (the
//                previous step's query in, the departing one out, both
//                recomputed from the same S tile), raw logits kept for the
//                V pass (heads 0..G-2 in TMEM, head G-1 in shared memory);
//                V pass: weights with the final statistics, features, the
//                policy's input row, score; then the output and the select.
//
// TMEM columns: S tiles [0, 32), O [32, 48), policy layer of warpgroup w
// [128 + 128 w, 256 + 128 w), logit stash [48, 128) and [384, 512).
//
// Per-token state rides along with the K tiles: TMA bulk copies bring the
// positions and window sums. The K pass writes the updated window sums back;
// the V pass re-reads them, with the positions and |v| (L2-resident), in loads
// issued two tiles ahead of use.
//
// Barrier phases: a parity wait is only sound when the waiting thread cannot
// be two phases ahead of the barrier. Every barrier here has one waiter that
// waits its phases in order (the producer, the MMA issuer, one warpgroup), or,
// for the K pass's stage reads, waits after a signal that implies the phase:
// the tile's S, committed by the MMA issuer after its own in-order wait. The
// stages alternate between the warpgroups, so the V pass does not wait on
// them at all.
#include <cuda.h>

#include "dc_common.cuh"
#include "dc_fused.h"
#include "dc_kernels.h"
#include "dc_select.cuh"
#include "dc_sm100.cuh"

namespace dc {
using namespace sm100;

namespace {

constexpr int kStages = 4;
// stage: K or V tile (32 KB, two 64-dim column blocks, 1024-byte aligned);
// K tiles also bring the tile's positions (512 B) and window sums (2 KB) into
// the stage's slot of the per-token area
constexpr int kStageBytes = 32768;
constexpr int kAuxBytes = 2560;
constexpr int kAuxPos = 0;                    // int32 [128] (K tiles)
constexpr int kAuxSZ = 512;                   // fp32x4 [128] (K tiles)
constexpr int kTok = 128;
constexpr int kThreads = 352;
constexpr int kEpi = 256;                     // two warpgroups
constexpr uint32_t kTmemCols = 512;
constexpr int kColS = 0, kColM = 128;
constexpr int kStashAEnd = 128, kStashB = 384, kStashBEnd = 512;

// The query tile holds the current, previous-step and departing queries (3G
// rows) padded to the QK MMA's N: 16 rows, or 32 for eight query heads per KV
// head. The S tiles (two buffers of N columns) come first in TMEM, then O (16
// columns), then the first logit stash area.
template <int G>
constexpr int q_rows() {
  return G == 8 ? 32 : 16;
}
template <int G>
constexpr int col_o() {
  return kColS + 2 * q_rows<G>();
}
template <int G>
constexpr int stash_a() {
  return col_o<G>() + 16;
}
// Tokens whose head-(G-1) logits, then scores, the fused kernel keeps in
// shared memory (a G = 8 row's larger query tiles take 8 KB of it).
template <int G>
constexpr int max_tok() {
  return G == 8 ? 8192 : kFusedMaxTok;
}

// Row pairs (PAIR): an item is two rows of at most kPairTiles tiles, one per
// warpgroup; their K and V tiles alternate in the stage ring.
constexpr int kPairTiles = 21;
constexpr int kPairTok = kPairTiles * kTok;
constexpr int kColOB = 48;                                 // the second row's O (PAIR)
constexpr int kPairStashA = 64;                            // the first row's logit stash (PAIR)

// Shared memory layout; PAIR keeps four query tiles (two per item, double
// buffered) and a smaller logit/score array per row.
template <bool PAIR, int G>
struct Smem {
  static constexpr int QBYTES = q_rows<G>() * 256;         // one query tile: two 64-dim blocks
  static constexpr int STAGE = 0;
  static constexpr int Q = STAGE + kStages * kStageBytes;   // (2 or 4) query tiles
  static constexpr int P = Q + (PAIR ? 4 : 2) * QBYTES;     // 2 x 4 KB (one per warpgroup)
  static constexpr int A = P + 2 * 4096;                    // 2 x 8 KB (one per warpgroup)
  static constexpr int W = A + 2 * 8192;                    // 8 KB
  static constexpr int AUX = W + 8192;                      // kStages x 2560 B
  static constexpr int SC = AUX + kStages * kAuxBytes;      // head G-1 logits, then scores
  static constexpr int MISC = SC + (PAIR ? 2 * kPairTok : max_tok<G>()) * 4;
  static constexpr int BYTES = MISC + 4096 + 1024;          // misc area + alignment slack
  static_assert(BYTES <= 232448, "more shared memory than a CTA may have");
};
constexpr int MISC_BYTES = 4096;

// barrier indices in the misc area
enum {
  B_FULL = 0, B_EMPTY = kStages, B_QFULL = 2 * kStages, B_QEMPTY = B_QFULL + 2, B_SFULL = B_QFULL + 4,
  B_SEMPTY = B_QFULL + 6, B_PFULL = B_QFULL + 8, B_PEMPTY = B_QFULL + 10, B_MFULL = B_QFULL + 12,
  B_MEMPTY = B_QFULL + 14, B_AFULL = B_QFULL + 16, B_AEMPTY = B_QFULL + 18, B_OFULL = B_QFULL + 20,
  B_OEMPTY = B_QFULL + 21, B_DRAIN = B_QFULL + 22, B_DRAIN2 = B_QFULL + 23, B_COUNT = B_QFULL + 24
};

// Tiles whose logits stay on chip between the passes (heads 0..G-2 in TMEM,
// head G-1 in shared memory); later tiles of longer rows keep all G logits in
// the global scratch [R][stride][G] instead.
template <int G>
constexpr int onchip_tiles() {
  constexpr int GS = G - 1;
  constexpr int st = GS > 0 ? (kStashAEnd - stash_a<G>()) / GS + (kStashBEnd - kStashB) / GS : (1 << 20);
  return st < max_tok<G>() / kTok ? st : max_tok<G>() / kTok;
}

template <int G>
__device__ __forceinline__ void store_logits(float* dst, const float* v) {
  if constexpr (G == 8) {
    reinterpret_cast<float4*>(dst)[0] = make_float4(v[0], v[1], v[2], v[3]);
    reinterpret_cast<float4*>(dst)[1] = make_float4(v[4], v[5], v[6], v[7]);
  } else if constexpr (G == 4) *reinterpret_cast<float4*>(dst) = make_float4(v[0], v[1], v[2], v[3]);
  else if constexpr (G == 2) *reinterpret_cast<float2*>(dst) = make_float2(v[0], v[1]);
  else dst[0] = v[0];
}

template <int G>
__device__ __forceinline__ void load_logits(const float* src, float* v) {
  if constexpr (G == 8) {
    const float4 x = reinterpret_cast<const float4*>(src)[0], y = reinterpret_cast<const float4*>(src)[1];
    v[0] = x.x; v[1] = x.y; v[2] = x.z; v[3] = x.w;
    v[4] = y.x; v[5] = y.y; v[6] = y.z; v[7] = y.w;
  } else if constexpr (G == 4) {
    const float4 x = *reinterpret_cast<const float4*>(src);
    v[0] = x.x; v[1] = x.y; v[2] = x.z; v[3] = x.w;
  } else if constexpr (G == 2) {
    const float2 x = *reinterpret_cast<const float2*>(src);
    v[0] = x.x; v[1] = x.y;
  } else {
    v[0] = src[0];
  }
}

// TMEM column of the stashed logits of tile j (GS = G - 1 columns per tile).
template <int G>
__device__ __forceinline__ uint32_t stash_col(int j) {
  constexpr int GS = G - 1;
  constexpr int TA = GS > 0 ? (kStashAEnd - stash_a<G>()) / GS : 0;
  return j < TA ? (uint32_t)(stash_a<G>() + GS * j) : (uint32_t)(kStashB + GS * (j - TA));
}

// byte offset of 16-byte chunk `c` (0..7) of row `row` inside a 128-byte
// swizzled tile (8-row atoms of 1024 bytes)
__device__ __forceinline__ uint32_t sw128(int row, int c) {
  return (uint32_t)((row >> 3) * 1024 + (row & 7) * 128 + ((c ^ (row & 7)) << 4));
}

// byte offset of 16-byte chunk `c` (0..3) of row `row` inside a 64-byte
// swizzled tile (8-row atoms of 512 bytes)
__device__ __forceinline__ uint32_t sw64(int row, int c) {
  return (uint32_t)((row >> 3) * 512 + (row & 7) * 64 + ((c ^ ((row & 7) >> 1)) << 4));
}

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Stores / loads the first GS of the G logits of this thread's token.
template <int GS>
__device__ __forceinline__ void stash_store(uint32_t taddr, const float* v) {
  if constexpr (GS == 7) {
    asm volatile("tcgen05.st.sync.aligned.32x32b.x4.b32 [%0], {%1,%2,%3,%4};" ::"r"(taddr),
                 "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
                 "r"(__float_as_uint(v[3]))
                 : "memory");
    asm volatile("tcgen05.st.sync.aligned.32x32b.x2.b32 [%0], {%1,%2};" ::"r"(taddr + 4), "r"(__float_as_uint(v[4])),
                 "r"(__float_as_uint(v[5]))
                 : "memory");
    asm volatile("tcgen05.st.sync.aligned.32x32b.x1.b32 [%0], {%1};" ::"r"(taddr + 6), "r"(__float_as_uint(v[6]))
                 : "memory");
  } else if constexpr (GS == 3) {
    asm volatile("tcgen05.st.sync.aligned.32x32b.x2.b32 [%0], {%1,%2};" ::"r"(taddr), "r"(__float_as_uint(v[0])),
                 "r"(__float_as_uint(v[1]))
                 : "memory");
    asm volatile("tcgen05.st.sync.aligned.32x32b.x1.b32 [%0], {%1};" ::"r"(taddr + 2), "r"(__float_as_uint(v[2]))
                 : "memory");
  } else if constexpr (GS == 1) {
    asm volatile("tcgen05.st.sync.aligned.32x32b.x1.b32 [%0], {%1};" ::"r"(taddr), "r"(__float_as_uint(v[0]))
                 : "memory");
  }
}

template <int GS>
__device__ __forceinline__ void stash_load(uint32_t taddr, float* v) {
  if constexpr (GS == 7) {
    uint32_t a, b, c, d, e, f, g;
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x4.b32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(a), "=r"(b), "=r"(c), "=r"(d)
                 : "r"(taddr));
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x2.b32 {%0,%1}, [%2];" : "=r"(e), "=r"(f) : "r"(taddr + 4));
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];" : "=r"(g) : "r"(taddr + 6));
    v[0] = __uint_as_float(a);
    v[1] = __uint_as_float(b);
    v[2] = __uint_as_float(c);
    v[3] = __uint_as_float(d);
    v[4] = __uint_as_float(e);
    v[5] = __uint_as_float(f);
    v[6] = __uint_as_float(g);
  } else if constexpr (GS == 3) {
    uint32_t a, b, c;
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x2.b32 {%0,%1}, [%2];" : "=r"(a), "=r"(b) : "r"(taddr));
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];" : "=r"(c) : "r"(taddr + 2));
    v[0] = __uint_as_float(a);
    v[1] = __uint_as_float(b);
    v[2] = __uint_as_float(c);
  } else if constexpr (GS == 1) {
    uint32_t a;
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];" : "=r"(a) : "r"(taddr));
    v[0] = __uint_as_float(a);
  }
}

// Online softmax state of one head in log2 units (m = max raw logit,
// l = sum 2^x, u = sum 2^x x with x = (s - m) c), updated without branches.
// The state starts at m = kNoMax, a finite stand-in for -infinity: its first
// rescale factor underflows to 0.
constexpr float kNoMax = -1e30f;

__device__ __forceinline__ void online_add(float& m, float& l, float& u, float s, float c) {
  const float mn = fmaxf(m, s);
  const float dm = (m - mn) * c;
  const float f = ex2(dm);
  const float x = (s - mn) * c;
  const float pe = ex2(x);
  u = fmaf(pe, x, (u + l * dm) * f);
  l = fmaf(l, f, pe);
  m = mn;
}

__device__ __forceinline__ void online_merge(float& m, float& l, float& u, float mo, float lo, float uo, float c) {
  const float M = fmaxf(m, mo), da = (m - M) * c, db = (mo - M) * c;
  const float fa = ex2(da), fb = ex2(db);
  u = (u + l * da) * fa + (uo + lo * db) * fb;
  l = l * fa + lo * fb;
  m = M;
}

// Work items come from a queue shared by all CTAs (an atomic counter): the
// first R - half_rows rows whole, then both halves of each of the last
// half_rows rows (half 0: the first ceil(nT/2) tiles, half 1: the rest). A CTA
// that takes a half row takes nothing after it, so the halves of a row always
// go to two different CTAs, which then wait on each other (all CTAs are
// resident under a cooperative launch). Taking rows as CTAs become free keeps
// their finishing times together however their speeds drift.
struct Item {
  int row, t0, t1, half;  // row -1: no more work; half -1: the whole row
};

constexpr int kItemRing = 8;  // items published ahead of the slowest role (at most ~3)

template <bool PERROW, bool PAIR>
__device__ __forceinline__ Item take_item(const FusedStep& fs, const Dev& p, int nT) {
  const unsigned w = atomicAdd(fs.work + (fs.epoch & 1u), 1u);
  if constexpr (PAIR) return w < (unsigned)(p.R / 2) ? Item{(int)(2 * w), 0, nT, -1} : Item{-1, 0, 0, 0};
  const unsigned whole = (unsigned)(p.R - fs.half_rows);
  if (w < whole) {
    if (!PERROW) return Item{(int)w, 0, nT, -1};
    const int r = p.roworder ? p.roworder[w] : (int)w;
    return Item{r, 0, (p.rowlen[r] + kTok - 1) / kTok, -1};
  }
  const unsigned k = w - whole;
  if (k >= 2u * (unsigned)fs.half_rows) return Item{-1, 0, 0, 0};
  const int mid = (nT + 1) >> 1, h = (int)(k & 1u);
  return Item{(int)(whole + (k >> 1)), h ? mid : 0, h ? nT : mid, h};
}

// Producer: item `gr` into the shared ring for the other roles.
__device__ __forceinline__ void publish_item(volatile int* ring, int gr, const Item& it) {
  volatile int* e = ring + (gr % kItemRing) * 4;
  e[0] = it.row;
  e[1] = it.t0;
  e[2] = it.t1;
  e[3] = it.half;
  __threadfence_block();
  ring[4 * kItemRing + gr % kItemRing] = gr + 1;  // sequence number
}

// One thread: item `gr` once published; row -1 when the kernel winds down.
__device__ __forceinline__ Item read_item(volatile int* ring, int gr, volatile int* abort, unsigned* dbg,
                                          unsigned site) {
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 0;; ++i) {
    if (ring[4 * kItemRing + gr % kItemRing] == gr + 1) break;
    if (*abort) return Item{-1, 0, 0, 0};
    if ((i & 255u) == 255u && globaltimer_ns() - t0 > kWaitNs) {
      record_timeout(dbg, site, (unsigned)gr, 0u);
      *abort = 1;
      return Item{-1, 0, 0, 0};
    }
  }
  __threadfence_block();
  volatile int* e = ring + (gr % kItemRing) * 4;
  return Item{e[0], e[1], e[2], e[3]};
}

// LONG: the row may be longer than its on-chip logit capacity (a separate
// instantiation, so rows that fit run code without the spill branches).
// FULL: attention only, over the cache as it is (the full-cache comparator):
// no window state, features, policy, select, or writes to the cache's state.
// HEUR: a heuristic scorer (H2O or StreamingLLM, Dev::scorer) ranks the tokens
// instead of the policy MLP, whose tensor-core layer is then skipped.
// GLOB: global token mode: each row leaves its share of the per-token sums in
// Dev::gpart (mass, squared mass, entropy-weighted mass and |v|, in the V
// pass; the window sums come from the sequence's ring of pooled query terms);
// features, scores and the selection are made per sequence afterwards.
// GRAPH: device-counted steps: the step arguments are the host's base values
// plus the number of steps taken since (Dev::gcount[0], advanced by the last
// CTA to finish), so that a captured launch replays as the following steps.
// PAIR: items are row pairs (rows 2w and 2w + 1) of at most kPairTiles tiles,
// warpgroup w doing the whole of row 2w + w (its K and V tiles alternate with
// the other row's in the ring), so that one row's merge, output and select
// overlap the other's; policy scorer, whole rows, equal lengths only.
// PERROW: rows of different lengths and budgets (Dev::rowlen, Dev::rowbudget;
// FusedStep::B > 0 overrides every row's budget); the kernel writes each
// row's new length after its selection. No half rows.
template <int D, int G, bool LONG, bool FULL, bool HEUR, bool GLOB, bool PERROW, bool PAIR, bool GRAPH>
__global__ void __launch_bounds__(kThreads, 1)
    fused_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                 const __grid_constant__ CUtensorMap tmK16, const __grid_constant__ CUtensorMap tmV16, Dev p,
                 Step st, FusedStep fs, FusedPolicy fp) {
  constexpr int GS = G - 1;  // heads whose logits wait in TMEM between the passes
  static_assert(!PAIR || (!LONG && !FULL && !HEUR && !GLOB && !PERROW), "row pairs: the plain step only");
  static_assert(!PAIR || G <= 4, "row pairs: up to four query heads per KV head");
  constexpr int NQ = q_rows<G>();   // query-tile rows, S-tile columns
  constexpr int kColO = col_o<G>();
  // G = 8: the per-row statistics of the window's queries (the K pass) sit in
  // shared memory rather than in 6 x 8 registers per thread
  constexpr bool kWqSmem = G == 8;
  static_assert(!GRAPH || (!FULL && !HEUR && !GLOB && !PERROW), "device-counted steps: the plain step");
  if constexpr (GRAPH) {
    grid_dep_wait();  // the counter is the previous launch's
    // this launch's step: the base arguments advanced by the steps taken (in
    // the steady state a step appends one token, so positions, window slots
    // and the launch epoch all advance by one per step)
    const int t = *reinterpret_cast<volatile int*>(p.gcount);
    st.p_newest += t;
    st.p_prev += t;
    st.p_dep += t;
    st.slot = (st.slot + t) % p.w;
    st.slot_prev = (st.slot_prev + t) % p.w;
    fs.epoch += (unsigned)t;
  }
  using L = Smem<PAIR, G>;
  constexpr int OFF_STAGE = L::STAGE, OFF_Q = L::Q, OFF_P = L::P, OFF_A = L::A, OFF_W = L::W, OFF_AUX = L::AUX,
                OFF_SC = L::SC, OFF_MISC = L::MISC;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + OFF_MISC);
  static_assert(8 * B_COUNT <= 384, "barriers overlap the misc fields");
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + OFF_MISC + 384);
  volatile int* abort = reinterpret_cast<volatile int*>(smem + OFF_MISC + 388);
  // [8][G][3]; with G = 8 in the area the row pairs' scratch takes otherwise
  float* red = reinterpret_cast<float*>(smem + OFF_MISC + (G == 8 ? 2560 : 512));
  float* s_wq = reinterpret_cast<float*>(smem + OFF_MISC + 3328);          // G = 8: [6][8], then [3][8]
  static_assert(G != 8 || (!PAIR && 2560 + 8 * G * 3 * 4 <= 3328 && 3328 + 9 * 8 * 4 <= MISC_BYTES),
                "misc area layout");
  int* s_hist = reinterpret_cast<int*>(smem + OFF_MISC + 1024);           // [256]
  int* s_sh = reinterpret_cast<int*>(smem + OFF_MISC + 2048);             // [4]
  int* s_wsum = reinterpret_cast<int*>(smem + OFF_MISC + 2064);           // [8]
  unsigned long long* s_best = reinterpret_cast<unsigned long long*>(smem + OFF_MISC + 2112);  // [8]
  int* s_best_slot = reinterpret_cast<int*>(smem + OFF_MISC + 2176);      // [8]
  float* sc = reinterpret_cast<float*>(smem + OFF_SC);
  volatile int* items = reinterpret_cast<volatile int*>(smem + OFF_MISC + 2304);  // [8][4] + seq [8]
  // PAIR: the second warpgroup's select scratch
  int* s_hist2 = reinterpret_cast<int*>(smem + OFF_MISC + 2560);          // [256]
  int* s_sh2 = reinterpret_cast<int*>(smem + OFF_MISC + 3584);            // [4]
  int* s_wsum2 = reinterpret_cast<int*>(smem + OFF_MISC + 3600);          // [4]
  unsigned long long* s_best2 = reinterpret_cast<unsigned long long*>(smem + OFF_MISC + 3616);  // [4]
  int* s_best_slot2 = reinterpret_cast<int*>(smem + OFF_MISC + 3648);     // [4]

  const int warp = threadIdx.x / kWarp, lane = threadIdx.x % kWarp;
  const int n_step = st.n, nT = (n_step + kTok - 1) / kTok;
  constexpr uint32_t kTileBytes = (uint32_t)D * kTok * 2;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&bar[B_FULL + s], 1);
      mbar_init(&bar[B_EMPTY + s], 5);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bar[B_QFULL + b], 1);
      mbar_init(&bar[B_QEMPTY + b], 1);
      mbar_init(&bar[B_SFULL + b], 1);
      mbar_init(&bar[B_SEMPTY + b], 4);
      mbar_init(&bar[B_PFULL + b], 4);
      mbar_init(&bar[B_PEMPTY + b], 1);
      mbar_init(&bar[B_MFULL + b], 1);
      mbar_init(&bar[B_MEMPTY + b], 4);
      mbar_init(&bar[B_AFULL + b], 4);
      mbar_init(&bar[B_AEMPTY + b], 1);
    }
    mbar_init(&bar[B_OFULL], 1);
    mbar_init(&bar[B_OEMPTY], PAIR ? 8 : 4);
    mbar_init(&bar[B_DRAIN], 1);
    mbar_init(&bar[B_DRAIN2], 1);
    *abort = 0;
    for (int e = 0; e < kItemRing; ++e) items[4 * kItemRing + e] = 0;
    fence_mbar_init();
  }
  // zero the stages and their per-token areas (a row's ragged last tile loads
  // only its tokens: the rows past them then hold earlier tiles' finite data,
  // whose attention weights are zero), the query, weight and policy-input
  // tiles (unused rows and columns stay zero), then write the policy layer's
  // B operand (128 rows x 32 bf16, 64-byte swizzle)
  for (int e = threadIdx.x; e < (OFF_W - OFF_STAGE) / 16; e += kThreads)
    reinterpret_cast<uint4*>(smem + OFF_STAGE)[e] = make_uint4(0, 0, 0, 0);
  for (int e = threadIdx.x; e < kStages * kAuxBytes / 16; e += kThreads)
    reinterpret_cast<uint4*>(smem + OFF_AUX)[e] = make_uint4(0, 0, 0, 0);
  for (int e = threadIdx.x; e < 128 * 4; e += kThreads) {
    const int row = e >> 2, c = e & 3;
    *reinterpret_cast<uint4*>(smem + OFF_W + sw64(row, c)) = reinterpret_cast<const uint4*>(fp.wtile)[row * 4 + c];
  }
  fence_proxy_async();
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tmap(&tmK);
    prefetch_tmap(&tmV);
    prefetch_tmap(&tmK16);
    prefetch_tmap(&tmV16);
  }
  // everything above touches only shared memory, TMEM and read-only inputs:
  // with a programmatic launch it overlaps the kernel before (the append);
  // the cache and the queue counters are read and written after this wait
  grid_dep_wait();
  // the next launch's queue counter (this launch uses the other one)
  if (blockIdx.x == 0 && threadIdx.x == 0) fs.work[(fs.epoch + 1u) & 1u] = 0u;
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    const uint64_t pol = l2_evict_first_policy();
    int g = 0, issued = 0;
    bool last = false;  // a half row was taken: nothing more
    for (int gr = 0;; ++gr) {
      if (*abort) break;
      const int qb = gr & 1;
      if (!mbar_wait(&bar[B_QEMPTY + qb], ((gr >> 1) & 1) ^ 1, abort, p.dbg, 1u, (unsigned)gr)) break;
      // the next item, taken once this CTA's query buffer is free
      int4 iv = make_int4(-1, 0, 0, 0);
      if (lane == 0) {
        const Item t = last ? Item{-1, 0, 0, 0} : take_item<PERROW, PAIR>(fs, p, nT);
        publish_item(items, gr, t);
        iv = make_int4(t.row, t.t0, t.t1, t.half);
      }
      iv.x = __shfl_sync(0xffffffffu, iv.x, 0);
      iv.y = __shfl_sync(0xffffffffu, iv.y, 0);
      iv.z = __shfl_sync(0xffffffffu, iv.z, 0);
      iv.w = __shfl_sync(0xffffffffu, iv.w, 0);
      const Item it{iv.x, iv.y, iv.z, iv.w};
      if (it.row < 0) break;
      last = it.half >= 0;
      const int r = it.row;
      // query tile (PAIR: one per row): rows [0,G) current, [G,2G) previous
      // step, [2G,3G) departing
      if constexpr (PAIR) {
        // row pairs: a row's loads issued together (every element is read
        // before any is written, as the current query takes over the departing
        // query's ring slot), one global round trip per row
        constexpr int QCH = G * (D / 8);                 // 16-byte chunks of a row's G query heads
        constexpr int QIT = (QCH + kWarp - 1) / kWarp;   // per lane
        for (int qi = 0; qi < 2; ++qi) {
          const int rq = r + qi;
          uint8_t* qt = smem + OFF_Q + (2 * qb + qi) * L::QBYTES;
          const int qo = ((rq / p.kvh) * p.qh + (rq % p.kvh) * G) * D;
          const __nv_bfloat16* prev = p.ring_q + ((size_t)rq * p.w + st.slot_prev) * G * D;
          const __nv_bfloat16* dep = p.ring_q + ((size_t)rq * p.w + st.slot) * G * D;
          __nv_bfloat16* ring_slot = p.ring_q + ((size_t)rq * p.w + st.slot) * G * D;
          const bool q_ok = DC_INB(p, qo + G * D - 1, (long long)(p.R / p.kvh) * p.qh * D, 101) &&
                            DC_INB(p, ((long long)rq * p.w + st.slot) * G * D + G * D - 1, (long long)p.R * p.w * G * D, 102) &&
                            DC_INB(p, ((long long)rq * p.w + st.slot_prev) * G * D, (long long)p.R * p.w * G * D, 103);
          uint4 qcur[QIT], qprev[QIT], qdep[QIT];
#pragma unroll
          for (int u = 0; u < QIT; ++u) {
            const int e = lane + u * kWarp;
            const int h = e / (D / 8), kc = e % (D / 8);
            const bool ld = q_ok && e < QCH;
            qcur[u] = ld ? reinterpret_cast<const uint4*>(fs.q + qo + h * D)[kc] : make_uint4(0, 0, 0, 0);
            qprev[u] = ld && st.has_prev ? reinterpret_cast<const uint4*>(prev + h * D)[kc] : make_uint4(0, 0, 0, 0);
            qdep[u] = ld && st.has_dep ? reinterpret_cast<const uint4*>(dep + h * D)[kc] : make_uint4(0, 0, 0, 0);
          }
#pragma unroll
          for (int u = 0; u < QIT; ++u) {
            const int e = lane + u * kWarp;
            if (!q_ok || e >= QCH) continue;
            const int h = e / (D / 8), kc = e % (D / 8);
            *reinterpret_cast<uint4*>(qt + (kc >> 3) * (NQ * 128) + sw128(h, kc & 7)) = qcur[u];
            *reinterpret_cast<uint4*>(qt + (kc >> 3) * (NQ * 128) + sw128(G + h, kc & 7)) = qprev[u];
            *reinterpret_cast<uint4*>(qt + (kc >> 3) * (NQ * 128) + sw128(2 * G + h, kc & 7)) = qdep[u];
            if (!FULL && it.half < 0) reinterpret_cast<uint4*>(ring_slot + h * D)[kc] = qcur[u];  // halves: see the epilogue
          }
        }
      } else {
        // whole rows: one chunk per lane at a time (on whole rows this measured
        // faster than issuing the row's loads together: 6.04 against 6.25 ms
        // per step at 64 x 16384 x 25%)
        {
          const int rq = r;
          uint8_t* qt = smem + OFF_Q + qb * L::QBYTES;
          const int qo = ((rq / p.kvh) * p.qh + (rq % p.kvh) * G) * D;
          const __nv_bfloat16* prev = p.ring_q + ((size_t)rq * p.w + st.slot_prev) * G * D;
          const __nv_bfloat16* dep = p.ring_q + ((size_t)rq * p.w + st.slot) * G * D;
          // The current query also takes over the departing query's ring slot:
          // each lane reads the departing element before it writes the same one.
          __nv_bfloat16* ring_slot = p.ring_q + ((size_t)rq * p.w + st.slot) * G * D;
          const bool q_ok = DC_INB(p, qo + G * D - 1, (long long)(p.R / p.kvh) * p.qh * D, 101) &&
                            DC_INB(p, ((long long)rq * p.w + st.slot) * G * D + G * D - 1, (long long)p.R * p.w * G * D, 102) &&
                            DC_INB(p, ((long long)rq * p.w + st.slot_prev) * G * D, (long long)p.R * p.w * G * D, 103);
          for (int e = lane; q_ok && e < G * (D / 8); e += kWarp) {
            const int h = e / (D / 8), kc = e % (D / 8);
            const uint4 cur = reinterpret_cast<const uint4*>(fs.q + qo + h * D)[kc];
            const uint4 pv = st.has_prev ? reinterpret_cast<const uint4*>(prev + h * D)[kc] : make_uint4(0, 0, 0, 0);
            const uint4 dv = st.has_dep ? reinterpret_cast<const uint4*>(dep + h * D)[kc] : make_uint4(0, 0, 0, 0);
            *reinterpret_cast<uint4*>(qt + (kc >> 3) * (NQ * 128) + sw128(h, kc & 7)) = cur;
            *reinterpret_cast<uint4*>(qt + (kc >> 3) * (NQ * 128) + sw128(G + h, kc & 7)) = pv;
            *reinterpret_cast<uint4*>(qt + (kc >> 3) * (NQ * 128) + sw128(2 * G + h, kc & 7)) = dv;
            if (!FULL && it.half < 0) reinterpret_cast<uint4*>(ring_slot + h * D)[kc] = cur;  // halves: see the epilogue
          }
        }
      }
      fence_proxy_async();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&bar[B_QFULL + qb]);
        // PAIR: the two rows' tiles alternate (x even: the first row)
        const int nx = (PAIR ? 2 : 1) * (it.t1 - it.t0);
        for (int pass = 0; pass < 2 && !*abort; ++pass) {
          const CUtensorMap* tm = pass ? &tmV : &tmK;
          for (int x = 0; x < nx; ++x, ++g) {
            const int j = it.t0 + (PAIR ? x >> 1 : x), rt = r + (PAIR ? x & 1 : 0);
            const int s = g % kStages;
            if (!mbar_wait(&bar[B_EMPTY + s], ((g / kStages) & 1) ^ 1, abort, p.dbg, 2u, (unsigned)g)) break;
            // the tile's tokens: all 128, or the row's ragged last tile, loaded
            // in boxes of 16 tokens
            const int nrow = PERROW ? p.rowlen[rt] : n_step;
            const int valid = nrow - j * kTok < kTok ? nrow - j * kTok : kTok;
            const int nbox = valid < kTok ? (valid + 15) >> 4 : 0;
            const uint32_t kv_bytes = nbox ? (uint32_t)nbox * 16u * (uint32_t)D * 2u : kTileBytes;
            const uint32_t pos_bytes = ((uint32_t)valid * 4u + 15u) & ~15u, sz_bytes = (uint32_t)valid * 16u;
            const uint32_t aux_bytes = (pass || FULL) ? 0u : pos_bytes + (GLOB ? 0u : sz_bytes);
            uint8_t* dst = smem + OFF_STAGE + s * kStageBytes;
            uint8_t* aux = smem + OFF_AUX + s * kAuxBytes;
            const int y = rt * p.stride + j * kTok;
            if (!DC_INB(p, (long long)y + kTok - 1, (long long)p.R * p.stride, 104)) {
              // (debug builds) the tile lies outside the buffers: no copy; a
              // plain arrival completes the stage's phase with stale contents
              mbar_arrive(&bar[B_FULL + s]);
              issued = g + 1;
              continue;
            }
            mbar_expect_tx(&bar[B_FULL + s], kv_bytes + aux_bytes);
            if (nbox == 0) {
              tma_load_2d(dst, tm, 0, y, &bar[B_FULL + s], pol);
              if (D == 128) tma_load_2d(dst + 16384, tm, 64, y, &bar[B_FULL + s], pol);
            } else {
              // a 16-token box fills 2 KB (two 1 KB swizzle atoms) of each
              // 64-dim half, where the whole tile's load would put those rows
              const CUtensorMap* tm16 = pass ? &tmV16 : &tmK16;
              for (int b = 0; b < nbox; ++b) {
                tma_load_2d(dst + b * 2048, tm16, 0, y + 16 * b, &bar[B_FULL + s], pol);
                if (D == 128) tma_load_2d(dst + 16384 + b * 2048, tm16, 64, y + 16 * b, &bar[B_FULL + s], pol);
              }
            }
            if (!FULL && !pass) {
              bulk_load(aux + kAuxPos, p.pos + y, pos_bytes, &bar[B_FULL + s]);
              if (!GLOB) bulk_load(aux + kAuxSZ, p.SZ + y, sz_bytes, &bar[B_FULL + s]);
            }
            issued = g + 1;
          }
        }
      }
      g = __shfl_sync(0xffffffffu, g, 0);
      issued = __shfl_sync(0xffffffffu, issued, 0);
    }
    // every issued load must land before the CTA may exit
    if (lane == 0) {
      for (int t = issued - kStages < 0 ? 0 : issued - kStages; t < issued; ++t)
        mbar_wait_drain(&bar[B_FULL + t % kStages], (t / kStages) & 1);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t id_qk = idesc_bf16(128, NQ, 0, 0);
      const uint32_t id_pv = idesc_bf16(128, 16, 1, 1);
      int g = 0, gs = 0, gv = 0;
      for (int gr = 0;; ++gr) {
        const Item it = read_item(items, gr, abort, p.dbg, 23u);
        if (it.row < 0) break;
        const int qb = gr & 1;
        if (!mbar_wait(&bar[B_QFULL + qb], (gr >> 1) & 1, abort, p.dbg, 3u, (unsigned)gr)) break;
        tc_fence_after();
        const int nx = (PAIR ? 2 : 1) * (it.t1 - it.t0);  // PAIR: the rows' tiles alternate
        for (int x = 0; x < nx; ++x, ++g, ++gs) {
          const uint32_t qaddr = smem_u32(smem + OFF_Q + (PAIR ? 2 * qb + (x & 1) : qb) * L::QBYTES);
          const int s = g % kStages, b = gs & 1;
          if (!mbar_wait(&bar[B_FULL + s], (g / kStages) & 1, abort, p.dbg, 4u, (unsigned)g)) break;
          if (!mbar_wait(&bar[B_SEMPTY + b], ((gs >> 1) & 1) ^ 1, abort, p.dbg, 5u, (unsigned)gs)) break;
          tc_fence_after();
          const uint32_t kaddr = smem_u32(smem + OFF_STAGE + s * kStageBytes);
#pragma unroll
          for (int ks = 0; ks < D / 16; ++ks) {
            const uint32_t off = (uint32_t)(ks >> 2) * 16384u + (uint32_t)(ks & 3) * 32u;
            const uint32_t qoff = (uint32_t)(ks >> 2) * (uint32_t)(NQ * 128) + (uint32_t)(ks & 3) * 32u;
            mma_bf16(tmem + kColS + b * NQ, sdesc_sw128(kaddr + off, 16, 1024), sdesc_sw128(qaddr + qoff, 16, 1024),
                     id_qk, ks > 0);
          }
          mma_commit(&bar[B_SFULL + b]);
          mma_commit(&bar[B_EMPTY + s]);
        }
        mma_commit(&bar[B_QEMPTY + qb]);
        // V pass: PV MMAs in tile order; a V stage is released as soon as its
        // tile's weights are in (the policy-layer MMAs run on warp 10)
        for (int x = 0; x < nx; ++x, ++g, ++gv) {
          const int s = g % kStages, pb = gv & 1;
          // the first tile of each row starts its accumulator
          const bool first = PAIR ? x < 2 : x == 0;
          const uint32_t ocol = kColO + (PAIR && (x & 1) ? (uint32_t)(kColOB - kColO) : 0u);
          if (!mbar_wait(&bar[B_FULL + s], (g / kStages) & 1, abort, p.dbg, 13u, (unsigned)g)) break;
          // only these MMAs read a V stage: the four epilogue arrivals of the
          // stage's release are made here (its last one is the commit below)
          mbar_arrive_cnt(&bar[B_EMPTY + s], 4);
          if (!mbar_wait(&bar[B_PFULL + pb], (gv >> 1) & 1, abort, p.dbg, 14u, (unsigned)gv)) break;
          if (x == 0 && !mbar_wait(&bar[B_OEMPTY], (gr & 1) ^ 1, abort, p.dbg, 15u, (unsigned)gr)) break;
          tc_fence_after();
          const uint32_t vaddr = smem_u32(smem + OFF_STAGE + s * kStageBytes);
          const uint32_t paddr = smem_u32(smem + OFF_P + pb * 4096);
          // O^T[d x 16] += V^T[d x 128] P^T: V^T is MN-major (dims contiguous)
#pragma unroll
          for (int ks = 0; ks < kTok / 16; ++ks)
            mma_bf16(tmem + ocol, sdesc_sw128(vaddr + ks * 2048u, 16384, 1024),
                     sdesc_sw32(paddr + ks * 512u, 4096, 256), id_pv, (!first || ks > 0) ? 1u : 0u);
          mma_commit(&bar[B_PEMPTY + pb]);
          mma_commit(&bar[B_EMPTY + s]);
          if (x == nx - 1) mma_commit(&bar[B_OFULL]);
        }
      }
      // all issued MMAs complete before TMEM is released
      mma_commit(&bar[B_DRAIN]);
      mbar_wait_drain(&bar[B_DRAIN], 0);
    }
    __syncwarp();
  } else if (warp == 10) {
    // ------------------------------------------------------------ policy-layer MMA issuer
    if (!FULL && !HEUR && !GLOB && lane == 0) {
      const uint32_t id_m = idesc_bf16(128, 128, 0, 0);
      const uint32_t waddr = smem_u32(smem + OFF_W);
      int gv = 0;
      for (int gr = 0;; ++gr) {
        const Item it = read_item(items, gr, abort, p.dbg, 24u);
        if (it.row < 0) break;
        const int nx = (PAIR ? 2 : 1) * (it.t1 - it.t0);
        for (int x = 0; x < nx; ++x, ++gv) {
          const int pb = gv & 1;
          if (!mbar_wait(&bar[B_AFULL + pb], (gv >> 1) & 1, abort, p.dbg, 16u, (unsigned)gv)) break;
          if (!mbar_wait(&bar[B_MEMPTY + pb], ((gv >> 1) & 1) ^ 1, abort, p.dbg, 17u, (unsigned)gv)) break;
          tc_fence_after();
          const uint32_t aaddr = smem_u32(smem + OFF_A + pb * 8192);
          // Z[128 x 128] = A[128 x 32] W^T
#pragma unroll
          for (int ks = 0; ks < 2; ++ks)
            mma_bf16(tmem + kColM + pb * 128, sdesc_sw64(aaddr + ks * 32u, 16, 512),
                     sdesc_sw64(waddr + ks * 32u, 16, 512), id_m, ks > 0);
          mma_commit(&bar[B_MFULL + pb]);
          mma_commit(&bar[B_AEMPTY + pb]);
        }
      }
      mma_commit(&bar[B_DRAIN2]);
      mbar_wait_drain(&bar[B_DRAIN2], 0);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue
    const int ew = warp - 2;                    // 0..7
    const int wg = ew >> 2;                     // warpgroup 0 / 1
    const int quad = warp & 3;                  // TMEM lane quarter of this warp
    const int tok = quad * 32 + lane;           // token (TMEM lane) within a tile
    const int etid = ew * 32 + lane;            // 0..255
    const uint32_t lane_addr = tmem + ((uint32_t)(quad * 32) << 16);
    const float c = p.c;
    // the team that works on one row: both warpgroups, or (PAIR) one each
    constexpr int kTeam = PAIR ? kEpi / 2 : kEpi;
    const int tid = PAIR ? etid % kTeam : etid;    // thread within the team
    const int w0 = PAIR ? wg * (kTeam / kWarp) : 0;  // the team's first epilogue warp
    auto sync = [wg] {
      if constexpr (PAIR) named_bar(2 + wg, kTeam);
      else named_bar(1, kEpi);
    };
    const SelectScratch scr = (PAIR && wg == 1) ? SelectScratch{s_hist2, s_sh2, s_wsum2, s_best2, s_best_slot2}
                                                : SelectScratch{s_hist, s_sh, s_wsum, s_best, s_best_slot};
    // PAIR: this team's logits of head G-1, then scores
    float* const scw = sc + (PAIR ? wg * kPairTok : 0);
    // TMEM column of the stashed logits of this team's tile j
    auto stash_at = [wg](int j) -> uint32_t {
      if constexpr (PAIR) return (uint32_t)((wg ? kStashB : kPairStashA) + GS * j);
      else return stash_col<G>(j);
    };
    // position of this team's tile j in the item's tile sequence
    auto tpos = [wg](int j, int t0) { return PAIR ? 2 * j + wg : j - t0; };
    constexpr int JS = PAIR ? 1 : 2;  // step between a team's tiles
    int g = 0, gs = 0, gv = 0;
    for (int gr = 0;; ++gr) {
      int4 iv = make_int4(-1, 0, 0, 0);
      if (lane == 0) {
        const Item t = read_item(items, gr, abort, p.dbg, 25u);
        iv = make_int4(t.row, t.t0, t.t1, t.half);
      }
      iv.x = __shfl_sync(0xffffffffu, iv.x, 0);
      iv.y = __shfl_sync(0xffffffffu, iv.y, 0);
      iv.z = __shfl_sync(0xffffffffu, iv.z, 0);
      iv.w = __shfl_sync(0xffffffffu, iv.w, 0);
      if (named_bar_or(1, kEpi, *abort != 0 || iv.x < 0)) break;
      const Item it{iv.x, iv.y, iv.z, iv.w};
      const int r = it.row + (PAIR ? wg : 0), t0 = it.t0, t1 = it.t1, nTi = it.t1 - it.t0;
      const int nItem = (PAIR ? 2 : 1) * nTi;  // tiles of the item
      // this row's length (after the append) and budget
      const int n = PERROW ? p.rowlen[r] : n_step;
      const int Bsel = PERROW ? (fs.B > 0 ? fs.B : p.rowbudget[r]) : fs.B;
      const int ts = r - (p.R - fs.half_rows);  // exchange slot (half rows only)
      const size_t rbase = (size_t)r * p.stride;
      // (debug builds) slot i of this row inside the row and the buffers
      const long long RS = (long long)p.R * p.stride;
      auto slot_ok = [&](long long i, unsigned site) {
        return DC_INB(p, i, p.stride, site) && DC_INB(p, (long long)rbase + i, RS, site);
      };
      (void)RS;
      const bool x_ok = it.half < 0 || (DC_INB(p, ts, fs.xslots, 110) && DC_INB(p, ts, fs.half_rows, 110));
      // a row longer than the shared score array keeps its scores in HBM when
      // the radix select reads them (several evictions), or when asked to
      const bool spill_scores = LONG && n > max_tok<G>() && fs.do_evict && Bsel < n - 1;
      // statistics (m, -log2 l, H) of the previous and the departing query
      constexpr int GR = kWqSmem ? 1 : G;
      float pm[GR], pnl[GR], pH[GR], dm[GR], dnl[GR], dH[GR];
      if constexpr (kWqSmem) {
        // one thread per (query, head) loads them into shared memory; the
        // team's barrier publishes them (the previous item's K pass, their
        // last reader, ended before that item's statistics merge)
        if (tid < 2 * G) {
          const int h = tid % G, dep = tid / G;
          const float4 rs =
              reinterpret_cast<const float4*>(p.ring_stats)[((size_t)r * p.w + (dep ? st.slot : st.slot_prev)) * G + h];
          s_wq[(3 * dep + 0) * G + h] = rs.x;
          s_wq[(3 * dep + 1) * G + h] = rs.w;
          s_wq[(3 * dep + 2) * G + h] = rs.z;
        }
        sync();
      } else {
#pragma unroll
        for (int h = 0; h < G; ++h) {
          const float4 rp = reinterpret_cast<const float4*>(p.ring_stats)[((size_t)r * p.w + st.slot_prev) * G + h];
          const float4 rd = reinterpret_cast<const float4*>(p.ring_stats)[((size_t)r * p.w + st.slot) * G + h];
          pm[h] = rp.x; pnl[h] = rp.w; pH[h] = rp.z;
          dm[h] = rd.x; dnl[h] = rd.w; dH[h] = rd.z;
        }
      }
      float m[G], l[G], u[G];
#pragma unroll
      for (int h = 0; h < G; ++h) { m[h] = kNoMax; l[h] = 0.f; u[h] = 0.f; }

      // ---------------- K pass: this warpgroup's tiles (global index parity)
      for (int j = PAIR ? t0 : t0 + ((wg - gs) & 1); j < t1; j += JS) {
        const int gj = g + tpos(j, t0), gsj = gs + tpos(j, t0);
        const int s = gj % kStages, b = gsj & 1;
        mbar_wait(&bar[B_SFULL + b], (gsj >> 1) & 1, abort, p.dbg, 6u, (unsigned)gsj);
        mbar_wait(&bar[B_FULL + s], (gj / kStages) & 1, abort, p.dbg, 12u, (unsigned)gj);
        __syncwarp();
        tc_fence_after();
        float S16[NQ];  // the current, previous and departing queries' logits
        if constexpr (NQ == 32) tmem_ld32(lane_addr + kColS + b * NQ, S16);
        else tmem_ld16(lane_addr + kColS + b * NQ, S16);
        tmem_ld_wait();
        const uint8_t* aux = smem + OFF_AUX + s * kAuxBytes;
        const int pos = reinterpret_cast<const int*>(aux + kAuxPos)[tok];
        float4 sz = reinterpret_cast<const float4*>(aux + kAuxSZ)[tok];
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&bar[B_SEMPTY + b]);
          mbar_arrive(&bar[B_EMPTY + s]);
        }
        const int i = j * kTok + tok;
        if (i < n) {
#pragma unroll
          for (int h = 0; h < G; ++h) online_add(m[h], l[h], u[h], S16[h], c);
          if (!FULL && !GLOB && (st.has_prev || st.has_dep)) {
            // terms of the previous and the departing query, masked (x 1 or x 0,
            // both exact) where the token was not yet in the cache at that step
            float zp, sp, zd, sd;
            if constexpr (kWqSmem) {
              window_terms<G>(S16 + G, s_wq, s_wq + G, s_wq + 2 * G, c, zp, sp);
              window_terms<G>(S16 + 2 * G, s_wq + 3 * G, s_wq + 4 * G, s_wq + 5 * G, c, zd, sd);
            } else {
              window_terms<G>(S16 + G, pm, pnl, pH, c, zp, sp);
              window_terms<G>(S16 + 2 * G, dm, dnl, dH, c, zd, sd);
            }
            const float mp = (st.has_prev && pos <= st.p_prev) ? 1.f : 0.f;
            const float md = (st.has_dep && pos <= st.p_dep) ? 1.f : 0.f;
            sz = window_update(sz, sp * mp, sd * md, zp * mp, zd * md);
            if (slot_ok(i, 105)) p.SZ[rbase + i] = sz;
          }
        }
        if (!LONG || j < onchip_tiles<G>()) {
          scw[i] = S16[G - 1];
          __syncwarp();
          stash_store<GS>(lane_addr + stash_at(j), S16);
        } else if (slot_ok(i, 106)) {
          store_logits<G>(p.logit + (rbase + i) * G, S16);
        }
      }
      g += nItem;
      gs += nItem;
      // per-token state of this warpgroup's V-pass tiles (the same tiles as its
      // K pass), loaded two own tiles ahead: window sums (this thread wrote
      // them in the K pass), positions, |v|; the first two issued here, so that
      // their latency overlaps the statistics merge
      const int j0 = PAIR ? t0 : t0 + ((wg - gv) & 1);
      const float4* szrow = p.SZ + rbase + tok;
      const int* posrow = p.pos + rbase + tok;
      const float* vnrow = p.vnorm + rbase + tok;
      const float4 kZero4 = make_float4(0.f, 0.f, 0.f, 0.f);
      float4 szA = kZero4, szB = kZero4;
      int posA = 0, posB = 0;
      float vnA = 0.f, vnB = 0.f;
      // HEUR: cumulative alpha (H2O's score) loaded ahead the same way
      const bool ac_ahead = HEUR && p.alpha_mode == 1;
      const float* acrow = ac_ahead ? p.acc + rbase + tok : nullptr;
      float acA = 0.f, acB = 0.f;
      if (ac_ahead) {
        acA = j0 < t1 ? acrow[j0 * kTok] : 0.f;
        acB = j0 + JS < t1 ? acrow[(j0 + JS) * kTok] : 0.f;
      }
      if constexpr (!FULL && !GLOB) {
        szA = j0 < t1 ? szrow[j0 * kTok] : kZero4;
        szB = j0 + JS < t1 ? szrow[(j0 + JS) * kTok] : kZero4;
        posA = j0 < t1 ? posrow[j0 * kTok] : 0;
        posB = j0 + JS < t1 ? posrow[(j0 + JS) * kTok] : 0;
      }
      if constexpr (!FULL) {
        vnA = j0 < t1 ? vnrow[j0 * kTok] : 0.f;
        vnB = j0 + JS < t1 ? vnrow[(j0 + JS) * kTok] : 0.f;
      }
      if constexpr (GS > 0) tmem_st_wait();
      // ---------------- row softmax statistics (deterministic merge order):
      // the maximum first, then every partial (l, u) rescaled to it and summed
#pragma unroll
      for (int h = 0; h < G; ++h) {
        float mm = m[h];
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) mm = fmaxf(mm, __shfl_xor_sync(0xffffffffu, mm, off));
        const float dm = (m[h] - mm) * c, f = ex2(dm);
        float ll = l[h] * f, uu = (u[h] + l[h] * dm) * f;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
          ll += __shfl_xor_sync(0xffffffffu, ll, off);
          uu += __shfl_xor_sync(0xffffffffu, uu, off);
        }
        if (lane == 0) {
          red[(ew * G + h) * 3 + 0] = mm;
          red[(ew * G + h) * 3 + 1] = ll;
          red[(ew * G + h) * 3 + 2] = uu;
        }
      }
      sync();
      float Mm[G], Ll[G], Uu[G];
#pragma unroll
      for (int h = 0; h < G; ++h) {
        float mm = kNoMax;
#pragma unroll
        for (int w = w0; w < w0 + kTeam / kWarp; ++w) mm = fmaxf(mm, red[(w * G + h) * 3 + 0]);
        float ll = 0.f, uu = 0.f;
#pragma unroll
        for (int w = w0; w < w0 + kTeam / kWarp; ++w) {
          const float lw = red[(w * G + h) * 3 + 1];
          const float dm = (red[(w * G + h) * 3 + 0] - mm) * c, f = ex2(dm);
          ll = fmaf(lw, f, ll);
          uu = fmaf(red[(w * G + h) * 3 + 2] + lw * dm, f, uu);
        }
        Mm[h] = mm; Ll[h] = ll; Uu[h] = uu;
      }
      sync();  // red is rewritten by the next row
      const int half = it.half;
      unsigned* my_flag = half >= 0 ? fs.xflag + 2 * ts + half : nullptr;
      const unsigned* peer_flag = half >= 0 ? fs.xflag + 2 * ts + (half ^ 1) : nullptr;
      const unsigned ep = fs.epoch * 4u;
      if (half >= 0 && x_ok) {
        // half row: swap the partial statistics with the other half, then
        // both merge half 0's before half 1's (identical results on both)
        float4* xs = reinterpret_cast<float4*>(fs.xstats);
        if (etid < G) {
          xs[(2 * ts + half) * G + etid] = make_float4(Mm[etid], Ll[etid], Uu[etid], 0.f);
          __threadfence();
        }
        sync();
        if (etid == 0) {
          flag_release(my_flag, ep + 1u);
          flag_wait(peer_flag, ep + 1u, abort, p.dbg, 20u, (unsigned)r);
        }
        sync();
#pragma unroll
        for (int h = 0; h < G; ++h) {
          const float4 o = __ldcg(&xs[(2 * ts + (half ^ 1)) * G + h]);
          float mm = kNoMax, ll = 0.f, uu = 0.f;
          if (half == 0) {
            online_merge(mm, ll, uu, Mm[h], Ll[h], Uu[h], c);
            online_merge(mm, ll, uu, o.x, o.y, o.z, c);
          } else {
            online_merge(mm, ll, uu, o.x, o.y, o.z, c);
            online_merge(mm, ll, uu, Mm[h], Ll[h], Uu[h], c);
          }
          Mm[h] = mm; Ll[h] = ll; Uu[h] = uu;
        }
        // half 1 has read the departing query and statistics (it published
        // after its K pass): half 0 may now give their ring slot to this step
        if (!FULL && half == 0 && DC_INB(p, ((long long)r * p.w + st.slot) * G * D + G * D - 1,
                                         (long long)p.R * p.w * G * D, 119) &&
            DC_INB(p, (long long)((r / p.kvh) * p.qh + (r % p.kvh) * G) * D + G * D - 1,
                   (long long)(p.R / p.kvh) * p.qh * D, 119)) {
          const int qo = ((r / p.kvh) * p.qh + (r % p.kvh) * G) * D;
          uint4* ring_slot = reinterpret_cast<uint4*>(p.ring_q + ((size_t)r * p.w + st.slot) * G * D);
          for (int e = etid; e < G * (D / 8); e += kEpi) ring_slot[e] = reinterpret_cast<const uint4*>(fs.q + qo)[e];
        }
      }
      float M[G], NL[G], Hh[G];
      float L0 = 0.f;
#pragma unroll
      for (int h = 0; h < G; ++h) {
        M[h] = Mm[h];
        // H = ln l - ln 2 u / l. Whole rows take log2 l from the hardware log2
        // and divide (l >= 1: the row's largest logit contributes 2^0), row
        // pairs from log2f and logf: each measured the faster for its
        // schedule (the kernel's speed on these shapes moves by several
        // per cent with its code layout)
        if constexpr (PAIR) {
          NL[h] = -log2f(Ll[h]);
          Hh[h] = logf(Ll[h]) - 0.69314718055994531f * (Uu[h] / Ll[h]);
        } else {
          const float lg = lg2_approx(Ll[h]);
          NL[h] = -lg;
          Hh[h] = 0.69314718055994531f * (lg - __fdividef(Uu[h], Ll[h]));
        }
        if (tid == h) L0 = Ll[h];
      }
      // G = 8: the V pass reads the row's final statistics from shared memory
      float* s_st = s_wq + 6 * 8;  // [3][8]: M, -log2 l, H
      if constexpr (kWqSmem) {
        if (tid == 0) {
#pragma unroll
          for (int h = 0; h < G; ++h) {
            s_st[h] = M[h];
            s_st[G + h] = NL[h];
            s_st[2 * G + h] = Hh[h];
          }
        }
        sync();
      }
      // push (m, l, H, -log2 l) of this step into the ring slot it takes over
      // (the producer, or half 0 above, wrote the query there)
      if (!FULL && tid < G && half <= 0 && DC_INB(p, (long long)r * p.w + st.slot, (long long)p.R * p.w, 109)) {
        float4 v;
        v.x = M[tid]; v.y = L0; v.z = Hh[tid]; v.w = NL[tid];
        reinterpret_cast<float4*>(p.ring_stats)[((size_t)r * p.w + st.slot) * G + tid] = v;
        p.hq[(size_t)r * G + tid] = Hh[tid];
      }

      // One eviction (the steady state): slot B, the only mover, is loaded now
      // (its window sums were written before the merge barrier), so that the
      // select does not wait on it; what the V pass may still write is loaded
      // at the select.
      const bool single_evict = fs.do_evict && n == Bsel + 1 && slot_ok(Bsel, 116);
      SlotCopy mv{};
      if (single_evict && half != 0 && tid < kWarp) slot_load_settled(p, rbase + Bsel, tid, fs.write_scores, mv);

      // ---------------- V pass: this warpgroup's tiles; prep of the next one
      // overlaps the MMAs of the current one
      const float pos_den = (float)max(st.p_newest, 1);
      auto prep = [&](int j) {
        const int gvj = gv + tpos(j, t0), pb = gvj & 1;
        const float4 sz = szA;
        const int pos = posA;
        const float vn = vnA, ac = acA;
        szA = szB;
        posA = posB;
        vnA = vnB;
        acA = acB;
        if (!FULL && j + 2 * JS < t1 && slot_ok((j + 2 * JS) * kTok + tok, 107)) {
          if constexpr (!GLOB) {
            szB = szrow[(j + 2 * JS) * kTok];
            posB = posrow[(j + 2 * JS) * kTok];
          }
          vnB = vnrow[(j + 2 * JS) * kTok];
          if (ac_ahead) acB = acrow[(j + 2 * JS) * kTok];
        }
        const int i = j * kTok + tok;
        const bool valid = i < n;
        float sv[G];
        if (!LONG || j < onchip_tiles<G>()) {
          stash_load<GS>(lane_addr + stash_at(j), sv);
          if constexpr (GS > 0) tmem_ld_wait();
          sv[G - 1] = scw[i];
        } else if (slot_ok(i, 108)) {
          load_logits<G>(p.logit + (rbase + i) * G, sv);
        }
        float a[G], zc = 0.f, scur = 0.f;
#pragma unroll
        for (int h = 0; h < G; ++h) {
          a[h] = kWqSmem ? attn_weight(sv[h], s_st[h], c, s_st[G + h]) : attn_weight(sv[h], M[h], c, NL[h]);
          zc += a[h];
          scur = fmaf(a[h], kWqSmem ? s_st[2 * G + h] : Hh[h], scur);
        }
        // attention weights as the PV operand, MN-major (one 32-byte row of 16
        // columns per token, 32-byte swizzle): bf16 high parts in columns
        // [0, G), the residuals in [G, 2G), so that O = D[:, h] + D[:, G + h]
        // carries ~16 mantissa bits; columns [2G, 16) stay zero
        mbar_wait(&bar[B_PEMPTY + pb], ((gvj >> 1) & 1) ^ 1, abort, p.dbg, 8u, (unsigned)gvj);
        {
          constexpr int NP = G == 8 ? 16 : 8;  // columns written: one or both 16-byte chunks
          float pw[NP];
#pragma unroll
          for (int h = 0; h < NP; ++h) pw[h] = 0.f;
#pragma unroll
          for (int h = 0; h < G; ++h) {
            const float ah = valid ? a[h] : 0.f;
            const float hv = __bfloat162float(__float2bfloat16_rn(ah));
            pw[h] = hv;
            pw[G + h] = ah - hv;
          }
          uint8_t* prow = smem + OFF_P + pb * 4096 + (tok >> 3) * 256 + (tok & 7) * 32;
#pragma unroll
          for (int ck = 0; ck < NP / 8; ++ck)
            *reinterpret_cast<uint4*>(prow + ((ck ^ ((tok >> 2) & 1)) << 4)) =
                make_uint4(pack_bf16(pw[8 * ck + 0], pw[8 * ck + 1]), pack_bf16(pw[8 * ck + 2], pw[8 * ck + 3]),
                           pack_bf16(pw[8 * ck + 4], pw[8 * ck + 5]), pack_bf16(pw[8 * ck + 6], pw[8 * ck + 7]));
          fence_proxy_async();
          __syncwarp();
          if (lane == 0) mbar_arrive(&bar[B_PFULL + pb]);
        }
        if constexpr (FULL) return make_float2(0.f, 0.f);
        if constexpr (GLOB) {
          // this row's share of the token's pooled sums
          if (valid && slot_ok(i, 111)) {
            float a2 = 0.f;
#pragma unroll
            for (int h = 0; h < G; ++h) a2 = fmaf(a[h], a[h], a2);
            p.gpart[rbase + i] = make_float4(zc, a2, scur, vn);
          }
          return make_float2(0.f, 0.f);
        }
        const float mean = zc / (float)G;
        float var = 0.f;
#pragma unroll
        for (int h = 0; h < G; ++h) var = fmaf(a[h] - mean, a[h] - mean, var);
        var /= (float)G;
        const float Zt = __fadd_rn(__fadd_rn(sz.z, zc), sz.w);
        const float St = __fadd_rn(__fadd_rn(sz.x, scur), sz.y);
        float x[5] = {mean, vn, var, Zt > 0.f ? St / Zt : 0.f, (float)pos / pos_den};
        if (valid && slot_ok(i, 112)) {
          const size_t slot = rbase + i;
          if (p.alpha_mode == 1) {
            x[0] = (ac_ahead ? ac : p.acc[slot]) + mean;
            p.acc[slot] = x[0];
          }
          if (p.keep_features)
#pragma unroll
            for (int e = 0; e < 5; ++e) p.feat[slot * 5 + e] = x[e];
        }
        if constexpr (HEUR) return make_float2(heuristic_score(p, x[0], pos, st.p_newest), __int_as_float(pos));
        // the policy layer's input row: [r x, r, 1, 0] (LayerNorm folded into
        // the weights) or [x, 1, 0, 0], as bf16 hi | lo | hi parts
        float av[8];
        if (fp.layernorm) {
          const float xt[6] = {x[0], x[1], x[2], x[3], x[4], 1.f};
          float q2 = 0.f;
          int k = 0;
#pragma unroll
          for (int aa = 0; aa < 6; ++aa)
#pragma unroll
            for (int bb = aa; bb < 6; ++bb) q2 = fmaf(fp.M[k++] * xt[aa], xt[bb], q2);
          const float rs = rsqrtf(fmaxf(q2, 0.f) + 1e-5f);
#pragma unroll
          for (int e = 0; e < 6; ++e) av[e] = rs * xt[e];
          av[6] = 1.f;
          av[7] = 0.f;
        } else {
#pragma unroll
          for (int e = 0; e < 5; ++e) av[e] = x[e];
          av[5] = 1.f;
          av[6] = 0.f;
          av[7] = 0.f;
        }
        uint32_t hi[4], lo[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const __nv_bfloat16 h0 = __float2bfloat16_rn(av[2 * e]), h1 = __float2bfloat16_rn(av[2 * e + 1]);
          const float r0 = av[2 * e] - __bfloat162float(h0), r1 = av[2 * e + 1] - __bfloat162float(h1);
          hi[e] = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
          lo[e] = pack_bf16(r0, r1);
        }
        mbar_wait(&bar[B_AEMPTY + pb], ((gvj >> 1) & 1) ^ 1, abort, p.dbg, 9u, (unsigned)gvj);
        uint8_t* at = smem + OFF_A + pb * 8192;
        *reinterpret_cast<uint4*>(at + sw64(tok, 0)) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
        *reinterpret_cast<uint4*>(at + sw64(tok, 1)) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
        *reinterpret_cast<uint4*>(at + sw64(tok, 2)) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
        fence_proxy_async();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bar[B_AFULL + pb]);
        // the linear part of the score, sum_j sgn_j z_j, on the CUDA cores
        float lin = 0.f;
#pragma unroll
        for (int e = 0; e < 8; ++e) lin = fmaf(av[e], fp.u[e], lin);
        return make_float2(lin, __int_as_float(pos));
      };
      uint32_t ev_key = 0xFFFFFFFFu;
      int ev_slot = -1, ev_pos = -1;
      auto finish = [&](int j, float lin, int pos) {
        const int gvj = gv + tpos(j, t0), pb = gvj & 1;
        mbar_wait(&bar[B_MFULL + pb], (gvj >> 1) & 1, abort, p.dbg, 10u, (unsigned)gvj);
        __syncwarp();
        tc_fence_after();
        // score = b2 + sum_j sgn_j max(z_j, 0) = b2 + (lin + sum_j sgn_j |z_j|) / 2;
        // eight independent partial sums
        float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int c8 = 0; c8 < 2; ++c8) {
          float z2[2][32];
          tmem_ld32(lane_addr + kColM + pb * 128 + c8 * 64, z2[0]);
          tmem_ld32(lane_addr + kColM + pb * 128 + c8 * 64 + 32, z2[1]);
          tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 64; ++e)
            acc[e & 7] = fmaf(fp.sgn[c8 * 64 + e], fabsf(z2[e >> 5][e & 31]), acc[e & 7]);
        }
        const float abs_sum = ((acc[0] + acc[1]) + (acc[2] + acc[3])) + ((acc[4] + acc[5]) + (acc[6] + acc[7]));
        const float relu_sum = 0.5f * (lin + abs_sum);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bar[B_MEMPTY + pb]);
        const int i = j * kTok + tok;
        if (i < n && slot_ok(i, 113)) {
          const float score = fp.b2 + relu_sum;
          if constexpr (LONG) {
            if (spill_scores || fs.write_scores) p.score[rbase + i] = score;
            if (n <= max_tok<G>()) scw[i] = score;
          } else {
            scw[i] = score;
            if (fs.write_scores) p.score[rbase + i] = score;
          }
          // this thread's lowest-ranked token so far (lower key, then the later position)
          const uint32_t kk = score_key(score);
          if (ev_slot < 0 || kk < ev_key || (kk == ev_key && pos > ev_pos)) {
            ev_key = kk;
            ev_slot = i;
            ev_pos = pos;
          }
        }
      };
      // the score of a heuristic scorer, recorded like finish() records the policy's
      auto record_h = [&](int j, float score, int pos) {
        const int i = j * kTok + tok;
        if (i < n && slot_ok(i, 114)) {
          if (spill_scores || fs.write_scores) p.score[rbase + i] = score;
          if (n <= max_tok<G>()) scw[i] = score;
          const uint32_t kk = score_key(score);
          if (ev_slot < 0 || kk < ev_key || (kk == ev_key && pos > ev_pos)) {
            ev_key = kk;
            ev_slot = i;
            ev_pos = pos;
          }
        }
      };
      // prep(j) returns (the linear score part, or a heuristic score; the
      // position) for finish(j), which runs after prep(j + JS); one call site
      // each (the first pass of the loop only preps the first tile), so that
      // the loop's code is inlined once
      float2 pf_cur = make_float2(0.f, 0.f);
      for (int j = j0 - JS; j < t1; j += JS) {
        const float2 pf_next = j + JS < t1 ? prep(j + JS) : make_float2(0.f, 0.f);
        if (j >= j0) {
          if constexpr (HEUR) record_h(j, pf_cur.x, __float_as_int(pf_cur.y));
          else if constexpr (!FULL && !GLOB) finish(j, pf_cur.x, __float_as_int(pf_cur.y));
        }
        pf_cur = pf_next;
      }
      g += nItem;
      gv += nItem;
      // ---------------- attention output (warpgroup 0); a half row's two
      // partial sums (weights already normalised by the whole row) add up
      float ov[G];
      if (PAIR || wg == 0) {
        mbar_wait(&bar[B_OFULL], gr & 1, abort, p.dbg, 11u, (unsigned)gr);
        __syncwarp();
        tc_fence_after();
        float o16[16];
        tmem_ld16(lane_addr + (PAIR && wg ? kColOB : kColO), o16);
        tmem_ld_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bar[B_OEMPTY]);
#pragma unroll
        for (int h = 0; h < G; ++h) ov[h] = o16[h] + o16[G + h];
        if (half == 1 && tok < D && x_ok) {
#pragma unroll
          for (int h = 0; h < G; ++h) fs.xo[((size_t)ts * G + h) * D + tok] = ov[h];
          __threadfence();
        }
      }
      if (half >= 0 && x_ok) {
        sync();
        if (etid == 0) {
          if (half == 1) flag_release(my_flag, ep + 2u);
          else flag_wait(peer_flag, ep + 2u, abort, p.dbg, 21u, (unsigned)r);
        }
        sync();
      }
      if ((PAIR || wg == 0) && half <= 0 && tok < D && x_ok &&
          DC_INB(p, (long long)((r / p.kvh) * p.qh + (r % p.kvh) * G) * D + (G - 1) * D + tok,
                 (long long)(p.R / p.kvh) * p.qh * D, 115)) {
        float* op = fs.out + ((r / p.kvh) * p.qh + (r % p.kvh) * G) * D;
#pragma unroll
        for (int h = 0; h < G; ++h)
          op[h * D + tok] = half == 0 ? ov[h] + __ldcg(&fs.xo[((size_t)ts * G + h) * D + tok]) : ov[h];
      }
      // ---------------- argtop_B and prune
      if (single_evict) {
        // one eviction (the steady state): the lowest-ranked token, from each
        // thread's running candidate; slot B (the last, held by the whole row
        // or by half 1) is the only mover and fills the evicted slot. Half
        // rows swap their candidates first.
        const bool mover = half != 0;
        if (mover && tid < kWarp) slot_load_late(p, rbase + Bsel, tid, fs.write_scores, mv);
        auto lower = [](uint32_t ka, int sa, int pa, uint32_t kb, int sb, int pb) {  // (kb, sb) ranks lower?
          if (sb < 0) return false;
          if (sa < 0) return true;
          return kb < ka || (kb == ka && pb > pa);
        };
        uint32_t bk = ev_key;
        int bs = ev_slot, bp = ev_pos;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
          const uint32_t ok = __shfl_xor_sync(0xffffffffu, bk, off);
          const int os = __shfl_xor_sync(0xffffffffu, bs, off);
          const int op = __shfl_xor_sync(0xffffffffu, bp, off);
          if (lower(bk, bs, bp, ok, os, op)) { bk = ok; bs = os; bp = op; }
        }
        if (half >= 0) sync();
        const int tw = tid / kWarp;  // warp within the team
        if (lane == 0) { scr.best[tw] = bk; scr.best_slot[tw] = bs; scr.hist[tw] = bp; }
        sync();
        if (half < 0) {
          // whole rows and row pairs: the warp that holds slot B reduces the
          // team's candidates itself (in warp order, as one thread would) and
          // fills the evicted slot; no further barrier (the candidates' next
          // writers are behind the next item's barriers)
          if (tid < kWarp) {
            uint32_t fk = (uint32_t)scr.best[0];
            int fe = scr.best_slot[0], fpos = scr.hist[0];
            for (int w = 1; w < kTeam / kWarp; ++w)
              if (lower(fk, fe, fpos, (uint32_t)scr.best[w], scr.best_slot[w], scr.hist[w])) {
                fk = (uint32_t)scr.best[w]; fe = scr.best_slot[w]; fpos = scr.hist[w];
              }
            if (fe >= 0 && fe < Bsel && slot_ok(fe, 117)) slot_store(p, rbase + fe, tid, mv);
          }
        } else {
        if (tid == 0) {
          uint32_t fk = (uint32_t)scr.best[0];
          int fe = scr.best_slot[0], fpos = scr.hist[0];
          for (int w = 1; w < kTeam / kWarp; ++w)
            if (lower(fk, fe, fpos, (uint32_t)scr.best[w], scr.best_slot[w], scr.hist[w])) {
              fk = (uint32_t)scr.best[w]; fe = scr.best_slot[w]; fpos = scr.hist[w];
            }
          if (half >= 0 && x_ok) {
            int* xs = fs.xsel + (2 * ts + half) * 4;
            xs[0] = (int)fk; xs[1] = fe; xs[2] = fpos;
            __threadfence();
            flag_release(my_flag, ep + 3u);
            if (flag_wait(peer_flag, ep + 3u, abort, p.dbg, 22u, (unsigned)r)) {
              const int* ys = fs.xsel + (2 * ts + (half ^ 1)) * 4;
              const uint32_t ok = (uint32_t)__ldcg(&ys[0]);
              const int oe = __ldcg(&ys[1]), opos = __ldcg(&ys[2]);
              // the same total order on both halves: lower key, then the later position
              if (lower(fk, fe, fpos, ok, oe, opos)) fe = oe;
            } else {
              fe = -1;
            }
          }
          scr.sh[0] = fe;
        }
        sync();
        const int e = scr.sh[0];
        if (mover && e >= 0 && e < Bsel && tid < kWarp && slot_ok(e, 117)) slot_store(p, rbase + e, tid, mv);
        sync();
        }
      } else if (fs.do_evict && Bsel < n) {
        // several evictions (whole rows only): radix select over the scores
        sync();
        team_select_compact<kTeam>(p, r, n, Bsel, LONG && n > max_tok<G>() ? p.score + rbase : scw, tid, scr,
                                   sync);
      }
      if (PERROW && fs.do_evict && tid == 0 && DC_INB(p, r, p.R, 118)) p.rowlen[r] = n < Bsel ? n : Bsel;
    }
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
  if (threadIdx.x == 0 && *abort) atomicOr(p.status, kStatusTimeout);
  if constexpr (GRAPH) {
    // the last CTA to finish (every CTA has read the counter by then)
    // advances the step count for the next launch
    if (threadIdx.x == 0 && atomicAdd(p.gcount + 1, 1) == (int)gridDim.x - 1) {
      p.gcount[1] = 0;
      __threadfence();
      atomicAdd(p.gcount, 1);
    }
  }
}


template <int D, int G, bool LONG, bool FULL = false, bool HEUR = false, bool GLOB = false, bool PERROW = false,
          bool PAIR = false, bool GRAPH = false>
static cudaError_t launch_t(const FusedMaps& maps, const Dev& p, const Step& st, const FusedStep& fs,
                            const FusedPolicy& fp, int grid, cudaStream_t s) {
  constexpr int kSmemBytes = Smem<PAIR, G>::BYTES;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(fused_kernel<D, G, LONG, FULL, HEUR, GLOB, PERROW, PAIR, GRAPH>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  if (fs.half_rows == 0 && !GRAPH)
    return launch_pdl(fused_kernel<D, G, LONG, FULL, HEUR, GLOB, PERROW, PAIR, GRAPH>, dim3(grid), dim3(kThreads),
                      kSmemBytes, s, maps.k, maps.v, maps.k16, maps.v16, p, st, fs, fp);
  if (fs.half_rows == 0) {
    fused_kernel<D, G, LONG, FULL, HEUR, GLOB, PERROW, PAIR, GRAPH>
        <<<grid, kThreads, kSmemBytes, s>>>(maps.k, maps.v, maps.k16, maps.v16, p, st, fs, fp);
    return cudaGetLastError();
  }
  // the two CTAs of a half row wait on each other: a cooperative launch
  // guarantees that the whole grid is resident at once
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmemBytes;
  cfg.stream = s;
  cudaLaunchAttribute la[1];
  la[0].id = cudaLaunchAttributeCooperative;
  la[0].val.cooperative = 1;
  cfg.attrs = la;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, fused_kernel<D, G, LONG, FULL, HEUR, GLOB, PERROW, PAIR, GRAPH>, maps.k, maps.v,
                            maps.k16, maps.v16, p, st, fs, fp);
}

// One CTA per SM, or per row when rows are fewer; two per row when every row
// is split in halves (at most half as many rows as SMs).
inline int fused_grid(const Dev& p, const FusedStep& fs, int num_sms) {
  if (fs.half_rows > 0 && fs.half_rows == p.R && 2 * p.R <= num_sms) return 2 * p.R;
  return p.R < num_sms ? p.R : num_sms;
}

}  // namespace
}  // namespace dc
