// dc_global.cu -- the global token mode (Sec. 3.1.1: a token's features pool
// every attention head of every layer; one policy score and one argtop_B per
// sequence). The rows of a sequence (its layers x KV heads) share one token
// set, slot for slot. The per-row kernels (fused or split engine) leave each
// row's share of the per-token sums in Dev::gpart; here they are pooled per
// sequence, turned into features and scores, and the sequence's selection is
// applied to every one of its rows.
//
// Per-sequence state lives in the sequence's home row (layer 0, KV head 0):
// window sums, cumulative alpha, features and scores; beside it, the ring of
// the last w queries' pooled terms per token (Dev::gring), which moves with
// the tokens.
#include "dc_common.cuh"
#include "dc_kernels.h"
#include "dc_select.cuh"

namespace dc {
namespace {

// The pooling is bound by the latency of each thread's chain of loads (one
// per row it sums), so every token gets 16 threads, each summing 1/16 of the
// sequence's rows (16 of 256 at the Mistral-7B shape).
constexpr int kFeatTok = 32;     // tokens per block
constexpr int kFeatGroups = 16;  // threads per token, each summing 1/16 of the rows
constexpr int kFeatThreads = kFeatTok * kFeatGroups;
constexpr int kPoolBatch = 8;    // rows whose partial sums a thread loads at once
constexpr int kSelThreads = 1024;
constexpr int kMoveThreads = 256;

// A streaming 16-byte load (evict-first: read once) that the compiler keeps
// in program order with the other loads of its batch.
__device__ __forceinline__ float4 ld_stream(const float4* a) {
  float4 v;
  asm volatile("ld.global.cs.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "l"(a));
  return v;
}

__device__ __forceinline__ int seq_row(const Dev& p, int b, int l, int g) { return (l * p.batch + b) * p.kvh + g; }

// grid (ceil(n / kFeatTok), batch), block kFeatTok tokens x kFeatGroups row
// groups; dynamic shared memory: the policy blob, then the groups' partial
// sums. The rows of a sequence are taken in a fixed order (layer-major, then
// KV head): group q sums rows [q S / kFeatGroups, (q + 1) S / kFeatGroups) in
// that order, and the partials are added in group order.
__global__ void __launch_bounds__(kFeatThreads) glob_feature_kernel(Dev p, Step st) {
  extern __shared__ float wsm[];
  const int H = p.hidden, nblob = 9 * H + 1;
  float4* part = reinterpret_cast<float4*>(wsm + ((nblob + 3) & ~3));  // [groups][kFeatTok]
  const int b = blockIdx.y, t = threadIdx.x % kFeatTok, grp = threadIdx.x / kFeatTok;
  const int i = blockIdx.x * kFeatTok + t;
  for (int e = threadIdx.x; e < nblob; e += blockDim.x) wsm[e] = p.policy[e];
  float4 P = make_float4(0.f, 0.f, 0.f, 0.f);
  if (i < st.n) {
    const int S = p.seq_rows, r0 = grp * S / kFeatGroups, r1 = (grp + 1) * S / kFeatGroups;
    int l = r0 / p.kvh, g = r0 % p.kvh;
    // the partial sums of kPoolBatch rows are loaded before any is added (the
    // loads are independent; only the adds are ordered), so that a thread
    // keeps that many loads in flight
    int rr = r0;
    for (; rr + kPoolBatch <= r1; rr += kPoolBatch) {
      float4 q[kPoolBatch];
#pragma unroll
      for (int u = 0; u < kPoolBatch; ++u) {
        q[u] = ld_stream(&p.gpart[(size_t)seq_row(p, b, l, g) * p.stride + i]);
        // the next row without a branch, so that the batch's loads can issue
        // back to back
        const int wrap = (g + 1 == p.kvh) ? 1 : 0;
        g = wrap ? 0 : g + 1;
        l += wrap;
      }
#pragma unroll
      for (int u = 0; u < kPoolBatch; ++u) {
        P.x += q[u].x; P.y += q[u].y; P.z += q[u].z; P.w += q[u].w;
      }
    }
    for (; rr < r1; ++rr) {
      const float4 q = __ldcs(&p.gpart[(size_t)seq_row(p, b, l, g) * p.stride + i]);
      P.x += q.x; P.y += q.y; P.z += q.z; P.w += q.w;
      if (++g == p.kvh) { g = 0; ++l; }
    }
  }
  part[grp * kFeatTok + t] = P;
  __syncthreads();
  if (grp != 0 || i >= st.n) return;
  for (int q = 1; q < kFeatGroups; ++q) {
    const float4 pp = part[q * kFeatTok + t];
    P.x += pp.x; P.y += pp.y; P.z += pp.z; P.w += pp.w;
  }
  const size_t s0 = (size_t)seq_row(p, b, 0, 0) * p.stride + i;
  float4 sz = p.SZ[s0];
  if (st.has_prev || st.has_dep) {
    // the previous step's query joins the stored sums, the departing one
    // (whose ring slot this step's query takes) leaves them: both read from
    // the ring, so the departing terms are exactly those once added
    const float2 pv = st.has_prev ? *gring_at(p, b, st.slot_prev, i) : make_float2(0.f, 0.f);
    const float2 dp = st.has_dep ? *gring_at(p, b, st.slot, i) : make_float2(0.f, 0.f);
    sz = window_update(sz, pv.y, dp.y, pv.x, dp.x);
    p.SZ[s0] = sz;
  }
  // this step's query: total mass and entropy-weighted mass over every head
  *gring_at(p, b, st.slot, i) = make_float2(P.x, P.z);
  const float N = (float)(p.seq_rows * p.G);
  const float mean = P.x / N;
  const float var = fmaxf(P.y / N - mean * mean, 0.f);
  const float Zt = __fadd_rn(__fadd_rn(sz.z, P.x), sz.w);
  const float St = __fadd_rn(__fadd_rn(sz.x, P.z), sz.y);
  float alpha = mean;
  if (p.alpha_mode == 1) {
    alpha = p.acc[s0] + mean;
    p.acc[s0] = alpha;
  }
  const float pos_den = (float)max(st.p_newest, 1);
  const int pos = p.pos[s0];
  float x[5] = {alpha, P.w / (float)p.seq_rows, var, Zt > 0.f ? St / Zt : 0.f, (float)pos / pos_den};
  if (p.keep_features)
#pragma unroll
    for (int e = 0; e < 5; ++e) p.feat[s0 * 5 + e] = x[e];
  p.score[s0] = p.scorer == 0 ? policy_score(wsm, H, p.layernorm, x) : heuristic_score(p, alpha, pos, st.p_newest);
}

// grid (batch), block 1024: the sequence's selection as a move list.
__global__ void __launch_bounds__(kSelThreads) glob_select_kernel(Dev p, int n, int B) {
  __shared__ int hist[256];
  __shared__ int sh[4];
  __shared__ int wsum[kSelThreads / kWarp];
  __shared__ unsigned long long best[kSelThreads / kWarp];
  __shared__ int best_slot[kSelThreads / kWarp];
  const SelectScratch scr{hist, sh, wsum, best, best_slot};
  auto sync = [] { __syncthreads(); };
  const int b = blockIdx.x;
  const size_t base = (size_t)seq_row(p, b, 0, 0) * p.stride;
  int* moves = p.gmoves + (size_t)b * (1 + 2 * (size_t)p.stride);
  team_select_moves<kSelThreads>(p.score + base, p.pos + base, n, B, p.holes + base, moves, threadIdx.x, scr, sync);
}

// grid (R), block 256: every row applies its sequence's moves (one warp per
// move); the home row also moves the sequence's state.
__global__ void __launch_bounds__(kMoveThreads) glob_compact_kernel(Dev p) {
  const int r = blockIdx.x;
  const int b = (r / p.kvh) % p.batch;
  const bool home = r == seq_row(p, b, 0, 0);
  const int* moves = p.gmoves + (size_t)b * (1 + 2 * (size_t)p.stride);
  const int count = moves[0];
  const int lane = threadIdx.x % kWarp, warp = threadIdx.x / kWarp, nwarps = blockDim.x / kWarp;
  const int VPR = p.d / 8;
  const size_t base = (size_t)r * p.stride;
  for (int k = warp; k < count; k += nwarps) {
    const size_t dst = base + moves[1 + 2 * k], src = base + moves[2 + 2 * k];
    uint4 kv = make_uint4(0, 0, 0, 0);
    if (lane < VPR) kv = reinterpret_cast<const uint4*>(p.K)[src * VPR + lane];
    else if (lane < 2 * VPR) kv = reinterpret_cast<const uint4*>(p.V)[src * VPR + lane - VPR];
    const int ps = p.pos[src];
    const float vn = p.vnorm[src];
    float4 sz = make_float4(0.f, 0.f, 0.f, 0.f);
    float ac = 0.f, sc = 0.f, ft = 0.f;
    if (home) {
      sz = p.SZ[src];
      sc = p.score[src];
      if (p.acc) ac = p.acc[src];
      if (p.keep_features && lane < 5) ft = p.feat[src * 5 + lane];
    }
    if (lane < VPR) reinterpret_cast<uint4*>(p.K)[dst * VPR + lane] = kv;
    else if (lane < 2 * VPR) reinterpret_cast<uint4*>(p.V)[dst * VPR + lane - VPR] = kv;
    if (lane == 0) {
      p.pos[dst] = ps;
      p.vnorm[dst] = vn;
      if (home) {
        p.SZ[dst] = sz;
        p.score[dst] = sc;
        if (p.acc) p.acc[dst] = ac;
      }
    }
    if (home && p.keep_features && lane < 5) p.feat[dst * 5 + lane] = ft;
    if (home) {
      const size_t id = dst - base, is = src - base;
      for (int e = lane; e < p.w; e += kWarp) *gring_at(p, b, e, id) = *gring_at(p, b, e, is);
    }
  }
}

}  // namespace

void launch_glob_features(const Dev& p, const Step& st, cudaStream_t s) {
  const dim3 grid((st.n + kFeatTok - 1) / kFeatTok, p.batch);
  const size_t smem = (size_t)((9 * p.hidden + 1 + 3) & ~3) * sizeof(float) + kFeatGroups * kFeatTok * sizeof(float4);
  glob_feature_kernel<<<grid, kFeatThreads, smem, s>>>(p, st);
}

void launch_glob_evict(const Dev& p, int n, int B, cudaStream_t s) {
  glob_select_kernel<<<p.batch, kSelThreads, 0, s>>>(p, n, B);
  glob_compact_kernel<<<p.R, kMoveThreads, 0, s>>>(p);
}

}  // namespace dc
