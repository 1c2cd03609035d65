// dc_common.cuh -- device-side layout, parameters and shared arithmetic of the
// DistillCache decode step (sm_103a).
//
// Row r = (layer * batch + b) * kv_heads + g owns `cap` slots, laid out with a
// row stride of `stride` slots (cap rounded up to 128, so that every 128-token
// tile of a row is 16-byte aligned and stays inside the row). Per-slot data:
//   K, V   bf16 [R][stride][d]   keys / values
//   pos    int32 [R][stride]     absolute position (tokens seen before it)
//   vnorm  fp32 [R][stride]      |v_i|_2, computed once when the token is appended
//   SZ     fp32x4 [R][stride]    window sums of the entropy feature H_i as
//                                double-float pairs (S_hi, S_lo, Z_hi, Z_lo),
//                                over the window's queries BEFORE the last step
//                                (the last step's terms are added, and the
//                                departing query's subtracted, by the next
//                                step's attention pass; both are recomputed
//                                by the same code, so they cancel bit for bit)
//   acc    fp32 [R][stride]      cumulative alpha (alpha_mode 1 only)
//   score  fp32 [R][stride]      policy score of the last decode step
// Per-row ring of the last w decode queries (the window of H_i, Sec. 3.1.1):
//   ring_q     bf16 [R][w][G][d] the query vectors
//   ring_stats fp32 [R][w][G][4] (m, l, H, nl): max raw logit, softmax
//              denominator sum of 2^((s-m)c), entropy in nats, -log2(l)
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace dc {

constexpr int kWarp = 32;

// Device status word bits (read back by dc_sync).
constexpr unsigned kStatusBadShape = 1u;
constexpr unsigned kStatusTimeout = 2u;
constexpr unsigned kStatusBounds = 4u;  // debug builds: an index check failed

// Debug builds (DC_DEBUG_BOUNDS) check computed global-memory indices before
// the access: DC_INB(p, i, lim, site) is false when i is outside [0, lim),
// after raising kStatusBounds and recording the first failure (site, low 32
// bits of the index, limit) in dbg[5..7]; the caller then skips the access.
// Release builds compile it to `true`.
#ifdef DC_DEBUG_BOUNDS
__device__ __forceinline__ bool in_bounds(long long i, long long lim, unsigned* status, unsigned* dbg,
                                          unsigned site) {
  if (i >= 0 && i < lim) return true;
  if (status) atomicOr(status, kStatusBounds);
  if (dbg && atomicCAS(dbg + 5, 0u, site) == 0u) {
    dbg[6] = (unsigned)i;
    dbg[7] = (unsigned)lim;
  }
  return false;
}
#define DC_INB(p, i, lim, site) ::dc::in_bounds((long long)(i), (long long)(lim), (p).status, (p).dbg, (site))
#else
#define DC_INB(p, i, lim, site) true
#endif

struct Dev {
  int R, cap, stride, d, G, qh, kvh, w, hidden, layernorm, alpha_mode, keep_features;
  int scorer, n_sinks;  // 0 policy MLP, 1 H2O (cumulative alpha), 2 StreamingLLM
  // global token mode: rows per sequence (layers x KV heads), 0 = per-row mode;
  // batch = sequences. Per-token partial sums of each row ([R][stride]
  // float4: this step's attention mass, squared mass, entropy-weighted mass
  // and |v|); per sequence, the pooled contribution (mass, entropy-weighted
  // mass) of each of the last w queries to every token ([batch][w][stride]
  // float2, ring slot = step mod w, zero for a token not yet cached at that
  // step), from which the window sums gain the previous query's terms and lose
  // the departing query's exactly; and each sequence's move list
  // ([batch][1 + 2 stride]: count, then hole/mover pairs).
  int seq_rows, batch;
  float4* gpart;
  float2* gring;
  int* gmoves;
  // per-row budgets (head-level hybrid): each row's length and budget on the
  // device ([R] each); null when every row has the same length
  int* rowlen;
  int* rowbudget;
  // per-row mode: the order in which the fused engine's queue hands out rows
  // (longest first, so that no long row starts last); null: row order
  const int* roworder;
  // device-counted steps (CUDA-graph replay): [0] steps taken since the mode
  // was entered, added by the append and fused kernels to the host's base
  // step arguments; [1] CTAs of the current fused launch that have finished
  // (the last one advances [0]); null outside the mode
  int* gcount;
  __nv_bfloat16* K;
  __nv_bfloat16* V;
  int* pos;
  float* vnorm;
  float4* SZ;
  float* acc;
  float* score;
  float* feat;
  float* hq;
  __nv_bfloat16* ring_q;
  float* ring_stats;
  const float* policy;
  unsigned* status;
  unsigned* dbg;  // [8]: first wait timeout of a launch (site, block, parity, info)
  // scratch of the split engine
  float* logit;   // [R][stride][G]
  float* part;    // [R][smax][G][4]: per-split (m, l, u2, 0)
  float* opart;   // [R][smax][G][d]
  int* holes;     // [R][stride]
  int* nmoves;    // [R][2]: the eviction kernel's move count and hole count per row
  int smax;
  float c;        // log2(e) / sqrt(d): raw logit difference -> log2 units
};

// Ring entry (ring slot k, token slot i) of sequence b.
__host__ __device__ inline float2* gring_at(const Dev& p, int b, int k, size_t i) {
  return p.gring + ((size_t)b * p.w + k) * p.stride + i;
}

// Arguments that change every step.
struct Step {
  int n;          // tokens per row after the append
  int p_newest;   // position of the newest token
  int slot;       // ring slot of this step (= slot of the departing query)
  int has_dep;    // a query leaves the window this step (step t - w)
  int p_dep;      // newest position at the departing query's step
  int has_prev;   // the previous step's query joins the stored sums (step t - 1)
  int slot_prev;  // its ring slot
  int p_prev;     // newest position at the previous step
  int nsplit;     // splits per row (split engine)
  int chunk;      // tokens per split
};

// Programmatic dependent launch (a grid launched with the programmatic
// stream serialization attribute may start while the grid before it in the
// stream still runs): grid_dep_wait returns once the grids this one depends
// on have completed and their writes are visible (at once when there are
// none); grid_dep_launch lets the grid after this one start launching.
__device__ __forceinline__ void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_dep_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Launches f with programmatic stream serialization: the grid may start while
// the grid before it in the stream runs, and waits for it in grid_dep_wait.
template <class... KArgs, class... Args>
inline cudaError_t launch_pdl(void (*f)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                              Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute la[1];
  la[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  la[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = la;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, f, static_cast<Args&&>(args)...);
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Hardware base-2 logarithm (lg2.approx, relative error ~2^-22).
__device__ __forceinline__ float lg2_approx(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Attention weight a = 2^((s - m) c) / l = 2^((s - m) c + nl), nl = -log2(l),
// of a token with raw logit s under a query whose max raw logit is m. Written
// with explicitly rounded operations so that the value is bit-identical
// wherever it is evaluated: the term a query adds to the window sums one step
// after its own is subtracted again, bit for bit, when it leaves the window.
__device__ __forceinline__ float attn_weight(float s, float m, float c, float nl) {
  return ex2(__fmaf_rn(__fsub_rn(s, m), c, nl));
}

// (Z, S) terms of one query step for one token: sum over heads of a_h and of
// a_h * H_h, accumulated in head order with rounded adds (see attn_weight).
template <int G>
__device__ __forceinline__ void window_terms(const float* s, const float* m, const float* nl,
                                             const float* H, float c, float& z, float& sh) {
  z = 0.f;
  sh = 0.f;
#pragma unroll
  for (int h = 0; h < G; ++h) {
    float a = attn_weight(s[h], m[h], c, nl[h]);
    z = __fadd_rn(z, a);
    sh = __fadd_rn(sh, __fmul_rn(a, H[h]));
  }
}

// Double-float accumulation (a value held as an unevaluated sum hi + lo, about
// 48 significant bits): (hi, lo) += x with Knuth's TwoSum and a renormalising
// Fast2Sum. The window sums stay exact enough that adding a term and
// subtracting the same term many steps later leaves no visible residue.
__device__ __forceinline__ void df_add(float& hi, float& lo, float x) {
  const float s = __fadd_rn(hi, x);
  const float bb = __fsub_rn(s, hi);
  const float e = __fadd_rn(__fsub_rn(hi, __fsub_rn(s, bb)), __fsub_rn(x, bb));
  const float t = __fadd_rn(e, lo);
  hi = __fadd_rn(s, t);
  lo = __fsub_rn(t, __fsub_rn(hi, s));
}

// Window sums after this step's update: S += sp - sd, Z += zp - zd.
__device__ __forceinline__ float4 window_update(float4 sz, float sp, float sd, float zp, float zd) {
  df_add(sz.x, sz.y, sp);
  df_add(sz.x, sz.y, -sd);
  df_add(sz.z, sz.w, zp);
  df_add(sz.z, sz.w, -zd);
  return sz;
}

// Order-preserving 32-bit key of a score for the top-B selection: larger key =
// higher rank. -0 maps to +0's key; NaN maps to 0, below every number.
__device__ __forceinline__ uint32_t score_key(float s) {
  if (s != s) return 0u;
  uint32_t b = __float_as_uint(s);
  if (b == 0x80000000u) b = 0u;
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

__device__ __forceinline__ float bf16lo(uint32_t u) { return __uint_as_float(u << 16); }
__device__ __forceinline__ float bf16hi(uint32_t u) { return __uint_as_float(u & 0xFFFF0000u); }

// Policy MLP on one feature vector (Sec. 3.1.2; App. D): weights in shared
// memory, blob layout [W1 (H x 5) | b1 | gamma | beta | w2 | b2].
__device__ __forceinline__ float policy_score(const float* __restrict__ wsm, int H, int layernorm,
                                              const float x[5]) {
  const float* W1 = wsm;
  const float* b1 = W1 + 5 * H;
  const float* gamma = b1 + H;
  const float* beta = gamma + H;
  const float* w2 = beta + H;
  float out = w2[H];
  if (layernorm) {
    float sum = 0.f, sq = 0.f;
    for (int j = 0; j < H; ++j) {
      float h = b1[j];
#pragma unroll
      for (int c = 0; c < 5; ++c) h = fmaf(W1[j * 5 + c], x[c], h);
      sum += h;
      sq = fmaf(h, h, sq);
    }
    float mu = sum / (float)H;
    float var = fmaxf(sq / (float)H - mu * mu, 0.f);
    float rstd = rsqrtf(var + 1e-5f);
    for (int j = 0; j < H; ++j) {
      float h = b1[j];
#pragma unroll
      for (int c = 0; c < 5; ++c) h = fmaf(W1[j * 5 + c], x[c], h);
      float y = fmaf((h - mu) * rstd, gamma[j], beta[j]);
      out = fmaf(w2[j], fmaxf(y, 0.f), out);
    }
  } else {
    for (int j = 0; j < H; ++j) {
      float h = b1[j];
#pragma unroll
      for (int c = 0; c < 5; ++c) h = fmaf(W1[j * 5 + c], x[c], h);
      out = fmaf(w2[j], fmaxf(h, 0.f), out);
    }
  }
  return out;
}

// Scores of the heuristic scorers on the same path: H2O ranks by the
// cumulative attention mass (alpha, accumulated since insertion); StreamingLLM
// keeps the first n_sinks positions, then the most recent tokens (the score is
// the position relative to the newest, exact in fp32 for the last 2^24).
__device__ __forceinline__ float heuristic_score(const Dev& p, float alpha_cum, int pos, int p_newest) {
  if (p.scorer == 1) return alpha_cum;
  return pos < p.n_sinks ? 3.0e38f : (float)(pos - p_newest);
}

}  // namespace dc
