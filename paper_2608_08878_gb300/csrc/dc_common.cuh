// dc_common.cuh -- device-side layout, parameters and shared arithmetic of the
// DistillCache decode step (sm_103a).
//
// Row r = (layer * batch + b) * kv_heads + g owns `cap` slots. Per-slot data:
//   K, V   bf16 [R][cap][d]      keys / values
//   pos    int32 [R][cap]        absolute position (tokens seen before it)
//   S, Z   fp64 [R][cap]         window sums of the entropy feature H_i over
//                                the window's queries BEFORE the last step
//                                (the last step's terms are added, and the
//                                departing query's subtracted, by the next
//                                step's attention pass; both are recomputed
//                                by the same code, so they cancel bit for bit)
//   acc    fp32 [R][cap]         cumulative alpha (alpha_mode 1 only)
//   score  fp32 [R][cap]         policy score of the last decode step
// Per-row ring of the last w decode queries (the window of H_i, Sec. 3.1.1):
//   ring_q     bf16 [R][w][G][d] the query vectors
//   ring_stats fp32 [R][w][G][4] (m, l, H, 0): max raw logit, softmax
//              denominator 2^((s-m)c) summed, entropy in nats
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace dc {

constexpr int kWarp = 32;

// Device status word bits (read back by dc_sync).
constexpr unsigned kStatusBadShape = 1u;
constexpr unsigned kStatusTimeout = 2u;

struct Dev {
  int R, cap, d, G, qh, kvh, w, hidden, layernorm, alpha_mode, keep_features;
  __nv_bfloat16* K;
  __nv_bfloat16* V;
  int* pos;
  double* S;
  double* Z;
  float* acc;
  float* score;
  float* feat;
  float* hq;
  __nv_bfloat16* ring_q;
  float* ring_stats;
  const float* policy;
  unsigned* status;
  // scratch of the split engine
  float* logit;   // [R][cap][G]
  float* part;    // [R][smax][G][4]: per-split (m, l, u2, 0)
  float* opart;   // [R][smax][G][d]
  int* holes;     // [R][cap]
  int smax;
  float c;        // log2(e) / sqrt(d): raw logit difference -> log2 units
};

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

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Attention weight a = 2^((s - m) c) / l of a token with raw logit s under a
// query whose max raw logit is m and whose denominator is l. Written with
// explicitly rounded operations so that the value is bit-identical wherever
// it is evaluated: the term a query adds to Z_i and S_i at its own step is
// subtracted again, bit for bit, when it leaves the window w steps later.
__device__ __forceinline__ float attn_weight(float s, float m, float c, float l) {
  return __fdiv_rn(ex2(__fmul_rn(__fsub_rn(s, m), c)), l);
}

// (Z, S) terms of one query step for one token: sum over heads of a_h and of
// a_h * H_h, accumulated in head order with rounded adds (see attn_weight).
template <int G>
__device__ __forceinline__ void window_terms(const float* s, const float* m, const float* l,
                                             const float* H, float c, float& z, float& sh) {
  z = 0.f;
  sh = 0.f;
#pragma unroll
  for (int h = 0; h < G; ++h) {
    float a = attn_weight(s[h], m[h], c, l[h]);
    z = __fadd_rn(z, a);
    sh = __fadd_rn(sh, __fmul_rn(a, H[h]));
  }
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

}  // namespace dc
