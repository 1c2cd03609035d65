// synth.cu -- device implementation of the seeded synthetic-input generator
// (a separate library, libdc_synth.so; it is not part of the decode step and
// holds none of its arithmetic). It follows the same published definition as
// the host generator in synth.py, so both produce identical bits:
//   splitmix64 (Steele, Lea, Flood); stream key mix(tag, w...) folds each word
//   as h = splitmix64(h ^ w); a normal is the Irwin-Hall sum of twelve 16-bit
//   uniforms from splitmix64(key + 3j + c), c = 0..2, as (sum - 393210) / 65536;
//   bf16 by round-to-nearest-even; fp32 products and sums each rounded once.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

extern "C" {
typedef struct {
  int layers, batch, kv_heads, q_heads, head_dim;
  int n_sinks, hot_sets, epoch_len;
  float sink_scale, hh_scale, q_align;
  unsigned long long seed;
} dcs_workload;
}

namespace {

constexpr uint64_t TAG_KEY = 0x4B455900ull, TAG_VAL = 0x56414C00ull, TAG_DIR = 0x44495200ull,
                   TAG_HOT = 0x484F5400ull, TAG_QRY = 0x51525900ull, TAG_KNEW = 0x4B4E5700ull,
                   TAG_VNEW = 0x564E5700ull;

__device__ __forceinline__ uint64_t sm64(uint64_t x) {
  uint64_t z = x + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__device__ __forceinline__ uint64_t mix4(uint64_t tag, uint64_t a, uint64_t b, uint64_t c, uint64_t d) {
  uint64_t h = sm64(tag);
  h = sm64(h ^ a);
  h = sm64(h ^ b);
  h = sm64(h ^ c);
  h = sm64(h ^ d);
  return h;
}

__device__ __forceinline__ float normal(uint64_t key, uint64_t j) {
  const uint64_t base = key + 3ull * j;
  int64_t total = 0;
#pragma unroll
  for (int c = 0; c < 3; ++c) {
    const uint64_t w = sm64(base + (uint64_t)c);
    total += (int64_t)(w & 0xFFFF) + (int64_t)((w >> 16) & 0xFFFF) + (int64_t)((w >> 32) & 0xFFFF) +
             (int64_t)(w >> 48);
  }
  return (float)(total - 393210) / 65536.0f;
}

__device__ __forceinline__ void row_coords(const dcs_workload& w, int r, int& layer, int& b, int& g) {
  g = r % w.kv_heads;
  b = (r / w.kv_heads) % w.batch;
  layer = r / (w.kv_heads * w.batch);
}

// One thread = 8 consecutive dims of one (row, token).
__global__ void prompt_kernel(dcs_workload w, long long t0, int T, __nv_bfloat16* __restrict__ k,
                              __nv_bfloat16* __restrict__ v, long long total) {
  const int vpr = w.head_dim / 8;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const int j8 = (int)(e % vpr);
    const long long rt = e / vpr;
    const int tt = (int)(rt % T);
    const int r = (int)(rt / T);
    const uint64_t t = (uint64_t)(t0 + tt);
    int layer, b, g;
    row_coords(w, r, layer, b, g);
    const uint64_t kkey = sm64(mix4(TAG_KEY, w.seed, layer, b, g) ^ t);
    const uint64_t vkey = sm64(mix4(TAG_VAL, w.seed, layer, b, g) ^ t);
    int hot = -1;
    if ((long long)t >= w.n_sinks && w.hot_sets > 0) {
      const uint64_t hh = sm64(mix4(TAG_HOT, w.seed, layer, b, g) + t) % 100ull;
      if ((int)hh < w.hot_sets) hot = (int)hh;
    }
    uint64_t dkey = 0;
    if (hot >= 0) {
      uint64_t h = mix4(TAG_DIR, w.seed, layer, b, g);
      dkey = sm64(h ^ (uint64_t)hot);
    }
    __align__(16) __nv_bfloat16 kb[8], vb[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const uint64_t j = (uint64_t)(j8 * 8 + q);
      const float nk = normal(kkey, j);
      float kv;
      if ((long long)t < w.n_sinks) kv = __fmul_rn(w.sink_scale, nk);
      else if (hot >= 0) kv = __fadd_rn(__fmul_rn(w.hh_scale, normal(dkey, j)), nk);
      else kv = nk;
      kb[q] = __float2bfloat16_rn(kv);
      vb[q] = __float2bfloat16_rn(normal(vkey, j));
    }
    const size_t o = (size_t)rt * w.head_dim + j8 * 8;
    *reinterpret_cast<uint4*>(k + o) = *reinterpret_cast<const uint4*>(kb);
    *reinterpret_cast<uint4*>(v + o) = *reinterpret_cast<const uint4*>(vb);
  }
}

// One thread = one element of q [L][b][qh][d] (or of k_new/v_new when e >= nq).
__global__ void step_kernel(dcs_workload w, long long step, __nv_bfloat16* __restrict__ q,
                            __nv_bfloat16* __restrict__ kn, __nv_bfloat16* __restrict__ vn) {
  const int d = w.head_dim, G = w.q_heads / w.kv_heads;
  const long long nq = (long long)w.layers * w.batch * w.q_heads * d;
  const long long nk = (long long)w.layers * w.batch * w.kv_heads * d;
  const int hs = w.hot_sets > 0 ? w.hot_sets : 1;
  const uint64_t epoch = (uint64_t)((step / w.epoch_len) % hs);
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < nq + nk;
       e += (long long)gridDim.x * blockDim.x) {
    if (e < nq) {
      const int j = (int)(e % d);
      const long long hrow = e / d;  // (layer, b, head)
      const int head = (int)(hrow % w.q_heads);
      const int b = (int)((hrow / w.q_heads) % w.batch);
      const int layer = (int)(hrow / ((long long)w.q_heads * w.batch));
      const int g = head / G;
      const uint64_t dkey = sm64(mix4(TAG_DIR, w.seed, layer, b, g) ^ epoch);
      const uint64_t qkey = sm64(mix4(TAG_QRY, w.seed, layer, b, head) ^ (uint64_t)step);
      const float u = normal(dkey, j);
      q[e] = __float2bfloat16_rn(__fadd_rn(__fmul_rn(w.q_align, u), normal(qkey, j)));
    } else {
      const long long f = e - nq;
      const int j = (int)(f % d);
      const int r = (int)(f / d);
      int layer, b, g;
      row_coords(w, r, layer, b, g);
      kn[f] = __float2bfloat16_rn(normal(sm64(mix4(TAG_KNEW, w.seed, layer, b, g) ^ (uint64_t)step), j));
      vn[f] = __float2bfloat16_rn(normal(sm64(mix4(TAG_VNEW, w.seed, layer, b, g) ^ (uint64_t)step), j));
    }
  }
}

}  // namespace

extern "C" {

// Fills k, v (bf16 [R][T][d], device) with the prompt tokens at positions
// [t0, t0 + T) of every row. Returns a cudaError_t value (0 = success).
int dcs_prompt(const dcs_workload* w, long long t0, int T, void* k, void* v, void* stream) {
  const long long total = (long long)w->layers * w->batch * w->kv_heads * T * (w->head_dim / 8);
  if (total <= 0) return 0;
  prompt_kernel<<<152 * 16, 256, 0, (cudaStream_t)stream>>>(*w, t0, T, (__nv_bfloat16*)k,
                                                             (__nv_bfloat16*)v, total);
  return (int)cudaGetLastError();
}

// Fills q (bf16 [L][b][qh][d]), k_new and v_new (bf16 [L][b][kvh][d]) of a decode step.
int dcs_step(const dcs_workload* w, long long step, void* q, void* k_new, void* v_new, void* stream) {
  step_kernel<<<152 * 8, 256, 0, (cudaStream_t)stream>>>(*w, step, (__nv_bfloat16*)q,
                                                          (__nv_bfloat16*)k_new, (__nv_bfloat16*)v_new);
  return (int)cudaGetLastError();
}

}  // extern "C"
