// dc_split.cu -- the split engine: the decode step as separate kernels
// (append; attention logits + window-sum update; softmax statistics;
// attention output + features + policy scores; output combine). Each row's
// tokens are cut into `nsplit` chunks that run as separate CTAs; logits go
// through a global scratch buffer between the passes.
//
// Paper: Algorithm 1 (forward pass over C_t including the new pair, feature
// extraction, scoring); Sec. 3.1.1 (features); Sec. 3.1.2 and App. D (policy).
#include "dc_common.cuh"
#include "dc_kernels.h"

namespace dc {

constexpr int kTile = 128;  // tokens per tile = threads per CTA

// ---------------------------------------------------------------------------
// Append T tokens to every row: slot n0 + t gets k/v[r][t], position
// seen0 + t, |v|_2, zeroed window sums and cumulative alpha.
// grid (T, R), block d/8 threads (one 16-byte vector each of K and V).
// ---------------------------------------------------------------------------
// One (row, token) pair per group of d/8 lanes (16-byte chunks), 256 threads
// per block: pair e = r * T + t goes to slot n0 + t of row r.
__global__ void __launch_bounds__(256) append_kernel(Dev p, const uint4* __restrict__ k,
                                                     const uint4* __restrict__ v, long long pairs, int T,
                                                     int n0, int seen0) {
  // launched after the kernels that wrote k and v, or after the previous
  // step's kernels, which still read the slots written here
  grid_dep_wait();
  // the fused step kernel after this one may start its set-up meanwhile
  grid_dep_launch();
  const int vpr = p.d / 8;
  const long long e = ((long long)blockIdx.x * blockDim.x + threadIdx.x) / vpr;
  const int c = threadIdx.x % vpr;
  const bool live = e < pairs;
  const long long ee = live ? e : pairs - 1;
  const int r = (int)(ee / T), t = (int)(ee % T);
  const size_t src = (size_t)ee * vpr + c;
  const int col = (p.rowlen ? p.rowlen[r] : n0) + t;
  const size_t slot = (size_t)r * p.stride + col;
  const uint4 kv = k[src], vv = v[src];
  if (live && DC_INB(p, col, p.cap, 301) && DC_INB(p, r, p.R, 301)) {
    reinterpret_cast<uint4*>(p.K)[slot * vpr + c] = kv;
    reinterpret_cast<uint4*>(p.V)[slot * vpr + c] = vv;
  }
  const uint32_t w4[4] = {vv.x, vv.y, vv.z, vv.w};
  float ss = 0.f;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const float x0 = bf16lo(w4[q]), x1 = bf16hi(w4[q]);
    ss = fmaf(x0, x0, ss);
    ss = fmaf(x1, x1, ss);
  }
  // xor offsets below vpr stay inside the pair's aligned lane group
  for (int off = 1; off < vpr; off <<= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
  if (live && c == 0 && DC_INB(p, col, p.cap, 302)) {
    // device-counted steps: positions continue from the steps taken since
    p.pos[slot] = seen0 + t + (p.gcount ? *reinterpret_cast<volatile int*>(p.gcount) : 0);
    p.vnorm[slot] = sqrtf(ss);
    p.SZ[slot] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (p.acc) p.acc[slot] = 0.f;
    if (p.seq_rows && r < p.batch * p.kvh && r % p.kvh == 0) {
      // global token mode, the sequence's home row: no past query saw this token
      const int b = r / p.kvh;
      const size_t i = slot - (size_t)r * p.stride;
      for (int k = 0; k < p.w; ++k) *gring_at(p, b, k, i) = make_float2(0.f, 0.f);
    }
  }
}

// Cooperative copy of `rows` rows of d bf16 into shared memory with a row
// pitch of d + 8 elements (conflict-free 16-byte reads by row).
template <int D>
__device__ __forceinline__ void load_tile(__nv_bfloat16 (*dst)[D + 8], const __nv_bfloat16* src,
                                          int rows) {
  constexpr int VPR = D / 8;
  for (int e = threadIdx.x; e < rows * VPR; e += blockDim.x) {
    int rr = e / VPR, cc = e % VPR;
    *reinterpret_cast<uint4*>(&dst[rr][cc * 8]) =
        __ldg(reinterpret_cast<const uint4*>(src) + (size_t)rr * VPR + cc);
  }
}

// Dot products of one key row (shared memory) with NQ fp32 query rows
// (shared memory, [NQ][D]), accumulated in dimension order with fmaf.
template <int D, int NQ>
__device__ __forceinline__ void dots(const __nv_bfloat16* krow, const float (*qs)[D], float* s) {
#pragma unroll
  for (int j = 0; j < NQ; ++j) s[j] = 0.f;
#pragma unroll 2
  for (int c8 = 0; c8 < D / 8; ++c8) {
    uint4 u = *reinterpret_cast<const uint4*>(krow + c8 * 8);
    float kf[8] = {bf16lo(u.x), bf16hi(u.x), bf16lo(u.y), bf16hi(u.y),
                   bf16lo(u.z), bf16hi(u.z), bf16lo(u.w), bf16hi(u.w)};
#pragma unroll
    for (int e = 0; e < 8; ++e)
#pragma unroll
      for (int j = 0; j < NQ; ++j) s[j] = fmaf(qs[j][c8 * 8 + e], kf[e], s[j]);
  }
}

// Online softmax state of one head in log2 units: m = max raw logit,
// l = sum 2^x, u = sum 2^x * x with x = (s - m) * c.
__device__ __forceinline__ void online_add(float& m, float& l, float& u, float s, float c) {
  if (s > m) {
    if (m == -INFINITY) {
      l = 1.f;
      u = 0.f;
    } else {
      const float dl = (m - s) * c, f = ex2(dl);
      u = (u + l * dl) * f;
      l = fmaf(l, f, 1.f);
    }
    m = s;
  } else {
    const float x = (s - m) * c, pe = ex2(x);
    l += pe;
    u = fmaf(pe, x, u);
  }
}

__device__ __forceinline__ void online_merge(float& m, float& l, float& u, float mo, float lo, float uo,
                                             float c) {
  if (mo == -INFINITY) return;
  if (m == -INFINITY) { m = mo; l = lo; u = uo; return; }
  const float M = fmaxf(m, mo), da = (m - M) * c, db = (mo - M) * c;
  const float fa = ex2(da), fb = ex2(db);
  u = (u + l * da) * fa + (uo + lo * db) * fb;
  l = l * fa + lo * fb;
  m = M;
}

__device__ __forceinline__ int row_q_offset(const Dev& p, int r) {
  // q / out index of head 0 of row r's group: [L][b][qh][d] with r = lb*kvh + g
  return ((r / p.kvh) * p.qh + (r % p.kvh) * p.G) * p.d;
}

// ---------------------------------------------------------------------------
// Pass 1: raw logits of the current queries (to scratch), per-split softmax
// statistics (m, l, u2) and the window-sum update: the previous step's query
// joins the stored sums S, Z and the departing one (step t - w) leaves them,
// both recomputed here from their ring entries.
// grid (nsplit, R), block kTile.
// ---------------------------------------------------------------------------
template <int D, int G>
__global__ void __launch_bounds__(kTile) split_qk_kernel(Dev p, Step st,
                                                         const __nv_bfloat16* __restrict__ q) {
  __shared__ float qs[3 * G][D];  // current, previous, departing
  __shared__ __align__(16) __nv_bfloat16 kt[kTile][D + 8];
  __shared__ float ring_ml[2][G][3];  // (m, nl, H) of previous / departing
  __shared__ float red[kTile / kWarp][G][3];
  const int r = blockIdx.y, sp = blockIdx.x, tid = threadIdx.x;
  const int c0 = sp * st.chunk, c1 = min(p.rowlen ? p.rowlen[r] : st.n, c0 + st.chunk);
  const int qo = row_q_offset(p, r);
  const __nv_bfloat16* rq_prev = p.ring_q + ((size_t)r * p.w + st.slot_prev) * G * D;
  const __nv_bfloat16* rq_dep = p.ring_q + ((size_t)r * p.w + st.slot) * G * D;
  for (int e = tid; e < G * D; e += blockDim.x) {
    qs[e / D][e % D] = __bfloat162float(q[qo + e]);
    qs[G + e / D][e % D] = st.has_prev ? __bfloat162float(rq_prev[e]) : 0.f;
    qs[2 * G + e / D][e % D] = st.has_dep ? __bfloat162float(rq_dep[e]) : 0.f;
  }
  if (tid < 2 * G) {
    const int which = tid / G, h = tid % G;
    const int slot = which == 0 ? st.slot_prev : st.slot;
    const float* rs = p.ring_stats + (((size_t)r * p.w + slot) * G + h) * 4;
    ring_ml[which][h][0] = rs[0];
    ring_ml[which][h][1] = rs[3];
    ring_ml[which][h][2] = rs[2];
  }
  float m[G], l[G], u[G];
#pragma unroll
  for (int h = 0; h < G; ++h) { m[h] = -INFINITY; l[h] = 0.f; u[h] = 0.f; }
  const float c = p.c;
  for (int base = c0; base < c1; base += kTile) {
    const int rows = min(kTile, c1 - base);
    __syncthreads();
    load_tile<D>(kt, p.K + ((size_t)r * p.stride + base) * D, rows);
    __syncthreads();
    if (tid < rows && DC_INB(p, base + tid, p.stride, 311) && DC_INB(p, r, p.R, 311)) {
      const size_t slot = (size_t)r * p.stride + base + tid;
      float s[3 * G];
      dots<D, 3 * G>(&kt[tid][0], qs, s);
      float* lo = p.logit + slot * G;
#pragma unroll
      for (int h = 0; h < G; ++h) {
        lo[h] = s[h];
        online_add(m[h], l[h], u[h], s[h], c);
      }
      // global token mode: the window sums come from the sequence's ring
      if (!p.seq_rows && (st.has_prev || st.has_dep)) {
        const int pos = p.pos[slot];
        float zp = 0.f, sp_ = 0.f, zd = 0.f, sd = 0.f;
        float rm[G], rnl[G], rH[G];
        if (st.has_prev && pos <= st.p_prev) {
#pragma unroll
          for (int h = 0; h < G; ++h) { rm[h] = ring_ml[0][h][0]; rnl[h] = ring_ml[0][h][1]; rH[h] = ring_ml[0][h][2]; }
          window_terms<G>(s + G, rm, rnl, rH, c, zp, sp_);
        }
        if (st.has_dep && pos <= st.p_dep) {
#pragma unroll
          for (int h = 0; h < G; ++h) { rm[h] = ring_ml[1][h][0]; rnl[h] = ring_ml[1][h][1]; rH[h] = ring_ml[1][h][2]; }
          window_terms<G>(s + 2 * G, rm, rnl, rH, c, zd, sd);
        }
        p.SZ[slot] = window_update(p.SZ[slot], sp_, sd, zp, zd);
      }
    }
  }
  // Merge the per-thread (m, l, u2) of each head across the CTA.
  const int lane = tid % kWarp, wid = tid / kWarp;
#pragma unroll
  for (int h = 0; h < G; ++h) {
    float mm = m[h], ll = l[h], uu = u[h];
    for (int off = 16; off > 0; off >>= 1) {
      float mo = __shfl_xor_sync(0xffffffffu, mm, off);
      float lo_ = __shfl_xor_sync(0xffffffffu, ll, off);
      float uo = __shfl_xor_sync(0xffffffffu, uu, off);
      online_merge(mm, ll, uu, mo, lo_, uo, c);
    }
    if (lane == 0) { red[wid][h][0] = mm; red[wid][h][1] = ll; red[wid][h][2] = uu; }
  }
  __syncthreads();
  if (tid < G) {
    const int h = tid;
    float M = -INFINITY, L = 0.f, U = 0.f;
    for (int wv = 0; wv < kTile / kWarp; ++wv) online_merge(M, L, U, red[wv][h][0], red[wv][h][1], red[wv][h][2], c);
    float* pp = p.part + (((size_t)r * p.smax + sp) * G + h) * 4;
    if (DC_INB(p, sp, p.smax, 312)) { pp[0] = M; pp[1] = L; pp[2] = U; pp[3] = 0.f; }
  }
}

// ---------------------------------------------------------------------------
// Softmax statistics of the whole row: merge the splits, entropy
// H = ln l - ln2 * u2 / l, push (q, m, l, H) into the ring slot of this step.
// grid (R), block 128.
// ---------------------------------------------------------------------------
template <int D, int G>
__global__ void split_stats_kernel(Dev p, Step st, const __nv_bfloat16* __restrict__ q) {
  const int r = blockIdx.x, tid = threadIdx.x;
  const int qo = row_q_offset(p, r);
  __nv_bfloat16* rq = p.ring_q + ((size_t)r * p.w + st.slot) * G * D;
  if (!(DC_INB(p, (long long)r * p.w + st.slot, (long long)p.R * p.w, 316) &&
        DC_INB(p, (long long)qo + G * D - 1, (long long)(p.R / p.kvh) * p.qh * D, 316)))
    return;
  for (int e = tid; e < G * D; e += blockDim.x) rq[e] = q[qo + e];
  if (tid < G) {
    const int h = tid;
    const float c = p.c;
    float M = -INFINITY, L = 0.f, U = 0.f;
    for (int sp = 0; sp < st.nsplit; ++sp) {
      const float* pp = p.part + (((size_t)r * p.smax + sp) * G + h) * 4;
      online_merge(M, L, U, pp[0], pp[1], pp[2], c);
    }
    float H = logf(L) - 0.69314718055994531f * (U / L);
    float* rs = p.ring_stats + (((size_t)r * p.w + st.slot) * G + h) * 4;
    rs[0] = M; rs[1] = L; rs[2] = H; rs[3] = -log2f(L);
    p.hq[(size_t)r * G + h] = H;
  }
}

// ---------------------------------------------------------------------------
// Pass 2: attention weights with the row's final statistics, per-split
// attention output, the five features, window-sum update and policy score.
// grid (nsplit, R), block kTile. Dynamic shared memory: policy blob.
// ---------------------------------------------------------------------------
template <int D, int G>
__global__ void __launch_bounds__(kTile) split_v_kernel(Dev p, Step st) {
  extern __shared__ float wsm[];
  __shared__ __align__(16) __nv_bfloat16 vt[kTile][D + 8];
  __shared__ float at[kTile][G];
  __shared__ float stat[G][3];  // (m, nl, H)
  const int r = blockIdx.y, sp = blockIdx.x, tid = threadIdx.x;
  const int c0 = sp * st.chunk, c1 = min(p.rowlen ? p.rowlen[r] : st.n, c0 + st.chunk);
  const int H = p.hidden, nblob = 9 * H + 1;
  for (int e = tid; e < nblob; e += blockDim.x) wsm[e] = p.policy[e];
  if (tid < G) {
    const float* rs = p.ring_stats + (((size_t)r * p.w + st.slot) * G + tid) * 4;
    stat[tid][0] = rs[0]; stat[tid][1] = rs[3]; stat[tid][2] = rs[2];
  }
  constexpr int NOUT = G * D;
  constexpr int OPT = NOUT >= kTile ? NOUT / kTile : 1;  // outputs per thread
  const int o0 = tid * OPT;
  const bool owns = o0 < NOUT;
  const int oh = owns ? o0 / D : 0, oc = owns ? o0 % D : 0;
  float oacc[OPT];
#pragma unroll
  for (int e = 0; e < OPT; ++e) oacc[e] = 0.f;
  const float c = p.c;
  const float pos_den = (float)max(st.p_newest, 1);
  for (int base = c0; base < c1; base += kTile) {
    const int rows = min(kTile, c1 - base);
    __syncthreads();
    load_tile<D>(vt, p.V + ((size_t)r * p.stride + base) * D, rows);
    __syncthreads();
    if (tid < rows && DC_INB(p, base + tid, p.stride, 313) && DC_INB(p, r, p.R, 313)) {
      const size_t slot = (size_t)r * p.stride + base + tid;
      const float* lo = p.logit + slot * G;
      float a[G], mean = 0.f;
      float zc = 0.f, sc = 0.f;
      {
        float s[G], mm[G], nl[G], hh[G];
#pragma unroll
        for (int h = 0; h < G; ++h) { s[h] = lo[h]; mm[h] = stat[h][0]; nl[h] = stat[h][1]; hh[h] = stat[h][2]; }
        window_terms<G>(s, mm, nl, hh, c, zc, sc);
#pragma unroll
        for (int h = 0; h < G; ++h) {
          a[h] = attn_weight(s[h], mm[h], c, nl[h]);
          at[tid][h] = a[h];
          mean += a[h];
        }
      }
      if (p.seq_rows) {
        // global token mode: this row's share of the pooled per-token sums
        float a2 = 0.f;
#pragma unroll
        for (int h = 0; h < G; ++h) a2 = fmaf(a[h], a[h], a2);
        p.gpart[slot] = make_float4(mean, a2, sc, p.vnorm[slot]);
      } else {
      mean /= (float)G;
      float var = 0.f;
#pragma unroll
      for (int h = 0; h < G; ++h) var = fmaf(a[h] - mean, a[h] - mean, var);
      var /= (float)G;
      const float vn = p.vnorm[slot];
      // H_i over the whole window: stored sums (earlier queries) + this step
      const float4 sz = p.SZ[slot];
      const float Zt = __fadd_rn(__fadd_rn(sz.z, zc), sz.w);
      const float St = __fadd_rn(__fadd_rn(sz.x, sc), sz.y);
      float alpha = mean;
      if (p.alpha_mode == 1) {
        alpha = p.acc[slot] + mean;
        p.acc[slot] = alpha;
      }
      float Hi = Zt > 0.f ? St / Zt : 0.f;
      float x[5] = {alpha, vn, var, Hi, (float)p.pos[slot] / pos_den};
      if (p.keep_features) {
#pragma unroll
        for (int e = 0; e < 5; ++e) p.feat[slot * 5 + e] = x[e];
      }
      p.score[slot] = p.scorer == 0 ? policy_score(wsm, H, p.layernorm, x)
                                    : heuristic_score(p, alpha, p.pos[slot], st.p_newest);
      }
    }
    __syncthreads();
    if (owns) {
      for (int i = 0; i < rows; ++i) {
        const float ai = at[i][oh];
        if constexpr (OPT % 2 == 0) {
#pragma unroll
          for (int e = 0; e < OPT; e += 2) {
            uint32_t u2 = *reinterpret_cast<const uint32_t*>(&vt[i][oc + e]);
            oacc[e] = fmaf(ai, bf16lo(u2), oacc[e]);
            oacc[e + 1] = fmaf(ai, bf16hi(u2), oacc[e + 1]);
          }
        } else {
#pragma unroll
          for (int e = 0; e < OPT; ++e) oacc[e] = fmaf(ai, __bfloat162float(vt[i][oc + e]), oacc[e]);
        }
      }
    }
  }
  if (owns && DC_INB(p, sp, p.smax, 314)) {
    float* op = p.opart + (((size_t)r * p.smax + sp) * G) * D + o0;
#pragma unroll
    for (int e = 0; e < OPT; ++e) op[e] = oacc[e];
  }
}

// ---------------------------------------------------------------------------
// out = sum over splits of the per-split outputs (weights were normalised with
// the final statistics). grid (R), block G*D.
// ---------------------------------------------------------------------------
template <int D, int G>
__global__ void split_out_kernel(Dev p, Step st, float* __restrict__ out) {
  const int r = blockIdx.x;
  for (int e = threadIdx.x; e < G * D; e += blockDim.x) {
    float s = 0.f;
    for (int sp = 0; sp < st.nsplit; ++sp) s += p.opart[(((size_t)r * p.smax + sp) * G) * D + e];
    if (DC_INB(p, row_q_offset(p, r) + e, (long long)(p.R / p.kvh) * p.qh * D, 315)) out[row_q_offset(p, r) + e] = s;
  }
}

// ---------------------------------------------------------------------------
// Window sums as fp64 [nrows][cap] (hi + lo of the stored double-float pairs)
// for inspection. grid-stride over the elements.
// ---------------------------------------------------------------------------
__global__ void convert_sz_kernel(Dev p, int row0, int nrows, int which, double* __restrict__ dst) {
  const long long total = (long long)nrows * p.cap;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const int r = row0 + (int)(e / p.cap), i = (int)(e % p.cap);
    const float4 v = p.SZ[(size_t)r * p.stride + i];
    dst[e] = which == 0 ? (double)v.x + (double)v.y : (double)v.z + (double)v.w;
  }
}

void launch_convert_sz(const Dev& p, int row0, int nrows, int which, double* dst, cudaStream_t s) {
  convert_sz_kernel<<<1024, 256, 0, s>>>(p, row0, nrows, which, dst);
}

// ---------------------------------------------------------------------------
// Host launchers
// ---------------------------------------------------------------------------
// Per-row lengths: every row grew by T tokens.
__global__ void rowlen_add_kernel(Dev p, int T) {
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r < p.R) p.rowlen[r] += T;
}

void launch_rowlen_add(const Dev& p, int T, cudaStream_t s) {
  rowlen_add_kernel<<<(p.R + 255) / 256, 256, 0, s>>>(p, T);
}

void launch_append(const Dev& p, const void* k, const void* v, int T, int n0, int seen0,
                   cudaStream_t s) {
  const long long pairs = (long long)T * p.R;
  if (pairs == 0) return;
  const long long per_block = 256 / (p.d / 8);
  const unsigned blocks = (unsigned)((pairs + per_block - 1) / per_block);
  launch_pdl(append_kernel, dim3(blocks), dim3(256), 0, s, p, (const uint4*)k, (const uint4*)v, pairs, T, n0, seen0);
}

#define DC_DISPATCH(EXPR)                                                   \
  do {                                                                      \
    if (p.d == 64) {                                                        \
      constexpr int D = 64;                                                 \
      if (p.G == 1) { constexpr int G = 1; EXPR; }                          \
      else if (p.G == 2) { constexpr int G = 2; EXPR; }                     \
      else if (p.G == 4) { constexpr int G = 4; EXPR; }                     \
      else { constexpr int G = 8; EXPR; }                                   \
    } else {                                                                \
      constexpr int D = 128;                                                \
      if (p.G == 1) { constexpr int G = 1; EXPR; }                          \
      else if (p.G == 2) { constexpr int G = 2; EXPR; }                     \
      else if (p.G == 4) { constexpr int G = 4; EXPR; }                     \
      else { constexpr int G = 8; EXPR; }                                   \
    }                                                                       \
  } while (0)

bool split_supported(const Dev& p) {
  return (p.d == 64 || p.d == 128) && (p.G == 1 || p.G == 2 || p.G == 4 || p.G == 8);
}

void launch_split_qk(const Dev& p, const Step& st, const void* q, cudaStream_t s) {
  dim3 grid(st.nsplit, p.R);
  DC_DISPATCH((split_qk_kernel<D, G><<<grid, kTile, 0, s>>>(p, st, (const __nv_bfloat16*)q)));
}

void launch_split_stats(const Dev& p, const Step& st, const void* q, cudaStream_t s) {
  DC_DISPATCH((split_stats_kernel<D, G><<<p.R, 128, 0, s>>>(p, st, (const __nv_bfloat16*)q)));
}

void launch_split_v(const Dev& p, const Step& st, cudaStream_t s) {
  dim3 grid(st.nsplit, p.R);
  const size_t wbytes = sizeof(float) * (9 * p.hidden + 1);
  DC_DISPATCH((split_v_kernel<D, G><<<grid, kTile, wbytes, s>>>(p, st)));
}

void launch_split_out(const Dev& p, const Step& st, float* out, cudaStream_t s) {
  const int threads = p.G * p.d < 1024 ? p.G * p.d : 1024;
  DC_DISPATCH((split_out_kernel<D, G><<<p.R, threads, 0, s>>>(p, st, out)));
}

}  // namespace dc
