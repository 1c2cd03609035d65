// dc_fused.cu -- the fused engine's host side and its main instantiations
// (per-row selection with the policy MLP; rows within and past the on-chip
// logit capacity). The kernel itself is in dc_fused_kernel.cuh.
#include "dc_fused_kernel.cuh"

namespace dc {

int fused_onchip_tokens(int G) {
  const int t = G == 8 ? onchip_tiles<8>() : G == 4 ? onchip_tiles<4>() : G == 2 ? onchip_tiles<2>() : onchip_tiles<1>();
  return t * kTok;
}

bool fused_eligible(const Dev& p, int n) {
  return (p.d == 64 || p.d == 128) && (p.G == 1 || p.G == 2 || p.G == 4 || p.G == 8) && p.hidden <= 128 && n >= 1 &&
         p.logit != nullptr && p.score != nullptr;
}

int fused_smem_bytes() { return Smem<false, 4>::BYTES; }

bool fused_pairs(const Dev& p, int n, int num_sms) {
  const int nT = (n + kTok - 1) / kTok;
  if (!(p.seq_rows == 0 && p.rowlen == nullptr && p.scorer == 0 && p.G <= 4 && p.R % 2 == 0 && p.R > num_sms &&
        nT >= 1 && nT <= kPairTiles))
    return false;
  // Critical path of a CTA in units of one token's streaming time at an SM's
  // share of the bandwidth (measured with per-row timestamps): a row costs its
  // n tokens plus ~350 of serial epilogue (statistics merge, output, select), a
  // pair 2n plus ~410. Pairs halve the serial part per row but make the last
  // wave coarser: the cheaper schedule wins.
  const int rem = p.R % num_sms;
  const double waves1 = p.R / num_sms + (rem == 0 ? 0.0 : 2 * rem <= num_sms ? 0.5 : 1.0);
  const double waves2 = (p.R / 2 + num_sms - 1) / num_sms;
  return waves2 * (2.0 * n + 410.0) < waves1 * (n + 350.0);
}

int fused_half_rows(const Dev& p, int n, const FusedStep& fs, int num_sms) {
  if (fused_pairs(p, n, num_sms)) return 0;
  const int grid = p.R < num_sms ? p.R : num_sms, rem = p.R % grid;
  const int nT = (n + kTok - 1) / kTok;
  const bool ok = fs.xflag && fs.xstats && fs.xo && fs.xsel && nT >= 2 && (!fs.do_evict || fs.B >= n || fs.B == n - 1);
  if (!ok) return 0;
  // at most half as many rows as SMs: every row of 12 tiles or more over two
  // CTAs (shorter halves cost more in exchanges than they save: 129-token
  // rows measured 25 us per step whole, 30 us halved; 2049-token rows 44 and
  // 41 us, 4097-token rows 64 and 51 us)
  if (2 * p.R <= num_sms) return nT >= 12 ? p.R : 0;
  return rem > 0 && 2 * rem <= grid ? rem : 0;
}

cudaError_t launch_fused_step(const FusedMaps& maps, const Dev& p, const Step& st, const FusedStep& fs,
                              const FusedPolicy& fp, int num_sms, cudaStream_t s) {
  // the other variants are instantiated in their own translation units
  if (p.seq_rows) return launch_fused_glob(maps, p, st, fs, fp, num_sms, s);
  if (p.rowlen || p.scorer != 0) return launch_fused_heur_perrow(maps, p, st, fs, fp, num_sms, s);
  if (fs.half_rows == 0 && fused_pairs(p, st.n, num_sms)) return launch_fused_pair(maps, p, st, fs, fp, num_sms, s);
  const int grid = fused_grid(p, fs, num_sms);
  const bool lg = st.n > fused_onchip_tokens(p.G);
#define DC_FUSED_LAUNCH(D, G) \
  return lg ? launch_t<D, G, true>(maps, p, st, fs, fp, grid, s) : launch_t<D, G, false>(maps, p, st, fs, fp, grid, s)
  if (p.d == 128) {
    if (p.G == 8) DC_FUSED_LAUNCH(128, 8);
    if (p.G == 4) DC_FUSED_LAUNCH(128, 4);
    if (p.G == 2) DC_FUSED_LAUNCH(128, 2);
    DC_FUSED_LAUNCH(128, 1);
  }
  if (p.G == 8) DC_FUSED_LAUNCH(64, 8);
  if (p.G == 4) DC_FUSED_LAUNCH(64, 4);
  if (p.G == 2) DC_FUSED_LAUNCH(64, 2);
  DC_FUSED_LAUNCH(64, 1);
#undef DC_FUSED_LAUNCH
}

}  // namespace dc

// ---------------------------------------------------------------------------
// Host-side preparation
// ---------------------------------------------------------------------------
#include <algorithm>
#include <cmath>
#include <numeric>

namespace dc {

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

cudaError_t make_fused_maps(const Dev& p, FusedMaps* maps, const char** why) {
  static EncodeTiledFn encode = nullptr;
  if (!encode) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn) {
      *why = "cuTensorMapEncodeTiled is unavailable";
      return e != cudaSuccess ? e : cudaErrorNotSupported;
    }
    encode = reinterpret_cast<EncodeTiledFn>(fn);
  }
  const cuuint64_t dims[2] = {(cuuint64_t)p.d, (cuuint64_t)p.R * (cuuint64_t)p.stride};
  const cuuint64_t strides[1] = {(cuuint64_t)p.d * 2};
  const cuuint32_t estr[2] = {1, 1};
  CUtensorMap* const out[4] = {&maps->k, &maps->v, &maps->k16, &maps->v16};
  for (int which = 0; which < 4; ++which) {
    const cuuint32_t box[2] = {64, which < 2 ? 128u : 16u};
    CUresult r = encode(out[which], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (which & 1) ? (void*)p.V : (void*)p.K,
                        dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
      *why = "cuTensorMapEncodeTiled rejected the K/V layout";
      return cudaErrorInvalidValue;
    }
  }
  return cudaSuccess;
}

void prepare_policy(const float* blob, int H, int layernorm, FusedPolicy* fp, std::vector<__nv_bfloat16>* wtile) {
  const float* W1 = blob;
  const float* b1 = W1 + 5 * H;
  const float* gamma = b1 + H;
  const float* beta = gamma + H;
  const float* w2 = beta + H;
  const double b2 = w2[H];
  // rows w_j (8 values) of the folded first layer, in double precision
  std::vector<double> rows((size_t)H * 8, 0.0);
  double Mq[6][6] = {};
  if (layernorm) {
    double mW[5] = {}, mb = 0.0;
    for (int j = 0; j < H; ++j) {
      for (int k = 0; k < 5; ++k) mW[k] += W1[j * 5 + k];
      mb += b1[j];
    }
    for (int k = 0; k < 5; ++k) mW[k] /= H;
    mb /= H;
    for (int j = 0; j < H; ++j) {
      double cj[6];
      for (int k = 0; k < 5; ++k) cj[k] = (double)W1[j * 5 + k] - mW[k];
      cj[5] = (double)b1[j] - mb;
      for (int a = 0; a < 6; ++a)
        for (int b = 0; b < 6; ++b) Mq[a][b] += cj[a] * cj[b] / H;
      const double aw = std::fabs((double)w2[j]);
      const double s = aw * (double)gamma[j];
      for (int k = 0; k < 6; ++k) rows[(size_t)j * 8 + k] = s * cj[k];
      rows[(size_t)j * 8 + 6] = aw * (double)beta[j];
    }
  } else {
    for (int j = 0; j < H; ++j) {
      const double aw = std::fabs((double)w2[j]);
      for (int k = 0; k < 5; ++k) rows[(size_t)j * 8 + k] = aw * (double)W1[j * 5 + k];
      rows[(size_t)j * 8 + 5] = aw * (double)b1[j];
    }
  }
  int k = 0;
  for (int a = 0; a < 6; ++a)
    for (int b = a; b < 6; ++b) fp->M[k++] = (float)(a == b ? Mq[a][b] : 2.0 * Mq[a][b]);
  fp->b2 = (float)b2;
  fp->layernorm = layernorm ? 1 : 0;
  // hidden units with w2 >= 0 first (the order is immaterial to the sum)
  std::vector<int> perm(H);
  std::iota(perm.begin(), perm.end(), 0);
  std::stable_partition(perm.begin(), perm.end(), [&](int j) { return w2[j] >= 0.f; });
  fp->npos = (int)std::count_if(w2, w2 + H, [](float x) { return x >= 0.f; });
  wtile->assign(128 * 32, __float2bfloat16_rn(0.f));
  for (int jj = 0; jj < 128; ++jj) fp->sgn[jj] = jj < H ? (w2[perm[jj]] >= 0.f ? 1.f : -1.f) : 0.f;
  double u[8] = {};
  for (int jj = 0; jj < H; ++jj) {
    const double* rj = &rows[(size_t)perm[jj] * 8];
    for (int e = 0; e < 8; ++e) {
      const __nv_bfloat16 hi = __float2bfloat16_rn((float)rj[e]);
      const __nv_bfloat16 lo = __float2bfloat16_rn((float)(rj[e] - (double)__bfloat162float(hi)));
      (*wtile)[jj * 32 + e] = hi;
      (*wtile)[jj * 32 + 8 + e] = hi;
      (*wtile)[jj * 32 + 16 + e] = lo;
      u[e] += (double)fp->sgn[jj] * ((double)__bfloat162float(hi) + (double)__bfloat162float(lo));
    }
  }
  for (int e = 0; e < 8; ++e) fp->u[e] = (float)u[e];
  fp->wtile = nullptr;
}

}  // namespace dc
