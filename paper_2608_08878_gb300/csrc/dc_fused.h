// dc_fused.h -- host-visible pieces of the fused engine: launch arguments,
// the policy network in the form the fused kernel consumes, TMA descriptors.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <vector>

#include "dc_common.cuh"

namespace dc {

// Tokens of a row whose head-(G-1) logits and scores the fused kernel keeps in
// shared memory; longer rows keep them in HBM (Dev::logit, Dev::score).
constexpr int kFusedMaxTok = 10240;

struct FusedMaps {
  CUtensorMap k, v;      // [R * cap][d] bf16, boxes of 64 dims x 128 tokens, 128-byte swizzle
  CUtensorMap k16, v16;  // the same with boxes of 64 dims x 16 tokens (a row's ragged last tile)
};

struct FusedStep {
  const __nv_bfloat16* q;
  float* out;
  int do_evict;      // 1: select and compact in the same kernel
  int B;             // tokens to keep when do_evict
  int write_scores;  // 1: also store scores in Dev::score (for dc_evict)
  // Rows are taken from a queue (an atomic counter) as CTAs become free. With
  // half_rows > 0 the last half_rows rows are each taken as two halves by two
  // CTAs, which exchange softmax statistics, the output and the eviction
  // candidate through global memory. Needs a cooperative launch (all CTAs
  // resident), 2 * half_rows <= grid and, with do_evict, one eviction per row.
  int half_rows;
  unsigned epoch;    // increases every launch; queue and exchange flags key on it
  unsigned* work;    // [2] queue counters, used by alternate launches
  float* xstats;     // [half_rows][2][G][4]
  float* xo;         // [half_rows][G][d]
  int* xsel;         // [half_rows][2][4]
  unsigned* xflag;   // [half_rows][2]
  int xslots;        // exchange slots allocated (bounds of the four above)
};

// Exchange buffer sizes (floats / ints) for a grid of `grid` CTAs.
inline size_t fused_xstats_len(int grid, int G) { return (size_t)(grid / 2 + 1) * 2 * G * 4; }
inline size_t fused_xo_len(int grid, int G, int d) { return (size_t)(grid / 2 + 1) * G * d; }
inline size_t fused_xsel_len(int grid) { return (size_t)(grid / 2 + 1) * 2 * 4; }
inline size_t fused_xflag_len(int grid) { return (size_t)(grid / 2 + 1) * 2; }

// The policy MLP folded for the tensor cores (see prepare_policy):
//   z_j = <a, w_j> with a = [r x, r, 1, 0] (LayerNorm) or [x, 1, 0, 0], where
//   w_j carries |w2_j| (and the LayerNorm gain and shift);
//   score = b2 + sum_j sgn_j max(z_j, 0), sgn_j = sign(w2_j);
//   r = 1 / sqrt(x~^T M x~ + 1e-5), x~ = [x, 1] (LayerNorm variance).
struct FusedPolicy {
  float M[21];                   // upper triangle, off-diagonal terms doubled
  float b2;
  int npos;
  int layernorm;
  const __nv_bfloat16* wtile;    // device [128][32]: rows w_j as bf16 hi | hi | lo | 0
  float sgn[128];                // +1 / -1 per hidden unit, 0 for unused columns
  float u[8];                    // sum_j sgn_j w_j: the policy input row dotted with
                                 // it is sum_j sgn_j z_j (relu(z) = (z + |z|) / 2)
};

// Tokens per row whose logits the fused kernel keeps on chip between its two
// passes (G query heads per KV head); beyond that a row's logits go through
// the global scratch Dev::logit (16 bytes per token written and read back)
// and its scores through Dev::score.
int fused_onchip_tokens(int G);
bool fused_eligible(const Dev& p, int n);
int fused_smem_bytes();

// Builds the two TMA descriptors of the K and V buffers.
cudaError_t make_fused_maps(const Dev& p, FusedMaps* maps, const char** why);

// Folds a policy blob [W1 | b1 | gamma | beta | w2 | b2] (hidden H) into
// FusedPolicy fields and the host copy of the weight tile (128 * 32 bf16).
void prepare_policy(const float* blob, int H, int layernorm, FusedPolicy* fp, std::vector<__nv_bfloat16>* wtile);

// Whether a step over n tokens runs on row pairs (each warpgroup of a CTA on
// its own row): short rows (at most kPairTiles tiles), more rows than SMs, an
// even row count, the plain step (policy scorer, equal lengths, per-row
// selection).
bool fused_pairs(const Dev& p, int n, int num_sms);

// How many rows a step over n tokens splits into halves (see FusedStep): every
// row when rows are at most half the SMs and at least 12 tiles long, else the
// remainder of R over the grid when it is at most half the grid, else 0 (and 0
// on row pairs).
int fused_half_rows(const Dev& p, int n, const FusedStep& fs, int num_sms);

cudaError_t launch_fused_step(const FusedMaps& maps, const Dev& p, const Step& st, const FusedStep& fs,
                              const FusedPolicy& fp, int num_sms, cudaStream_t s);

// The variants with a heuristic scorer or per-row budgets (dc_fused_modes.cu)
// and with the global token mode (dc_fused_glob.cu); launch_fused_step
// dispatches to them.
cudaError_t launch_fused_heur_perrow(const FusedMaps& maps, const Dev& p, const Step& st, const FusedStep& fs,
                                     const FusedPolicy& fp, int num_sms, cudaStream_t s);
cudaError_t launch_fused_glob(const FusedMaps& maps, const Dev& p, const Step& st, const FusedStep& fs,
                              const FusedPolicy& fp, int num_sms, cudaStream_t s);
// Row pairs (dc_fused_pair.cu).
cudaError_t launch_fused_pair(const FusedMaps& maps, const Dev& p, const Step& st, const FusedStep& fs,
                              const FusedPolicy& fp, int num_sms, cudaStream_t s);
// Device-counted steps (dc_fused_graph.cu): st and fs.epoch are base values
// that the kernel advances by Dev::gcount[0]; whole rows, halves or row pairs
// (as the plain step would take them), policy scorer, one eviction per step.
cudaError_t launch_fused_graph(const FusedMaps& maps, const Dev& p, const Step& st, const FusedStep& fs,
                               const FusedPolicy& fp, int num_sms, cudaStream_t s);

// Attention only over the first n tokens of every row as they are (the
// full-cache comparator): writes fs.out, touches no cache state (the logit
// scratch aside). fs.do_evict and fs.write_scores must be 0.
cudaError_t launch_fused_full(const FusedMaps& maps, const Dev& p, int n, const FusedStep& fs,
                              const FusedPolicy& fp, int num_sms, cudaStream_t s);

}  // namespace dc
