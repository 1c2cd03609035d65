// dc_kernels.h -- host-side launchers of the decode-step kernels.
#pragma once

#include <cuda_runtime.h>

#include "dc_common.cuh"

namespace dc {

void launch_append(const Dev& p, const void* k, const void* v, int T, int n0, int seen0,
                   cudaStream_t s);
// Per-row lengths (Dev::rowlen): add T to every row's length after an append.
void launch_rowlen_add(const Dev& p, int T, cudaStream_t s);

// Split engine: attention + features + scores of one decode step (after the
// append), one launcher per kernel.
bool split_supported(const Dev& p);
void launch_split_qk(const Dev& p, const Step& st, const void* q, cudaStream_t s);
void launch_split_stats(const Dev& p, const Step& st, const void* q, cudaStream_t s);
void launch_split_v(const Dev& p, const Step& st, cudaStream_t s);
void launch_split_out(const Dev& p, const Step& st, float* out, cudaStream_t s);

// argtop_B and prune of every row (B <= 0: per-row budgets): a select kernel
// and, when slots have to move, a move kernel (evict_kernel_count of them).
void launch_evict(const Dev& p, int n, int B, cudaStream_t s);
int evict_kernel_count(int n, int B);

// Global token mode: pooled per-sequence features and scores after the split
// engine's per-row pass; the sequence's selection applied to all its rows.
void launch_glob_features(const Dev& p, const Step& st, cudaStream_t s);
void launch_glob_evict(const Dev& p, int n, int B, cudaStream_t s);

// Window sums S (which 0) or Z (which 1) of rows [row0, row0 + nrows) as fp64
// [nrows][cap].
void launch_convert_sz(const Dev& p, int row0, int nrows, int which, double* dst, cudaStream_t s);

bool launch_full_decode(const Dev& p, int n, int nsplit, int chunk, const void* q, float* out,
                        cudaStream_t s);

}  // namespace dc
