/*
 * distillcache.h -- C ABI of the GB300 (sm_103a) DistillCache decode step.
 *
 * A cache holds R = layers * batch * kv_heads independent rows. Each row is the
 * key/value cache of one (layer, sequence, KV head) plus per-token eviction
 * state. One decode step of the paper's inference loop (Algorithm 1) is
 *
 *     dc_decode_step   forward pass over C_t (the cache including the new
 *                      pair), token features x_i and policy scores s_i;
 *     dc_evict         argtop_B of the scores and prune of the cache.
 *
 * The problem statement (Sec. 3.1, Problem Formulation) asks for a pruned cache
 * C'_t of at most B tokens; the features are those of Sec. 3.1.1 (State Space)
 * and the policy is the MLP of Sec. 3.1.2 (Action Space) with the widths of
 * App. D (Training Details).
 *
 * Conventions for every call:
 *   - Pointers are DEVICE pointers unless the name says host. bf16 tensors are
 *     passed as `const void*` holding IEEE bfloat16 values, row-major, densely
 *     packed. The caller owns inputs and outputs; the library owns the cache,
 *     its state, its scratch and the policy weights.
 *   - Work is enqueued on the stream given at creation (cfg->stream, a
 *     cudaStream_t; NULL is the legacy default stream) and is asynchronous,
 *     except where a call says it synchronises.
 *   - Every call returns a dc_status. No C++ exception crosses the ABI. A CUDA
 *     error makes the handle unusable: later calls return DC_ERR_CUDA and
 *     dc_last_error() gives the message. Invalid arguments leave the cache
 *     unchanged.
 *   - Calls on one handle must not run concurrently from several host threads.
 *   - The handle keeps the step's host-side state (row lengths, the window
 *     slot, the launch epoch that keys the fused kernel's work queue and
 *     exchange flags) and advances it on every call; the launches it enqueues
 *     carry that step's values. A stream capture of a call therefore records
 *     one particular step: replaying it repeats that step's arguments. In
 *     graph mode (dc_set_graph_mode) dc_step counts steps on the device
 *     instead, and a captured dc_step replays as the following decode steps.
 */
#ifndef DISTILLCACHE_H
#define DISTILLCACHE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  DC_OK = 0,
  DC_ERR_INVALID_ARG = 1, /* bad pointer, size or shape; nothing was done */
  DC_ERR_CAPACITY = 2,    /* the rows would exceed `capacity` tokens */
  DC_ERR_OOM = 3,         /* device allocation failed at creation */
  DC_ERR_CUDA = 4,        /* a CUDA call failed; the handle is now unusable */
  DC_ERR_DEVICE = 5,      /* a kernel reported an error through its status word */
  DC_ERR_STATE = 6        /* call out of order (e.g. evict with no scores) */
} dc_status;

typedef struct dc_cache dc_cache;

typedef struct {
  int batch;          /* sequences per layer (default 1) */
  int q_heads;        /* query heads per layer (default 4 * kv_heads) */
  int window;         /* w of the entropy feature H_i (default 64, Sec. 3.1.1) */
  int mlp_hidden;     /* hidden width of the policy MLP (default 128, App. D) */
  int layernorm;      /* 1: LayerNorm after the first layer (default, App. D) */
  int alpha_mode;     /* 0: alpha_i from the most recent pass (Sec. 3.1.1, default);
                         1: cumulative since insertion */
  int engine;         /* 0: auto (default): the fused kernel whenever the step
                            fits it, unless a few long rows run faster on the
                            split engine (a latency model of the two);
                         1: split (separate attention, feature and scoring kernels);
                         2: fused whenever the step fits it (one CTA per row
                            streams K/V once and does the whole step) */
  int keep_features;  /* 1: also store x_i [R][capacity][5] fp32 for inspection */
  unsigned long long seed; /* policy weight seed (dc_policy_init) */
  void* stream;       /* cudaStream_t */
  int tail_split;     /* fused engine, rows not a multiple of the grid: 1 (default)
                         splits each row of the last, partly filled wave over two
                         CTAs, which exchange softmax statistics, output and the
                         eviction candidate through global memory under a
                         cooperative launch (steps that evict one token or none);
                         0: whole rows only */
  int scorer;         /* what ranks the tokens for argtop_B:
                         0: the policy MLP (default, Sec. 3.1.2);
                         1: H2O, cumulative attention mass since insertion (the
                            heavy-hitter baseline of Sec. 2 / Sec. 4; implies
                            alpha_mode 1);
                         2: StreamingLLM, the first n_sinks positions (attention
                            sinks) and then the most recent tokens */
  int n_sinks;        /* sink tokens kept by scorer 2 (default 4) */
  float budget_ratio; /* > 0: dynamic budget B_t = max(floor(r * L_t), budget_min)
                         whenever a call passes budget <= 0 (App. D); 0 (default):
                         the fixed budget given to dc_cache_create */
  int budget_min;     /* B_min of the dynamic budget (default 32) */
  int budget_basis;   /* L_t of the dynamic budget: 0 (default) tokens seen so far
                         (the sequence length), 1 the tokens cached before the
                         eviction, |C_t| */
  int global_tokens;  /* 1: global token mode (Sec. 3.1.1, "across all heads and
                         layers"): a token's features pool the attention of every
                         query head of every layer of its sequence, one policy
                         score and one argtop_B per sequence, and all rows of a
                         sequence keep the same tokens. The sequence's window
                         sums, cumulative alpha, features and scores are kept in
                         its home row (layer 0, KV head 0). dc_step runs as
                         dc_decode_step + dc_evict. 0 (default): one selection
                         per row. */
} dc_config;

/* Fills *cfg with the defaults above (batch 1, q_heads 0 meaning 4 * kv_heads,
 * seed 0, stream NULL). */
dc_status dc_config_default(dc_config* cfg);

/* Creates a cache of `layers` x cfg->batch x `kv_heads` rows, each able to hold
 * `capacity` tokens of `head_dim` dimensions, with default budget `budget`.
 * Requirements: head_dim in {64, 128}; q_heads % kv_heads == 0 and
 * q_heads / kv_heads in {1, 2, 4, 8}; 1 <= budget < capacity; window in
 * [1, 1024]; mlp_hidden in [1, 256] and a multiple of 32 when >= 32.
 * The policy weights are initialised from cfg->seed as dc_policy_init does.
 * Synchronises the device once (allocation). cfg may be NULL (defaults). */
dc_status dc_cache_create(int layers, int kv_heads, int head_dim, int capacity, int budget,
                          const dc_config* cfg, dc_cache** out);

/* Frees every device buffer of the handle (synchronises its stream). NULL is a
 * no-op. A handle must not be used after it is destroyed. */
dc_status dc_cache_destroy(dc_cache* h);

/* Number of floats in a policy blob of hidden width H: 9 * H + 1. Layout
 * (fp32): [W1 (H x 5, row-major) | b1 (H) | gamma (H) | beta (H) | w2 (H) | b2],
 * i.e. s = w2 . relu(LN(W1 x + b1) * gamma + beta) + b2, with the feature order
 * x = [alpha, |v|_2, sigma, H, pos] (Sec. 3.1.1). */
size_t dc_policy_blob_len(int hidden);

/* Host-only: the seeded initial weights. Linear layers draw uniformly from
 * [-1/sqrt(fan_in), 1/sqrt(fan_in)] (PyTorch's default rule) from a
 * SplitMix64 stream; gamma = 1, beta = 0. `host_out` holds n >= blob_len
 * floats. Needs no GPU. */
dc_status dc_policy_init(unsigned long long seed, int hidden, float* host_out, size_t n);

/* Replaces the policy weights with a host fp32 blob of dc_policy_blob_len(H)
 * floats (H = cfg->mlp_hidden): the network f_phi of Sec. 3.1.2 (Action Space,
 * scores s_i = f_phi(x_i)) with the two-layer, LayerNorm, ReLU shape of App. D
 * (Training Details), e.g. trained weights. The blob is copied before the call
 * returns; DC_ERR_INVALID_ARG if n differs from dc_policy_blob_len(H). */
dc_status dc_policy_set_weights(dc_cache* h, const float* host_blob, size_t n);

/* Appends n_tokens tokens to every row without queries (prompt loading).
 * Algorithm 1 takes the prompt as the cache at t = 0; later decode steps add
 * one pair each (C_t includes the new key/value pair before the forward pass,
 * Sec. 3.1, Problem Formulation).
 * k, v: bf16 [layers][batch][kv_heads][n_tokens][head_dim]. Positions continue
 * from the number of tokens seen. DC_ERR_CAPACITY (cache unchanged) if the
 * rows would exceed capacity. */
dc_status dc_append(dc_cache* h, const void* k, const void* v, int n_tokens);

/* One decode step (Algorithm 1, forward pass, feature extraction and scoring):
 * appends (k_new, v_new) to every row, attends with q over the whole unpruned
 * row (the new token included), writes the attention output, updates the
 * token features and scores every cached token. The scores stay on the device
 * for dc_evict.
 *   q:     bf16 [layers][batch][q_heads][head_dim]; query head j uses KV head
 *          j / (q_heads / kv_heads).
 *   k_new, v_new: bf16 [layers][batch][kv_heads][head_dim].
 *   out:   fp32 [layers][batch][q_heads][head_dim].
 * DC_ERR_CAPACITY (cache unchanged) if a row is full. */
dc_status dc_decode_step(dc_cache* h, const void* q, const void* k_new, const void* v_new,
                         float* out);

/* The same step with HOST buffers of the same shapes (pinned memory is fastest);
 * the copies run on the handle's stream and the call synchronises it before it
 * returns, so `out_host` is ready. */
dc_status dc_decode_step_host(dc_cache* h, const void* q_host, const void* k_new_host,
                              const void* v_new_host, float* out_host);

/* One whole step of Algorithm 1: dc_decode_step followed by dc_evict(budget),
 * as one kernel when the fused engine takes the step (no scores are stored
 * then; DC_BUF_SCORE is not updated). Exceptions, which run as the two
 * calls: with split rows (see tail_split) a step that evicts more than one
 * token per row, and a step that evicts more than 1024 tokens per row (a
 * prompt compression). The result is bit-identical to the two calls either
 * way. Same arguments as dc_decode_step. */
dc_status dc_step(dc_cache* h, const void* q, const void* k_new, const void* v_new, float* out,
                  int budget);

/* dc_step with HOST buffers (copies on the handle's stream; synchronises). */
dc_status dc_step_host(dc_cache* h, const void* q_host, const void* k_new_host,
                       const void* v_new_host, float* out_host, int budget);

/* dc_step_host without the final synchronisation. The input copies run on a
 * copy stream of the handle's own, the step on the handle's stream, the output
 * copy on a second copy stream, with two device staging sets used in turn: the
 * inputs of step s + 1 and the output of step s move while kernels run. The
 * call returns at once; out_host holds the output after dc_sync (which also
 * waits for the copy streams), and every host buffer must stay untouched until
 * then. Pinned host memory keeps the copies asynchronous. */
dc_status dc_step_host_async(dc_cache* h, const void* q_host, const void* k_new_host,
                             const void* v_new_host, float* out_host, int budget);

/* Graph mode (enable = 1): dc_step (and dc_step_host, dc_step_host_async)
 * counts its steps in device memory: the kernels advance positions, window
 * slots and the launch epoch by that count, so the same enqueued work -- a
 * CUDA graph captured from one dc_step call -- performs the following decode
 * steps when replayed, with the inputs the captured buffers hold at each
 * replay. Needs the steady state of the fused engine: the policy scorer, the
 * fixed budget, every row at the budget (one eviction per step), at least a
 * window of consecutive decode steps taken, no per-row budgets or global
 * token mode (DC_ERR_STATE otherwise). Other calls that change the cache
 * return DC_ERR_STATE while the mode is on; dc_get_length reports the tokens
 * seen as of entering the mode. enable = 0 synchronises the stream, reads the
 * count and brings the handle's state up to date; then every call works as
 * before. */
dc_status dc_set_graph_mode(dc_cache* h, int enable);

/* Per-row budgets, the head-level hybrid of Sec. 5 (Table tab:hybrid: the most
 * important heads keep the full cache, token selection in the others):
 * budgets[r] for every row r = (layer * batch + b) * kv_heads + g (host array of
 * n = rows ints, each >= 1). dc_evict / dc_step calls with budget <= 0 then keep
 * min(n_r, budgets[r]) tokens in row r (a budget >= capacity keeps the row's full
 * cache up to its capacity); a positive budget argument still applies to every
 * row; per-row budgets take precedence over budget_ratio. Rows then hold
 * different lengths (dc_get_row_lengths; dc_get_length reports the longest);
 * the fused engine takes them with the policy scorer (heuristic scorers run
 * on the split engine); dc_full_decode needs equal lengths (else
 * DC_ERR_STATE). budgets == NULL returns to one budget when every row has the
 * same length (else DC_ERR_STATE). Not with global_tokens (DC_ERR_STATE).
 * Synchronises the handle's stream. */
dc_status dc_set_row_budgets(dc_cache* h, const int* budgets_host, int n);

/* Every row's current length (host array of n = rows ints). */
dc_status dc_get_row_lengths(dc_cache* h, int* lengths_host, int n);

/* Which engine a step over n tokens per row would use (n <= 0: the next
 * decode step): 1 split, 2 fused (one CTA per row), 3 fused on row pairs (each
 * warpgroup of a CTA on a row of its own; short rows, more rows than SMs, when
 * that schedule is expected to be faster). */
dc_status dc_engine(dc_cache* h, int n, int* engine);

/* argtop_B and prune (Algorithm 1): every row keeps its min(n, B) highest-scored
 * tokens (ties: lower position first; -0 equals +0; NaN ranks last) and
 * compacts them into its first min(n, B) slots. Survivors below that bound do
 * not move; each survivor above it moves into the lowest free slot, in
 * ascending slot order. budget <= 0 uses the configured budget: the dynamic
 * max(floor(budget_ratio * L_t), budget_min) when budget_ratio > 0 (capped at
 * capacity - 1), else the fixed one. Needs the scores of a decode step since
 * the last append/evict (else DC_ERR_STATE). */
dc_status dc_evict(dc_cache* h, int budget);

/* Full-cache comparator: softmax attention of q over the current rows with no
 * append, features or eviction (the "Full" row of the paper's latency table).
 * q and out as in dc_decode_step. */
dc_status dc_full_decode(dc_cache* h, const void* q, float* out);

/* Current tokens per row (every row holds the same number) and tokens seen. */
dc_status dc_get_length(dc_cache* h, int* n, long long* seen);

typedef enum {
  DC_BUF_K = 0,     /* bf16 [R][capacity][head_dim] */
  DC_BUF_V = 1,     /* bf16 [R][capacity][head_dim] */
  DC_BUF_POS = 2,   /* int32 [R][capacity] absolute position of each slot */
  DC_BUF_S = 3,     /* fp64 [R][capacity] entropy-weighted window mass S_i over the
                       window's queries before the last step (Sec. 3.1.1, H_i) */
  DC_BUF_Z = 4,     /* fp64 [R][capacity] window mass Z_i, same queries */
  DC_BUF_ACC = 5,   /* fp32 [R][capacity] cumulative alpha (alpha_mode 1) */
  DC_BUF_SCORE = 6, /* fp32 [R][capacity] policy scores of the last step */
  DC_BUF_FEAT = 7,  /* fp32 [R][capacity][5] features (keep_features only) */
  DC_BUF_HQ = 8,    /* fp32 [R][q_heads / kv_heads] entropy of each head, last step */
  DC_BUF_VNORM = 9  /* fp32 [R][capacity] |v_i|_2 of each slot */
} dc_buffer;

/* Size in bytes of one row of an internal buffer (0 if the handle has none of
 * it); every buffer above is laid out as [R][row]. */
dc_status dc_buffer_bytes(dc_cache* h, dc_buffer which, size_t* row_bytes);

/* Copies rows [row0, row0 + nrows) of an internal buffer into device memory
 * `dst` of `bytes` bytes (bytes must equal nrows * row_bytes) on the handle's
 * stream. DC_ERR_INVALID_ARG if the range is outside [0, R). */
dc_status dc_copy_buffer(dc_cache* h, dc_buffer which, int row0, int nrows, void* dst, size_t bytes);

/* Kernel phases of the calls above, for launch counting and timing. */
typedef enum {
  DC_PHASE_APPEND = 0,  /* new pairs written into the rows */
  DC_PHASE_ATTEND = 1,  /* attention pass over K (split) or the whole fused step */
  DC_PHASE_STATS = 2,   /* softmax statistics and window-ring push (split) */
  DC_PHASE_SCORE = 3,   /* attention output, features and policy scores (split) */
  DC_PHASE_COMBINE = 4, /* per-split output merge (split) */
  DC_PHASE_EVICT = 5,   /* top-B select and compaction */
  DC_PHASE_FULL = 6,    /* full-cache comparator */
  DC_PHASE_COUNT = 7
} dc_phase;

/* Name of a phase ("append", "attend", ...), or "" if out of range. */
const char* dc_phase_name(int phase);

/* Turns per-launch CUDA-event timing on (1) or off (0) and zeroes the
 * counters. Events are recorded on the handle's stream around every kernel. */
dc_status dc_profile_enable(dc_cache* h, int on);

/* Synchronises the stream and reads, per phase, the summed kernel time in ms
 * (timed launches only) and the number of launches since the last enable.
 * ms and launches each hold DC_PHASE_COUNT values (either may be NULL). */
dc_status dc_profile_read(dc_cache* h, double* ms, long long* launches);

/* Waits for all work enqueued on the handle's stream (and on the copy streams
 * of dc_step_host_async); reports any device status the kernels raised
 * (DC_ERR_DEVICE). */
dc_status dc_sync(dc_cache* h);

/* Full-cache decode attention that allocates no device memory, for callers
 * that cannot call cudaMalloc: runtimes that reserve all device memory up
 * front and allow no allocation afterwards (a fixed-footprint serving
 * process), and paths that cannot afford the implicit device synchronisation
 * of cudaMalloc/cudaFree. The handle-based calls do not suit them, because
 * dc_cache_create allocates. The paper has no counterpart; this is the
 * dc_full_decode computation on caller-provided buffers, with no handle.
 *   q:   bf16 [rows][group][head_dim]; k, v: bf16 [rows][n][head_dim]
 *        (16-byte aligned); out: fp32 [rows][group][head_dim]; all device.
 *   stream: cudaStream_t (NULL: legacy default stream).
 * The split-K partial results go to a 16 MiB file-scope device array that
 * stays reserved, on every GPU where this library's device code is loaded,
 * until the process exits. With CUDA's lazy module loading (the default since
 * CUDA 12.2) that code, and so the array, is loaded on a device at the first
 * call there: a caller that reserves the rest of device memory up front must
 * make one call (a warm-up) on each device before it does, or that first call
 * can fail with DC_ERR_CUDA (out of memory while loading the module).
 * DC_ERR_CAPACITY if one split of all rows does not fit it, i.e. if
 * rows * group * (head_dim + 4) * 4 > 16 MiB; DC_ERR_INVALID_ARG for bad
 * shapes (head_dim 64 or 128, group 1, 2, 4 or 8, 1 <= rows <= 65535, n >= 1).
 * The first call on a device looks up the array's device address (once per
 * device, with that device current); make that first call before any stream
 * capture. Every call shares the array, which keeps the last call's
 * contents; nothing in it has to start at zero, because each call writes every
 * partial result before it reads it. Calls that overlap on the GPU (two
 * streams, or two host threads) race on the array and must be serialised by
 * the caller. Asynchronous on `stream`; dc_noalloc_last_error() describes a
 * failure. */
dc_status dc_attend_noalloc(const void* q, const void* k, const void* v, int rows, int n,
                            int head_dim, int group, float* out, void* stream);

/* Message of the last failed dc_attend_noalloc call on this host thread. */
const char* dc_noalloc_last_error(void);

/* Self-test of the bounded waits every kernel relies on (a wait that cannot be
 * satisfied gives up after its time limit, records where and lets the kernel
 * return an error status instead of hanging): one thread waits limit_ns on a
 * flag in global memory that nothing sets, then limit_ns on an mbarrier that
 * nothing arrives on. result (host, 7 values): [0] bit 0 the flag wait gave
 * up, bit 1 the mbarrier wait gave up (3 = both, as they must); [1..4] the first
 * timeout's record (claim flag, site 901 for the flag, block, waited value);
 * [5], [6] each wait's duration in microseconds. limit_ns within [1 ms, 1 s].
 * Synchronises the stream; the CUDA context stays usable. */
dc_status dc_wait_selftest(unsigned long long limit_ns, unsigned* result, void* stream);

/* Message of the last failed dc_wait_selftest call on this host thread. */
const char* dc_selftest_last_error(void);

/* ---------------------------------------------------------------------------
 * Testing hooks: for the library's own tests, not for production use. None
 * of them can make a kernel fault.
 * ------------------------------------------------------------------------- */

/* Allocation-failure injection: the device allocation with index nth, counted
 * from this call over every allocation the library makes for a handle
 * (dc_cache_create and the buffers some calls add later), fails as if the
 * device were out of memory, once; nth < 0 disarms. Host-only; DC_OK. A
 * create that meets the failure returns DC_ERR_OOM after freeing what it
 * took; a later call that needs a new buffer returns DC_ERR_OOM and leaves
 * the handle usable and unchanged. */
dc_status dc_debug_fail_alloc(long long nth);

/* 1 if this library is a debug build (compiled with DC_DEBUG_BOUNDS), else 0.
 * A debug build checks computed global-memory indices in its kernels before
 * each access (a failed check raises a status bit that dc_sync reports as
 * DC_ERR_DEVICE, records the first site, index and limit, and skips the
 * access), and puts a guard region before and after every device buffer of
 * a handle, which dc_sync checks. */
int dc_debug_checks(void);

/* Debug builds: one kernel checks an index one past its limit; result (host,
 * 5 values): [0] the status word it raised (bit 2: a failed index check),
 * [1] the site recorded (903), [2] the index, [3] the limit, [4] 1 if the
 * access was skipped. Synchronises the stream. Release builds: DC_ERR_STATE
 * (message in dc_selftest_last_error()). */
dc_status dc_debug_bounds_selftest(unsigned* result, void* stream);

/* Debug builds: overwrites one byte of the guard region after the handle's
 * first buffer (memory the handle owns, outside every buffer) on its stream,
 * so that the next dc_sync reports DC_ERR_DEVICE. Release builds:
 * DC_ERR_STATE. */
dc_status dc_debug_corrupt_guard(dc_cache* h);

/* Message of the last error on the handle (or of the last failed create when
 * h is NULL). Valid until the next call on the handle. */
const char* dc_last_error(const dc_cache* h);

/* ---------------------------------------------------------------------------
 * Training-side kernels (App. C). Handle-free; device pointers, asynchronous on
 * `stream` (a cudaStream_t, NULL for the default stream).
 * ------------------------------------------------------------------------- */

/* Exact log-partition function of the Plackett-Luce distribution over size-B
 * subsets (App. C): out[r] = log sum_{a subset of [L], |a| = B}
 * exp(sum_{i in a} scores[r][i] / tau), for `rows` independent rows.
 * scores: fp32 [rows][L]; out: fp32 [rows]. Computed by the O(L B) dynamic
 * programme over the elementary symmetric polynomials, in base-2 log space,
 * fp32 with the hardware exp2/log2 (the error grows at most linearly in L:
 * |error| <= 2 L 2^-24 (|log Z| + max |s| / tau) + L 2^-21). Needs
 * 1 <= B <= L, rows <= 65535, B <= 25599, tau > 0;
 * else DC_ERR_INVALID_ARG (message in dc_train_last_error()). */
dc_status dc_pl_log_partition(const float* scores, int rows, int L, int B, float tau, float* out,
                              void* stream);

/* Gumbel-top-B sampling (Sec. 3.1.2, App. C): per row, the perturbed scores
 * scores[r][i] / tau + gumbel[r][i] (each operation rounded to fp32; gumbel
 * holds caller-drawn Gumbel(0, 1) noise, fp32 [rows][L]); the B largest are
 * kept (ties: lower index first) and their indices written to idx[r][0..B) in
 * ascending order (int32 [rows][B]). If logp is not NULL, logp[r] =
 * sum_{i in a} scores[r][i] / tau - log Z, the log-probability of the sampled
 * subset under the Plackett-Luce distribution; logz_scratch (fp32 [rows])
 * receives log Z. Same argument rules as dc_pl_log_partition. */
dc_status dc_gumbel_top_b(const float* scores, const float* gumbel, int rows, int L, int B, float tau,
                          int* idx, float* logp, float* logz_scratch, void* stream);

/* Message of the last failed training-side call of this thread. */
const char* dc_train_last_error(void);

#ifdef __cplusplus
}
#endif
#endif
