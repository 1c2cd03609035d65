/*
 * dc_oracle.h -- plain fp64 CPU oracle of the DistillCache budgeted KV-eviction
 * decode step (one cache row = one (layer, batch, KV head)).
 *
 * TEST INFRASTRUCTURE ONLY. Nothing in the product path may include, link or
 * call this code: only the tests, the package's smoke check and the benchmark's
 * CPU-baseline leg use it. It shares no code with the CUDA path.
 *
 * What it computes (paper section in brackets):
 *   - append of the new key/value pair before attention [Algorithm 1: the
 *     forward pass's cache already holds the new pair];
 *   - softmax attention of each query head of the KV group over every cached
 *     token, its output and its entropy [Sec. 3.1.1 entropy definition;
 *     Sec. 3.1 Reward, normalised attention weights];
 *   - the five token features x_i = [alpha_i, |v_i|_2, sigma_i, H_i, pos_i]
 *     [Sec. 3.1.1 State Space];
 *   - the policy score s_i = f_phi(x_i) of the two-layer MLP with LayerNorm and
 *     ReLU [Sec. 3.1.2 Action Space; App. D Training Details];
 *   - deterministic top-B retention and pruning [Algorithm 1, argtop_B and prune].
 *
 * Everything is double precision; bf16 inputs are widened exactly.
 */
#ifndef DC_ORACLE_H
#define DC_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct dco_row dco_row;

/* d: head_dim; G: query heads per KV head; w: entropy window (w = 64 in the
 * paper); alpha_mode 0: attention mass of the most recent pass, 1: cumulative
 * since insertion. cap: most tokens the row may hold. Returns NULL on bad
 * arguments or allocation failure. */
dco_row* dco_row_new(int d, int G, int w, int alpha_mode, int cap);
void dco_row_free(dco_row* r);

/* Appends T tokens (bf16 bit patterns, [T][d]) without queries; positions
 * continue from the number of tokens seen. Returns 0, or -1 if cap would be
 * exceeded (the row is then unchanged). */
int dco_row_append(dco_row* r, const uint16_t* k, const uint16_t* v, int T);

/* One decode step: append (k_new, v_new), attend with the G query heads
 * q [G][d], compute features and policy scores of all n tokens (ascending
 * position order). Outputs (any may be NULL):
 *   o [G][d] attention output, Hq [G] entropy of each head's distribution,
 *   feat [n][5], score [n].
 * mlp: fp32 blob [W1 (hidden x 5) | b1 | gamma | beta | w2 | b2];
 * layernorm 0 skips the LayerNorm. Returns n, or -1 on capacity overflow. */
int dco_row_step(dco_row* r, const uint16_t* q, const uint16_t* k_new, const uint16_t* v_new,
                 const float* mlp, int hidden, int layernorm,
                 double* o, double* Hq, double* feat, double* score);

/* Keeps the top min(n, budget) tokens by (score descending, position
 * ascending). Scores: `scores_f32` (n values in ascending-position order) if
 * not NULL, else the scores of the last step. Returns the new length, or -1 if
 * no scores are available. */
int dco_row_evict(dco_row* r, int budget, const float* scores_f32);

int dco_row_len(const dco_row* r);
/* Positions [n] (ascending). */
void dco_row_positions(const dco_row* r, int64_t* pos);
/* bf16 bit patterns of the cached keys and values, [n][d] each. */
void dco_row_kv_bits(const dco_row* r, uint16_t* k, uint16_t* v);
/* Window sums of the last step, [n] each: Z_i (attention mass over the window)
 * and S_i (entropy-weighted mass); cumulative alpha (alpha_mode 1) in acc. */
void dco_row_window_sums(const dco_row* r, double* S, double* Z, double* acc);

/* Heuristic scores of the row's tokens (ascending positions): scorer 1 H2O
 * (cumulative attention mass; needs alpha_mode 1), scorer 2 StreamingLLM
 * (n_sinks first positions, then the most recent). Returns 0 or -1. */
int dco_row_heuristic_scores(const dco_row* r, int scorer, int n_sinks, double* score);

/* The same window sums without the most recent step's query (the window's
 * earlier min(w, steps) - 1 queries), [n] each. */
void dco_row_window_sums_prior(const dco_row* r, double* S, double* Z);

/* Plain softmax attention of G query heads over n keys (no state): the
 * full-cache decode comparator. q [G][d], k/v [n][d] bf16 bits, o [G][d]. */
void dco_attend(const uint16_t* q, const uint16_t* k, const uint16_t* v, int n, int d, int G,
                double* o, double* Hq);

/* The policy MLP on m feature vectors x [m][5] -> score [m]. */
void dco_policy(const double* x, int m, const float* mlp, int hidden, int layernorm, double* score);

/* Global token mode (Sec. 3.1.1, "across all heads and layers"): a sequence of
 * R rows (its layers x KV heads) sharing one token set. The features of a
 * token pool all R x G attention heads: alpha (mean mass), sigma (population
 * variance), H (entropy-weighted window mass over the pooled heads), |v| (mean
 * over the rows of the value norm) and pos; one policy score and one argtop_B
 * per sequence; every row pruned the same way. k/v/q arrays are row-major
 * over the rows: append k [R][T][d]; step q [R][G][d], k_new/v_new [R][d],
 * o [R][G][d], feat [n][5], score [n]. */
typedef struct dco_seq dco_seq;
dco_seq* dco_seq_new(int R, int d, int G, int w, int alpha_mode, int cap);
void dco_seq_free(dco_seq* s);
int dco_seq_append(dco_seq* s, const uint16_t* k, const uint16_t* v, int T);
int dco_seq_step(dco_seq* s, const uint16_t* q, const uint16_t* k_new, const uint16_t* v_new,
                 const float* mlp, int hidden, int layernorm, double* o, double* feat, double* score);
int dco_seq_evict(dco_seq* s, int budget, const float* scores_f32);
int dco_seq_len(const dco_seq* s);
void dco_seq_positions(const dco_seq* s, int64_t* pos);
void dco_seq_kv_bits(const dco_seq* s, int r, uint16_t* k, uint16_t* v);
void dco_seq_window_sums_prior(const dco_seq* s, double* S, double* Z);

/* Training side (App. C). log Z of the Plackett-Luce distribution over
 * size-B subsets of the L scores s at temperature tau (fp64). */
double dco_pl_logz(const double* s, int L, int B, double tau);

/* Gumbel-top-B: indices (ascending) of the B largest fp32 perturbed scores
 * s_i / tau + g_i (ties: lower index). Returns 0 or -1. */
int dco_gumbel_topb(const float* s, const float* g, int L, int B, float tau, int* idx);

#ifdef __cplusplus
}
#endif
#endif
