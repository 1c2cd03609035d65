// dc_cache.cu -- host side of the C ABI (include/distillcache.h): the cache
// handle, its device buffers, argument checks, status codes and the launch
// sequence of each call.
#include <cuda_runtime.h>

#include <atomic>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "../../include/distillcache.h"
#include "dc_common.cuh"
#include "dc_fused.h"
#include "dc_kernels.h"

namespace {

constexpr unsigned kMagic = 0x44434331u;  // "DCC1"
// dc_step evicts more tokens per row than this with the eviction kernel (a
// separate launch after the decode kernel) rather than in the fused kernel.
constexpr int kFusedEvictMax = 1024;
constexpr unsigned kDead = 0xDEADDEADu;

thread_local std::string g_create_error;

// SplitMix64 output function (Steele, Lea, Flood).
uint64_t splitmix64(uint64_t x) {
  uint64_t z = x + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

constexpr uint64_t kTagPolicy = 0x504F4C00ull;

}  // namespace

struct dc_cache {
  unsigned magic = kMagic;
  int layers = 0, kv_heads = 0, head_dim = 0, capacity = 0, budget = 0;
  dc_config cfg{};
  cudaStream_t stream = nullptr;
  int num_sms = 0;
  dc::Dev dev{};
  // host-side state (every row holds the same number of tokens)
  int n = 0;
  long long seen = 0;
  long long steps = 0;
  bool have_scores = false;
  std::vector<int> ring_pnew;  // newest position at the step held by each ring slot
  // staging for dc_decode_step_host
  void* st_q = nullptr;
  void* st_k = nullptr;
  void* st_v = nullptr;
  float* st_out = nullptr;
  // dc_step_host_async: a second staging set, copy streams and events, so that
  // step s + 1's input copy and step s's output copy overlap the kernels
  void* st2_q = nullptr;
  void* st2_k = nullptr;
  void* st2_v = nullptr;
  float* st2_out = nullptr;
  cudaStream_t h2d = nullptr, d2h = nullptr;
  cudaEvent_t ev_in[2] = {}, ev_done[2] = {}, ev_out[2] = {};
  long long host_seq = 0;
  // fused engine: TMA descriptors of K/V and the folded policy
  bool fused_ok = false;
  std::string fused_why;
  dc::FusedMaps maps{};
  dc::FusedPolicy fpol{};
  __nv_bfloat16* wtile = nullptr;
  // queue counters and exchange buffers of the half rows (FusedStep)
  unsigned* work = nullptr;
  float* xstats = nullptr;
  float* xo = nullptr;
  int* xsel = nullptr;
  unsigned* xflag = nullptr;
  unsigned epoch = 0;
  int* rowlen_dev = nullptr;
  int* rowbudget_dev = nullptr;
  // per-row budgets (head-level hybrid): host mirror of every row's length
  // (kept in step with Dev::rowlen) and the budgets; n is then the longest row
  bool per_row = false;
  std::vector<int> hlen, hbudget;
  // the fused queue's row order in per-row mode (longest rows first): pinned
  // host copy, device copy, and the event of its last upload
  int* horder = nullptr;
  int* roworder_dev = nullptr;
  cudaEvent_t ev_order = nullptr;
  bool order_valid = false;
  // device-counted steps (dc_set_graph_mode): the base step arguments and
  // epoch that the kernels advance by the device's step count
  bool graph = false;
  dc::Step gstep{};
  unsigned gepoch = 0;
  int* gcount_dev = nullptr;
  struct Alloc {
    void* base;    // what cudaMalloc returned (guard regions included in debug builds)
    size_t bytes;  // the buffer's own size
  };
  std::vector<Alloc> allocs;
  std::string err;
  bool broken = false;
  // launch counting and optional per-launch event timing
  long long launches[DC_PHASE_COUNT] = {};
  bool profiling = false;
  struct Timed { int phase; cudaEvent_t a, b; };
  std::vector<Timed> timed;
  std::vector<cudaEvent_t> event_pool;
  double ms[DC_PHASE_COUNT] = {};
};

namespace {

dc_status fail(dc_cache* h, dc_status s, const std::string& msg) {
  if (h) h->err = msg; else g_create_error = msg;
  return s;
}

dc_status cuda_fail(dc_cache* h, cudaError_t e, const char* what) {
  std::string m = std::string(what) + ": " + cudaGetErrorString(e);
  if (h) { h->broken = true; h->err = m; } else g_create_error = m;
  return DC_ERR_CUDA;
}

bool valid(const dc_cache* h) { return h && h->magic == kMagic; }

#define DC_CHECK_HANDLE(h)                                                     \
  do {                                                                         \
    if (!valid(h)) return DC_ERR_INVALID_ARG;                                  \
    if ((h)->broken) return DC_ERR_CUDA;                                       \
  } while (0)

#define DC_CUDA(h, call)                                                       \
  do {                                                                         \
    cudaError_t e_ = (call);                                                   \
    if (e_ != cudaSuccess) return cuda_fail((h), e_, #call);                   \
  } while (0)

// Allocation-failure injection (dc_debug_fail_alloc): the allocation with this
// index, counted from when the hook was armed, fails as if the device were out
// of memory; -1: disarmed. Host-only.
std::atomic<long long> g_fail_alloc_at{-1};
std::atomic<long long> g_alloc_index{0};

// Debug builds put a guard region of kGuardBytes before and after every device
// buffer of a handle, filled with kGuardByte; dc_sync checks that both are intact.
#ifdef DC_DEBUG_BOUNDS
constexpr size_t kGuardBytes = 256;
#else
constexpr size_t kGuardBytes = 0;
#endif
constexpr unsigned char kGuardByte = 0xA5;

template <class T>
cudaError_t dalloc(dc_cache* h, T** p, size_t bytes) {
  if (g_fail_alloc_at.load() >= 0 && g_alloc_index.fetch_add(1) == g_fail_alloc_at.load()) {
    g_fail_alloc_at.store(-1);  // one-shot
    return cudaErrorMemoryAllocation;
  }
  const size_t nb = bytes ? bytes : 16;
  void* q = nullptr;
  cudaError_t e = cudaMalloc(&q, nb + 2 * kGuardBytes);
  if (e != cudaSuccess) return e;
  h->allocs.push_back(dc_cache::Alloc{q, nb});
  if (kGuardBytes) {
    e = cudaMemsetAsync(q, kGuardByte, kGuardBytes, h->stream);
    if (e == cudaSuccess) e = cudaMemsetAsync((char*)q + kGuardBytes + nb, kGuardByte, kGuardBytes, h->stream);
    if (e != cudaSuccess) return e;
  }
  *p = (T*)((char*)q + kGuardBytes);
  return cudaMemsetAsync(*p, 0, nb, h->stream);
}

// Frees one buffer of the handle (nullptr: nothing) and clears the pointer.
template <class T>
void dfree(dc_cache* h, T** p) {
  if (!*p) return;
  char* base = (char*)*p - kGuardBytes;
  for (size_t i = 0; i < h->allocs.size(); ++i)
    if (h->allocs[i].base == base) {
      cudaFree(base);
      h->allocs.erase(h->allocs.begin() + (long)i);
      break;
    }
  *p = nullptr;
}

void free_all(dc_cache* h) {
  for (const auto& a : h->allocs) cudaFree(a.base);
  h->allocs.clear();
}

// A failed allocation after creation: DC_ERR_OOM (the handle stays usable and
// unchanged), any other CUDA error as usual.
dc_status alloc_fail(dc_cache* h, cudaError_t e, const char* what) {
  if (e == cudaErrorMemoryAllocation) {
    cudaGetLastError();
    return fail(h, DC_ERR_OOM, std::string(what) + ": device allocation failed: " + cudaGetErrorString(e));
  }
  return cuda_fail(h, e, what);
}

// Split count and chunk (a multiple of 128 tokens) for n tokens per row.
void split_plan(const dc_cache* h, int n, int* nsplit, int* chunk) {
  int want = std::max(1, std::min(h->dev.smax, (n + 127) / 128));
  int c = (n + want - 1) / want;
  c = (c + 127) / 128 * 128;
  if (c < 128) c = 128;
  *chunk = c;
  *nsplit = std::max(1, (n + c - 1) / c);
}

cudaEvent_t take_event(dc_cache* h) {
  if (!h->event_pool.empty()) {
    cudaEvent_t e = h->event_pool.back();
    h->event_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

// Brackets the kernels of one phase: counts them and, when profiling, records
// CUDA events around them on the handle's stream.
struct Phase {
  dc_cache* h;
  int phase;
  cudaEvent_t a = nullptr;
  Phase(dc_cache* h_, int ph, int kernels) : h(h_), phase(ph) {
    h->launches[ph] += kernels;
    if (h->profiling) {
      a = take_event(h);
      cudaEventRecord(a, h->stream);
    }
  }
  ~Phase() {
    if (a) {
      cudaEvent_t b = take_event(h);
      cudaEventRecord(b, h->stream);
      h->timed.push_back({phase, a, b});
    }
  }
};

dc_status launch_error(dc_cache* h, const char* what) {
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(h, e, what);
  return DC_OK;
}

// Fused engine for a step over n tokens per row? (auto: whenever the rows fill
// at least half the SMs, else by the latency estimates below)
bool use_fused(const dc_cache* h, int n) {
  // rows of different lengths: the fused kernel ranks them with the policy only
  if (h->per_row && h->dev.scorer != 0) return false;
  if (!h->fused_ok || !dc::fused_eligible(h->dev, n)) return false;
  if (h->cfg.engine == 2) return true;
  if (h->cfg.engine != 0) return false;
  if (2 * h->dev.R >= h->num_sms) return true;
  // Few rows: the fused kernel gives each its own CTA, which streams a tile in
  // ~0.75 us after ~11 us of fixed cost (K and V: 1.5 us per 128 tokens), or
  // two CTAs (rows of 12 tiles or more, at most half as many rows as SMs: ~16
  // us with the exchange, 0.75 us per 128 tokens); the split engine spreads
  // the rows over the GPU but costs ~57 us of launches plus ~0.55 ns per
  // token-row (all measured on Mistral-7B head shapes). The split engine wins
  // only for a few very long rows.
  const double nT = (double)((n + 127) / 128);
  const bool halves = h->xflag != nullptr && 2 * h->dev.R <= h->num_sms && nT >= 12;
  const double fused_us = halves ? 16.0 + 0.75 * nT : 11.0 + 1.5 * nT;
  return fused_us < 57.0 + 0.00055 * (double)h->dev.R * (double)n;
}

cudaError_t upload_fused_policy(dc_cache* h, const float* blob) {
  std::vector<__nv_bfloat16> wt;
  dc::prepare_policy(blob, h->cfg.mlp_hidden, h->cfg.layernorm, &h->fpol, &wt);
  h->fpol.wtile = h->wtile;
  cudaError_t e = cudaMemcpyAsync(h->wtile, wt.data(), wt.size() * sizeof(__nv_bfloat16), cudaMemcpyHostToDevice,
                                  h->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(h->stream);
  return e;
}

// The step's common part: append the new pair, fill the step arguments.
dc::Step begin_step(dc_cache* h) {
  dc::Step st{};
  st.n = h->n + 1;
  st.p_newest = (int)h->seen;
  st.slot = (int)(h->steps % h->cfg.window);
  st.has_dep = h->steps >= h->cfg.window ? 1 : 0;
  st.p_dep = h->ring_pnew[st.slot];
  st.has_prev = h->steps >= 1 ? 1 : 0;
  st.slot_prev = (int)((h->steps + h->cfg.window - 1) % h->cfg.window);
  st.p_prev = h->ring_pnew[st.slot_prev];
  split_plan(h, st.n, &st.nsplit, &st.chunk);
  return st;
}

void end_step(dc_cache* h, const dc::Step& st) {
  h->n += 1;
  for (int& x : h->hlen) x += 1;
  h->seen += 1;
  h->ring_pnew[st.slot] = st.p_newest;
  h->steps += 1;
  h->have_scores = true;
}

bool run_split_step(dc_cache* h, const dc::Step& st, const void* q, float* out) {
  const dc::Dev& p = h->dev;
  if (!dc::split_supported(p)) return false;
  { Phase ph(h, DC_PHASE_ATTEND, 1); dc::launch_split_qk(p, st, q, h->stream); }
  { Phase ph(h, DC_PHASE_STATS, 1); dc::launch_split_stats(p, st, q, h->stream); }
  { Phase ph(h, DC_PHASE_SCORE, 1); dc::launch_split_v(p, st, h->stream); }
  { Phase ph(h, DC_PHASE_COMBINE, 1); dc::launch_split_out(p, st, out, h->stream); }
  if (p.seq_rows) {
    // global token mode: pool the rows' partial sums per sequence
    Phase ph(h, DC_PHASE_SCORE, 1);
    dc::launch_glob_features(p, st, h->stream);
  }
  return true;
}

}  // namespace

extern "C" {

dc_status dc_config_default(dc_config* cfg) {
  if (!cfg) return DC_ERR_INVALID_ARG;
  std::memset(cfg, 0, sizeof *cfg);
  cfg->batch = 1;
  cfg->q_heads = 0;
  cfg->window = 64;
  cfg->mlp_hidden = 128;
  cfg->layernorm = 1;
  cfg->alpha_mode = 0;
  cfg->engine = 0;
  cfg->keep_features = 0;
  cfg->seed = 0;
  cfg->stream = nullptr;
  cfg->tail_split = 1;
  cfg->scorer = 0;
  cfg->n_sinks = 4;
  cfg->budget_ratio = 0.f;
  cfg->budget_min = 32;
  cfg->budget_basis = 0;
  cfg->global_tokens = 0;
  return DC_OK;
}

size_t dc_policy_blob_len(int hidden) { return hidden > 0 ? (size_t)9 * hidden + 1 : 0; }

dc_status dc_policy_init(unsigned long long seed, int hidden, float* out, size_t n) {
  if (hidden <= 0 || !out || n < dc_policy_blob_len(hidden)) return DC_ERR_INVALID_ARG;
  const int H = hidden;
  uint64_t key = splitmix64(kTagPolicy);
  key = splitmix64(key ^ (uint64_t)seed);
  key = splitmix64(key ^ (uint64_t)H);
  const float b1 = (float)(1.0 / std::sqrt(5.0));
  const float b2 = (float)(1.0 / std::sqrt((double)H));
  auto draw = [&](uint64_t j) {
    float u = (float)(splitmix64(key + j) >> 40) / 16777216.0f;
    return 2.0f * u - 1.0f;  // exact: u has 24 bits
  };
  uint64_t j = 0;
  for (int i = 0; i < 5 * H; ++i) out[i] = draw(j++) * b1;            // W1
  for (int i = 0; i < H; ++i) out[5 * H + i] = draw(j++) * b1;        // b1
  for (int i = 0; i < H; ++i) out[6 * H + i] = 1.0f;                  // gamma
  for (int i = 0; i < H; ++i) out[7 * H + i] = 0.0f;                  // beta
  for (int i = 0; i < H; ++i) out[8 * H + i] = draw(j++) * b2;        // w2
  out[9 * H] = draw(j++) * b2;                                        // b2
  return DC_OK;
}

dc_status dc_cache_create(int layers, int kv_heads, int head_dim, int capacity, int budget,
                          const dc_config* cfg_in, dc_cache** out) {
  if (!out) return fail(nullptr, DC_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  dc_config cfg;
  if (cfg_in) cfg = *cfg_in; else dc_config_default(&cfg);
  if (cfg.q_heads == 0) cfg.q_heads = 4 * kv_heads;
  if (layers < 1 || kv_heads < 1 || cfg.batch < 1)
    return fail(nullptr, DC_ERR_INVALID_ARG, "layers, kv_heads and batch must be >= 1");
  if (head_dim != 64 && head_dim != 128) return fail(nullptr, DC_ERR_INVALID_ARG, "head_dim must be 64 or 128");
  if (cfg.q_heads % kv_heads) return fail(nullptr, DC_ERR_INVALID_ARG, "q_heads % kv_heads != 0");
  const int G = cfg.q_heads / kv_heads;
  if (G != 1 && G != 2 && G != 4 && G != 8) return fail(nullptr, DC_ERR_INVALID_ARG, "group must be 1, 2, 4 or 8");
  if (budget < 1 || capacity <= budget) return fail(nullptr, DC_ERR_INVALID_ARG, "need 1 <= budget < capacity");
  if (cfg.window < 1 || cfg.window > 1024) return fail(nullptr, DC_ERR_INVALID_ARG, "window must be in [1, 1024]");
  if (cfg.mlp_hidden < 1 || cfg.mlp_hidden > 256 || (cfg.mlp_hidden >= 32 && cfg.mlp_hidden % 32))
    return fail(nullptr, DC_ERR_INVALID_ARG, "mlp_hidden must be in [1, 256], a multiple of 32 when >= 32");
  if (cfg.alpha_mode != 0 && cfg.alpha_mode != 1) return fail(nullptr, DC_ERR_INVALID_ARG, "alpha_mode must be 0 or 1");
  if (cfg.scorer < 0 || cfg.scorer > 2) return fail(nullptr, DC_ERR_INVALID_ARG, "scorer must be 0, 1 or 2");
  if (cfg.n_sinks < 0) return fail(nullptr, DC_ERR_INVALID_ARG, "n_sinks must be >= 0");
  if (!(cfg.budget_ratio >= 0.f && cfg.budget_ratio <= 1.f) || cfg.budget_min < 1 ||
      (cfg.budget_basis != 0 && cfg.budget_basis != 1))
    return fail(nullptr, DC_ERR_INVALID_ARG, "need 0 <= budget_ratio <= 1, budget_min >= 1, budget_basis 0 or 1");
  if (cfg.scorer == 1) cfg.alpha_mode = 1;  // H2O ranks by the cumulative mass
  if (cfg.global_tokens != 0 && cfg.global_tokens != 1)
    return fail(nullptr, DC_ERR_INVALID_ARG, "global_tokens must be 0 or 1");
  if (cfg.engine < 0 || cfg.engine > 2) return fail(nullptr, DC_ERR_INVALID_ARG, "engine must be 0, 1 or 2");
  const long long R = (long long)layers * cfg.batch * kv_heads;
  if (R > 65535 || (long long)capacity * R > (1ll << 40) || capacity > (1 << 30))
    return fail(nullptr, DC_ERR_INVALID_ARG, "cache too large");

  dc_cache* h = new dc_cache();
  h->layers = layers; h->kv_heads = kv_heads; h->head_dim = head_dim;
  h->capacity = capacity; h->budget = budget; h->cfg = cfg;
  h->stream = (cudaStream_t)cfg.stream;
  h->ring_pnew.assign(cfg.window, -1);
  int dev_id = 0;
  cudaError_t e = cudaGetDevice(&dev_id);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, dev_id);
  if (e != cudaSuccess) {
    dc_status s = cuda_fail(nullptr, e, "cudaGetDevice");
    delete h;
    return s;
  }
  dc::Dev& p = h->dev;
  p.R = (int)R; p.cap = capacity; p.stride = (capacity + 127) / 128 * 128; p.d = head_dim; p.G = G; p.qh = cfg.q_heads; p.kvh = kv_heads;
  p.w = cfg.window; p.hidden = cfg.mlp_hidden; p.layernorm = cfg.layernorm ? 1 : 0;
  p.alpha_mode = cfg.alpha_mode; p.keep_features = cfg.keep_features ? 1 : 0;
  p.scorer = cfg.scorer; p.n_sinks = cfg.n_sinks;
  p.batch = cfg.batch;
  p.seq_rows = cfg.global_tokens ? layers * kv_heads : 0;
  p.c = (float)(1.4426950408889634 / std::sqrt((double)head_dim));
  p.smax = (int)std::max(1ll, std::min(64ll, (8ll * h->num_sms + R - 1) / R));
  const size_t RC = (size_t)R * p.stride;
  const size_t kv = RC * head_dim * sizeof(__nv_bfloat16);
  const size_t blob = dc_policy_blob_len(cfg.mlp_hidden);
  cudaError_t ae = cudaSuccess;
  auto A = [&](auto** ptr, size_t bytes) { if (ae == cudaSuccess) ae = dalloc(h, ptr, bytes); };
  A(&p.K, kv);
  A(&p.V, kv);
  A(&p.pos, RC * sizeof(int));
  A(&p.vnorm, RC * sizeof(float));
  A(&p.SZ, RC * sizeof(float4));
  if (cfg.alpha_mode == 1) A(&p.acc, RC * sizeof(float));
  A(&p.score, RC * sizeof(float));
  if (p.keep_features) A(&p.feat, RC * 5 * sizeof(float));
  A(&p.hq, (size_t)R * G * sizeof(float));
  A(&p.ring_q, (size_t)R * cfg.window * G * head_dim * sizeof(__nv_bfloat16));
  A(&p.ring_stats, (size_t)R * cfg.window * G * 4 * sizeof(float));
  float* pol = nullptr;
  A(&pol, blob * sizeof(float));
  p.policy = pol;
  A(&p.status, sizeof(unsigned));
  A(&p.dbg, 8 * sizeof(unsigned));
  A(&p.logit, RC * G * sizeof(float));
  A(&p.part, (size_t)R * p.smax * G * 4 * sizeof(float));
  A(&p.opart, (size_t)R * p.smax * G * head_dim * sizeof(float));
  A(&p.holes, RC * sizeof(int));
  A(&p.nmoves, (size_t)R * 2 * sizeof(int));
  if (p.seq_rows) {
    A(&p.gpart, RC * sizeof(float4));
    A(&p.gring, (size_t)cfg.batch * cfg.window * p.stride * sizeof(float2));
    A(&p.gmoves, (size_t)cfg.batch * (1 + 2 * (size_t)p.stride) * sizeof(int));
  }
  A(&h->st_q, (size_t)R * G * head_dim * 2);
  A(&h->st_k, (size_t)R * head_dim * 2);
  A(&h->st_v, (size_t)R * head_dim * 2);
  A(&h->st_out, (size_t)R * G * head_dim * sizeof(float));
  if (ae != cudaSuccess) {
    cudaGetLastError();
    cudaStreamSynchronize(h->stream);  // the zeroing of what was taken
    free_all(h);
    std::string m = std::string("device allocation failed: ") + cudaGetErrorString(ae);
    delete h;
    return fail(nullptr, ae == cudaErrorMemoryAllocation ? DC_ERR_OOM : DC_ERR_CUDA, m);
  }
  std::vector<float> w(blob);
  dc_policy_init(cfg.seed, cfg.mlp_hidden, w.data(), blob);
  e = cudaMemcpyAsync(pol, w.data(), blob * sizeof(float), cudaMemcpyHostToDevice, h->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(h->stream);
  if (e == cudaSuccess && cfg.engine != 1 && dc::fused_eligible(p, 1) && R * (long long)p.stride < (1ll << 31)) {
    const char* why = "";
    cudaError_t fe = dalloc(h, &h->wtile, 128 * 32 * sizeof(__nv_bfloat16));
    if (fe == cudaSuccess) fe = dc::make_fused_maps(p, &h->maps, &why);
    if (fe == cudaSuccess) fe = upload_fused_policy(h, w.data());
    if (fe == cudaSuccess) fe = dalloc(h, &h->work, 2 * sizeof(unsigned));
    if (fe == cudaSuccess) fe = cudaMemsetAsync(h->work, 0, 2 * sizeof(unsigned), h->stream);
    if (fe == cudaSuccess && cfg.tail_split) {
      // exchange slots: the last wave's half rows, or every row when rows are
      // at most half the SMs (fused_*_len(x) has x / 2 + 1 slots)
      const int grid = 2 * (int)std::min<long long>(R, h->num_sms);
      fe = dalloc(h, &h->xstats, dc::fused_xstats_len(grid, G) * sizeof(float));
      if (fe == cudaSuccess) fe = dalloc(h, &h->xo, dc::fused_xo_len(grid, G, head_dim) * sizeof(float));
      if (fe == cudaSuccess) fe = dalloc(h, &h->xsel, dc::fused_xsel_len(grid) * sizeof(int));
      if (fe == cudaSuccess) fe = dalloc(h, &h->xflag, dc::fused_xflag_len(grid) * sizeof(unsigned));
      if (fe == cudaSuccess)
        fe = cudaMemsetAsync(h->xflag, 0, dc::fused_xflag_len(grid) * sizeof(unsigned), h->stream);
      if (fe == cudaSuccess) fe = cudaStreamSynchronize(h->stream);
    }
    if (fe == cudaSuccess) {
      h->fused_ok = true;
    } else {
      cudaGetLastError();
      h->fused_why = why;
      // out of memory is reported as such; another failure (e.g. a tensor
      // map the driver rejects) leaves the split engine, unless the fused
      // engine was asked for
      if (cfg.engine == 2 || fe == cudaErrorMemoryAllocation) e = fe;
    }
  }
  if (e != cudaSuccess) {
    const bool oom = e == cudaErrorMemoryAllocation;
    dc_status s = oom ? fail(nullptr, DC_ERR_OOM, std::string("device allocation failed: ") + cudaGetErrorString(e))
                      : cuda_fail(nullptr, e, "policy upload");
    cudaGetLastError();
    cudaStreamSynchronize(h->stream);
    free_all(h);
    delete h;
    return s;
  }
  *out = h;
  return DC_OK;
}

dc_status dc_cache_destroy(dc_cache* h) {
  if (!h) return DC_OK;
  if (!valid(h)) return DC_ERR_INVALID_ARG;
  cudaStreamSynchronize(h->stream);
  if (h->h2d) {
    cudaStreamSynchronize(h->h2d);
    cudaStreamSynchronize(h->d2h);
    for (int i = 0; i < 2; ++i) {
      cudaEventDestroy(h->ev_in[i]);
      cudaEventDestroy(h->ev_done[i]);
      cudaEventDestroy(h->ev_out[i]);
    }
    cudaStreamDestroy(h->h2d);
    cudaStreamDestroy(h->d2h);
  }
  for (auto& t : h->timed) { cudaEventDestroy(t.a); cudaEventDestroy(t.b); }
  for (auto e : h->event_pool) cudaEventDestroy(e);
  if (h->ev_order) cudaEventDestroy(h->ev_order);
  if (h->horder) cudaFreeHost(h->horder);
  free_all(h);
  h->magic = kDead;
  delete h;
  return DC_OK;
}

dc_status dc_policy_set_weights(dc_cache* h, const float* blob, size_t n) {
  DC_CHECK_HANDLE(h);
  if (h->graph) return fail(h, DC_ERR_STATE, "graph mode: only dc_step and its host forms until dc_set_graph_mode(h, 0)");
  if (!blob || n != dc_policy_blob_len(h->cfg.mlp_hidden))
    return fail(h, DC_ERR_INVALID_ARG, "policy blob must hold 9 * mlp_hidden + 1 floats");
  DC_CUDA(h, cudaMemcpyAsync((void*)h->dev.policy, blob, n * sizeof(float), cudaMemcpyHostToDevice,
                             h->stream));
  DC_CUDA(h, cudaStreamSynchronize(h->stream));  // the caller may free the blob on return
  if (h->fused_ok) DC_CUDA(h, upload_fused_policy(h, blob));
  return DC_OK;
}

dc_status dc_append(dc_cache* h, const void* k, const void* v, int n_tokens) {
  DC_CHECK_HANDLE(h);
  if (h->graph) return fail(h, DC_ERR_STATE, "graph mode: only dc_step and its host forms until dc_set_graph_mode(h, 0)");
  if (n_tokens < 0 || (n_tokens > 0 && (!k || !v))) return fail(h, DC_ERR_INVALID_ARG, "bad append arguments");
  if (((uintptr_t)k | (uintptr_t)v) & 15) return fail(h, DC_ERR_INVALID_ARG, "k and v must be 16-byte aligned");
  if (n_tokens == 0) return DC_OK;
  if ((long long)h->n + n_tokens > h->capacity) return fail(h, DC_ERR_CAPACITY, "append exceeds capacity");
  if (h->seen + n_tokens > 0x7FFFFFFFll) return fail(h, DC_ERR_CAPACITY, "position counter overflow");
  {
    Phase ph(h, DC_PHASE_APPEND, h->per_row ? 2 : 1);
    dc::launch_append(h->dev, k, v, n_tokens, h->n, (int)h->seen, h->stream);
    if (h->per_row) dc::launch_rowlen_add(h->dev, n_tokens, h->stream);
  }
  dc_status s = launch_error(h, "append");
  if (s != DC_OK) return s;
  h->n += n_tokens;
  for (int& x : h->hlen) x += n_tokens;
  h->seen += n_tokens;
  h->have_scores = false;
  return DC_OK;
}

namespace {

// The budget of a step: the caller's if > 0, else the dynamic budget
// B_t = max(floor(r * L_t), B_min) (App. D) when configured, else the fixed
// one. L_t: tokens seen (basis 0) or tokens cached before the eviction
// (basis 1). Kept below the capacity so the next append fits.
int effective_budget(const dc_cache* h, int budget, int n_cached, long long seen) {
  if (budget > 0) return budget;
  if (h->cfg.budget_ratio <= 0.f) return h->budget;
  const double L = h->cfg.budget_basis == 0 ? (double)seen : (double)n_cached;
  long long B = (long long)std::floor((double)h->cfg.budget_ratio * L);
  if (B < h->cfg.budget_min) B = h->cfg.budget_min;
  if (B > h->capacity - 1) B = h->capacity - 1;
  return (int)B;
}

// Arguments of one fused launch; enables the half-row tail split when the
// handle has exchange buffers and the step qualifies.
dc::FusedStep fused_args(dc_cache* h, const dc::Step& st, const void* q, float* out, int do_evict, int B,
                         int write_scores) {
  dc::FusedStep fs{};
  fs.q = (const __nv_bfloat16*)q;
  fs.out = out;
  fs.do_evict = do_evict;
  fs.B = B;
  fs.write_scores = write_scores;
  fs.xstats = h->xstats;
  fs.xo = h->xo;
  fs.xsel = h->xsel;
  fs.xflag = h->xflag;
  fs.xslots = h->xflag ? (int)std::min<long long>(h->dev.R, h->num_sms) + 1 : 0;
  fs.work = h->work;
  fs.half_rows = (h->xflag && !h->per_row) ? dc::fused_half_rows(h->dev, st.n, fs, h->num_sms) : 0;
  // launch epoch: the queue counter is work[epoch & 1]; exchange flags hold
  // epoch * 4 + phase (1..3), so a flag left by an earlier launch never matches
  fs.epoch = ++h->epoch;
  return fs;
}

// One device-counted step (graph mode): the append and the fused step with the
// base arguments, which the kernels advance by the device's step count; the
// host's mirror of the step state stays at the base until the mode ends.
dc_status graph_step(dc_cache* h, const void* q, const void* k_new, const void* v_new, float* out, int budget) {
  if (budget > 0 && budget != h->budget) return fail(h, DC_ERR_INVALID_ARG, "graph mode keeps the configured budget");
  {
    Phase ph(h, DC_PHASE_APPEND, 1);
    dc::launch_append(h->dev, k_new, v_new, 1, h->n, h->gstep.p_newest, h->stream);
  }
  dc::FusedStep fs{};
  fs.q = (const __nv_bfloat16*)q;
  fs.out = out;
  fs.do_evict = 1;
  fs.B = h->budget;
  fs.xstats = h->xstats;
  fs.xo = h->xo;
  fs.xsel = h->xsel;
  fs.xflag = h->xflag;
  fs.xslots = h->xflag ? (int)std::min<long long>(h->dev.R, h->num_sms) + 1 : 0;
  fs.work = h->work;
  fs.half_rows = h->xflag ? dc::fused_half_rows(h->dev, h->gstep.n, fs, h->num_sms) : 0;
  fs.epoch = h->gepoch;
  cudaError_t e;
  {
    Phase ph(h, DC_PHASE_ATTEND, 1);
    e = dc::launch_fused_graph(h->maps, h->dev, h->gstep, fs, h->fpol, h->num_sms, h->stream);
  }
  if (e != cudaSuccess) return cuda_fail(h, e, "fused step (graph mode)");
  return DC_OK;
}

// Whether a decode step over n tokens would split the fused grid's last wave.
bool tail_split_applies(dc_cache* h, int n) {
  if (!h->xflag) return false;
  dc::FusedStep fs{};
  fs.xstats = h->xstats;
  fs.xo = h->xo;
  fs.xsel = h->xsel;
  fs.xflag = h->xflag;
  return dc::fused_half_rows(h->dev, n, fs, h->num_sms) > 0;
}

}  // namespace

dc_status dc_decode_step(dc_cache* h, const void* q, const void* k_new, const void* v_new, float* out) {
  DC_CHECK_HANDLE(h);
  if (h->graph) return fail(h, DC_ERR_STATE, "graph mode: only dc_step and its host forms until dc_set_graph_mode(h, 0)");
  if (!q || !k_new || !v_new || !out) return fail(h, DC_ERR_INVALID_ARG, "NULL pointer");
  if (((uintptr_t)q | (uintptr_t)k_new | (uintptr_t)v_new) & 15)
    return fail(h, DC_ERR_INVALID_ARG, "q, k_new and v_new must be 16-byte aligned");
  if (h->n + 1 > h->capacity) return fail(h, DC_ERR_CAPACITY, "decode step exceeds capacity");
  if (h->seen + 1 > 0x7FFFFFFFll) return fail(h, DC_ERR_CAPACITY, "position counter overflow");
  {
    Phase ph(h, DC_PHASE_APPEND, h->per_row ? 2 : 1);
    dc::launch_append(h->dev, k_new, v_new, 1, h->n, (int)h->seen, h->stream);
    if (h->per_row) dc::launch_rowlen_add(h->dev, 1, h->stream);
  }
  const dc::Step st = begin_step(h);
  if (use_fused(h, st.n)) {
    const dc::FusedStep fs = fused_args(h, st, q, out, 0, 0, h->dev.seq_rows ? 0 : 1);
    cudaError_t e;
    {
      Phase ph(h, DC_PHASE_ATTEND, 1);
      e = dc::launch_fused_step(h->maps, h->dev, st, fs, h->fpol, h->num_sms, h->stream);
    }
    if (e != cudaSuccess) return cuda_fail(h, e, "fused step");
    if (h->dev.seq_rows) {
      // global token mode: pool the rows' partial sums per sequence
      Phase ph(h, DC_PHASE_SCORE, 1);
      dc::launch_glob_features(h->dev, st, h->stream);
    }
  } else if (!run_split_step(h, st, q, out)) {
    return fail(h, DC_ERR_INVALID_ARG, "unsupported head_dim / group");
  }
  dc_status s = launch_error(h, "decode step");
  if (s != DC_OK) return s;
  end_step(h, st);
  return DC_OK;
}

namespace {

// Per-row mode: rows of many tiles first in the fused engine's queue, so that
// the CTAs finish together (a long row taken last would run alone). The order
// is rebuilt only when a row's tile count overtakes the one before it, and
// uploaded from a pinned buffer (the previous upload has finished before the
// buffer is rewritten).
dc_status update_row_order(dc_cache* h) {
  const int R = h->dev.R;
  auto tiles = [&](int r) { return (h->hlen[r] + 1 + 127) / 128; };  // after the step's append
  if (h->order_valid) {
    bool sorted = true;
    for (int i = 0; i + 1 < R && sorted; ++i) sorted = tiles(h->horder[i]) >= tiles(h->horder[i + 1]);
    if (sorted) return DC_OK;
  }
  // the buffers come with the per-row budgets (dc_set_row_budgets)
  DC_CUDA(h, cudaEventSynchronize(h->ev_order));
  for (int r = 0; r < R; ++r) h->horder[r] = r;
  std::stable_sort(h->horder, h->horder + R, [&](int a, int b) { return tiles(a) > tiles(b); });
  DC_CUDA(h, cudaMemcpyAsync(h->roworder_dev, h->horder, (size_t)R * sizeof(int), cudaMemcpyHostToDevice,
                             h->stream));
  DC_CUDA(h, cudaEventRecord(h->ev_order, h->stream));
  h->dev.roworder = h->roworder_dev;
  h->order_valid = true;
  return DC_OK;
}

}  // namespace

dc_status dc_step(dc_cache* h, const void* q, const void* k_new, const void* v_new, float* out, int budget) {
  DC_CHECK_HANDLE(h);
  if (!q || !k_new || !v_new || !out) return fail(h, DC_ERR_INVALID_ARG, "NULL pointer");
  if (((uintptr_t)q | (uintptr_t)k_new | (uintptr_t)v_new) & 15)
    return fail(h, DC_ERR_INVALID_ARG, "q, k_new and v_new must be 16-byte aligned");
  if (h->n + 1 > h->capacity) return fail(h, DC_ERR_CAPACITY, "decode step exceeds capacity");
  if (h->graph) return graph_step(h, q, k_new, v_new, out, budget);
  const int n1 = h->n + 1;
  if (!use_fused(h, n1) || h->dev.seq_rows) {  // global mode: per-sequence selection after the rows
    dc_status s = dc_decode_step(h, q, k_new, v_new, out);
    if (s != DC_OK) return s;
    return dc_evict(h, budget);
  }
  const int B = effective_budget(h, budget, n1, h->seen + 1);
  if (!h->per_row && B < n1 - 1 && (tail_split_applies(h, n1) || n1 - B > kFusedEvictMax)) {
    // several evictions need the whole row's scores in one CTA: with half
    // rows this step runs as the decode kernel plus the eviction kernel; so
    // does a step with many evictions (a prompt compression), whose moves the
    // eviction kernel makes with many more bytes in flight than the fused
    // kernel's epilogue
    dc_status s = dc_decode_step(h, q, k_new, v_new, out);
    if (s != DC_OK) return s;
    return dc_evict(h, budget);
  }
  if (h->seen + 1 > 0x7FFFFFFFll) return fail(h, DC_ERR_CAPACITY, "position counter overflow");
  {
    Phase ph(h, DC_PHASE_APPEND, h->per_row ? 2 : 1);
    dc::launch_append(h->dev, k_new, v_new, 1, h->n, (int)h->seen, h->stream);
    if (h->per_row) dc::launch_rowlen_add(h->dev, 1, h->stream);
  }
  if (h->per_row) {
    if (dc_status o = update_row_order(h); o != DC_OK) return o;
  }
  const dc::Step st = begin_step(h);
  if (h->per_row) {
    // every row to its own budget (B = 0), or all to `budget` when > 0; the
    // kernel writes the new lengths, the host mirrors them
    const dc::FusedStep fs = fused_args(h, st, q, out, 1, budget > 0 ? budget : 0, 0);
    cudaError_t e;
    {
      Phase ph(h, DC_PHASE_ATTEND, 1);
      e = dc::launch_fused_step(h->maps, h->dev, st, fs, h->fpol, h->num_sms, h->stream);
    }
    if (e != cudaSuccess) return cuda_fail(h, e, "fused step");
    end_step(h, st);
    int mx = 0;
    for (size_t r = 0; r < h->hlen.size(); ++r) {
      h->hlen[r] = std::min(h->hlen[r], budget > 0 ? budget : h->hbudget[r]);
      mx = std::max(mx, h->hlen[r]);
    }
    h->n = mx;
    h->have_scores = false;
    return DC_OK;
  }
  const int keep = std::min(st.n, B);
  const dc::FusedStep fs = fused_args(h, st, q, out, keep < st.n ? 1 : 0, keep, 0);
  cudaError_t e;
  {
    Phase ph(h, DC_PHASE_ATTEND, 1);
    e = dc::launch_fused_step(h->maps, h->dev, st, fs, h->fpol, h->num_sms, h->stream);
  }
  if (e != cudaSuccess) return cuda_fail(h, e, "fused step");
  end_step(h, st);
  h->n = keep;
  h->have_scores = false;
  return DC_OK;
}

namespace {

// The first staging set is shared with the asynchronous path, whose output
// copies run on their own stream: the handle's stream waits for them.
dc_status wait_async_copies(dc_cache* h) {
  if (h->h2d)
    for (int i = 0; i < 2; ++i) DC_CUDA(h, cudaStreamWaitEvent(h->stream, h->ev_out[i], 0));
  return DC_OK;
}

// dc_step with host buffers: inputs copied into the device staging buffers,
// the step, the output copied back, all in the handle's stream order (so the
// staging buffers are reused safely by the next call).
dc_status step_host(dc_cache* h, const void* q, const void* k_new, const void* v_new, float* out, int budget,
                    bool synchronise) {
  DC_CHECK_HANDLE(h);
  if (!q || !k_new || !v_new || !out) return fail(h, DC_ERR_INVALID_ARG, "NULL pointer");
  const size_t R = h->dev.R, G = h->dev.G, d = h->dev.d;
  if (dc_status w = wait_async_copies(h); w != DC_OK) return w;
  DC_CUDA(h, cudaMemcpyAsync(h->st_q, q, R * G * d * 2, cudaMemcpyHostToDevice, h->stream));
  DC_CUDA(h, cudaMemcpyAsync(h->st_k, k_new, R * d * 2, cudaMemcpyHostToDevice, h->stream));
  DC_CUDA(h, cudaMemcpyAsync(h->st_v, v_new, R * d * 2, cudaMemcpyHostToDevice, h->stream));
  dc_status s = dc_step(h, h->st_q, h->st_k, h->st_v, h->st_out, budget);
  if (s != DC_OK) return s;
  DC_CUDA(h, cudaMemcpyAsync(out, h->st_out, R * G * d * sizeof(float), cudaMemcpyDeviceToHost, h->stream));
  if (synchronise) DC_CUDA(h, cudaStreamSynchronize(h->stream));
  return DC_OK;
}

}  // namespace

dc_status dc_step_host(dc_cache* h, const void* q, const void* k_new, const void* v_new, float* out, int budget) {
  return step_host(h, q, k_new, v_new, out, budget, true);
}

// Two staging sets used in turn; the input copies of step s + 1 and the output
// copy of step s run on copy streams while step s (or s + 1) computes.

dc_status dc_step_host_async(dc_cache* h, const void* q, const void* k_new, const void* v_new, float* out,
                             int budget) {
  DC_CHECK_HANDLE(h);
  if (!q || !k_new || !v_new || !out) return fail(h, DC_ERR_INVALID_ARG, "NULL pointer");
  const size_t R = h->dev.R, G = h->dev.G, d = h->dev.d;
  if (!h->h2d) {
    cudaError_t ae = dalloc(h, &h->st2_q, R * G * d * 2);
    if (ae == cudaSuccess) ae = dalloc(h, &h->st2_k, R * d * 2);
    if (ae == cudaSuccess) ae = dalloc(h, &h->st2_v, R * d * 2);
    if (ae == cudaSuccess) ae = dalloc(h, &h->st2_out, R * G * d * sizeof(float));
    if (ae != cudaSuccess) {
      cudaStreamSynchronize(h->stream);
      dfree(h, &h->st2_q);
      dfree(h, &h->st2_k);
      dfree(h, &h->st2_v);
      dfree(h, &h->st2_out);
      return alloc_fail(h, ae, "second staging set");
    }
    DC_CUDA(h, cudaStreamCreateWithFlags(&h->h2d, cudaStreamNonBlocking));
    DC_CUDA(h, cudaStreamCreateWithFlags(&h->d2h, cudaStreamNonBlocking));
    for (int i = 0; i < 2; ++i) {
      DC_CUDA(h, cudaEventCreateWithFlags(&h->ev_in[i], cudaEventDisableTiming));
      DC_CUDA(h, cudaEventCreateWithFlags(&h->ev_done[i], cudaEventDisableTiming));
      DC_CUDA(h, cudaEventCreateWithFlags(&h->ev_out[i], cudaEventDisableTiming));
    }
    // the first uses of each buffer wait on events that have completed
    for (int i = 0; i < 2; ++i) {
      DC_CUDA(h, cudaEventRecord(h->ev_done[i], h->stream));
      DC_CUDA(h, cudaEventRecord(h->ev_out[i], h->stream));
    }
  }
  const int b = (int)(h->host_seq & 1);
  void* sq = b ? h->st2_q : h->st_q;
  void* sk = b ? h->st2_k : h->st_k;
  void* sv = b ? h->st2_v : h->st_v;
  float* so = b ? h->st2_out : h->st_out;
  // inputs: once the step two calls back has read this staging set
  DC_CUDA(h, cudaStreamWaitEvent(h->h2d, h->ev_done[b], 0));
  DC_CUDA(h, cudaMemcpyAsync(sq, q, R * G * d * 2, cudaMemcpyHostToDevice, h->h2d));
  DC_CUDA(h, cudaMemcpyAsync(sk, k_new, R * d * 2, cudaMemcpyHostToDevice, h->h2d));
  DC_CUDA(h, cudaMemcpyAsync(sv, v_new, R * d * 2, cudaMemcpyHostToDevice, h->h2d));
  DC_CUDA(h, cudaEventRecord(h->ev_in[b], h->h2d));
  // the step: after its inputs, and after the output of two calls back has left
  DC_CUDA(h, cudaStreamWaitEvent(h->stream, h->ev_in[b], 0));
  DC_CUDA(h, cudaStreamWaitEvent(h->stream, h->ev_out[b], 0));
  dc_status s = dc_step(h, sq, sk, sv, so, budget);
  if (s != DC_OK) return s;
  DC_CUDA(h, cudaEventRecord(h->ev_done[b], h->stream));
  // the output, on its own stream
  DC_CUDA(h, cudaStreamWaitEvent(h->d2h, h->ev_done[b], 0));
  DC_CUDA(h, cudaMemcpyAsync(out, so, R * G * d * sizeof(float), cudaMemcpyDeviceToHost, h->d2h));
  DC_CUDA(h, cudaEventRecord(h->ev_out[b], h->d2h));
  h->host_seq += 1;
  return DC_OK;
}

dc_status dc_engine(dc_cache* h, int n, int* engine) {
  if (!valid(h) || !engine) return DC_ERR_INVALID_ARG;
  const int nn = n > 0 ? n : h->n + 1;
  *engine = !use_fused(h, nn) ? 1 : dc::fused_pairs(h->dev, nn, h->num_sms) ? 3 : 2;
  return DC_OK;
}

dc_status dc_decode_step_host(dc_cache* h, const void* q, const void* k_new, const void* v_new,
                              float* out) {
  DC_CHECK_HANDLE(h);
  if (h->graph) return fail(h, DC_ERR_STATE, "graph mode: only dc_step and its host forms until dc_set_graph_mode(h, 0)");
  if (!q || !k_new || !v_new || !out) return fail(h, DC_ERR_INVALID_ARG, "NULL pointer");
  const size_t R = h->dev.R, G = h->dev.G, d = h->dev.d;
  if (dc_status w = wait_async_copies(h); w != DC_OK) return w;
  DC_CUDA(h, cudaMemcpyAsync(h->st_q, q, R * G * d * 2, cudaMemcpyHostToDevice, h->stream));
  DC_CUDA(h, cudaMemcpyAsync(h->st_k, k_new, R * d * 2, cudaMemcpyHostToDevice, h->stream));
  DC_CUDA(h, cudaMemcpyAsync(h->st_v, v_new, R * d * 2, cudaMemcpyHostToDevice, h->stream));
  dc_status s = dc_decode_step(h, h->st_q, h->st_k, h->st_v, h->st_out);
  if (s != DC_OK) return s;
  DC_CUDA(h, cudaMemcpyAsync(out, h->st_out, R * G * d * sizeof(float), cudaMemcpyDeviceToHost, h->stream));
  DC_CUDA(h, cudaStreamSynchronize(h->stream));
  return DC_OK;
}

dc_status dc_evict(dc_cache* h, int budget) {
  DC_CHECK_HANDLE(h);
  if (h->graph) return fail(h, DC_ERR_STATE, "graph mode: only dc_step and its host forms until dc_set_graph_mode(h, 0)");
  if (!h->have_scores) return fail(h, DC_ERR_STATE, "evict needs the scores of a decode step");
  if (h->per_row) {
    // every row to its own budget (or all to `budget` when > 0)
    {
      Phase ph(h, DC_PHASE_EVICT, dc::evict_kernel_count(h->n, budget > 0 ? budget : 0));
      dc::launch_evict(h->dev, h->n, budget > 0 ? budget : 0, h->stream);
    }
    dc_status s = launch_error(h, "evict");
    if (s != DC_OK) return s;
    int mx = 0;
    for (size_t r = 0; r < h->hlen.size(); ++r) {
      h->hlen[r] = std::min(h->hlen[r], budget > 0 ? budget : h->hbudget[r]);
      mx = std::max(mx, h->hlen[r]);
    }
    h->n = mx;
    h->have_scores = false;
    return DC_OK;
  }
  const int B = effective_budget(h, budget, h->n, h->seen);
  const int keep = std::min(h->n, B);
  if (keep < h->n) {
    Phase ph(h, DC_PHASE_EVICT, h->dev.seq_rows ? 2 : dc::evict_kernel_count(h->n, keep));
    if (h->dev.seq_rows) dc::launch_glob_evict(h->dev, h->n, keep, h->stream);
    else dc::launch_evict(h->dev, h->n, keep, h->stream);
    dc_status s = launch_error(h, "evict");
    if (s != DC_OK) return s;
  }
  h->n = keep;
  h->have_scores = false;
  return DC_OK;
}

dc_status dc_full_decode(dc_cache* h, const void* q, float* out) {
  DC_CHECK_HANDLE(h);
  if (h->graph) return fail(h, DC_ERR_STATE, "graph mode: only dc_step and its host forms until dc_set_graph_mode(h, 0)");
  if (!q || !out) return fail(h, DC_ERR_INVALID_ARG, "NULL pointer");
  if (h->n < 1) return fail(h, DC_ERR_STATE, "the cache is empty");
  if (h->per_row && std::any_of(h->hlen.begin(), h->hlen.end(), [&](int x) { return x != h->n; }))
    return fail(h, DC_ERR_STATE, "full decode needs rows of equal length (per-row budgets differ)");
  if (h->fused_ok && dc::fused_eligible(h->dev, h->n)) {
    // the fused kernel's attention-only variant (TMA + tensor cores)
    dc::Step st{};
    st.n = h->n;
    const dc::FusedStep fs = fused_args(h, st, q, out, 0, 0, 0);
    cudaError_t e;
    {
      Phase ph(h, DC_PHASE_FULL, 1);
      e = dc::launch_fused_full(h->maps, h->dev, h->n, fs, h->fpol, h->num_sms, h->stream);
    }
    if (e != cudaSuccess) return cuda_fail(h, e, "full decode");
    return launch_error(h, "full decode");
  }
  int nsplit, chunk;
  split_plan(h, h->n, &nsplit, &chunk);
  bool ok;
  {
    Phase ph(h, DC_PHASE_FULL, 2);
    ok = dc::launch_full_decode(h->dev, h->n, nsplit, chunk, q, out, h->stream);
  }
  if (!ok) return fail(h, DC_ERR_INVALID_ARG, "unsupported head_dim / group");
  return launch_error(h, "full decode");
}

dc_status dc_set_row_budgets(dc_cache* h, const int* budgets, int n) {
  DC_CHECK_HANDLE(h);
  if (h->graph) return fail(h, DC_ERR_STATE, "graph mode: only dc_step and its host forms until dc_set_graph_mode(h, 0)");
  dc::Dev& p = h->dev;
  if (!budgets) {
    if (!h->per_row) return DC_OK;
    for (int x : h->hlen)
      if (x != h->n) return fail(h, DC_ERR_STATE, "rows hold different lengths: per-row budgets stay on");
    h->per_row = false;
    h->hlen.clear();
    p.rowlen = nullptr;
    p.rowbudget = nullptr;
    p.roworder = nullptr;
    h->order_valid = false;
    return DC_OK;
  }
  if (n != p.R) return fail(h, DC_ERR_INVALID_ARG, "one budget per row (layers x batch x kv_heads)");
  if (p.seq_rows) return fail(h, DC_ERR_STATE, "per-row budgets do not apply to the global token mode");
  for (int r = 0; r < n; ++r)
    if (budgets[r] < 1) return fail(h, DC_ERR_INVALID_ARG, "budgets must be >= 1");
  if (!h->rowlen_dev) {
    // row lengths, budgets and the fused queue's row order (device), with the
    // order's pinned host copy and the event of its last upload
    cudaError_t ae = dalloc(h, &h->rowlen_dev, (size_t)n * sizeof(int));
    if (ae == cudaSuccess) ae = dalloc(h, &h->rowbudget_dev, (size_t)n * sizeof(int));
    if (ae == cudaSuccess) ae = dalloc(h, &h->roworder_dev, (size_t)n * sizeof(int));
    if (ae != cudaSuccess) {
      cudaStreamSynchronize(h->stream);
      dfree(h, &h->rowlen_dev);
      dfree(h, &h->rowbudget_dev);
      dfree(h, &h->roworder_dev);
      return alloc_fail(h, ae, "per-row budgets");
    }
    DC_CUDA(h, cudaHostAlloc(reinterpret_cast<void**>(&h->horder), (size_t)n * sizeof(int), cudaHostAllocDefault));
    DC_CUDA(h, cudaEventCreateWithFlags(&h->ev_order, cudaEventDisableTiming));
    DC_CUDA(h, cudaEventRecord(h->ev_order, h->stream));
  }
  if (!h->per_row) {
    h->hlen.assign(n, h->n);
    DC_CUDA(h, cudaMemcpyAsync(h->rowlen_dev, h->hlen.data(), (size_t)n * sizeof(int), cudaMemcpyHostToDevice,
                               h->stream));
  }
  h->hbudget.assign(budgets, budgets + n);
  DC_CUDA(h, cudaMemcpyAsync(h->rowbudget_dev, budgets, (size_t)n * sizeof(int), cudaMemcpyHostToDevice, h->stream));
  DC_CUDA(h, cudaStreamSynchronize(h->stream));  // the caller may free `budgets` on return
  p.rowlen = h->rowlen_dev;
  p.rowbudget = h->rowbudget_dev;
  h->per_row = true;
  return DC_OK;
}

dc_status dc_set_graph_mode(dc_cache* h, int enable) {
  DC_CHECK_HANDLE(h);
  const int w = h->cfg.window;
  if (enable) {
    if (h->graph) return DC_OK;
    if (h->per_row || h->dev.seq_rows || h->dev.scorer != 0 || h->cfg.budget_ratio > 0.f)
      return fail(h, DC_ERR_STATE, "graph mode needs the policy scorer, one fixed budget for every row, per-row selection");
    if (h->n != h->budget || h->n + 1 > h->capacity)
      return fail(h, DC_ERR_STATE, "graph mode needs the steady state: the cache at its budget, one eviction per step");
    if (h->steps < w) return fail(h, DC_ERR_STATE, "graph mode needs a full window of decode steps first");
    // the window's queries of consecutive steps (no appends in between)
    for (int k = 1; k <= w; ++k)
      if (h->ring_pnew[(size_t)((h->steps - k) % w)] != (int)(h->seen - k))
        return fail(h, DC_ERR_STATE, "graph mode needs the window's last steps to be consecutive decode steps");
    if (!use_fused(h, h->n + 1)) return fail(h, DC_ERR_STATE, "graph mode runs on the fused engine only");
    if (h->seen + (1ll << 30) > 0x7FFFFFFFll) return fail(h, DC_ERR_CAPACITY, "position counter too close to its limit");
    if (!h->gcount_dev) {
      cudaError_t ae = dalloc(h, &h->gcount_dev, 2 * sizeof(int));
      if (ae != cudaSuccess) {
        cudaStreamSynchronize(h->stream);
        dfree(h, &h->gcount_dev);
        return alloc_fail(h, ae, "graph mode step counter");
      }
    }
    DC_CUDA(h, cudaMemsetAsync(h->gcount_dev, 0, 2 * sizeof(int), h->stream));
    h->gstep = begin_step(h);
    h->gepoch = h->epoch + 1;
    h->dev.gcount = h->gcount_dev;
    h->graph = true;
    return DC_OK;
  }
  if (!h->graph) return DC_OK;
  int t = 0;
  DC_CUDA(h, cudaStreamSynchronize(h->stream));
  DC_CUDA(h, cudaMemcpy(&t, h->gcount_dev, sizeof t, cudaMemcpyDeviceToHost));
  // the host mirror takes the t steps the device counted
  const long long steps0 = h->steps, seen0 = h->seen;
  for (long long k = (t > w ? t - w : 0); k < t; ++k) h->ring_pnew[(size_t)((steps0 + k) % w)] = (int)(seen0 + k);
  h->seen += t;
  h->steps += t;
  h->epoch = h->gepoch + (unsigned)t - 1u;
  h->have_scores = false;
  h->dev.gcount = nullptr;
  h->graph = false;
  return DC_OK;
}

dc_status dc_get_row_lengths(dc_cache* h, int* lengths, int n) {
  DC_CHECK_HANDLE(h);
  if (!lengths || n != h->dev.R) return fail(h, DC_ERR_INVALID_ARG, "one length per row");
  for (int r = 0; r < n; ++r) lengths[r] = h->per_row ? h->hlen[r] : h->n;
  return DC_OK;
}

dc_status dc_get_length(dc_cache* h, int* n, long long* seen) {
  if (!valid(h)) return DC_ERR_INVALID_ARG;
  if (n) *n = h->n;
  if (seen) *seen = h->seen;
  return DC_OK;
}

// Base pointer, element size and elements per slot of an internal buffer
// (stored with the padded row stride; the ABI view is [R][capacity]).
static char* buffer_ptr(dc_cache* h, dc_buffer which, size_t* elem, size_t* per_slot) {
  const dc::Dev& p = h->dev;
  *per_slot = 1;
  switch (which) {
    case DC_BUF_K: *elem = 2; *per_slot = p.d; return (char*)p.K;
    case DC_BUF_V: *elem = 2; *per_slot = p.d; return (char*)p.V;
    case DC_BUF_POS: *elem = 4; return (char*)p.pos;
    case DC_BUF_S: *elem = 8; return (char*)p.SZ;
    case DC_BUF_Z: *elem = 8; return (char*)p.SZ;
    case DC_BUF_ACC: *elem = 4; return (char*)p.acc;
    case DC_BUF_SCORE: *elem = 4; return (char*)p.score;
    case DC_BUF_FEAT: *elem = 4; *per_slot = 5; return (char*)p.feat;
    case DC_BUF_HQ: *elem = 4; *per_slot = p.G; return (char*)p.hq;
    case DC_BUF_VNORM: *elem = 4; return (char*)p.vnorm;
  }
  *elem = 0;
  return nullptr;
}

static size_t row_bytes(dc_cache* h, dc_buffer which) {
  size_t elem = 0, per = 0;
  char* b = buffer_ptr(h, which, &elem, &per);
  if (!b) return 0;
  return which == DC_BUF_HQ ? elem * per : elem * per * (size_t)h->capacity;
}

dc_status dc_buffer_bytes(dc_cache* h, dc_buffer which, size_t* rb) {
  if (!valid(h) || !rb) return DC_ERR_INVALID_ARG;
  *rb = row_bytes(h, which);
  return DC_OK;
}

dc_status dc_copy_buffer(dc_cache* h, dc_buffer which, int row0, int nrows, void* dst, size_t bytes) {
  DC_CHECK_HANDLE(h);
  size_t elem = 0, per = 0;
  char* src = buffer_ptr(h, which, &elem, &per);
  const size_t rb = row_bytes(h, which);
  if (!src || rb == 0 || !dst) return fail(h, DC_ERR_INVALID_ARG, "the cache has no such buffer");
  if (row0 < 0 || nrows < 0 || row0 + nrows > h->dev.R || bytes != rb * (size_t)nrows)
    return fail(h, DC_ERR_INVALID_ARG, "row range or size mismatch");
  if (nrows == 0) return DC_OK;
  if (which == DC_BUF_S || which == DC_BUF_Z) {
    dc::launch_convert_sz(h->dev, row0, nrows, which == DC_BUF_S ? 0 : 1, (double*)dst, h->stream);
    return launch_error(h, "window-sum copy");
  }
  if (which == DC_BUF_HQ) {
    DC_CUDA(h, cudaMemcpyAsync(dst, src + rb * (size_t)row0, bytes, cudaMemcpyDeviceToDevice, h->stream));
    return DC_OK;
  }
  const size_t spitch = elem * per * (size_t)h->dev.stride;
  DC_CUDA(h, cudaMemcpy2DAsync(dst, rb, src + spitch * (size_t)row0, spitch, rb, (size_t)nrows,
                               cudaMemcpyDeviceToDevice, h->stream));
  return DC_OK;
}

dc_status dc_sync(dc_cache* h) {
  DC_CHECK_HANDLE(h);
  DC_CUDA(h, cudaStreamSynchronize(h->stream));
  if (h->h2d) {
    DC_CUDA(h, cudaStreamSynchronize(h->h2d));
    DC_CUDA(h, cudaStreamSynchronize(h->d2h));
  }
  unsigned st = 0, dbg[8] = {};
  DC_CUDA(h, cudaMemcpy(&st, h->dev.status, sizeof st, cudaMemcpyDeviceToHost));
  DC_CUDA(h, cudaMemcpy(dbg, h->dev.dbg, sizeof dbg, cudaMemcpyDeviceToHost));
  if (st) {
    char buf[256];
    std::snprintf(buf, sizeof buf,
                  "kernel status word 0x%x (first wait timeout: site %u block %u parity %u info 0x%x; "
                  "first failed index check: site %u index %u limit %u)",
                  st, dbg[1], dbg[2], dbg[3], dbg[4], dbg[5], dbg[6], dbg[7]);
    return fail(h, DC_ERR_DEVICE, buf);
  }
  if (kGuardBytes) {
    // debug builds: the guard regions around every buffer are intact
    std::vector<unsigned char> g(kGuardBytes);
    for (size_t a = 0; a < h->allocs.size(); ++a) {
      for (int side = 0; side < 2; ++side) {
        const char* at = (const char*)h->allocs[a].base + (side ? kGuardBytes + h->allocs[a].bytes : 0);
        DC_CUDA(h, cudaMemcpy(g.data(), at, kGuardBytes, cudaMemcpyDeviceToHost));
        for (size_t i = 0; i < kGuardBytes; ++i)
          if (g[i] != kGuardByte) {
            char buf[160];
            std::snprintf(buf, sizeof buf, "guard region %s buffer %zu (%zu bytes) overwritten at byte %zu",
                          side ? "after" : "before", a, h->allocs[a].bytes, i);
            return fail(h, DC_ERR_DEVICE, buf);
          }
      }
    }
  }
  return DC_OK;
}

dc_status dc_debug_fail_alloc(long long nth) {
  g_alloc_index.store(0);
  g_fail_alloc_at.store(nth < 0 ? -1 : nth);
  return DC_OK;
}

int dc_debug_checks(void) { return kGuardBytes ? 1 : 0; }

dc_status dc_debug_corrupt_guard(dc_cache* h) {
  DC_CHECK_HANDLE(h);
  if (!kGuardBytes || h->allocs.empty()) return fail(h, DC_ERR_STATE, "not a debug build (DC_DEBUG_BOUNDS)");
  // the first byte of the guard region after the first buffer (K): memory the
  // handle owns, outside every buffer
  char* at = (char*)h->allocs[0].base + kGuardBytes + h->allocs[0].bytes;
  DC_CUDA(h, cudaMemsetAsync(at, (unsigned char)~kGuardByte, 1, h->stream));
  return DC_OK;
}

const char* dc_phase_name(int phase) {
  static const char* names[DC_PHASE_COUNT] = {"append", "attend", "stats", "score", "combine", "evict", "full"};
  return (phase >= 0 && phase < DC_PHASE_COUNT) ? names[phase] : "";
}

dc_status dc_profile_enable(dc_cache* h, int on) {
  DC_CHECK_HANDLE(h);
  DC_CUDA(h, cudaStreamSynchronize(h->stream));
  for (auto& t : h->timed) { h->event_pool.push_back(t.a); h->event_pool.push_back(t.b); }
  h->timed.clear();
  for (int i = 0; i < DC_PHASE_COUNT; ++i) { h->launches[i] = 0; h->ms[i] = 0.0; }
  h->profiling = on != 0;
  return DC_OK;
}

dc_status dc_profile_read(dc_cache* h, double* ms, long long* launches) {
  DC_CHECK_HANDLE(h);
  DC_CUDA(h, cudaStreamSynchronize(h->stream));
  for (auto& t : h->timed) {
    float x = 0.f;
    DC_CUDA(h, cudaEventElapsedTime(&x, t.a, t.b));
    h->ms[t.phase] += x;
    h->event_pool.push_back(t.a);
    h->event_pool.push_back(t.b);
  }
  h->timed.clear();
  for (int i = 0; i < DC_PHASE_COUNT; ++i) {
    if (ms) ms[i] = h->ms[i];
    if (launches) launches[i] = h->launches[i];
  }
  return DC_OK;
}

const char* dc_last_error(const dc_cache* h) {
  if (!h) return g_create_error.c_str();
  if (!valid(h)) return "invalid handle";
  return h->err.c_str();
}

}  // extern "C"
