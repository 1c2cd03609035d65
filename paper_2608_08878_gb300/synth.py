"""Seeded synthetic inputs for the budgeted KV-eviction decode step.

This module only makes inputs. It holds none of the method's arithmetic: no
attention, no features, no policy scoring, no selection. Both the fp64 CPU
oracle (through the tests) and the CUDA path consume what it produces, and the
CUDA side has its own implementation of the same generator (``csrc/synth.cu``)
for inputs too large to build on the host. Both follow the definition below,
so sampled rows of a device-generated cache can be rebuilt here bit for bit.

Generator definition
--------------------
* ``splitmix64`` is Steele, Lea and Flood's SplitMix64 output function
  (golden-gamma increment followed by the two xor-shift-multiply rounds).
* A stream key is ``mix(tag, w1, w2, ...)``: start from ``splitmix64(tag)`` and
  fold each word in as ``h = splitmix64(h ^ w)``.
* Element ``j`` of a normal stream draws three words
  ``splitmix64(key + 3j + c)`` for ``c = 0, 1, 2`` (mod 2^64), splits each into
  four 16-bit unsigned integers and sums the twelve (Irwin-Hall, k = 12). The
  value ``(sum - 393210) / 65536`` has mean 0 and variance ``1 - 2^-32`` and is
  exact in fp32.
* Element ``j`` of a uniform stream is ``(splitmix64(key + j) >> 40) / 2^24``.
* bf16 values are the fp32 value rounded to nearest even (the bits are kept as
  ``uint16``).

Workload recipe (the synthetic stand-in for the paper's LongBench, GSM8K and
BBH prompts on Mistral-7B, none of which are available here)
------------------------------------------------------------------------------
Per row (layer, batch, kv_head):

* ``u_e``: a per-row "query direction" for hot-set epoch ``e``, N(0, I_d).
* prompt key of token ``t``:
    - sink (``t < n_sinks``): ``sink_scale * N(0, I)``;
    - heavy hitter (position hash ``% 100 < hot_sets`` and not a sink): hot set
      ``e = hash % 100`` gets ``hh_scale * u_e + N(0, I)``;
    - otherwise ``N(0, I)``.
* prompt value: ``N(0, I)``.
* decode step ``s``: every query head of the group gets
  ``q_align * u_e + N(0, I)`` with ``e = (s // epoch_len) % hot_sets``;
  the new key and value are ``N(0, I)``.

The fp32 arithmetic above is one multiply by an fp32 constant followed by one
add, each rounded separately (no fused multiply-add), then bf16 rounding.
"""

from __future__ import annotations

from dataclasses import dataclass, field, replace
import math

import numpy as np

MASK64 = (1 << 64) - 1
_GAMMA = 0x9E3779B97F4A7C15
_M1 = 0xBF58476D1CE4E5B9
_M2 = 0x94D049BB133111EB

# Stream tags (arbitrary distinct constants, shared with csrc/synth.cu).
TAG_KEY = 0x4B455900  # "KEY"
TAG_VAL = 0x56414C00  # "VAL"
TAG_DIR = 0x44495200  # "DIR"
TAG_HOT = 0x484F5400  # "HOT"
TAG_QRY = 0x51525900  # "QRY"
TAG_KNEW = 0x4B4E5700  # "KNW"
TAG_VNEW = 0x564E5700  # "VNW"
TAG_POLICY = 0x504F4C00  # "POL"


def splitmix64_int(x: int) -> int:
    """SplitMix64 output function on a Python int (mod 2^64)."""
    z = (x + _GAMMA) & MASK64
    z = ((z ^ (z >> 30)) * _M1) & MASK64
    z = ((z ^ (z >> 27)) * _M2) & MASK64
    return z ^ (z >> 31)


def splitmix64(x: np.ndarray) -> np.ndarray:
    """Vectorised SplitMix64 output function on uint64 arrays (wrapping)."""
    x = np.asarray(x, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = x + np.uint64(_GAMMA)
        z = (z ^ (z >> np.uint64(30))) * np.uint64(_M1)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(_M2)
    return z ^ (z >> np.uint64(31))


def mix(tag: int, *words: int) -> int:
    """Stream key: fold each word into the tag's hash."""
    h = splitmix64_int(tag & MASK64)
    for w in words:
        h = splitmix64_int(h ^ (int(w) & MASK64))
    return h


def normal_f32(key: int, n: int, start: int = 0) -> np.ndarray:
    """Elements ``start .. start+n-1`` of the Irwin-Hall normal stream ``key``."""
    j = np.arange(start, start + n, dtype=np.uint64)
    base = (np.uint64(key) + np.uint64(3) * j) if n else j
    total = np.zeros(n, dtype=np.int64)
    with np.errstate(over="ignore"):
        for c in range(3):
            w = splitmix64(base + np.uint64(c))
            for s in (0, 16, 32, 48):
                total += ((w >> np.uint64(s)) & np.uint64(0xFFFF)).astype(np.int64)
    return ((total - 393210).astype(np.float32) / np.float32(65536.0)).astype(np.float32)


def normal_rows_f32(keys: np.ndarray, n: int) -> np.ndarray:
    """Elements ``0 .. n-1`` of the normal streams ``keys`` (one row per key)."""
    keys = np.asarray(keys, dtype=np.uint64).reshape(-1, 1)
    j = np.arange(n, dtype=np.uint64).reshape(1, -1)
    total = np.zeros((keys.shape[0], n), dtype=np.int64)
    with np.errstate(over="ignore"):
        base = keys + np.uint64(3) * j
        for c in range(3):
            w = splitmix64(base + np.uint64(c))
            for s in (0, 16, 32, 48):
                total += ((w >> np.uint64(s)) & np.uint64(0xFFFF)).astype(np.int64)
    return ((total - 393210).astype(np.float32) / np.float32(65536.0)).astype(np.float32)


def fold(prefix: int, words: np.ndarray) -> np.ndarray:
    """``mix(..., w)`` for many last words ``w`` sharing the key ``prefix``."""
    with np.errstate(over="ignore"):
        return splitmix64(np.uint64(prefix) ^ np.asarray(words, dtype=np.uint64))


def uniform_f32(key: int, n: int) -> np.ndarray:
    """First ``n`` elements of the uniform [0, 1) stream ``key`` (24-bit)."""
    j = np.arange(n, dtype=np.uint64)
    with np.errstate(over="ignore"):
        w = splitmix64(np.uint64(key) + j)
    return ((w >> np.uint64(40)).astype(np.float32) / np.float32(16777216.0)).astype(np.float32)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 to bf16 (nearest even); returns the 16-bit patterns."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    rounded = (b + np.uint64(0x7FFF) + ((b >> np.uint64(16)) & np.uint64(1))) >> np.uint64(16)
    return rounded.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Widen bf16 bit patterns to fp32 (exact)."""
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


@dataclass(frozen=True)
class Workload:
    """Shape and structure of one synthetic decode workload."""

    name: str
    layers: int
    batch: int
    kv_heads: int
    q_heads: int
    head_dim: int
    prompt_len: int
    budget: int
    steps: int
    n_sinks: int = 4
    sink_scale: float = 4.0
    hot_sets: int = 1          # hot sets of 1% of positions each (0: none)
    hh_scale: float = 4.0
    q_align: float = 0.1
    epoch_len: int = 1 << 30   # steps per hot-set epoch
    mlp_hidden: int = 128
    layernorm: int = 1
    window: int = 64
    alpha_mode: int = 0
    seed: int = 1              # workload seed (policy weights use policy_seed)
    policy_seed: int = 0
    extra: dict = field(default_factory=dict, compare=False)

    @property
    def group(self) -> int:
        return self.q_heads // self.kv_heads

    @property
    def rows(self) -> int:
        return self.layers * self.batch * self.kv_heads

    @property
    def capacity(self) -> int:
        return max(self.prompt_len, self.budget) + 1

    def row_index(self, layer: int, b: int, g: int) -> int:
        return (layer * self.batch + b) * self.kv_heads + g

    def row_coords(self, r: int):
        g = r % self.kv_heads
        b = (r // self.kv_heads) % self.batch
        layer = r // (self.kv_heads * self.batch)
        return layer, b, g

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


def round_half_up(x: float) -> int:
    return int(math.floor(x + 0.5))


# The five workloads of the decode-step benchmark (shapes are Mistral-7B's KV
# layout: 32 layers, 32 query / 8 KV heads, head_dim 128).
TINY = Workload("tiny: 1 layer, 4q/2kv, d64, prompt 512, budget 128", 1, 1, 2, 4, 64, 512, 128, 16,
                n_sinks=2, hot_sets=0, q_align=0.0, mlp_hidden=64, layernorm=0, seed=11)
MISTRAL_1L = Workload("mistral-7b single layer: 32q/8kv, d128, prompt 8192, budget 2048", 1, 1, 8, 32,
                      128, 8192, 2048, 128, seed=12)
MISTRAL_FULL = Workload("mistral-7b 32 layers, batch 8, context 32768, budget 8192", 32, 8, 8, 32, 128,
                        32768, 8192, 64, seed=13)
AGGRESSIVE = Workload("mistral-7b 32 layers, batch 16, context 32768, budget 3277 (10%)", 32, 16, 8,
                      32, 128, 32768, 3277, 64, hot_sets=4, epoch_len=16, seed=14)


def sweep_point(batch: int, ctx: int, ratio: float) -> Workload:
    """One point of the throughput sweep: 32 layers, budget round-half-up(ratio*ctx)."""
    return Workload(f"sweep b{batch} ctx{ctx} r{ratio}", 32, batch, 8, 32, 128, ctx,
                    round_half_up(ratio * ctx), 32, seed=15)


# ----------------------------------------------------------------------------
# Row streams
# ----------------------------------------------------------------------------

def direction(wl: Workload, layer: int, b: int, g: int, epoch: int = 0) -> np.ndarray:
    return normal_f32(mix(TAG_DIR, wl.seed, layer, b, g, epoch), wl.head_dim)


def hot_set(wl: Workload, layer: int, b: int, g: int, t: np.ndarray) -> np.ndarray:
    """Hot-set id of each prompt position (-1 if none)."""
    t = np.asarray(t, dtype=np.uint64)
    key = mix(TAG_HOT, wl.seed, layer, b, g)
    with np.errstate(over="ignore"):
        h = (splitmix64(np.uint64(key) + t) % np.uint64(100)).astype(np.int64)
    out = np.where(h < wl.hot_sets, h, -1)
    out[t.astype(np.int64) < wl.n_sinks] = -1
    return out


def prompt_row(wl: Workload, layer: int, b: int, g: int, t0: int = 0, t1: int | None = None):
    """bf16 bits of prompt keys and values of one row for positions [t0, t1)."""
    if t1 is None:
        t1 = wl.prompt_len
    d = wl.head_dim
    t = np.arange(t0, t1, dtype=np.int64)
    nk = normal_rows_f32(fold(mix(TAG_KEY, wl.seed, layer, b, g), t), d)
    v = normal_rows_f32(fold(mix(TAG_VAL, wl.seed, layer, b, g), t), d)
    hs = hot_set(wl, layer, b, g, t)
    k = nk.copy()
    sink = t < wl.n_sinks
    k[sink] = np.float32(wl.sink_scale) * nk[sink]
    for e in range(wl.hot_sets):
        sel = hs == e
        if sel.any():
            u = direction(wl, layer, b, g, e)
            k[sel] = (np.float32(wl.hh_scale) * u)[None, :] + nk[sel]
    return f32_to_bf16_bits(k), f32_to_bf16_bits(v)


def step_row(wl: Workload, step: int, layer: int, b: int, g: int):
    """bf16 bits of (q [G][d], k_new [d], v_new [d]) of one row at decode step ``step``."""
    d, G = wl.head_dim, wl.group
    e = (step // wl.epoch_len) % max(wl.hot_sets, 1)
    u = direction(wl, layer, b, g, e)
    q = np.empty((G, d), dtype=np.float32)
    for j in range(G):
        n = normal_f32(mix(TAG_QRY, wl.seed, layer, b, g * G + j, step), d)
        q[j] = (np.float32(wl.q_align) * u) + n
    kn = normal_f32(mix(TAG_KNEW, wl.seed, layer, b, g, step), d)
    vn = normal_f32(mix(TAG_VNEW, wl.seed, layer, b, g, step), d)
    return f32_to_bf16_bits(q), f32_to_bf16_bits(kn), f32_to_bf16_bits(vn)


def prompt_all(wl: Workload):
    """bf16 bits of the whole prompt, [L][b][kvh][T][d] (small workloads only)."""
    L, B, KV, T, d = wl.layers, wl.batch, wl.kv_heads, wl.prompt_len, wl.head_dim
    k = np.empty((L, B, KV, T, d), dtype=np.uint16)
    v = np.empty_like(k)
    for layer in range(L):
        for b in range(B):
            for g in range(KV):
                k[layer, b, g], v[layer, b, g] = prompt_row(wl, layer, b, g)
    return k, v


def step_all(wl: Workload, step: int):
    """bf16 bits of (q [L][b][qh][d], k_new [L][b][kvh][d], v_new [L][b][kvh][d])."""
    L, B, KV, G, d = wl.layers, wl.batch, wl.kv_heads, wl.group, wl.head_dim
    q = np.empty((L, B, KV * G, d), dtype=np.uint16)
    kn = np.empty((L, B, KV, d), dtype=np.uint16)
    vn = np.empty_like(kn)
    for layer in range(L):
        for b in range(B):
            for g in range(KV):
                qq, kk, vv = step_row(wl, step, layer, b, g)
                q[layer, b, g * G:(g + 1) * G] = qq
                kn[layer, b, g] = kk
                vn[layer, b, g] = vv
    return q, kn, vn


# ----------------------------------------------------------------------------
# Policy weights (the policy network's parameters are an input: random from a
# seed, as no trained weights exist)
# ----------------------------------------------------------------------------

N_FEATURES = 5


def policy_blob_len(hidden: int) -> int:
    return 9 * hidden + 1


def policy_weights(seed: int, hidden: int) -> np.ndarray:
    """fp32 blob ``[W1 (hidden x 5, row-major) | b1 | gamma | beta | w2 | b2]``.

    Linear layers follow PyTorch's default rule: weights and biases uniform in
    ``[-1/sqrt(fan_in), 1/sqrt(fan_in)]``. LayerNorm gain 1, shift 0. Draw
    order: W1, b1, w2, b2 from one uniform stream.
    """
    H = hidden
    n_draw = 5 * H + H + H + 1
    u = uniform_f32(mix(TAG_POLICY, seed, H), n_draw)
    two, one = np.float32(2.0), np.float32(1.0)
    sym = (two * u) - one  # in [-1, 1)
    bound1 = np.float32(1.0 / math.sqrt(N_FEATURES))
    bound2 = np.float32(1.0 / math.sqrt(H))
    W1 = sym[: 5 * H] * bound1
    b1 = sym[5 * H: 6 * H] * bound1
    w2 = sym[6 * H: 7 * H] * bound2
    b2 = sym[7 * H: 7 * H + 1] * bound2
    gamma = np.ones(H, dtype=np.float32)
    beta = np.zeros(H, dtype=np.float32)
    return np.concatenate([W1, b1, gamma, beta, w2, b2]).astype(np.float32)
