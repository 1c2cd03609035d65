"""Python binding of the C ABI in ``include/distillcache.h`` (argument
marshalling only: every step of the decode path runs in the CUDA library).

Device memory and streams come from PyTorch; tensors are passed to the library
as raw device pointers. There is no CPU fallback: if ``libdistillcache.so`` is
missing, opening it raises.
"""

from __future__ import annotations

import ctypes as C
import os
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
# DC_LIBRARY=debug selects the build with device-side index checks and guard
# regions (build.build_debug); the default is the release library.
LIB_PATH = os.path.join(_HERE, "libdistillcache_debug.so" if os.environ.get("DC_LIBRARY") == "debug"
                        else "libdistillcache.so")

DC_OK, DC_ERR_INVALID_ARG, DC_ERR_CAPACITY, DC_ERR_OOM, DC_ERR_CUDA, DC_ERR_DEVICE, DC_ERR_STATE = range(7)
STATUS_NAMES = ["DC_OK", "DC_ERR_INVALID_ARG", "DC_ERR_CAPACITY", "DC_ERR_OOM", "DC_ERR_CUDA",
                "DC_ERR_DEVICE", "DC_ERR_STATE"]

BUF_K, BUF_V, BUF_POS, BUF_S, BUF_Z, BUF_ACC, BUF_SCORE, BUF_FEAT, BUF_HQ, BUF_VNORM = range(10)

# Every function the header declares (checked by the tests).
EXPORTS = ["dc_config_default", "dc_cache_create", "dc_cache_destroy", "dc_policy_blob_len",
           "dc_policy_init", "dc_policy_set_weights", "dc_append", "dc_decode_step",
           "dc_decode_step_host", "dc_evict", "dc_full_decode", "dc_get_length", "dc_buffer_bytes",
           "dc_copy_buffer", "dc_sync", "dc_last_error", "dc_phase_name", "dc_profile_enable",
           "dc_profile_read", "dc_step", "dc_step_host", "dc_step_host_async", "dc_engine", "dc_attend_noalloc",
           "dc_noalloc_last_error", "dc_pl_log_partition", "dc_gumbel_top_b", "dc_train_last_error",
           "dc_set_row_budgets", "dc_get_row_lengths", "dc_wait_selftest", "dc_selftest_last_error",
           "dc_set_graph_mode", "dc_debug_fail_alloc", "dc_debug_checks", "dc_debug_bounds_selftest",
           "dc_debug_corrupt_guard"]
PHASES = ["append", "attend", "stats", "score", "combine", "evict", "full"]


class dc_config(C.Structure):
    _fields_ = [("batch", C.c_int), ("q_heads", C.c_int), ("window", C.c_int),
                ("mlp_hidden", C.c_int), ("layernorm", C.c_int), ("alpha_mode", C.c_int),
                ("engine", C.c_int), ("keep_features", C.c_int), ("seed", C.c_ulonglong),
                ("stream", C.c_void_p), ("tail_split", C.c_int), ("scorer", C.c_int),
                ("n_sinks", C.c_int), ("budget_ratio", C.c_float), ("budget_min", C.c_int),
                ("budget_basis", C.c_int), ("global_tokens", C.c_int)]


class DCError(RuntimeError):
    def __init__(self, status: int, msg: str):
        self.status = status
        name = STATUS_NAMES[status] if 0 <= status < len(STATUS_NAMES) else str(status)
        super().__init__(f"{name}: {msg}")


_lib = None
_lock = threading.Lock()


def lib():
    """Opens libdistillcache.so (raises if it has not been built)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise OSError(f"{LIB_PATH} is missing: build it with "
                              "`python -m paper_2608_08878_gb300.build`")
            L = C.CDLL(LIB_PATH)
            P, I, S = C.c_void_p, C.c_int, C.c_size_t
            L.dc_config_default.argtypes = [C.POINTER(dc_config)]
            L.dc_cache_create.argtypes = [I, I, I, I, I, C.POINTER(dc_config), C.POINTER(P)]
            L.dc_cache_destroy.argtypes = [P]
            L.dc_policy_blob_len.argtypes = [I]
            L.dc_policy_blob_len.restype = S
            L.dc_policy_init.argtypes = [C.c_ulonglong, I, P, S]
            L.dc_policy_set_weights.argtypes = [P, P, S]
            L.dc_append.argtypes = [P, P, P, I]
            L.dc_decode_step.argtypes = [P, P, P, P, P]
            L.dc_decode_step_host.argtypes = [P, P, P, P, P]
            L.dc_evict.argtypes = [P, I]
            L.dc_step.argtypes = [P, P, P, P, P, I]
            L.dc_step_host.argtypes = [P, P, P, P, P, I]
            L.dc_step_host_async.argtypes = [P, P, P, P, P, I]
            L.dc_engine.argtypes = [P, I, C.POINTER(I)]
            L.dc_attend_noalloc.argtypes = [P, P, P, I, I, I, I, P, P]
            L.dc_noalloc_last_error.argtypes = []
            L.dc_noalloc_last_error.restype = C.c_char_p
            L.dc_full_decode.argtypes = [P, P, P]
            L.dc_set_row_budgets.argtypes = [P, P, I]
            L.dc_set_graph_mode.argtypes = [P, I]
            L.dc_get_row_lengths.argtypes = [P, P, I]
            L.dc_pl_log_partition.argtypes = [P, I, I, I, C.c_float, P, P]
            L.dc_gumbel_top_b.argtypes = [P, P, I, I, I, C.c_float, P, P, P, P]
            L.dc_train_last_error.argtypes = []
            L.dc_train_last_error.restype = C.c_char_p
            L.dc_wait_selftest.argtypes = [C.c_ulonglong, P, P]
            L.dc_debug_fail_alloc.argtypes = [C.c_longlong]
            L.dc_debug_checks.argtypes = []
            L.dc_debug_bounds_selftest.argtypes = [P, P]
            L.dc_debug_corrupt_guard.argtypes = [P]
            L.dc_selftest_last_error.argtypes = []
            L.dc_selftest_last_error.restype = C.c_char_p
            L.dc_get_length.argtypes = [P, C.POINTER(I), C.POINTER(C.c_longlong)]
            L.dc_buffer_bytes.argtypes = [P, I, C.POINTER(S)]
            L.dc_copy_buffer.argtypes = [P, I, I, I, P, S]
            L.dc_sync.argtypes = [P]
            L.dc_last_error.argtypes = [P]
            L.dc_last_error.restype = C.c_char_p
            L.dc_phase_name.argtypes = [I]
            L.dc_phase_name.restype = C.c_char_p
            L.dc_profile_enable.argtypes = [P, I]
            L.dc_profile_read.argtypes = [P, P, P]
            for name in EXPORTS:
                if name not in ("dc_policy_blob_len", "dc_last_error", "dc_phase_name", "dc_noalloc_last_error",
                                "dc_train_last_error", "dc_selftest_last_error"):
                    getattr(L, name).restype = I
            _lib = L
    return _lib


def policy_blob_len(hidden: int) -> int:
    return int(lib().dc_policy_blob_len(hidden))


def policy_init(seed: int, hidden: int) -> np.ndarray:
    """The library's seeded initial policy weights (host-only, no GPU needed)."""
    n = policy_blob_len(hidden)
    out = np.empty(n, dtype=np.float32)
    st = lib().dc_policy_init(seed, hidden, out.ctypes.data_as(C.c_void_p), n)
    if st != DC_OK:
        raise DCError(st, "dc_policy_init rejected its arguments")
    return out


def attend_noalloc(q, k, v, out=None, stream=None):
    """Full-cache decode attention with no device allocation by the library:
    q [rows][group][d], k/v [rows][n][d] bf16 CUDA tensors -> out fp32.

    The library takes the device from the current CUDA device, so the call
    runs with q's device made current, on `stream` (which must belong to that
    device) or that device's current stream."""
    import torch
    if not isinstance(q, torch.Tensor) or q.dim() != 3 or not isinstance(k, torch.Tensor) or k.dim() != 3:
        raise DCError(DC_ERR_INVALID_ARG, "q must be [rows][group][head_dim] and k, v [rows][n][head_dim]")
    if not isinstance(v, torch.Tensor) or tuple(v.shape) != tuple(k.shape):
        raise DCError(DC_ERR_INVALID_ARG, f"v must have k's shape {tuple(k.shape)}")
    if not q.is_cuda:
        raise DCError(DC_ERR_INVALID_ARG, "q must be a CUDA tensor")
    rows, group, d = q.shape
    n = k.shape[1]
    if k.shape[0] != rows or k.shape[2] != d:
        raise DCError(DC_ERR_INVALID_ARG, f"k has shape {tuple(k.shape)}, expected ({rows}, n, {d})")
    dev = q.device.index
    pq = _arg(q, "q", torch.bfloat16, rows * group * d, device=dev)
    pk = _arg(k, "k", torch.bfloat16, rows * n * d, device=dev)
    pv = _arg(v, "v", torch.bfloat16, rows * n * d, device=dev)
    if out is None:
        out = torch.empty((rows, group, d), dtype=torch.float32, device=q.device)
    po = _arg(out, "out", torch.float32, rows * group * d, device=dev)
    if stream is not None and stream.device != q.device:
        raise DCError(DC_ERR_INVALID_ARG, f"stream is on {stream.device}, the tensors on {q.device}")
    with torch.cuda.device(q.device):
        s = (stream or torch.cuda.current_stream(q.device)).cuda_stream
        st = lib().dc_attend_noalloc(pq, pk, pv, rows, n, d, group, po, s)
    if st != DC_OK:
        raise DCError(st, lib().dc_noalloc_last_error().decode())
    return out


def debug_fail_alloc(nth: int) -> None:
    """Testing hook: the nth device allocation from now on fails as if the
    device were out of memory (once); nth < 0 disarms."""
    lib().dc_debug_fail_alloc(int(nth))


def debug_checks() -> bool:
    """Whether the loaded library is the debug build (index checks, guards)."""
    return bool(lib().dc_debug_checks())


def debug_bounds_selftest(stream=None) -> dict:
    """Debug builds: an index one past its limit must fail its check, raise
    the status bit, record site 903 and skip the access."""
    import torch
    res = np.zeros(5, dtype=np.uint32)
    s = (stream or torch.cuda.current_stream()).cuda_stream
    st = lib().dc_debug_bounds_selftest(res.ctypes.data_as(C.c_void_p), s)
    if st != DC_OK:
        raise DCError(st, lib().dc_selftest_last_error().decode())
    return {"status": int(res[0]), "site": int(res[1]), "index": int(res[2]), "limit": int(res[3]),
            "skipped": bool(res[4])}


def wait_selftest(limit_ms: float = 50.0, stream=None) -> dict:
    """Runs the bounded-wait self-test (a flag nothing sets, an mbarrier
    nothing arrives on, each waited for limit_ms) and returns what the kernel
    recorded."""
    import torch
    res = np.zeros(7, dtype=np.uint32)
    s = (stream or torch.cuda.current_stream()).cuda_stream
    st = lib().dc_wait_selftest(C.c_ulonglong(int(limit_ms * 1e6)), res.ctypes.data_as(C.c_void_p), s)
    if st != DC_OK:
        raise DCError(st, lib().dc_selftest_last_error().decode())
    return {"flag_gave_up": bool(res[0] & 1), "barrier_gave_up": bool(res[0] & 2), "site": int(res[2]),
            "flag_wait_us": int(res[5]), "barrier_wait_us": int(res[6])}


def pl_log_partition(scores, B: int, tau: float = 1.0, out=None, stream=None):
    """Exact log Z of the Plackett-Luce distribution over size-B subsets for
    each row of scores (fp32 CUDA tensor [rows][L]) -> fp32 [rows] (App. C)."""
    import torch
    if not isinstance(scores, torch.Tensor) or scores.dim() != 2:
        raise DCError(DC_ERR_INVALID_ARG, "scores must be a [rows][L] tensor")
    rows, L = scores.shape
    dev = scores.device.index if scores.is_cuda else None
    ps = _arg(scores, "scores", torch.float32, rows * L, device=dev)
    if out is None:
        out = torch.empty(rows, dtype=torch.float32, device=scores.device)
    po = _arg(out, "out", torch.float32, rows, device=dev)
    s = (stream or torch.cuda.current_stream()).cuda_stream
    st = lib().dc_pl_log_partition(ps, rows, L, B, tau, po, s)
    if st != DC_OK:
        raise DCError(st, lib().dc_train_last_error().decode())
    return out


def gumbel_top_b(scores, gumbel, B: int, tau: float = 1.0, with_logp: bool = True, stream=None):
    """Gumbel-top-B sample per row (scores, gumbel: fp32 CUDA tensors [rows][L]):
    the B kept indices ascending (int32 [rows][B]) and, if with_logp, the
    subset's Plackett-Luce log-probability (fp32 [rows]) (App. C)."""
    import torch
    if not isinstance(scores, torch.Tensor) or scores.dim() != 2:
        raise DCError(DC_ERR_INVALID_ARG, "scores must be a [rows][L] tensor")
    rows, L = scores.shape
    dev = scores.device.index if scores.is_cuda else None
    _arg(scores, "scores", torch.float32, rows * L, device=dev)
    _arg(gumbel, "gumbel", torch.float32, rows * L, device=dev)
    if B < 1:
        raise DCError(DC_ERR_INVALID_ARG, "B must be >= 1")
    idx = torch.empty((rows, B), dtype=torch.int32, device=scores.device)
    logp = torch.empty(rows, dtype=torch.float32, device=scores.device) if with_logp else None
    logz = torch.empty(rows, dtype=torch.float32, device=scores.device) if with_logp else None
    s = (stream or torch.cuda.current_stream()).cuda_stream
    st = lib().dc_gumbel_top_b(scores.data_ptr(), gumbel.data_ptr(), rows, L, B, tau, idx.data_ptr(),
                               _ptr(logp), _ptr(logz), s)
    if st != DC_OK:
        raise DCError(st, lib().dc_train_last_error().decode())
    return idx, logp


def head_level_hybrid_budgets(rows: int, context: int, full_rows, overall_ratio: float = 0.25):
    """Per-row budgets of the head-level hybrid (Sec. 5): the rows in
    `full_rows` keep the whole context, the others share what is left of an
    overall budget of overall_ratio x context per row, equally (at least 1)."""
    import numpy as np
    full = np.zeros(rows, dtype=bool)
    full[list(full_rows)] = True
    nf = int(full.sum())
    total = overall_ratio * context * rows
    rest = max(1, int((total - nf * context) // max(rows - nf, 1)))
    return np.where(full, context, rest).astype(np.int32)


def _ptr(t) -> int:
    return 0 if t is None else int(t.data_ptr())


def _arg(t, name: str, dtype, numel: int, cuda: bool = True, device: int | None = None) -> int:
    """The address of tensor argument `name` after checking what the C ABI
    assumes of it: device memory (or host memory for the *_host calls) on the
    expected device, the element type, a dense row-major layout and the element
    count. The library sees only the pointer, so a tensor that fails one of
    these would be read or written out of bounds (on the GPU: a memory fault).
    Raises DCError(DC_ERR_INVALID_ARG) before anything is enqueued."""
    import torch
    if not isinstance(t, torch.Tensor):
        raise DCError(DC_ERR_INVALID_ARG, f"{name} must be a torch tensor")
    if t.is_cuda != cuda:
        raise DCError(DC_ERR_INVALID_ARG, f"{name} must be a {'CUDA' if cuda else 'host (CPU)'} tensor")
    if cuda and device is not None and t.device.index != device:
        raise DCError(DC_ERR_INVALID_ARG, f"{name} is on cuda:{t.device.index}, expected cuda:{device}")
    if t.dtype != dtype:
        raise DCError(DC_ERR_INVALID_ARG, f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise DCError(DC_ERR_INVALID_ARG, f"{name} must be contiguous (dense row-major)")
    if t.numel() != numel:
        raise DCError(DC_ERR_INVALID_ARG, f"{name} has {t.numel()} elements, expected {numel}")
    return int(t.data_ptr())


class DistillCache:
    """A budgeted KV cache of ``layers x batch x kv_heads`` rows on the current
    CUDA device, driven through the C ABI on one CUDA stream."""

    def __init__(self, layers: int, kv_heads: int, head_dim: int, capacity: int, budget: int, *,
                 batch: int = 1, q_heads: int | None = None, window: int = 64,
                 mlp_hidden: int = 128, layernorm: int = 1, alpha_mode: int = 0, engine: int = 0,
                 keep_features: bool = False, seed: int = 0, stream=None, tail_split: bool = True,
                 scorer: int = 0, n_sinks: int = 4, budget_ratio: float = 0.0, budget_min: int = 32,
                 budget_basis: int = 0, global_tokens: bool = False):
        import torch
        L = lib()
        cfg = dc_config()
        L.dc_config_default(C.byref(cfg))
        cfg.batch, cfg.q_heads, cfg.window = batch, q_heads or 4 * kv_heads, window
        cfg.mlp_hidden, cfg.layernorm, cfg.alpha_mode = mlp_hidden, layernorm, alpha_mode
        cfg.engine, cfg.keep_features, cfg.seed = engine, int(bool(keep_features)), seed
        cfg.tail_split = int(bool(tail_split))
        cfg.scorer, cfg.n_sinks = scorer, n_sinks
        cfg.budget_ratio, cfg.budget_min, cfg.budget_basis = budget_ratio, budget_min, budget_basis
        cfg.global_tokens = int(bool(global_tokens))
        if stream is None:
            stream = torch.cuda.current_stream()
        self.stream = stream
        cfg.stream = stream.cuda_stream
        h = C.c_void_p()
        st = L.dc_cache_create(layers, kv_heads, head_dim, capacity, budget, C.byref(cfg), C.byref(h))
        if st != DC_OK:
            raise DCError(st, L.dc_last_error(None).decode())
        self._h = h
        self.layers, self.kv_heads, self.head_dim = layers, kv_heads, head_dim
        self.capacity, self.budget, self.batch = capacity, budget, batch
        self.q_heads = cfg.q_heads
        self.group = self.q_heads // kv_heads
        self.rows = layers * batch * kv_heads
        self.mlp_hidden = mlp_hidden
        self.device = torch.cuda.current_device()

    # -- lifetime ----------------------------------------------------------
    def close(self) -> None:
        if getattr(self, "_h", None):
            lib().dc_cache_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *a):
        self.close()

    def _check(self, st: int) -> None:
        if st != DC_OK:
            raise DCError(st, lib().dc_last_error(self._h).decode())

    # -- the ABI -----------------------------------------------------------
    def set_policy(self, blob: np.ndarray) -> None:
        blob = np.ascontiguousarray(blob, dtype=np.float32)
        self._check(lib().dc_policy_set_weights(self._h, blob.ctypes.data_as(C.c_void_p), blob.size))

    def _step_args(self, q, k_new, v_new, out, cuda: bool = True):
        """Addresses of one decode step's tensors: q bf16 [layers][batch][q_heads][d],
        k_new, v_new bf16 [layers][batch][kv_heads][d], out fp32 like q."""
        import torch
        nq, nkv = self.layers * self.batch * self.q_heads * self.head_dim, self.rows * self.head_dim
        dev = self.device if cuda else None
        return (_arg(q, "q", torch.bfloat16, nq, cuda, dev), _arg(k_new, "k_new", torch.bfloat16, nkv, cuda, dev),
                _arg(v_new, "v_new", torch.bfloat16, nkv, cuda, dev), _arg(out, "out", torch.float32, nq, cuda, dev))

    def _out_like(self, q, out):
        import torch
        if out is None and isinstance(q, torch.Tensor):
            out = torch.empty(q.shape, dtype=torch.float32, device=q.device)
        return out

    def append(self, k, v) -> None:
        """k, v: bf16 CUDA tensors [layers][batch][kv_heads][T][head_dim]."""
        import torch
        if not isinstance(k, torch.Tensor) or not isinstance(v, torch.Tensor) or k.shape != v.shape:
            raise DCError(DC_ERR_INVALID_ARG, "k and v must be tensors of the same shape")
        T = int(k.shape[-2]) if k.numel() else 0
        n = self.rows * T * self.head_dim
        pk = _arg(k, "k", torch.bfloat16, n, device=self.device)
        pv = _arg(v, "v", torch.bfloat16, n, device=self.device)
        self._check(lib().dc_append(self._h, pk, pv, T))

    def decode_step(self, q, k_new, v_new, out=None):
        out = self._out_like(q, out)
        self._check(lib().dc_decode_step(self._h, *self._step_args(q, k_new, v_new, out)))
        return out

    def decode_step_host(self, q, k_new, v_new, out) -> None:
        """Host (preferably pinned) tensors; synchronises before returning."""
        self._check(lib().dc_decode_step_host(self._h, *self._step_args(q, k_new, v_new, out, cuda=False)))

    def step(self, q, k_new, v_new, out=None, budget: int = 0):
        """decode_step + evict (one kernel on the fused engine)."""
        out = self._out_like(q, out)
        self._check(lib().dc_step(self._h, *self._step_args(q, k_new, v_new, out), budget))
        return out

    def step_host(self, q, k_new, v_new, out, budget: int = 0) -> None:
        self._check(lib().dc_step_host(self._h, *self._step_args(q, k_new, v_new, out, cuda=False), budget))

    def step_host_async(self, q, k_new, v_new, out, budget: int = 0) -> None:
        """step_host without the final synchronisation (pinned host tensors;
        `out` is valid after sync())."""
        self._check(lib().dc_step_host_async(self._h, *self._step_args(q, k_new, v_new, out, cuda=False), budget))

    def debug_corrupt_guard(self) -> None:
        """Debug builds: damages a guard region so the next sync() must fail."""
        self._check(lib().dc_debug_corrupt_guard(self._h))

    def set_graph_mode(self, enable: bool = True) -> None:
        """Device-counted steps: a CUDA graph captured from one step() replays
        as the following steps (see dc_set_graph_mode)."""
        self._check(lib().dc_set_graph_mode(self._h, int(bool(enable))))

    def engine(self, n: int = 0) -> str:
        e = C.c_int()
        self._check(lib().dc_engine(self._h, n, C.byref(e)))
        return {1: "split", 2: "fused", 3: "fused-pairs"}[e.value]

    def evict(self, budget: int = 0) -> None:
        self._check(lib().dc_evict(self._h, budget))

    def full_decode(self, q, out=None):
        import torch
        out = self._out_like(q, out)
        nq = self.layers * self.batch * self.q_heads * self.head_dim
        pq = _arg(q, "q", torch.bfloat16, nq, device=self.device)
        po = _arg(out, "out", torch.float32, nq, device=self.device)
        self._check(lib().dc_full_decode(self._h, pq, po))
        return out

    def set_row_budgets(self, budgets) -> None:
        """Per-row budgets (head-level hybrid); None returns to one budget."""
        import numpy as np
        if budgets is None:
            self._check(lib().dc_set_row_budgets(self._h, None, 0))
            return
        b = np.ascontiguousarray(budgets, dtype=np.int32)
        self._check(lib().dc_set_row_budgets(self._h, b.ctypes.data_as(C.c_void_p), b.size))

    def row_lengths(self):
        import numpy as np
        out = np.empty(self.rows, dtype=np.int32)
        self._check(lib().dc_get_row_lengths(self._h, out.ctypes.data_as(C.c_void_p), out.size))
        return out

    def length(self):
        n, seen = C.c_int(), C.c_longlong()
        self._check(lib().dc_get_length(self._h, C.byref(n), C.byref(seen)))
        return n.value, seen.value

    def profile(self, on: bool = True) -> None:
        """Zeroes the launch counters; with on=True also times every launch."""
        self._check(lib().dc_profile_enable(self._h, int(on)))

    def profile_read(self) -> dict:
        """{phase: (total kernel ms, launches)} since the last profile() call."""
        ms = (C.c_double * len(PHASES))()
        n = (C.c_longlong * len(PHASES))()
        self._check(lib().dc_profile_read(self._h, ms, n))
        return {PHASES[i]: (ms[i], n[i]) for i in range(len(PHASES))}

    def sync(self) -> None:
        self._check(lib().dc_sync(self._h))

    def buffer(self, which: int, row0: int = 0, nrows: int | None = None):
        """A device copy of rows [row0, row0 + nrows) of an internal buffer."""
        import torch
        if nrows is None:
            nrows = self.rows - row0
        rb = C.c_size_t()
        self._check(lib().dc_buffer_bytes(self._h, which, C.byref(rb)))
        cap, d, G = self.capacity, self.head_dim, self.group
        spec = {BUF_K: (torch.bfloat16, (cap, d)), BUF_V: (torch.bfloat16, (cap, d)),
                BUF_POS: (torch.int32, (cap,)), BUF_S: (torch.float64, (cap,)),
                BUF_Z: (torch.float64, (cap,)), BUF_ACC: (torch.float32, (cap,)),
                BUF_SCORE: (torch.float32, (cap,)), BUF_FEAT: (torch.float32, (cap, 5)),
                BUF_HQ: (torch.float32, (G,)), BUF_VNORM: (torch.float32, (cap,))}[which]
        if rb.value == 0:
            raise DCError(DC_ERR_INVALID_ARG, "the cache has no such buffer")
        out = torch.empty((nrows,) + spec[1], dtype=spec[0], device="cuda")
        self._check(lib().dc_copy_buffer(self._h, which, row0, nrows, _ptr(out), rb.value * nrows))
        return out
