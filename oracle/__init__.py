"""ctypes binding of the fp64 CPU oracle (``dc_oracle.c``).

TEST INFRASTRUCTURE ONLY: the tests, the package smoke check and the
benchmark's CPU-baseline leg may import this module; the product path never
does. The oracle shares no code with the CUDA path.
"""

from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "dc_oracle.c")
_LIB_PATH = os.path.join(_HERE, "libdc_oracle.so")
# A separately compiled copy of the oracle to load instead (the mutation tests
# load copies with a planted mistake); never set outside the tests.
_LIB_OVERRIDE = os.environ.get("DC_ORACLE_LIB")
_lib = None
_lock = threading.Lock()


def build(force: bool = False) -> str:
    """Compiles the oracle with gcc (plain C11, -O2, no fast-math)."""
    if _LIB_OVERRIDE:
        return _LIB_OVERRIDE
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < max(
            os.path.getmtime(_SRC), os.path.getmtime(os.path.join(_HERE, "dc_oracle.h"))):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math",
                               "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def lib():
    global _lib
    with _lock:
        if _lib is None:
            L = C.CDLL(build())
            P = C.c_void_p
            L.dco_row_new.restype = P
            L.dco_row_new.argtypes = [C.c_int] * 5
            L.dco_row_free.argtypes = [P]
            L.dco_row_append.argtypes = [P, P, P, C.c_int]
            L.dco_row_step.argtypes = [P, P, P, P, P, C.c_int, C.c_int, P, P, P, P]
            L.dco_row_evict.argtypes = [P, C.c_int, P]
            L.dco_row_len.argtypes = [P]
            L.dco_row_positions.argtypes = [P, P]
            L.dco_row_kv_bits.argtypes = [P, P, P]
            L.dco_row_window_sums.argtypes = [P, P, P, P]
            L.dco_row_window_sums_prior.argtypes = [P, P, P]
            L.dco_row_heuristic_scores.argtypes = [P, C.c_int, C.c_int, P]
            L.dco_seq_new.restype = P
            L.dco_seq_new.argtypes = [C.c_int] * 6
            L.dco_seq_free.argtypes = [P]
            L.dco_seq_append.argtypes = [P, P, P, C.c_int]
            L.dco_seq_step.argtypes = [P, P, P, P, P, C.c_int, C.c_int, P, P, P]
            L.dco_seq_evict.argtypes = [P, C.c_int, P]
            L.dco_seq_len.argtypes = [P]
            L.dco_seq_positions.argtypes = [P, P]
            L.dco_seq_kv_bits.argtypes = [P, C.c_int, P, P]
            L.dco_seq_window_sums_prior.argtypes = [P, P, P]
            L.dco_pl_logz.argtypes = [P, C.c_int, C.c_int, C.c_double]
            L.dco_pl_logz.restype = C.c_double
            L.dco_gumbel_topb.argtypes = [P, P, C.c_int, C.c_int, C.c_float, P]
            L.dco_attend.argtypes = [P, P, P, C.c_int, C.c_int, C.c_int, P, P]
            L.dco_policy.argtypes = [P, C.c_int, P, C.c_int, C.c_int, P]
            _lib = L
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


def _u16(a):
    return np.ascontiguousarray(a, dtype=np.uint16)


class OracleRow:
    """One cache row (layer, batch, KV head) of the oracle."""

    def __init__(self, head_dim: int, group: int, window: int, alpha_mode: int, capacity: int):
        self.d, self.G = head_dim, group
        self._h = lib().dco_row_new(head_dim, group, window, alpha_mode, capacity)
        if not self._h:
            raise ValueError("dco_row_new rejected its arguments")

    def __del__(self):
        h = getattr(self, "_h", None)
        if h:
            lib().dco_row_free(h)
            self._h = None

    def append(self, k_bits: np.ndarray, v_bits: np.ndarray) -> None:
        k, v = _u16(k_bits), _u16(v_bits)
        T = k.shape[0] if k.ndim == 2 else 0
        if lib().dco_row_append(self._h, _ptr(k), _ptr(v), T) != 0:
            raise OverflowError("oracle row capacity exceeded")

    def step(self, q_bits, k_new_bits, v_new_bits, mlp: np.ndarray, hidden: int, layernorm: int):
        """Returns dict(o [G][d], Hq [G], feat [n][5], score [n], pos [n])."""
        q, kn, vn = _u16(q_bits), _u16(k_new_bits), _u16(v_new_bits)
        mlp = np.ascontiguousarray(mlp, dtype=np.float32)
        n_max = len(self) + 1
        o = np.empty((self.G, self.d))
        Hq = np.empty(self.G)
        feat = np.empty((n_max, 5))
        score = np.empty(n_max)
        n = lib().dco_row_step(self._h, _ptr(q), _ptr(kn), _ptr(vn), _ptr(mlp), hidden, layernorm,
                               _ptr(o), _ptr(Hq), _ptr(feat), _ptr(score))
        if n < 0:
            raise OverflowError("oracle row capacity exceeded")
        return dict(o=o, Hq=Hq, feat=feat[:n], score=score[:n], pos=self.positions())

    def evict(self, budget: int, scores_f32: np.ndarray | None = None) -> int:
        s = None if scores_f32 is None else np.ascontiguousarray(scores_f32, dtype=np.float32)
        if s is not None and s.shape[0] != len(self):
            raise ValueError("scores must have one value per cached token")
        n = lib().dco_row_evict(self._h, budget, _ptr(s))
        if n < 0:
            raise RuntimeError("no scores to evict with")
        return n

    def heuristic_scores(self, scorer: int, n_sinks: int = 4) -> np.ndarray:
        """H2O (scorer 1: cumulative attention mass) or StreamingLLM (scorer 2:
        sinks, then recency) scores of the row's tokens, ascending positions."""
        out = np.empty(len(self))
        if lib().dco_row_heuristic_scores(self._h, scorer, n_sinks, _ptr(out)) != 0:
            raise ValueError("unknown scorer, or H2O without cumulative attention mass")
        return out

    def __len__(self) -> int:
        return lib().dco_row_len(self._h)

    def positions(self) -> np.ndarray:
        out = np.empty(len(self), dtype=np.int64)
        lib().dco_row_positions(self._h, _ptr(out))
        return out

    def kv_bits(self):
        n = len(self)
        k = np.empty((n, self.d), dtype=np.uint16)
        v = np.empty((n, self.d), dtype=np.uint16)
        lib().dco_row_kv_bits(self._h, _ptr(k), _ptr(v))
        return k, v

    def window_sums(self):
        n = len(self)
        S, Z, acc = np.empty(n), np.empty(n), np.empty(n)
        lib().dco_row_window_sums(self._h, _ptr(S), _ptr(Z), _ptr(acc))
        return S, Z, acc

    def window_sums_prior(self):
        """Window sums without the most recent step's query."""
        n = len(self)
        S, Z = np.empty(n), np.empty(n)
        lib().dco_row_window_sums_prior(self._h, _ptr(S), _ptr(Z))
        return S, Z


def attend(q_bits, k_bits, v_bits):
    """Full softmax attention (the full-cache comparator): o [G][d], Hq [G]."""
    q, k, v = _u16(q_bits), _u16(k_bits), _u16(v_bits)
    G, d = q.shape
    n = k.shape[0]
    o = np.empty((G, d))
    Hq = np.empty(G)
    lib().dco_attend(_ptr(q), _ptr(k), _ptr(v), n, d, G, _ptr(o), _ptr(Hq))
    return o, Hq


def policy(x: np.ndarray, mlp: np.ndarray, hidden: int, layernorm: int) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float64)
    mlp = np.ascontiguousarray(mlp, dtype=np.float32)
    out = np.empty(x.shape[0])
    lib().dco_policy(_ptr(x), x.shape[0], _ptr(mlp), hidden, layernorm, _ptr(out))
    return out


def pl_logz(scores, B: int, tau: float = 1.0) -> float:
    """log Z of the Plackett-Luce distribution over size-B subsets (App. C)."""
    s = np.ascontiguousarray(scores, dtype=np.float64)
    return lib().dco_pl_logz(_ptr(s), s.shape[0], B, tau)


def gumbel_topb(scores, gumbel, B: int, tau: float = 1.0) -> np.ndarray:
    """Indices (ascending) of the B largest fp32 perturbed scores s/tau + g."""
    s = np.ascontiguousarray(scores, dtype=np.float32)
    g = np.ascontiguousarray(gumbel, dtype=np.float32)
    out = np.empty(B, dtype=np.int32)
    if lib().dco_gumbel_topb(_ptr(s), _ptr(g), s.shape[0], B, tau, _ptr(out)) != 0:
        raise ValueError("bad arguments")
    return out


class OracleSeq:
    """Global token mode (Sec. 3.1.1): one sequence of R rows (layers x KV
    heads) sharing its token set; features pooled over all R x G heads, one
    score and one argtop_B per sequence."""

    def __init__(self, rows: int, head_dim: int, group: int, window: int, alpha_mode: int, capacity: int):
        self.R, self.d, self.G = rows, head_dim, group
        self._h = lib().dco_seq_new(rows, head_dim, group, window, alpha_mode, capacity)
        if not self._h:
            raise ValueError("dco_seq_new rejected its arguments")

    def __del__(self):
        h = getattr(self, "_h", None)
        if h:
            lib().dco_seq_free(h)
            self._h = None

    def append(self, k_bits, v_bits) -> None:
        """k, v: [R][T][d] bf16 bits."""
        k, v = _u16(k_bits), _u16(v_bits)
        if lib().dco_seq_append(self._h, _ptr(k), _ptr(v), k.shape[1]) != 0:
            raise ValueError("capacity exceeded")

    def step(self, q_bits, k_new_bits, v_new_bits, mlp, hidden: int, layernorm: int):
        """q [R][G][d], k_new/v_new [R][d] -> dict(o [R][G][d], feat, score, pos)."""
        q, kn, vn = _u16(q_bits), _u16(k_new_bits), _u16(v_new_bits)
        mlp = np.ascontiguousarray(mlp, dtype=np.float32)
        n_max = len(self) + 1
        o = np.empty((self.R, self.G, self.d))
        feat = np.empty((n_max, 5))
        score = np.empty(n_max)
        n = lib().dco_seq_step(self._h, _ptr(q), _ptr(kn), _ptr(vn), _ptr(mlp), hidden, layernorm,
                               _ptr(o), _ptr(feat), _ptr(score))
        if n < 0:
            raise ValueError("capacity exceeded")
        return {"o": o, "feat": feat[:n], "score": score[:n], "pos": self.positions()}

    def evict(self, budget: int, scores_f32=None) -> int:
        s = None if scores_f32 is None else np.ascontiguousarray(scores_f32, dtype=np.float32)
        n = lib().dco_seq_evict(self._h, budget, _ptr(s))
        if n < 0:
            raise RuntimeError("no scores to evict with")
        return n

    def __len__(self) -> int:
        return lib().dco_seq_len(self._h)

    def positions(self) -> np.ndarray:
        out = np.empty(len(self), dtype=np.int64)
        lib().dco_seq_positions(self._h, _ptr(out))
        return out

    def kv_bits(self, row: int):
        n = len(self)
        k = np.empty((n, self.d), dtype=np.uint16)
        v = np.empty((n, self.d), dtype=np.uint16)
        lib().dco_seq_kv_bits(self._h, row, _ptr(k), _ptr(v))
        return k, v

    def window_sums_prior(self):
        n = len(self)
        S, Z = np.empty(n), np.empty(n)
        lib().dco_seq_window_sums_prior(self._h, _ptr(S), _ptr(Z))
        return S, Z
