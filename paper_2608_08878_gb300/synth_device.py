"""Device side of the seeded input generator (``libdc_synth.so``): builds the
same bits as :mod:`synth` directly in GPU memory, for workloads too large to
generate on the host. Inputs only; none of the decode step's arithmetic."""

from __future__ import annotations

import ctypes as C
import os

from . import synth

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libdc_synth.so")
_lib = None


class dcs_workload(C.Structure):
    _fields_ = [("layers", C.c_int), ("batch", C.c_int), ("kv_heads", C.c_int), ("q_heads", C.c_int),
                ("head_dim", C.c_int), ("n_sinks", C.c_int), ("hot_sets", C.c_int),
                ("epoch_len", C.c_int), ("sink_scale", C.c_float), ("hh_scale", C.c_float),
                ("q_align", C.c_float), ("seed", C.c_ulonglong)]


def _l():
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise OSError(f"{LIB_PATH} is missing: build it with `python -m paper_2608_08878_gb300.build`")
        _lib = C.CDLL(LIB_PATH)
        _lib.dcs_prompt.argtypes = [C.POINTER(dcs_workload), C.c_longlong, C.c_int, C.c_void_p,
                                    C.c_void_p, C.c_void_p]
        _lib.dcs_step.argtypes = [C.POINTER(dcs_workload), C.c_longlong, C.c_void_p, C.c_void_p,
                                  C.c_void_p, C.c_void_p]
    return _lib


def _wl(wl: synth.Workload) -> dcs_workload:
    return dcs_workload(wl.layers, wl.batch, wl.kv_heads, wl.q_heads, wl.head_dim, wl.n_sinks,
                        wl.hot_sets, min(wl.epoch_len, 2 ** 31 - 1), wl.sink_scale, wl.hh_scale,
                        wl.q_align, wl.seed)


def prompt(wl: synth.Workload, t0: int, T: int, stream=None):
    """bf16 CUDA tensors k, v [L][b][kvh][T][d] of prompt positions [t0, t0+T)."""
    import torch
    shape = (wl.layers, wl.batch, wl.kv_heads, T, wl.head_dim)
    k = torch.empty(shape, dtype=torch.bfloat16, device="cuda")
    v = torch.empty_like(k)
    s = (stream or torch.cuda.current_stream()).cuda_stream
    w = _wl(wl)
    err = _l().dcs_prompt(C.byref(w), t0, T, k.data_ptr(), v.data_ptr(), s)
    if err:
        raise RuntimeError(f"dcs_prompt: CUDA error {err}")
    return k, v


def step_inputs(wl: synth.Workload, step: int, out=None, stream=None):
    """bf16 CUDA tensors (q [L][b][qh][d], k_new, v_new [L][b][kvh][d])."""
    import torch
    if out is None:
        q = torch.empty((wl.layers, wl.batch, wl.q_heads, wl.head_dim), dtype=torch.bfloat16, device="cuda")
        kn = torch.empty((wl.layers, wl.batch, wl.kv_heads, wl.head_dim), dtype=torch.bfloat16, device="cuda")
        vn = torch.empty_like(kn)
    else:
        q, kn, vn = out
    s = (stream or torch.cuda.current_stream()).cuda_stream
    w = _wl(wl)
    err = _l().dcs_step(C.byref(w), step, q.data_ptr(), kn.data_ptr(), vn.data_ptr(), s)
    if err:
        raise RuntimeError(f"dcs_step: CUDA error {err}")
    return q, kn, vn
