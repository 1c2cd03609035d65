"""Builds the CUDA libraries in-tree with nvcc for sm_103a.

* ``libdistillcache.so`` -- the decode-step kernels and the C ABI of
  ``include/distillcache.h``;
* ``libdc_synth.so``     -- the device side of the seeded input generator.

Each translation unit compiles in parallel; nothing is installed elsewhere.
"""

from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(HERE, "_build")
INCLUDE = os.path.join(os.path.dirname(HERE), "include")

LIB_MAIN = os.path.join(HERE, "libdistillcache.so")
LIB_SYNTH = os.path.join(HERE, "libdc_synth.so")
# the same library with device-side index checks and guard regions around the
# handle's buffers (DC_DEBUG_BOUNDS), for tests; the binding loads it when
# DC_LIBRARY=debug
LIB_DEBUG = os.path.join(HERE, "libdistillcache_debug.so")
BUILD_DEBUG = os.path.join(HERE, "_build_debug")

MAIN_SOURCES = ["dc_cache.cu", "dc_split.cu", "dc_evict.cu", "dc_full.cu", "dc_fused.cu", "dc_noalloc.cu",
                "dc_train.cu", "dc_global.cu", "dc_fused_modes.cu", "dc_fused_glob.cu",
                "dc_fused_pair.cu", "dc_selftest.cu", "dc_fused_graph.cu"]
SYNTH_SOURCES = ["synth.cu"]

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-O2",
                     "--expt-relaxed-constexpr", "-I", CSRC, "-I", INCLUDE]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def _deps() -> list[str]:
    out = []
    for d in (CSRC, INCLUDE):
        for f in os.listdir(d):
            if f.endswith((".cu", ".cuh", ".h")):
                out.append(os.path.join(d, f))
    return out


def _stale(target: str, inputs: list[str]) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(i) > t for i in inputs)


def _compile(src: str, extra: list[str], verbose: bool, build_dir: str = BUILD) -> str:
    obj = os.path.join(build_dir, os.path.basename(src).replace(".cu", ".o"))
    if _stale(obj, _deps()):
        cmd = [nvcc()] + NVCC_FLAGS + extra + ["-c", os.path.join(CSRC, src), "-o", obj]
        if verbose:
            cmd.insert(1, "-Xptxas=-v")
        res = subprocess.run(cmd, capture_output=True, text=True)
        if res.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{res.stdout}\n{res.stderr}")
        if verbose and res.stderr:
            sys.stderr.write(res.stderr)
    return obj


def _link(objs: list[str], target: str, libs: list[str]) -> None:
    if _stale(target, objs):
        tmp = target + f".tmp{os.getpid()}"
        cmd = [nvcc()] + ARCH + ["-shared", "-o", tmp] + objs + libs
        res = subprocess.run(cmd, capture_output=True, text=True)
        if res.returncode != 0:
            raise RuntimeError(f"link of {target} failed:\n{res.stdout}\n{res.stderr}")
        os.replace(tmp, target)


def build_debug(verbose: bool = False) -> str:
    """libdistillcache_debug.so: every kernel with its index checks compiled
    in (DC_DEBUG_BOUNDS) and guard regions around the handle's buffers."""
    os.makedirs(BUILD_DEBUG, exist_ok=True)
    with cf.ThreadPoolExecutor(max_workers=min(8, len(MAIN_SOURCES))) as ex:
        objs = list(ex.map(lambda s: _compile(s, ["-DDC_DEBUG_BOUNDS"], verbose, BUILD_DEBUG), MAIN_SOURCES))
    _link(objs, LIB_DEBUG, [])
    return LIB_DEBUG


def build(verbose: bool = False) -> tuple[str, str]:
    os.makedirs(BUILD, exist_ok=True)
    srcs = MAIN_SOURCES + SYNTH_SOURCES
    with cf.ThreadPoolExecutor(max_workers=min(8, len(srcs))) as ex:
        objs = dict(zip(srcs, ex.map(lambda s: _compile(s, [], verbose), srcs)))
    _link([objs[s] for s in MAIN_SOURCES], LIB_MAIN, [])
    _link([objs[s] for s in SYNTH_SOURCES], LIB_SYNTH, [])
    return LIB_MAIN, LIB_SYNTH


if __name__ == "__main__":
    print(build_debug(verbose="-v" in sys.argv) if "--debug" in sys.argv else build(verbose="-v" in sys.argv))
