"""Build ``libppas.so`` (CUDA for sm_103a + the C++ planner) in-tree.

Each translation unit is compiled in parallel with nvcc, then linked into a
shared library next to this file.  Usage: ``python -m
paper_2608_15171_gb300.build`` or ``build()`` from Python.
"""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD_DIR = os.path.join(HERE, "_build")
LIB_PATH = os.path.join(HERE, "libppas.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
SOURCES = ["planner.cpp", "attention_step.cu", "kv_append.cu", "attn_prefill.cu", "attn_decode.cu",
           "attention_noalloc.cu", "gateup.cu"]


def _nvcc() -> str:
    cand = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(cand):
        raise RuntimeError("nvcc not found")
    return cand


def _flags(extra=()):
    return [*ARCH, "-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC,-O3",
            f"-I{INCLUDE}", f"-I{CSRC}", *extra]


def _compile(src: str, extra=()) -> str:
    obj = os.path.join(BUILD_DIR, os.path.basename(src) + ".o")
    cmd = [_nvcc(), *_flags(extra), "-c", os.path.join(CSRC, src), "-o", obj]
    if src.endswith(".cpp"):
        cmd[len(cmd) - 4:len(cmd) - 4] = ["-x", "cu"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
    if r.stderr.strip():
        sys.stderr.write(r.stderr)
    return obj


def build(verbose: bool = False, extra=()) -> str:
    """Compile every source and link ``libppas.so``; returns its path."""
    os.makedirs(BUILD_DIR, exist_ok=True)
    with cf.ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        objs = list(ex.map(lambda s: _compile(s, extra), SOURCES))
    tmp = LIB_PATH + ".tmp"
    cmd = [_nvcc(), *ARCH, "-shared", "-cudart", "shared", "-Xlinker", "-rpath,/usr/local/cuda/lib64",
           "-o", tmp, *objs]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, LIB_PATH)
    if verbose:
        print(f"built {LIB_PATH}")
    fast = _build_fast(verbose)
    if verbose and fast is None:
        print("note: _ppasfast not built (no Python headers); the binding uses ctypes for every call")
    return LIB_PATH


def _build_fast(verbose: bool = False):
    """The CPython module with the per-layer calls (csrc/pyfast.c), linked
    against libppas.so; None when this Python has no headers to build it."""
    import sysconfig
    inc = sysconfig.get_paths().get("include")
    if not inc or not os.path.exists(os.path.join(inc, "Python.h")):
        return None
    gcc = shutil.which("gcc") or shutil.which("cc")
    if gcc is None:
        return None
    out = os.path.join(HERE, "_ppasfast" + (sysconfig.get_config_var("EXT_SUFFIX") or ".so"))
    tmp = out + ".tmp"
    cmd = [gcc, "-O2", "-shared", "-fPIC", f"-I{inc}", f"-I{INCLUDE}", os.path.join(CSRC, "pyfast.c"), "-o", tmp,
           f"-L{HERE}", "-lppas", f"-Wl,-rpath,{HERE}"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"building _ppasfast failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, out)
    if verbose:
        print(f"built {out}")
    return out


if __name__ == "__main__":
    build(verbose=True, extra=tuple(sys.argv[1:]))
