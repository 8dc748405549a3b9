"""Builds libtimebill_kv.so from csrc/*.cu for sm_103a with nvcc.

Each translation unit compiles in parallel into _build/, then nvcc links the
shared library next to this file. Only files whose sources changed are
recompiled. Run as ``python -m paper_2512_21859_gb300.build``.

``build(debug=True)`` (``python -m paper_2512_21859_gb300.build --debug``)
builds libtimebill_kv_debug.so instead, into _build_debug/, with TB_DEBUG=1:
the kernels then check invariants (index ranges, finite row normalisers and
split sums, the selected count) and raise the range bit of the workspace
status word when one fails. The binding loads it when TB_LIBRARY=debug.
"""
from __future__ import annotations

import concurrent.futures as cf
import glob
import hashlib
import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libtimebill_kv.so")
BUILD_DEBUG = os.path.join(PKG, "_build_debug")
LIB_DEBUG = os.path.join(PKG, "libtimebill_kv_debug.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-O2",
         "--expt-relaxed-constexpr", "-I" + INCLUDE, "-I" + CSRC]


def _nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libtimebill_kv.so")


def _digest(paths) -> str:
    h = hashlib.sha256()
    for p in sorted(paths):
        with open(p, "rb") as f:
            h.update(p.encode() + b"\0" + f.read())
    h.update(" ".join(ARCH + FLAGS).encode())
    return h.hexdigest()


def _compile(nvcc: str, src: str, headers, extra, build_dir=BUILD) -> str:
    obj = os.path.join(build_dir, os.path.basename(src)[:-3] + ".o")
    stamp = obj + ".sha"
    dig = _digest([src] + list(headers)) + " ".join(extra)
    if os.path.exists(obj) and os.path.exists(stamp) and open(stamp).read() == dig:
        return obj
    cmd = [nvcc, *ARCH, *FLAGS, *extra, "-c", src, "-o", obj]
    res = subprocess.run(cmd, capture_output=True, text=True)
    if res.returncode != 0:
        raise RuntimeError("nvcc failed for %s:\n%s\n%s" % (src, " ".join(cmd), res.stderr))
    if res.stderr.strip():
        sys.stderr.write(res.stderr)
    with open(stamp, "w") as f:
        f.write(dig)
    return obj


def build(verbose: bool = False, extra_flags=(), debug: bool = False) -> str:
    """Compiles every csrc/*.cu and links libtimebill_kv.so (with debug=True:
    libtimebill_kv_debug.so, TB_DEBUG=1); returns its path."""
    nvcc = _nvcc()
    build_dir, lib = (BUILD_DEBUG, LIB_DEBUG) if debug else (BUILD, LIB)
    extra = list(extra_flags) + (["-DTB_DEBUG=1"] if debug else [])
    os.makedirs(build_dir, exist_ok=True)
    sources = sorted(glob.glob(os.path.join(CSRC, "*.cu")))
    headers = sorted(glob.glob(os.path.join(CSRC, "*.cuh")) + glob.glob(os.path.join(INCLUDE, "*.h")))
    with cf.ThreadPoolExecutor(max_workers=max(1, min(len(sources), os.cpu_count() or 1))) as ex:
        objs = list(ex.map(lambda s: _compile(nvcc, s, headers, extra, build_dir), sources))
    link_dig = _digest(objs)
    stamp = lib + ".sha"
    if not (os.path.exists(lib) and os.path.exists(stamp) and open(stamp).read() == link_dig):
        tmp = lib + ".tmp"
        cmd = [nvcc, *ARCH, "-shared", "-cudart", "shared", "-o", tmp, *objs]
        res = subprocess.run(cmd, capture_output=True, text=True)
        if res.returncode != 0:
            raise RuntimeError("link failed:\n%s\n%s" % (" ".join(cmd), res.stderr))
        os.replace(tmp, lib)
        with open(stamp, "w") as f:
            f.write(link_dig)
    if verbose:
        print("built", lib)
    return lib


if __name__ == "__main__":
    args = sys.argv[1:]
    dbg = "--debug" in args
    build(verbose=True, extra_flags=[a for a in args if a != "--debug"], debug=dbg)
