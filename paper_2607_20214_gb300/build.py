"""Builds libelsaa.so (the C-ABI library) in-tree with nvcc for sm_103a.

Each .cu file compiles in its own nvcc process (in parallel), then one link
step produces paper_2607_20214_gb300/libelsaa.so. Objects go to
paper_2607_20214_gb300/_build/ (git-ignored).
"""
from __future__ import annotations

import glob
import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libelsaa.so")
# The checked variant: the sources that guard extra checks with
# ELSAA_CHECKED (recording out-of-range permutation entries in the forward
# kernels) compiled with it, linked with the other objects of the default
# build.
LIB_CHECKED = os.path.join(PKG, "libelsaa_checked.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC",
              "--expt-relaxed-constexpr", "-I" + os.path.join(ROOT, "include")]


def nvcc() -> str:
    path = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(path):
        raise RuntimeError("nvcc not found")
    return path


def _sources():
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")))


def _deps():
    return _sources() + sorted(glob.glob(os.path.join(CSRC, "*.h"))) + sorted(
        glob.glob(os.path.join(CSRC, "*.cuh"))) + [
            os.path.join(ROOT, "include", "elsaa.h")]


def up_to_date() -> bool:
    if not os.path.exists(LIB):
        return False
    t = os.path.getmtime(LIB)
    return all(os.path.getmtime(p) <= t for p in _deps())


def build(force: bool = False, verbose: bool = False, extra=()) -> str:
    if not force and up_to_date():
        return LIB
    os.makedirs(BUILD, exist_ok=True)
    cc = nvcc()

    def compile_one(src):
        obj = os.path.join(BUILD, os.path.basename(src) + ".o")
        cmd = [cc, *ARCH, *NVCC_FLAGS, *extra, "-c", src, "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError("nvcc failed on %s:\n%s%s" % (
                os.path.basename(src), r.stdout, r.stderr))
        if verbose and (r.stdout or r.stderr):
            sys.stderr.write(r.stdout + r.stderr)
        return obj

    with ThreadPoolExecutor(max_workers=max(1, len(_sources()))) as ex:
        objs = list(ex.map(compile_one, _sources()))
    tmp = LIB + ".tmp%d" % os.getpid()
    cmd = [cc, *ARCH, "-shared", "-o", tmp, *objs]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError("link failed:\n%s%s" % (r.stdout, r.stderr))
    os.replace(tmp, LIB)
    return LIB


def build_checked(force: bool = False) -> str:
    """Builds libelsaa_checked.so (after the default library)."""
    build()
    checked = [src for src in _sources()
               if "ELSAA_CHECKED" in open(src).read()]
    if (not force and os.path.exists(LIB_CHECKED) and
            os.path.getmtime(LIB_CHECKED) >= os.path.getmtime(LIB)):
        return LIB_CHECKED
    cc = nvcc()

    def compile_one(src):
        obj = os.path.join(BUILD, os.path.basename(src) + ".checked.o")
        cmd = [cc, *ARCH, *NVCC_FLAGS, "-DELSAA_CHECKED", "-c", src, "-o",
               obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError("nvcc failed on %s:\n%s%s" % (
                os.path.basename(src), r.stdout, r.stderr))
        return obj

    with ThreadPoolExecutor(max_workers=max(1, len(checked))) as ex:
        cobjs = list(ex.map(compile_one, checked))
    objs = [os.path.join(BUILD, os.path.basename(src) + ".o")
            for src in _sources() if src not in checked] + cobjs
    tmp = LIB_CHECKED + ".tmp%d" % os.getpid()
    r = subprocess.run([cc, *ARCH, "-shared", "-o", tmp, *objs],
                       capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError("link failed:\n%s%s" % (r.stdout, r.stderr))
    os.replace(tmp, LIB_CHECKED)
    return LIB_CHECKED


if __name__ == "__main__":
    v = "-v" in sys.argv
    extra = ["-Xptxas", "-v"] if "--ptxas" in sys.argv else []
    print(build(force=True, verbose=v or bool(extra), extra=extra))
