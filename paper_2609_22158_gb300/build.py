"""Build libstepkv.so in-tree: one nvcc per translation unit (in parallel), sm_103a only, then link.

    python -m paper_2609_22158_gb300.build          # or build_library() from Python
"""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

PKG_DIR = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(PKG_DIR, "csrc")
ROOT = os.path.dirname(PKG_DIR)
BUILD_DIR = os.path.join(PKG_DIR, "_build")
LIB_PATH = os.path.join(PKG_DIR, "libstepkv.so")

SOURCES = ["api.cu", "score.cu", "select.cu", "compact.cu", "decode.cu"]
ARCH_FLAGS = ["-gencode", "arch=compute_103a,code=sm_103a"]
COMMON_FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-Xcompiler", "-fvisibility=hidden",
                "-I" + os.path.join(ROOT, "include"), "--expt-relaxed-constexpr"]


def _nvcc() -> str:
    n = shutil.which("nvcc")
    if n:
        return n
    cand = "/usr/local/cuda/bin/nvcc"
    if os.path.exists(cand):
        return cand
    raise RuntimeError("nvcc not found")


def _run(cmd):
    r = subprocess.run(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
    return r.returncode, r.stdout


def build_library(verbose: bool = False, force: bool = False, extra_flags=None) -> str:
    """Compile every CUDA source for sm_103a and link libstepkv.so; returns the library path."""
    os.makedirs(BUILD_DIR, exist_ok=True)
    nvcc = _nvcc()
    flags = ARCH_FLAGS + COMMON_FLAGS + list(extra_flags or [])
    headers = [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".h", ".cuh"))]
    headers.append(os.path.join(ROOT, "include", "stepkv.h"))
    newest_header = max(os.path.getmtime(h) for h in headers)
    jobs = []
    for src in SOURCES:
        s = os.path.join(CSRC, src)
        o = os.path.join(BUILD_DIR, src.replace(".cu", ".o"))
        stale = force or not os.path.exists(o) or os.path.getmtime(o) < max(os.path.getmtime(s), newest_header)
        jobs.append((s, o, stale))
    cmds = [[nvcc] + flags + ["-c", s, "-o", o] for (s, o, stale) in jobs if stale]
    with cf.ThreadPoolExecutor(max_workers=max(1, min(len(cmds), os.cpu_count() or 1))) as ex:
        results = list(ex.map(_run, cmds))
    for cmd, (rc, out) in zip(cmds, results):
        if verbose or rc != 0:
            sys.stdout.write(" ".join(cmd) + "\n" + out)
        if rc != 0:
            raise RuntimeError(f"nvcc failed for {cmd[-3]}")
    objs = [o for (_, o, _) in jobs]
    if cmds or force or not os.path.exists(LIB_PATH) or os.path.getmtime(LIB_PATH) < max(os.path.getmtime(o) for o in objs):
        tmp = LIB_PATH + ".tmp"
        rc, out = _run([nvcc] + ARCH_FLAGS + ["-shared", "-o", tmp] + objs + ["-cudart", "static"])
        if verbose or rc != 0:
            sys.stdout.write(out)
        if rc != 0:
            raise RuntimeError("link of libstepkv.so failed")
        os.replace(tmp, LIB_PATH)
    return LIB_PATH


if __name__ == "__main__":
    print(build_library(verbose="-v" in sys.argv, force="-f" in sys.argv))
