"""Build libstepkv.so in-tree: one nvcc per translation unit (in parallel), sm_103a only, then link.

    python -m paper_2609_22158_gb300.build          # or build_library() from Python

Rebuilds are keyed on content, not on file times: each object's key is a SHA-256 over the compiler's
version, the host machine, the flags, the source and every header; the key and the object's own hash
are stored beside the object.  An object is reused only when both match, and the library is relinked
whenever the set of object hashes differs from the one recorded at its last link.  Objects or a library
carried over from another machine or build (whatever their time stamps) are therefore never mistaken
for a compile of the current sources.
"""
from __future__ import annotations

import concurrent.futures as cf
import hashlib
import json
import os
import platform
import shutil
import subprocess
import sys

PKG_DIR = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(PKG_DIR, "csrc")
ROOT = os.path.dirname(PKG_DIR)
BUILD_DIR = os.path.join(PKG_DIR, "_build")
LIB_PATH = os.path.join(PKG_DIR, "libstepkv.so")

SOURCES = ["api.cu", "score.cu", "select.cu", "compact.cu", "decode.cu", "signals.cu"]
ARCH_FLAGS = ["-gencode", "arch=compute_103a,code=sm_103a"]
COMMON_FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-Xcompiler", "-fvisibility=hidden",
                "-I" + os.path.join(ROOT, "include"), "--expt-relaxed-constexpr"]
LINK_FLAGS = ["-shared", "-cudart", "static"]


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


def _sha256_file(path: str) -> str:
    h = hashlib.sha256()
    with open(path, "rb") as f:
        for chunk in iter(lambda: f.read(1 << 20), b""):
            h.update(chunk)
    return h.hexdigest()


def _read_json(path: str):
    try:
        with open(path) as f:
            return json.load(f)
    except (OSError, ValueError):
        return None


def _write_json(path: str, obj) -> None:
    tmp = path + ".tmp"
    with open(tmp, "w") as f:
        json.dump(obj, f, sort_keys=True)
    os.replace(tmp, path)


def _toolchain_id(nvcc: str) -> str:
    rc, out = _run([nvcc, "--version"])
    return out.strip() if rc == 0 else nvcc


def build_library(verbose: bool = False, force: bool = False, extra_flags=None, build_dir: str = BUILD_DIR,
                  lib_path: str = LIB_PATH, sources=None, log=None) -> str:
    """Compile the CUDA sources for sm_103a and link the shared library; returns its path.

    ``log`` (a list) receives one dict per build: the library key and which sources were compiled."""
    os.makedirs(build_dir, exist_ok=True)
    nvcc = _nvcc()
    flags = ARCH_FLAGS + COMMON_FLAGS + list(extra_flags or [])
    headers = sorted(os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".h", ".cuh")))
    headers.append(os.path.join(ROOT, "include", "stepkv.h"))
    base = hashlib.sha256()
    base.update(_toolchain_id(nvcc).encode())
    base.update(platform.machine().encode())
    base.update("\0".join(flags).encode())
    for h in headers:
        base.update(os.path.basename(h).encode())
        base.update(_sha256_file(h).encode())
    jobs = []
    for src in (sources or SOURCES):
        s = os.path.join(CSRC, src)
        o = os.path.join(build_dir, src.replace(".cu", ".o"))
        key_h = base.copy()
        key_h.update(src.encode())
        key_h.update(_sha256_file(s).encode())
        key = key_h.hexdigest()
        rec = _read_json(o + ".key")
        fresh = (not force and rec is not None and rec.get("key") == key and os.path.exists(o)
                 and rec.get("object_sha256") == _sha256_file(o))
        jobs.append((s, o, key, not fresh))
    todo = [(s, o, key) for (s, o, key, stale) in jobs if stale]
    for _, o, _ in todo:  # a stale object and its key never survive a failed compile
        for p in (o, o + ".key"):
            if os.path.exists(p):
                os.remove(p)
    cmds = [[nvcc] + flags + ["-c", s, "-o", o] for (s, o, _) in todo]
    with cf.ThreadPoolExecutor(max_workers=max(1, min(len(cmds), os.cpu_count() or 1))) as ex:
        results = list(ex.map(_run, cmds))
    for cmd, (rc, out) in zip(cmds, results):
        if verbose or rc != 0:
            sys.stdout.write(" ".join(cmd) + "\n" + out)
        if rc != 0:
            raise RuntimeError(f"nvcc failed for {cmd[-3]}")
    for _, o, key in todo:
        _write_json(o + ".key", {"key": key, "object_sha256": _sha256_file(o)})
    obj_hashes = [_read_json(o + ".key")["object_sha256"] for (_, o, _, _) in jobs]
    lib_h = hashlib.sha256()
    lib_h.update("\0".join(ARCH_FLAGS + LINK_FLAGS).encode())
    for hsh in obj_hashes:
        lib_h.update(hsh.encode())
    lib_key = lib_h.hexdigest()
    rec = _read_json(lib_path + ".key")
    lib_fresh = (not force and rec is not None and rec.get("key") == lib_key and os.path.exists(lib_path)
                 and rec.get("lib_sha256") == _sha256_file(lib_path))
    if not lib_fresh:
        if os.path.exists(lib_path + ".key"):
            os.remove(lib_path + ".key")
        tmp = lib_path + ".tmp"
        objs = [o for (_, o, _, _) in jobs]
        rc, out = _run([nvcc] + ARCH_FLAGS + LINK_FLAGS[:1] + ["-o", tmp] + objs + LINK_FLAGS[1:])
        if verbose or rc != 0:
            sys.stdout.write(out)
        if rc != 0:
            raise RuntimeError("link of libstepkv.so failed")
        os.replace(tmp, lib_path)
        _write_json(lib_path + ".key", {"key": lib_key, "lib_sha256": _sha256_file(lib_path)})
    entry = {"library_key": lib_key[:16], "compiled": [os.path.basename(s) for (s, _, _) in todo],
             "linked": not lib_fresh}
    if log is not None:
        log.append(entry)
    if verbose or todo or not lib_fresh:
        sys.stderr.write(f"libstepkv build key {entry['library_key']}: compiled {len(todo)} of {len(jobs)} "
                         f"sources{', relinked' if not lib_fresh else ''}\n")
    return lib_path


if __name__ == "__main__":
    print(build_library(verbose="-v" in sys.argv, force="-f" in sys.argv))
