"""Build ``libltd.so`` in-tree with nvcc for sm_103a.

Each translation unit under ``csrc/`` compiles to an object in ``_build/`` in
parallel; the objects link into ``libltd.so`` next to this file.  A unit is
rebuilt only when it, a header it may include, or the flags changed.
"""

from __future__ import annotations

import concurrent.futures as cf
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
LIB = os.path.join(PKG, "libltd.so")

SOURCES = ["ltd_api.cu", "k_expand.cu", "k_select.cu", "k_policy.cu", "k_attn_simt.cu", "k_attn_tc.cu",
           "k_accept.cu", "k_selftest.cu", "k_accept_noalloc.cu", "k_lm_head.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-Xcompiler", "-Wall",
         "--expt-relaxed-constexpr", "-I", INCLUDE, "-I", CSRC] + ARCH


def _nvcc() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libltd.so")


def _headers_digest() -> str:
    h = hashlib.sha256()
    for d in (CSRC, INCLUDE):
        for name in sorted(os.listdir(d)):
            if name.endswith((".h", ".cuh")):
                with open(os.path.join(d, name), "rb") as f:
                    h.update(name.encode() + f.read())
    h.update(" ".join(FLAGS).encode())
    return h.hexdigest()[:16]


def _compile(nvcc: str, src: str, obj: str, extra: list) -> tuple:
    cmd = [nvcc, "-c", os.path.join(CSRC, src), "-o", obj] + FLAGS + extra
    r = subprocess.run(cmd, capture_output=True, text=True)
    return src, r.returncode, r.stdout + r.stderr, cmd


def build(force: bool = False, verbose: bool = False, extra_flags: list | None = None) -> str:
    """Compile every CUDA translation unit and link libltd.so; returns its path."""
    extra = list(extra_flags or [])
    nvcc = _nvcc()
    os.makedirs(BUILD, exist_ok=True)
    digest = _headers_digest() + hashlib.sha256(" ".join(extra).encode()).hexdigest()[:8]
    stamp = os.path.join(BUILD, "stamp")
    old = open(stamp).read().strip() if os.path.exists(stamp) else ""
    if old != digest:
        force = True
    jobs = []
    for src in SOURCES:
        obj = os.path.join(BUILD, src.replace(".cu", ".o"))
        if force or not os.path.exists(obj) or \
                os.path.getmtime(obj) < os.path.getmtime(os.path.join(CSRC, src)):
            jobs.append((src, obj))
    if jobs:
        with cf.ThreadPoolExecutor(max_workers=max(1, min(len(jobs), os.cpu_count() or 4))) as ex:
            futs = [ex.submit(_compile, nvcc, s, o, extra) for s, o in jobs]
            for fut in futs:
                src, rc, out, cmd = fut.result()
                if verbose or rc != 0:
                    sys.stderr.write(f"[ltd build] {' '.join(cmd)}\n{out}")
                if rc != 0:
                    raise RuntimeError(f"nvcc failed on {src}:\n{out}")
    objs = [os.path.join(BUILD, s.replace(".cu", ".o")) for s in SOURCES]
    if jobs or not os.path.exists(LIB) or any(os.path.getmtime(o) > os.path.getmtime(LIB) for o in objs):
        tmp = LIB + ".tmp"
        cmd = [nvcc, "-shared", "-o", tmp] + objs + ARCH + ["-cudart", "shared"]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{r.stdout}{r.stderr}")
        os.replace(tmp, LIB)
    with open(stamp, "w") as f:
        f.write(digest)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
