"""Builds libvase.so (the C-ABI library) in-tree with nvcc for sm_103a.

Usage: python -m paper_2606_03928_gb300.build [--force]
The translation units compile in parallel; the output lands in
paper_2606_03928_gb300/_lib/libvase.so (git-ignored).
"""

from __future__ import annotations

import concurrent.futures
import hashlib
import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
OUT_DIR = os.path.join(PKG, "_lib")
LIB = os.path.join(OUT_DIR, "libvase.so")
SOURCES = ["api.cu", "score_attn.cu", "dkv.cu", "misc.cu", "store.cu", "decode.cu", "decode_mixed.cu", "selftest.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-I", INCLUDE, "-I", CSRC]


def _nvcc():
    cand = os.environ.get("NVCC") or shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(cand):
        raise RuntimeError("nvcc not found; the VaSE CUDA library cannot be built")
    return cand


def source_digest():
    """Digest of the CUDA sources and the public header only (the same on every machine)."""
    h = hashlib.sha256()
    for name in sorted(os.listdir(CSRC)) + ["vase.h"]:
        path = os.path.join(CSRC, name) if name != "vase.h" else os.path.join(INCLUDE, name)
        if os.path.isfile(path):
            h.update(name.encode())
            with open(path, "rb") as f:
                h.update(f.read())
    return h.hexdigest()


# The source files each timed kernel is compiled from (its own translation unit and the headers it includes).
KERNEL_SOURCES = {
    "score_attn": ["score_attn.cu", "kernels.cuh", "ptx.cuh"],
    "select_compact": ["misc.cu", "kernels.cuh", "ptx.cuh", "quant.cuh"],
    "append": ["misc.cu", "kernels.cuh", "ptx.cuh", "quant.cuh"],
    "store_append": ["store.cu", "kernels.cuh", "ptx.cuh", "quant.cuh"],
    "store_evict": ["store.cu", "kernels.cuh", "ptx.cuh", "quant.cuh"],
    "dkv_score": ["dkv.cu", "kernels.cuh", "ptx.cuh"],
    "decode": ["decode.cu", "decode_simt.cuh", "decode_mixed.cu", "kernels.cuh", "ptx.cuh"],
}


def kernel_digest(kernel):
    """Digest of the sources of one kernel: ncu counters taken on it stay valid while this is unchanged."""
    h = hashlib.sha256()
    for name in KERNEL_SOURCES[kernel]:
        h.update(name.encode())
        with open(os.path.join(CSRC, name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def _digest():
    h = hashlib.sha256()
    for name in sorted(os.listdir(CSRC)) + ["vase.h"]:
        path = os.path.join(CSRC, name) if name != "vase.h" else os.path.join(INCLUDE, name)
        if os.path.isfile(path):
            h.update(name.encode())
            with open(path, "rb") as f:
                h.update(f.read())
    h.update(" ".join(ARCH + FLAGS).encode())
    h.update(os.uname().machine.encode())
    return h.hexdigest()


def build(force: bool = False, verbose: bool = False) -> str:
    os.makedirs(OUT_DIR, exist_ok=True)
    stamp = os.path.join(OUT_DIR, "libvase.stamp")
    digest = _digest()
    if not force and os.path.exists(LIB) and os.path.exists(stamp):
        with open(stamp) as f:
            if f.read().strip() == digest:
                return LIB
    nvcc = _nvcc()
    objs = []

    def compile_one(src):
        obj = os.path.join(OUT_DIR, os.path.splitext(src)[0] + ".o")
        cmd = [nvcc, *ARCH, *FLAGS, "-c", os.path.join(CSRC, src), "-o", obj]
        if verbose:
            cmd.insert(1, "-Xptxas=-v")
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}\n{r.stderr}")
        if verbose and r.stderr:
            sys.stderr.write(r.stderr)
        return obj

    with concurrent.futures.ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        objs = list(ex.map(compile_one, SOURCES))
    tmp = LIB + ".tmp"
    cmd = [nvcc, *ARCH, "-shared", "-o", tmp, *objs, "-lcudart_static", "-ldl", "-lrt", "-lpthread"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, LIB)
    with open(stamp, "w") as f:
        f.write(digest)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
