"""Build libpatconv.so in-tree: nvcc for the sm_103a kernels, g++ for the host packer.

The library is written to ``paper_2003_06513_gb300/_build/libpatconv.so`` (git-ignored) and is
rebuilt whenever a source file or a flag changes.  No CMake: two translation units compiled in
parallel and one link, so a fresh build takes well under a minute.
"""
from __future__ import annotations

import hashlib
import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(BUILD, "libpatconv.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-std=c++17", "-lineinfo", "--expt-relaxed-constexpr", "-Xcompiler", "-fPIC",
              "-Xcompiler", "-ffp-contract=off", "-I", os.path.join(ROOT, "include")] + ARCH
GXX_FLAGS = ["-O2", "-std=c++17", "-fPIC", "-ffp-contract=off", "-Wall", "-I",
             os.path.join(ROOT, "include")]
SOURCES = ["conv.cu", "pack.cpp", "layer.h", "gen_dispatch.py"]


def _nvcc() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libpatconv")


def _digest(extra) -> str:
    h = hashlib.sha256()
    for name in SOURCES + [os.path.join("..", "..", "include", "patconv.h")]:
        with open(os.path.join(CSRC, name), "rb") as f:
            h.update(f.read())
    h.update(repr((NVCC_FLAGS, GXX_FLAGS, extra)).encode())
    return h.hexdigest()


def build(force: bool = False, verbose: bool = False, extra_nvcc=()) -> str:
    """Compile (if stale) and return the path of libpatconv.so."""
    os.makedirs(BUILD, exist_ok=True)
    stamp = os.path.join(BUILD, "stamp")
    digest = _digest(tuple(extra_nvcc))
    if not force and os.path.exists(LIB) and os.path.exists(stamp):
        with open(stamp) as f:
            if f.read().strip() == digest:
                return LIB
    nvcc = _nvcc()
    subprocess.run([sys.executable, os.path.join(CSRC, "gen_dispatch.py"),
                    os.path.join(BUILD, "pattern_dispatch.h")], check=True)
    conv_o = os.path.join(BUILD, "conv.o")
    pack_o = os.path.join(BUILD, "pack.o")
    cmds = [
        [nvcc, "-c", os.path.join(CSRC, "conv.cu"), "-o", conv_o, "-I", BUILD] + NVCC_FLAGS + list(extra_nvcc),
        ["g++", "-c", os.path.join(CSRC, "pack.cpp"), "-o", pack_o] + GXX_FLAGS,
    ]

    def run(cmd):
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0 or verbose:
            sys.stderr.write(" ".join(cmd) + "\n" + r.stdout + r.stderr)
        if r.returncode != 0:
            raise RuntimeError(f"build step failed: {' '.join(cmd[:3])}")
        return r.stdout + r.stderr

    with ThreadPoolExecutor(max_workers=2) as ex:
        list(ex.map(run, cmds))
    tmp = LIB + ".tmp"
    run([nvcc, "-shared", "-o", tmp, conv_o, pack_o] + ARCH + ["-cudart", "static"])
    os.replace(tmp, LIB)
    with open(stamp, "w") as f:
        f.write(digest)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose=True))
