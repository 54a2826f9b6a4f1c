"""In-tree build of libsd.so for sm_103a with nvcc (no cmake, no torch extension).

Each translation unit under csrc/ compiles to an object in parallel, then the
objects link into paper_2606_31160_gb300/libsd.so with the CUDA runtime linked
statically, so the library loads on a machine without a GPU and needs nothing
but the driver at run time. floor/floor.cu (the launch and streaming floors
that `bench.py --floor` measures; not part of the verify path) builds beside
it into libsdfloor.so. Rebuilds only when a source, header or flag changed
(content hash stamp).

    python -m paper_2606_31160_gb300.build [--force] [--ptxas-info]
"""

import hashlib
import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libsd.so")
FLOOR_SRC = os.path.join(PKG, "floor", "floor.cu")
FLOOR_LIB = os.path.join(PKG, "libsdfloor.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC,-O2",
              "--expt-relaxed-constexpr", "-I" + INCLUDE] + ARCH
SOURCES = ["api.cu", "rope.cu", "kv.cu", "attention.cu", "attention_tc.cu", "layer.cu",
           "accept_greedy.cu", "accept_sample.cu", "budget.cu"]


def nvcc_path():
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: set NVCC or put the CUDA toolkit on PATH")


def _stamp(extra):
    h = hashlib.sha256()
    for name in sorted(os.listdir(CSRC)) + ["../../include/sd.h"]:
        path = os.path.normpath(os.path.join(CSRC, name))
        if os.path.isfile(path):
            h.update(name.encode())
            with open(path, "rb") as f:
                h.update(f.read())
    with open(FLOOR_SRC, "rb") as f:
        h.update(f.read())
    h.update(" ".join(NVCC_FLAGS + extra).encode())
    return h.hexdigest()


def build(force=False, ptxas_info=False, verbose=False):
    """Compile every CUDA source and link libsd.so; returns the library path."""
    extra = ["-Xptxas", "-v"] if ptxas_info else []
    stamp = _stamp(extra)
    stamp_file = os.path.join(BUILD, "stamp")
    if not force and os.path.exists(LIB) and os.path.exists(FLOOR_LIB) and os.path.exists(stamp_file):
        with open(stamp_file) as f:
            if f.read().strip() == stamp:
                return LIB
    os.makedirs(BUILD, exist_ok=True)
    nvcc = nvcc_path()

    def compile_one(src):
        obj = os.path.join(BUILD, src.replace(".cu", ".o"))
        cmd = [nvcc, "-c", os.path.join(CSRC, src), "-o", obj] + NVCC_FLAGS + extra
        res = subprocess.run(cmd, capture_output=True, text=True)
        if res.returncode != 0:
            raise RuntimeError("nvcc failed for %s:\n%s\n%s" % (src, " ".join(cmd), res.stderr))
        return obj, res.stderr

    def floor_lib():
        tmp = FLOOR_LIB + ".tmp"
        cmd = [nvcc, "-shared", FLOOR_SRC, "-o", tmp] + NVCC_FLAGS + extra + [
            "-cudart", "static", "-Xlinker", "--no-undefined", "-lrt", "-lpthread", "-ldl"]
        res = subprocess.run(cmd, capture_output=True, text=True)
        if res.returncode != 0:
            raise RuntimeError("nvcc failed for floor.cu:\n%s\n%s" % (" ".join(cmd), res.stderr))
        os.replace(tmp, FLOOR_LIB)

    with ThreadPoolExecutor(max_workers=min(len(SOURCES) + 1, os.cpu_count() or 4)) as ex:
        floor_job = ex.submit(floor_lib)
        results = list(ex.map(compile_one, SOURCES))
        floor_job.result()
    if verbose or ptxas_info:
        for (obj, err), src in zip(results, SOURCES):
            if err.strip():
                sys.stderr.write("== %s\n%s\n" % (src, err))
    tmp = LIB + ".tmp"
    cmd = [nvcc, "-shared", "-o", tmp] + [o for o, _ in results] + ARCH + [
        "-cudart", "static", "-Xlinker", "--no-undefined", "-lrt", "-lpthread", "-ldl"]
    res = subprocess.run(cmd, capture_output=True, text=True)
    if res.returncode != 0:
        raise RuntimeError("link failed:\n%s\n%s" % (" ".join(cmd), res.stderr))
    os.replace(tmp, LIB)
    with open(stamp_file, "w") as f:
        f.write(stamp)
    return LIB


if __name__ == "__main__":
    path = build(force="--force" in sys.argv, ptxas_info="--ptxas-info" in sys.argv, verbose=True)
    print(path)
