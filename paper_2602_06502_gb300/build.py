"""Build libdualmap.so (all CUDA kernels + the C ABI) for sm_103a with nvcc.

Each translation unit compiles in parallel; objects go to _build/ and the
shared library next to this file.  No torch extension machinery is used: the
library is a plain C-ABI shared object.
"""

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(ROOT, "_build", "dualmap")
LIB = os.path.join(HERE, "libdualmap.so")
# debug build: the same sources with -DDM_DEBUG (device index checks that
# record DM_ERR_BOUNDS), its own objects and library
BUILD_DEBUG = os.path.join(ROOT, "_build", "dualmap_debug")
LIB_DEBUG = os.path.join(HERE, "libdualmap_debug.so")
SOURCES = ["dm_api.cu", "dm_setup.cu", "dm_hash.cu", "dm_route.cu", "dm_choice.cu", "dm_commit.cu",
           "dm_rebalance.cu", "dm_ring.cu", "dm_noalloc.cu", "dm_potc.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-fvisibility=hidden",
         "--expt-relaxed-constexpr", "-I", os.path.join(ROOT, "include")]


def nvcc():
    p = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    return p


def _stale(out, deps):
    if not os.path.exists(out):
        return True
    t = os.path.getmtime(out)
    return any(os.path.getmtime(d) > t for d in deps)


def build(force=False, verbose=False, extra=(), debug=False):
    bdir, lib_path = (BUILD_DEBUG, LIB_DEBUG) if debug else (BUILD, LIB)
    if debug:
        extra = ("-DDM_DEBUG",) + tuple(extra)
    os.makedirs(bdir, exist_ok=True)
    headers = [os.path.join(CSRC, "dm_internal.cuh"), os.path.join(ROOT, "include", "dualmap.h")]
    objs, jobs = [], []
    for s in SOURCES:
        src = os.path.join(CSRC, s)
        obj = os.path.join(bdir, s.replace(".cu", ".o"))
        objs.append(obj)
        if force or _stale(obj, [src] + headers):
            jobs.append([nvcc(), *ARCH, *FLAGS, *extra, "-c", src, "-o", obj])
    with cf.ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        for cmd, res in zip(jobs, ex.map(lambda c: subprocess.run(c, capture_output=True, text=True), jobs)):
            if verbose or res.returncode:
                sys.stderr.write(res.stdout + res.stderr)
            if res.returncode:
                raise RuntimeError("nvcc failed: " + " ".join(cmd))
    if force or jobs or _stale(lib_path, objs):
        tmp = lib_path + f".tmp{os.getpid()}"
        cmd = [nvcc(), *ARCH, "-shared", "-o", tmp, *objs]
        res = subprocess.run(cmd, capture_output=True, text=True)
        if res.returncode:
            sys.stderr.write(res.stdout + res.stderr)
            raise RuntimeError("link failed")
        os.replace(tmp, lib_path)
    return lib_path


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose=True, debug="--debug" in sys.argv))
