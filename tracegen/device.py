"""Device-side token filling for traces (input generation only)."""

import ctypes as C
import os
import shutil
import subprocess

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "gen_tokens.cu")
LIB = os.path.join(HERE, "libdm_tracegen.so")
_lib = None


def build(force=False):
    if not force and os.path.exists(LIB) and os.path.getmtime(LIB) >= os.path.getmtime(SRC):
        return LIB
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    tmp = LIB + f".tmp{os.getpid()}"
    subprocess.check_call([nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-shared",
                           "-Xcompiler", "-fPIC", SRC, "-o", tmp])
    os.replace(tmp, LIB)
    return LIB


def lib():
    global _lib
    if _lib is None:
        if not os.path.exists(LIB):
            raise RuntimeError(f"{LIB} missing: run tracegen.device.build()")
        L = C.CDLL(LIB)
        L.tg_fill_tokens.restype = C.c_int
        L.tg_fill_tokens.argtypes = [C.c_void_p] * 5 + [C.c_uint64, C.c_uint64, C.c_uint64, C.c_void_p]
        _lib = L
    return _lib


def fill_range(trace, r0, r1, dst, stream=None):
    """Fill torch uint32-compatible (int32) device tensor `dst` with the tokens
    of requests [r0, r1) in the trace's aligned layout (offset 0 = request r0)."""
    import torch
    pd, ps, pst, pl = trace.pieces_for_range(r0, r1)
    dev = dst.device
    t = [torch.from_numpy(np.ascontiguousarray(a).view(np.int64 if a.dtype == np.uint64 else np.int32)).to(dev)
         for a in (pd, ps, pst, pl)]
    st = stream if stream is not None else torch.cuda.current_stream(dev)
    rc = lib().tg_fill_tokens(dst.data_ptr(), t[0].data_ptr(), t[1].data_ptr(), t[2].data_ptr(), t[3].data_ptr(),
                              len(pd), trace.token_seed, trace.vocab, st.cuda_stream)
    if rc:
        raise RuntimeError(f"tg_fill_tokens failed: {rc}")
    st.synchronize()
