"""Device-side twin of ``synth.values``: fills CUDA tensors with the same seeded
values (bit for bit) so large workloads need no host-side generation."""
from __future__ import annotations

import ctypes
import os
import shutil
import subprocess

import numpy as np

from . import values as V

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "cuda_gen.cu")
LIB = os.path.join(HERE, "libkvcsynth.so")

_lib = None


def build(force: bool = False) -> str:
    if not force and os.path.exists(LIB) and os.path.getmtime(LIB) >= os.path.getmtime(SRC):
        return LIB
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    tmp = LIB + ".tmp"
    cmd = [nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-std=c++17", "-shared",
           "-Xcompiler", "-fPIC", SRC, "-o", tmp]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed for {SRC}:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, LIB)
    return LIB


def _load():
    global _lib
    if _lib is None:
        if not os.path.exists(LIB):
            raise RuntimeError(f"{LIB} is missing: run synth.gpu.build() first")
        lib = ctypes.CDLL(LIB)
        lib.synth_fill.restype = ctypes.c_int
        lib.synth_fill.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_uint64, ctypes.c_int,
                                   ctypes.c_uint32, ctypes.c_float, ctypes.c_int, ctypes.c_int,
                                   ctypes.c_int, ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p,
                                   ctypes.c_void_p]
        _lib = lib
    return _lib


def fill(dst, dtype: str, seed: int, tag: int, tok_session, tok_pos, scale: float = 1.0,
         stream=None) -> None:
    """Fill ``dst`` ([L][T][H][D] CUDA tensor) with values at (session[t], l, pos[t], h, d).

    ``tok_session`` and ``tok_pos`` are int32 CUDA tensors of length T.
    """
    import torch
    layers, n_tok, heads, head_dim = dst.shape
    assert dst.is_contiguous() and tok_session.dtype == torch.int32 and tok_pos.dtype == torch.int32
    s = torch.cuda.current_stream().cuda_stream if stream is None else stream
    rc = _load().synth_fill(dst.data_ptr(), 1 if dtype == "bf16" else 0, seed, tag,
                            V.IH_SCALE_BITS, float(np.float32(scale)), layers, n_tok, heads,
                            head_dim, tok_session.data_ptr(), tok_pos.data_ptr(), s)
    if rc != 0:
        raise RuntimeError(f"synth_fill failed with CUDA error {rc}")
