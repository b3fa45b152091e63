"""Fill device buffers with the same synthetic values ``gen.py`` yields on the host."""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import gen

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libwmsynth.so")
_lib = None


def build(verbose: bool = False) -> str:
    import subprocess
    src = os.path.join(_HERE, "synth.cu")
    cmd = ["nvcc", "-O3", "-std=c++17", "-shared", "-Xcompiler", "-fPIC",
           "-gencode", "arch=compute_103a,code=sm_103a", "-lineinfo",
           "-o", LIB_PATH, src]
    if verbose:
        print(" ".join(cmd))
    subprocess.check_call(cmd)
    return LIB_PATH


def lib():
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} missing: run __graft_entry__.build()")
        L = ctypes.CDLL(LIB_PATH)
        L.wms_fill.restype = ctypes.c_int
        L.wms_fill.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_uint64, ctypes.c_uint64,
                               ctypes.c_uint64, ctypes.c_uint64, ctypes.c_float, ctypes.c_float,
                               ctypes.c_float, ctypes.c_void_p]
        _lib = L
    return _lib


def fill(tensor, dtype: str, seed: int, stream: int, std: float = 1.0, mean: float = 0.0,
         start: int = 0, cuda_stream=None) -> None:
    """Fill a contiguous CUDA tensor (fp32, or int16/bf16 storage) in flat order."""
    import torch
    assert tensor.is_cuda and tensor.is_contiguous()
    dt = 0 if dtype == "f32" else 1
    if cuda_stream is None:
        cuda_stream = torch.cuda.current_stream().cuda_stream
    rc = lib().wms_fill(ctypes.c_void_p(tensor.data_ptr()), dt, tensor.numel(), seed, stream,
                        start, float(gen.IRWIN_HALL4_SCALE), float(np.float32(std)),
                        float(np.float32(mean)), ctypes.c_void_p(cuda_stream))
    if rc != 0:
        raise RuntimeError(f"wms_fill failed with CUDA error {rc}")


def fill_spec(tensor, prob, name: str) -> None:
    s = prob.specs[name]
    assert tensor.numel() == s.count, (name, tensor.numel(), s.count)
    fill(tensor, prob.w.dtype, prob.seed, s.stream, s.std, s.mean)
