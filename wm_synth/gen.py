"""Counter-based seeded value generator shared by the oracle side and the GPU side.

This module holds no arithmetic of the method; it only turns
``(seed, stream, flat index)`` into a synthetic value, identically on the host
(numpy here, and the same definition compiled in ``gen_host.c``) and on the
device (``synth.cu`` in this folder).

Definition
----------
* Raw bits: the i-th output (i = 0, 1, ...) of a SplitMix64 generator
  (Steele, Lea & Flood, "Fast splittable pseudorandom number generators",
  OOPSLA 2014) whose state starts at ``key(seed, stream)``:
  ``raw(i) = mix64(key + (i + 1) * GAMMA)``.
* ``key(seed, stream) = mix64(seed * 2**32 + stream + GAMMA)`` (the first
  output of a SplitMix64 started at ``seed * 2**32 + stream``).
* Approximately normal value: the four 16-bit fields of ``raw(i)`` are summed
  (Irwin-Hall with four terms), centred and scaled to unit variance in fp32,
  then ``value = (n * std) + mean`` with each fp32 operation rounded to
  nearest separately (no fused multiply-add), so host and device agree bit
  for bit.  The distribution is bounded at +-3.46 sigma; its first two
  moments are those of N(mean, std^2).
* bf16 storage: round-to-nearest-even of the fp32 value.
"""
from __future__ import annotations

import concurrent.futures as cf
import ctypes
import os
import subprocess

import numpy as np

GAMMA = np.uint64(0x9E3779B97F4A7C15)
M1 = np.uint64(0xBF58476D1CE4E5B9)
M2 = np.uint64(0x94D049BB133111EB)
# 1 / sqrt(4 * (65536**2 - 1) / 12) rounded to fp32: unit variance for the
# sum of four uniform 16-bit integers.
IRWIN_HALL4_SCALE = np.float32(1.0 / np.sqrt(4.0 * (65536.0 ** 2 - 1.0) / 12.0))
IRWIN_HALL4_MEAN = 131070  # 4 * 65535 / 2

_S30 = np.uint64(30)
_S27 = np.uint64(27)
_S31 = np.uint64(31)


def mix64(z: np.ndarray) -> np.ndarray:
    """SplitMix64 output function on a uint64 array (wraps mod 2**64)."""
    z = np.asarray(z, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = (z ^ (z >> _S30)) * M1
        z = (z ^ (z >> _S27)) * M2
    return z ^ (z >> _S31)


def stream_key(seed: int, stream: int) -> np.uint64:
    with np.errstate(over="ignore"):
        s = np.uint64((int(seed) << 32) + int(stream)) + GAMMA
    return mix64(np.array([s], dtype=np.uint64))[0]


def raw_bits(seed: int, stream: int, index: np.ndarray) -> np.ndarray:
    key = stream_key(seed, stream)
    idx = np.asarray(index, dtype=np.uint64)
    with np.errstate(over="ignore"):
        return mix64(key + (idx + np.uint64(1)) * GAMMA)


def normal_f32(seed: int, stream: int, index: np.ndarray, std: float = 1.0,
               mean: float = 0.0) -> np.ndarray:
    """Approximately N(mean, std^2) fp32 values at the given flat indices."""
    z = raw_bits(seed, stream, index)
    m16 = np.uint64(0xFFFF)
    s = ((z & m16) + ((z >> np.uint64(16)) & m16) + ((z >> np.uint64(32)) & m16)
         + (z >> np.uint64(48))).astype(np.int64)
    c = (s - IRWIN_HALL4_MEAN).astype(np.float32)  # exact: |c| < 2**24
    n = c * IRWIN_HALL4_SCALE                     # fp32, one rounding
    v = n * np.float32(std)                         # fp32, one rounding
    v = v + np.float32(mean)                        # fp32, one rounding
    return v.astype(np.float32)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even fp32 -> bf16, returned as uint16 bit patterns."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    nan = (u & np.uint64(0x7FFFFFFF)) > np.uint64(0x7F800000)
    r = (u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))) >> np.uint64(16)
    r = np.where(nan, (u >> np.uint64(16)) | np.uint64(0x40), r)
    return r.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def _stored(dtype: str, seed: int, stream: int, idx: np.ndarray, std: float,
            mean: float) -> np.ndarray:
    v = normal_f32(seed, stream, idx, std, mean)
    return v if dtype == "f32" else f32_to_bf16_bits(v)


# Large requests are cut into chunks of this many values, filled by a few
# threads (numpy releases the GIL in its loops): the same bits as one pass,
# without gigabyte-sized temporaries.
_CHUNK = 1 << 20


def _chunked(dtype: str, count: int, fill) -> np.ndarray:
    if dtype not in ("f32", "bf16"):
        raise ValueError(f"unknown dtype {dtype!r}")
    out = np.empty(count, dtype=np.float32 if dtype == "f32" else np.uint16)

    def job(o):
        n = min(_CHUNK, count - o)
        out[o:o + n] = fill(o, n)

    starts = range(0, count, _CHUNK)
    if len(starts) <= 1:
        for o in starts:
            job(o)
        return out
    with cf.ThreadPoolExecutor(min(len(starts), os.cpu_count() or 1, 16)) as ex:
        list(ex.map(job, starts))
    return out


def values_np(dtype: str, seed: int, stream: int, start: int, count: int,
              std: float = 1.0, mean: float = 0.0) -> np.ndarray:
    """``count`` consecutive values of one stream, stored in ``dtype``, computed
    with numpy from the definition above.

    Returns float32 for ``"f32"`` and uint16 bf16 bit patterns for ``"bf16"``.
    """
    return _chunked(dtype, count, lambda o, n: _stored(
        dtype, seed, stream, np.arange(start + o, start + o + n, dtype=np.uint64), std, mean))


def values_at_np(dtype: str, seed: int, stream: int, index: np.ndarray,
                 std: float = 1.0, mean: float = 0.0) -> np.ndarray:
    """Values of one stream at arbitrary flat indices (numpy, same as ``values_np``)."""
    index = np.asarray(index, dtype=np.uint64)
    flat = index.reshape(-1)
    out = _chunked(dtype, flat.size, lambda o, n: _stored(dtype, seed, stream, flat[o:o + n],
                                                          std, mean))
    return out.reshape(index.shape)


# The same definition compiled (gen_host.c, OpenMP): tens of times faster than
# numpy for the gigabyte-sized regenerations of the full-size parity tests.
# Built on first use; without a C compiler the numpy functions serve.
_HERE = os.path.dirname(os.path.abspath(__file__))
HOST_SRC = os.path.join(_HERE, "gen_host.c")
HOST_LIB = os.path.join(_HERE, "libwmgen.so")
_host = None


def build_host(verbose: bool = False) -> str:
    cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-ffp-contract=off", "-shared", "-fPIC",
           "-o", HOST_LIB, HOST_SRC]
    if verbose:
        print(" ".join(cmd))
    subprocess.check_call(cmd)
    return HOST_LIB


def _host_lib():
    global _host
    if _host is None:
        try:
            if not os.path.exists(HOST_LIB) or os.path.getmtime(HOST_LIB) < os.path.getmtime(HOST_SRC):
                build_host()
            L = ctypes.CDLL(HOST_LIB)
            L.wmg_fill_runs.restype = None
            L.wmg_fill_runs.argtypes = [ctypes.c_int, ctypes.c_uint64, ctypes.c_void_p,
                                        ctypes.c_int64, ctypes.c_int64, ctypes.c_float,
                                        ctypes.c_float, ctypes.c_float, ctypes.c_void_p,
                                        ctypes.c_int]
            L.wmg_fill.restype = None
            L.wmg_fill.argtypes = [ctypes.c_int, ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int64,
                                   ctypes.c_void_p, ctypes.c_float, ctypes.c_float, ctypes.c_float,
                                   ctypes.c_void_p, ctypes.c_int]
            _host = L
        except Exception:
            _host = False
    return _host or None


def _fill_host(L, dtype, seed, stream, start, count, index, std, mean):
    if dtype not in ("f32", "bf16"):
        raise ValueError(f"unknown dtype {dtype!r}")
    out = np.empty(count, dtype=np.float32 if dtype == "f32" else np.uint16)
    key = int(stream_key(seed, stream))
    L.wmg_fill(0 if dtype == "f32" else 1, key, int(start), int(count),
               None if index is None else index.ctypes.data, float(IRWIN_HALL4_SCALE),
               float(np.float32(std)), float(np.float32(mean)), out.ctypes.data, 0)
    return out


def values(dtype: str, seed: int, stream: int, start: int, count: int,
           std: float = 1.0, mean: float = 0.0) -> np.ndarray:
    """``count`` consecutive values of one stream, stored in ``dtype``.

    Returns float32 for ``"f32"`` and uint16 bf16 bit patterns for ``"bf16"``.
    """
    L = _host_lib()
    if L is None:
        return values_np(dtype, seed, stream, start, count, std, mean)
    return _fill_host(L, dtype, seed, stream, start, count, None, std, mean)


def values_at(dtype: str, seed: int, stream: int, index: np.ndarray,
              std: float = 1.0, mean: float = 0.0) -> np.ndarray:
    """Values of one stream at arbitrary flat indices (same as ``values``)."""
    L = _host_lib()
    if L is None:
        return values_at_np(dtype, seed, stream, index, std, mean)
    index = np.ascontiguousarray(index, dtype=np.uint64)
    out = _fill_host(L, dtype, seed, stream, 0, index.size, index.reshape(-1), std, mean)
    return out.reshape(index.shape)


def values_runs(dtype: str, seed: int, stream: int, starts, run_len: int,
                std: float = 1.0, mean: float = 0.0) -> np.ndarray:
    """[len(starts)][run_len] values: row r holds the run of ``run_len``
    consecutive values from flat index ``starts[r]`` (same as ``values``)."""
    starts = np.ascontiguousarray(starts, dtype=np.uint64).reshape(-1)
    L = _host_lib()
    if L is None:
        return np.stack([values_np(dtype, seed, stream, int(s0), run_len, std, mean)
                         for s0 in starts]) if len(starts) else \
            np.empty((0, run_len), np.float32 if dtype == "f32" else np.uint16)
    if dtype not in ("f32", "bf16"):
        raise ValueError(f"unknown dtype {dtype!r}")
    out = np.empty((starts.size, run_len), dtype=np.float32 if dtype == "f32" else np.uint16)
    L.wmg_fill_runs(0 if dtype == "f32" else 1, int(stream_key(seed, stream)), starts.ctypes.data,
                    starts.size, int(run_len), float(IRWIN_HALL4_SCALE), float(np.float32(std)),
                    float(np.float32(mean)), out.ctypes.data, 0)
    return out


def to_f64(dtype: str, stored: np.ndarray) -> np.ndarray:
    """Widen stored values (fp32, or bf16 bit patterns) to float64."""
    if dtype == "f32":
        return np.asarray(stored, dtype=np.float32).astype(np.float64)
    return bf16_bits_to_f32(stored).astype(np.float64)
