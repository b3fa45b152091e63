"""Python access to the fp64 CPU oracle (``wm_oracle.c``).

TEST INFRASTRUCTURE ONLY: imported by tests/, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py``; never by the product package.

Arrays are passed in their storage dtype: ``float32`` for fp32 workloads and
``uint16`` bf16 bit patterns for bf16 workloads; the C code widens every read
to double.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(_HERE, "wm_oracle.c")
LIB_PATH = os.path.join(_HERE, "liboracle.so")
# A compiled copy of the oracle to load instead of liboracle.so: the mutation
# test (tests/test_oracle_mutants.py) points it at copies with a planted
# mistake to show that the pins catch each one.
ALT_LIB = os.environ.get("WM_ORACLE_LIB")
_lib = None

_dp = ctypes.POINTER(ctypes.c_double)
_vp = ctypes.c_void_p
_i64p = ctypes.POINTER(ctypes.c_int64)
_i32p = ctypes.POINTER(ctypes.c_int32)


def build(verbose: bool = False) -> str:
    cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-shared", "-fPIC", "-o", LIB_PATH, SRC, "-lm"]
    if verbose:
        print(" ".join(cmd))
    subprocess.check_call(cmd)
    return LIB_PATH


def lib():
    global _lib
    if _lib is None:
        if ALT_LIB:
            L = ctypes.CDLL(ALT_LIB)
        else:
            if not os.path.exists(LIB_PATH) or os.path.getmtime(LIB_PATH) < os.path.getmtime(SRC):
                build()
            L = ctypes.CDLL(LIB_PATH)
        L.orc_max_threads.restype = ctypes.c_int
        L.orc_rmsnorm.argtypes = [_dp, ctypes.c_int, ctypes.c_double, _dp, _dp]
        L.orc_rope.argtypes = [_dp, ctypes.c_int, ctypes.c_double, ctypes.c_double]
        L.orc_pool_route.argtypes = [ctypes.c_int] * 4 + [ctypes.c_double, ctypes.c_int] + \
            [_vp] * 4 + [_dp, _dp, _i64p]
        L.orc_pool_channel.argtypes = [ctypes.c_int] * 4 + [ctypes.c_double] * 3 + \
            [ctypes.c_int, ctypes.c_double, ctypes.c_int, _dp, _dp, _vp, _vp, _vp, _dp, _dp, _i64p]
        L.orc_kv_mix.argtypes = [ctypes.c_int] * 7 + [ctypes.c_double] * 3 + [ctypes.c_int] + \
            [_vp, _dp] + [_vp] * 6 + [_dp, _dp, _dp, _i64p, ctypes.c_int]
        L.orc_decode_attn.restype = ctypes.c_int
        L.orc_decode_attn.argtypes = [ctypes.c_int] * 8 + [_vp, _vp, _i32p, _i32p, _vp,
                                                           ctypes.c_int, _i32p, _dp, _i64p,
                                                           ctypes.c_int]
        L.orc_prefill_attn.restype = ctypes.c_int
        L.orc_prefill_attn.argtypes = [ctypes.c_int] * 8 + [_vp, _vp, _i32p, _i32p, ctypes.c_int,
                                                            _vp, ctypes.c_int, _i32p, _dp, _i64p,
                                                            ctypes.c_int]
        _lib = L
    return _lib


def _dtcode(a: np.ndarray) -> int:
    if a.dtype == np.float32:
        return 0
    if a.dtype == np.uint16:
        return 1
    raise TypeError(f"oracle inputs are float32 or uint16 (bf16 bits), got {a.dtype}")


def _c(a, dtype=None):
    return np.ascontiguousarray(a, dtype=dtype)


def _ptr(a):
    return a.ctypes.data_as(ctypes.c_void_p)


def _dptr(a):
    return a.ctypes.data_as(_dp)


def max_threads() -> int:
    return int(lib().orc_max_threads())


def rmsnorm(x, eps, g=None) -> np.ndarray:
    x = _c(x, np.float64)
    y = np.empty_like(x)
    gg = None if g is None else _c(g, np.float64)
    lib().orc_rmsnorm(_dptr(x), x.size, eps, None if gg is None else _dptr(gg), _dptr(y))
    return y


def rope(y, pos, theta) -> np.ndarray:
    y = _c(y, np.float64).copy()
    lib().orc_rope(_dptr(y), y.size, float(pos), float(theta))
    return y


def pool_route(h, pre_g, Wr, br, *, L, k, D, p, eps):
    """Sec. 3.1 Step 1 routing for one token.  Returns (hhat[2][L][D],
    alpha[2][k][L], router MACs)."""
    h, pre_g, Wr, br = (_c(a) for a in (h, pre_g, Wr, br))
    dt = _dtcode(h)
    hhat = np.empty((2, L, D))
    alpha = np.empty((2, k, L))
    macs = np.zeros(1, dtype=np.int64)
    lib().orc_pool_route(L, k, D, p, eps, dt, _ptr(h), _ptr(pre_g), _ptr(Wr), _ptr(br),
                         _dptr(hhat), _dptr(alpha), macs.ctypes.data_as(_i64p))
    return hhat, alpha, int(macs[0])


def pool_channel(hhat_X, alpha_Xj, ch_g_Xj, W_Xj, qk_g_j, *, is_key, pos, Hkv, d, eps,
                 eps_qk, theta):
    """Sec. 3.1 Steps 1 (mix) and 2 for one token, branch and channel.
    Returns (htilde[D], out[Hkv*d], (mix MACs, projection MACs))."""
    hhat_X = _c(hhat_X, np.float64)
    alpha_Xj = _c(alpha_Xj, np.float64)
    ch_g_Xj, W_Xj, qk_g_j = _c(ch_g_Xj), _c(W_Xj), _c(qk_g_j)
    L, D = hhat_X.shape
    ht = np.empty(D)
    out = np.empty(Hkv * d)
    macs = np.zeros(2, dtype=np.int64)
    lib().orc_pool_channel(L, D, Hkv, d, eps, eps_qk, theta, int(is_key), float(pos),
                           _dtcode(W_Xj), _dptr(hhat_X), _dptr(alpha_Xj), _ptr(ch_g_Xj),
                           _ptr(W_Xj), _ptr(qk_g_j), _dptr(ht), _dptr(out),
                           macs.ctypes.data_as(_i64p))
    return ht, out, (int(macs[0]), int(macs[1]))


def kv_mix(h, pos, pre_g, Wr, br, ch_g, Wkv, qk_g, *, L, k, D, Hkv, d, p, eps, eps_qk,
           theta, nthreads=1):
    """The pool for B tokens.  Returns (K[B][k][Hkv][d] rotated normed keys,
    V[B][k][Hkv][d], alpha[B][2][k][L], MACs (router, mix, projection))."""
    h = _c(h)
    B = h.shape[0]
    arrs = [_c(a) for a in (pre_g, Wr, br, ch_g, Wkv, qk_g)]
    pos = _c(pos, np.float64)
    K = np.empty((B, k, Hkv, d))
    V = np.empty((B, k, Hkv, d))
    alpha = np.empty((B, 2, k, L))
    macs = np.zeros(3, dtype=np.int64)
    lib().orc_kv_mix(B, L, k, D, Hkv, d, p, eps, eps_qk, theta, _dtcode(h), _ptr(h), _dptr(pos),
                     *[_ptr(a) for a in arrs], _dptr(K), _dptr(V), _dptr(alpha),
                     macs.ctypes.data_as(_i64p), int(nthreads))
    return K, V, alpha, tuple(int(m) for m in macs)


def decode_attn(q, k_pool, v_pool, page_table, seq_lens, *, chan, Hq, Hkv, d, P, units=None,
                nthreads=1, return_macs=False):
    """Sec. 3.1 Step 3 decode attention of layer-reading channel ``chan``.

    ``k_pool``/``v_pool`` are [kch][num_pages][Hkv][P][d]; ``q`` is [B][Hq][d].
    ``units`` lists (b, hq) pairs (default: all).  Returns out[nunits][d]
    (or [B][Hq][d] when ``units`` is None)."""
    q = _c(q)
    k_pool, v_pool = _c(k_pool), _c(v_pool)
    pt = _c(page_table, np.int32)
    sl = _c(seq_lens, np.int32)
    B = q.shape[0]
    num_pages = k_pool.shape[1]
    full = units is None
    if full:
        units = [(b, hq) for b in range(B) for hq in range(Hq)]
    u = _c(np.asarray(units, dtype=np.int32).reshape(-1, 2))
    out = np.empty((u.shape[0], d))
    macs = np.zeros(1, dtype=np.int64)
    rc = lib().orc_decode_attn(Hq, Hkv, d, P, num_pages, pt.shape[1], chan, _dtcode(q), _ptr(k_pool),
                               _ptr(v_pool), pt.ctypes.data_as(_i32p), sl.ctypes.data_as(_i32p),
                               _ptr(q), u.shape[0], u.ctypes.data_as(_i32p), _dptr(out),
                               macs.ctypes.data_as(_i64p), int(nthreads))
    if rc != 0:
        raise IndexError(f"oracle decode_attn: error {rc} (page id or length out of range)")
    if full:
        out = out.reshape(B, Hq, d)
    return (out, int(macs[0])) if return_macs else out


def prefill_attn(q, k_pool, v_pool, page_table, pos, *, chan, Hq, Hkv, d, P, units=None,
                 nthreads=1, return_macs=False):
    """Sec. 3.1 Step 3 causal attention with the dummy offset of Sec. 3.2, for
    query rows at given token positions (prefill; Jacobi / Gauss-Seidel passes
    of Sec. 3.3).  Row r of sequence b is the query of the token at position
    ``pos[b][r]`` and reads slots 0 .. pos of channel ``chan``.

    ``q`` is [B][Tq][Hq][d]; ``k_pool``/``v_pool`` are [kch][num_pages][Hkv][P][d].
    ``units`` lists (b, r, hq) triples (default: all).  Returns out[nunits][d]
    (or [B][Tq][Hq][d] when ``units`` is None)."""
    q = _c(q)
    k_pool, v_pool = _c(k_pool), _c(v_pool)
    pt = _c(page_table, np.int32)
    ps = _c(pos, np.int32)
    B, Tq = q.shape[0], q.shape[1]
    num_pages = k_pool.shape[1]
    full = units is None
    if full:
        units = [(b, r, hq) for b in range(B) for r in range(Tq) for hq in range(Hq)]
    u = _c(np.asarray(units, dtype=np.int32).reshape(-1, 3))
    out = np.empty((u.shape[0], d))
    macs = np.zeros(1, dtype=np.int64)
    rc = lib().orc_prefill_attn(Hq, Hkv, d, P, num_pages, pt.shape[1], chan, _dtcode(q),
                                _ptr(k_pool), _ptr(v_pool), pt.ctypes.data_as(_i32p),
                                ps.ctypes.data_as(_i32p), Tq, _ptr(q), u.shape[0],
                                u.ctypes.data_as(_i32p), _dptr(out), macs.ctypes.data_as(_i64p),
                                int(nthreads))
    if rc != 0:
        raise IndexError(f"oracle prefill_attn: error {rc} (position or page id out of range)")
    if full:
        out = out.reshape(B, Tq, Hq, d)
    return (out, int(macs[0])) if return_macs else out
