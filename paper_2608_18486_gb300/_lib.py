"""ctypes binding of libwm (include/wm.h): argument marshalling only.

Every function here has the name of the C entry point it calls and does no
computation of its own.  Loading fails loudly when libwm.so is missing: there
is no fallback path.
"""
from __future__ import annotations

import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libwm.so")

WM_MAX_L = 128
WM_OK, WM_ERR_INVALID_ARG, WM_ERR_UNSUPPORTED, WM_ERR_CUDA, WM_ERR_BOUNDS, WM_ERR_TIMEOUT = range(6)
WM_DT_F32, WM_DT_BF16 = 0, 1

EXPORTED = ["wm_status_string", "wm_config_check", "wm_cache_bytes", "wm_cache_alloc",
            "wm_kv_mix_workspace", "wm_kv_mix", "wm_decode_attn_workspace", "wm_decode_attn",
            "wm_decode_attn_flags", "wm_decode_attn_plan", "wm_prefill_attn",
            "wm_kv_mix_launches"]
WM_ATTN_INPUTS_READY = 1
WM_ATTN_DYNAMIC_SPLIT = 2
WM_ATTN_UNIT_SPLIT = 4


class wm_config(ctypes.Structure):
    _fields_ = [("L", ctypes.c_int32), ("k", ctypes.c_int32), ("D", ctypes.c_int32),
                ("Hq", ctypes.c_int32), ("Hkv", ctypes.c_int32), ("d", ctypes.c_int32),
                ("p", ctypes.c_int32), ("page_size", ctypes.c_int32), ("dtype", ctypes.c_int32),
                ("eps_rms", ctypes.c_float), ("eps_qk", ctypes.c_float),
                ("rope_theta", ctypes.c_double),
                ("chan_of_layer", ctypes.c_int32 * WM_MAX_L)]


class wm_cache(ctypes.Structure):
    _fields_ = [("k_pool", ctypes.c_void_p), ("v_pool", ctypes.c_void_p),
                ("num_pages", ctypes.c_int32), ("k", ctypes.c_int32), ("Hkv", ctypes.c_int32),
                ("page_size", ctypes.c_int32), ("d", ctypes.c_int32), ("dtype", ctypes.c_int32)]


class wm_mix_weights(ctypes.Structure):
    _fields_ = [("pre_g", ctypes.c_void_p * 2), ("Wr", ctypes.c_void_p * 2),
                ("br", ctypes.c_void_p * 2), ("ch_g", ctypes.c_void_p * 2),
                ("Wkv", ctypes.c_void_p * 2), ("qk_g", ctypes.c_void_p)]


class WMError(RuntimeError):
    def __init__(self, code: int, what: str):
        self.code = code
        super().__init__(f"{what}: {wm_status_string(code)} ({code})")


_lib = None


def lib():
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with __graft_entry__.build() "
                               "(there is no non-CUDA fallback)")
        L = ctypes.CDLL(LIB_PATH)
        cp, vp, sz, i32 = ctypes.POINTER(wm_config), ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int32
        L.wm_status_string.restype = ctypes.c_char_p
        L.wm_status_string.argtypes = [ctypes.c_int]
        L.wm_config_check.restype = ctypes.c_int
        L.wm_config_check.argtypes = [cp]
        L.wm_cache_bytes.restype = sz
        L.wm_cache_bytes.argtypes = [cp, i32]
        L.wm_cache_alloc.restype = ctypes.c_int
        L.wm_cache_alloc.argtypes = [cp, vp, sz, i32, ctypes.POINTER(wm_cache)]
        L.wm_kv_mix_workspace.restype = sz
        L.wm_kv_mix_workspace.argtypes = [cp, i32]
        L.wm_kv_mix.restype = ctypes.c_int
        L.wm_kv_mix.argtypes = [cp, ctypes.POINTER(wm_cache), ctypes.POINTER(wm_mix_weights), vp,
                                vp, vp, i32, i32, vp, sz, vp, vp]
        L.wm_decode_attn_workspace.restype = sz
        L.wm_decode_attn_workspace.argtypes = [cp, i32, i32]
        L.wm_decode_attn.restype = ctypes.c_int
        L.wm_decode_attn.argtypes = [cp, ctypes.POINTER(wm_cache), i32, vp, vp, vp, i32, i32, vp,
                                     vp, sz, vp, vp]
        L.wm_decode_attn_flags.restype = ctypes.c_int
        L.wm_decode_attn_flags.argtypes = [cp, ctypes.POINTER(wm_cache), i32, vp, vp, vp, i32, i32,
                                           vp, vp, sz, ctypes.c_uint32, vp, vp]
        L.wm_kv_mix_launches.restype = ctypes.c_int32
        L.wm_kv_mix_launches.argtypes = [cp, i32]
        L.wm_decode_attn_plan.restype = ctypes.c_int
        L.wm_decode_attn_plan.argtypes = [cp, i32, i32, ctypes.c_uint32,
                                          ctypes.POINTER(ctypes.c_int32)]
        L.wm_prefill_attn.restype = ctypes.c_int
        L.wm_prefill_attn.argtypes = [cp, ctypes.POINTER(wm_cache), i32, vp, vp, vp, i32, i32, i32,
                                      vp, vp, vp]
        _lib = L
    return _lib


def make_config(L, k, D, Hq, Hkv, d, p, page_size, dtype, chan_of_layer, eps_rms=1e-6,
                eps_qk=1e-6, rope_theta=1e6) -> wm_config:
    c = wm_config()
    c.L, c.k, c.D, c.Hq, c.Hkv, c.d, c.p, c.page_size = L, k, D, Hq, Hkv, d, p, page_size
    c.dtype = {"f32": WM_DT_F32, "bf16": WM_DT_BF16}.get(dtype, dtype)
    c.eps_rms, c.eps_qk, c.rope_theta = eps_rms, eps_qk, rope_theta
    if len(chan_of_layer) != L or L > WM_MAX_L:
        raise ValueError("chan_of_layer must have L entries, L <= WM_MAX_L")
    for i, ch in enumerate(chan_of_layer):
        c.chan_of_layer[i] = int(ch)
    return c


def _p(x) -> int | None:
    """Address of a tensor (or an int address, or None)."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def wm_status_string(code: int) -> str:
    return lib().wm_status_string(int(code)).decode()


def wm_config_check(cfg: wm_config) -> int:
    return lib().wm_config_check(ctypes.byref(cfg))


def wm_cache_bytes(cfg: wm_config, num_pages: int) -> int:
    return int(lib().wm_cache_bytes(ctypes.byref(cfg), int(num_pages)))


def wm_cache_alloc(cfg: wm_config, dev_buf, nbytes: int, num_pages: int) -> wm_cache:
    out = wm_cache()
    rc = lib().wm_cache_alloc(ctypes.byref(cfg), _p(dev_buf), int(nbytes), int(num_pages),
                              ctypes.byref(out))
    if rc != WM_OK:
        raise WMError(rc, "wm_cache_alloc")
    return out


def wm_kv_mix_workspace(cfg: wm_config, B: int) -> int:
    return int(lib().wm_kv_mix_workspace(ctypes.byref(cfg), int(B)))


def wm_decode_attn_workspace(cfg: wm_config, B: int, max_pages: int) -> int:
    return int(lib().wm_decode_attn_workspace(ctypes.byref(cfg), int(B), int(max_pages)))


def mix_weights(pre_g, Wr, br, ch_g, Wkv, qk_g) -> wm_mix_weights:
    """Pack per-branch pairs (index 0 = K, 1 = V) of device tensors."""
    w = wm_mix_weights()
    for X in range(2):
        w.pre_g[X], w.Wr[X], w.br[X] = _p(pre_g[X]), _p(Wr[X]), _p(br[X])
        w.ch_g[X], w.Wkv[X] = _p(ch_g[X]), _p(Wkv[X])
    w.qk_g = _p(qk_g)
    return w


def wm_kv_mix(cfg, cache, weights, h, page_table, slot, B, max_pages, workspace, ws_bytes,
              dev_status, stream) -> int:
    return lib().wm_kv_mix(ctypes.byref(cfg), ctypes.byref(cache), ctypes.byref(weights), _p(h),
                           _p(page_table), _p(slot), int(B), int(max_pages), _p(workspace),
                           int(ws_bytes), _p(dev_status), stream)


def wm_decode_attn(cfg, cache, layer, q, page_table, seq_lens, B, max_pages, out, workspace,
                   ws_bytes, dev_status, stream) -> int:
    return lib().wm_decode_attn(ctypes.byref(cfg), ctypes.byref(cache), int(layer), _p(q),
                                _p(page_table), _p(seq_lens), int(B), int(max_pages), _p(out),
                                _p(workspace), int(ws_bytes), _p(dev_status), stream)


def wm_decode_attn_flags(cfg, cache, layer, q, page_table, seq_lens, B, max_pages, out, workspace,
                         ws_bytes, flags, dev_status, stream) -> int:
    return lib().wm_decode_attn_flags(ctypes.byref(cfg), ctypes.byref(cache), int(layer), _p(q),
                                      _p(page_table), _p(seq_lens), int(B), int(max_pages),
                                      _p(out), _p(workspace), int(ws_bytes), int(flags),
                                      _p(dev_status), stream)


def wm_kv_mix_launches(cfg, B) -> int:
    """Kernels one wm_kv_mix call of B tokens enqueues (-1: invalid)."""
    return int(lib().wm_kv_mix_launches(ctypes.byref(cfg), int(B)))


def wm_decode_attn_plan(cfg, B, max_pages, flags=0) -> dict:
    """How a launch would be split: grid, warps, chunks, stages per chunk,
    CTAs per unit of the unit split (0: stream-K)."""
    plan = (ctypes.c_int32 * 5)()
    rc = lib().wm_decode_attn_plan(ctypes.byref(cfg), int(B), int(max_pages), int(flags), plan)
    if rc != WM_OK:
        raise WMError(rc, "wm_decode_attn_plan")
    return {"grid": plan[0], "warps": plan[1], "chunks": plan[2], "chunk_stages": plan[3],
            "unit_ctas": plan[4]}


def wm_prefill_attn(cfg, cache, layer, q, pos, page_table, B, Tq, max_pages, out, dev_status,
                    stream) -> int:
    return lib().wm_prefill_attn(ctypes.byref(cfg), ctypes.byref(cache), int(layer), _p(q), _p(pos),
                                 _p(page_table), int(B), int(Tq), int(max_pages), _p(out),
                                 _p(dev_status), stream)


def wm_decode_attn_noalloc(cfg, cache, layer, q, page_table, seq_lens, B, max_pages, out,
                           dev_status, stream) -> int:
    """Decode attention with the library's own fixed scratch (no workspace)."""
    L = lib()
    if not getattr(L, "_noalloc_typed", False):
        cp, vp, i32 = ctypes.POINTER(wm_config), ctypes.c_void_p, ctypes.c_int32
        L.wm_decode_attn_noalloc.restype = ctypes.c_int
        L.wm_decode_attn_noalloc.argtypes = [cp, ctypes.POINTER(wm_cache), i32, vp, vp, vp, i32,
                                             i32, vp, vp, vp]
        L._noalloc_typed = True
    return L.wm_decode_attn_noalloc(ctypes.byref(cfg), ctypes.byref(cache), int(layer), _p(q),
                                    _p(page_table), _p(seq_lens), int(B), int(max_pages), _p(out),
                                    _p(dev_status), stream)


def wm_selftest_bounded_wait(dev_status, limit_us: int, stream) -> int:
    """Run the bounded-wait self-test (see include/wm.h)."""
    L = lib()
    L.wm_selftest_bounded_wait.restype = ctypes.c_int
    L.wm_selftest_bounded_wait.argtypes = [ctypes.c_void_p, ctypes.c_uint32, ctypes.c_void_p]
    return L.wm_selftest_bounded_wait(_p(dev_status), int(limit_us), stream)
