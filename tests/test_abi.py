"""The C-ABI library loads, exports every entry point include/*.h declares,
and rejects bad arguments on the host (no GPU needed, nothing launched)."""
import ctypes
import glob
import os
import re

import pytest

from paper_2608_18486_gb300 import _lib as W
from wm_synth import configs

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _cuda_present() -> bool:
    try:
        import torch
        return torch.cuda.is_available()
    except Exception:  # pragma: no cover
        return False


# Tests that hand made-up device addresses to entry points that can launch:
# they check refusals made on the host before any launch, and run only where
# no GPU could ever receive a launch should a check regress.
host_refusals_only = pytest.mark.skipif(
    _cuda_present(), reason="passes made-up device addresses; host-side checks only, CPU only")


def declared_functions():
    names = set()
    for hdr in glob.glob(os.path.join(ROOT, "include", "*.h")):
        text = re.sub(r"/\*.*?\*/", "", open(hdr).read(), flags=re.S)
        names |= set(re.findall(r"\b(wm_\w+)\s*\(", text))
    return sorted(names)


def test_library_exports_every_declared_entry_point():
    lib = ctypes.CDLL(W.LIB_PATH)
    names = declared_functions()
    assert set(W.EXPORTED) <= set(names)
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing


def cfg(**kw):
    w = configs.get("large")
    c = W.make_config(w.L, w.k, w.D, w.Hq, w.Hkv, w.d, w.p, w.page, w.dtype, w.chan_of_layer())
    for k, v in kw.items():
        setattr(c, k, v)
    return c


@pytest.mark.parametrize("field,value,code", [
    ("k", 33, W.WM_ERR_INVALID_ARG), ("k", 0, W.WM_ERR_INVALID_ARG),
    ("Hq", 33, W.WM_ERR_INVALID_ARG), ("p", 0, W.WM_ERR_INVALID_ARG),
    ("dtype", 7, W.WM_ERR_INVALID_ARG), ("d", 80, W.WM_ERR_UNSUPPORTED),
    ("page_size", 24, W.WM_ERR_UNSUPPORTED), ("D", 8192, W.WM_ERR_UNSUPPORTED),
    ("Hq", 96, W.WM_ERR_UNSUPPORTED)])
def test_config_check_codes(field, value, code):
    assert W.wm_config_check(cfg()) == W.WM_OK
    assert W.wm_config_check(cfg(**{field: value})) == code


def test_channel_map_must_point_at_existing_channels():
    c = cfg()
    c.chan_of_layer[5] = c.k
    assert W.wm_config_check(c) == W.WM_ERR_INVALID_ARG


def test_cache_sizing_and_layout_without_gpu():
    c = cfg()
    n = W.wm_cache_bytes(c, 10)
    pool = c.k * 10 * c.Hkv * c.page_size * c.d * 2
    assert n == 2 * ((pool + 255) // 256 * 256)
    fake = 1 << 40  # never dereferenced: wm_cache_alloc only lays out views
    cache = W.wm_cache_alloc(c, fake, n, 10)
    assert cache.k_pool == fake and cache.v_pool == fake + n // 2
    with pytest.raises(W.WMError):
        W.wm_cache_alloc(c, fake, n - 1, 10)
    with pytest.raises(W.WMError):
        W.wm_cache_alloc(c, fake + 8, n, 10)
    assert W.wm_cache_bytes(c, 0) == 0


@host_refusals_only
def test_compute_calls_reject_bad_arguments_before_launching():
    c = cfg()
    n = W.wm_cache_bytes(c, 4)
    cache = W.wm_cache_alloc(c, 1 << 40, n, 4)
    fake = 1 << 41
    ws = W.wm_decode_attn_workspace(c, 2, 4)
    assert ws > 0
    # layer out of range, NULL query, misaligned output, short workspace
    assert W.wm_decode_attn(c, cache, c.L, fake, fake, fake, 2, 4, fake, fake, ws, None, None) == W.WM_ERR_INVALID_ARG
    assert W.wm_decode_attn(c, cache, 0, None, fake, fake, 2, 4, fake, fake, ws, None, None) == W.WM_ERR_INVALID_ARG
    assert W.wm_decode_attn(c, cache, 0, fake, fake, fake, 2, 4, fake + 2, fake, ws, None, None) == W.WM_ERR_INVALID_ARG
    assert W.wm_decode_attn(c, cache, 0, fake, fake, fake, 2, 4, fake, fake, ws - 1, None, None) == W.WM_ERR_INVALID_ARG
    # empty batch is a no-op even with NULL buffers
    assert W.wm_decode_attn(c, cache, 0, None, None, None, 0, 4, None, None, 0, None, None) == W.WM_OK
    # a cache laid out for another config is refused
    other = cfg(k=8)
    assert W.wm_decode_attn(other, cache, 0, fake, fake, fake, 2, 4, fake, fake, ws, None, None) == W.WM_ERR_INVALID_ARG
    assert W.wm_decode_attn_flags(c, cache, 0, fake, fake, fake, 2, 4, fake, fake, ws, 8, None,
                                  None) == W.WM_ERR_INVALID_ARG  # unknown flag bit
    both = W.WM_ATTN_DYNAMIC_SPLIT | W.WM_ATTN_UNIT_SPLIT  # two splits at once
    assert W.wm_decode_attn_flags(c, cache, 0, fake, fake, fake, 2, 4, fake, fake, ws, both, None,
                                  None) == W.WM_ERR_INVALID_ARG
    wts = W.mix_weights((fake, fake), (fake, fake), (fake, fake), (fake, fake), (fake, fake), fake)
    mws = W.wm_kv_mix_workspace(c, 2)
    assert W.wm_kv_mix(c, cache, wts, fake, fake, fake, 2, 4, fake, mws - 1, None, None) == W.WM_ERR_INVALID_ARG
    bad = W.mix_weights((fake, fake), (fake, None), (fake, fake), (fake, fake), (fake, fake), fake)
    assert W.wm_kv_mix(c, cache, bad, fake, fake, fake, 2, 4, fake, mws, None, None) == W.WM_ERR_INVALID_ARG
    assert W.wm_kv_mix(c, cache, wts, None, None, None, 0, 4, None, 0, None, None) == W.WM_OK


@host_refusals_only
def test_attention_refuses_output_rows_past_32_bits_before_launching():
    # 4096 sequences x 2^19 query heads: more output rows than the kernel's
    # 32-bit row index covers
    c = cfg(Hq=1 << 19, Hkv=1 << 16)
    assert W.wm_config_check(c) == W.WM_OK
    n = W.wm_cache_bytes(c, 1)
    cache = W.wm_cache_alloc(c, 1 << 40, n, 1)
    fake = 1 << 41
    ws = W.wm_decode_attn_workspace(c, 4096, 1)
    assert W.wm_decode_attn(c, cache, 0, fake, fake, fake, 4096, 1, fake, fake, ws, None,
                            None) == W.WM_ERR_UNSUPPORTED


def test_attention_workspace_grows_with_the_batch():
    # a workspace sized for the largest batch serves every smaller one
    c = cfg()
    sizes = [W.wm_decode_attn_workspace(c, b, 513) for b in (1, 2, 5, 16, 32, 100, 1000, 4096)]
    assert all(a <= b for a, b in zip(sizes, sizes[1:])), sizes
    assert all(s % 256 == 0 for s in sizes)


def test_status_strings():
    for code in range(6):
        assert W.wm_status_string(code) and W.wm_status_string(code) != "unknown status"


@host_refusals_only
def test_prefill_rejects_unsupported_and_bad_arguments_before_launching():
    c = cfg()
    n = W.wm_cache_bytes(c, 4)
    cache = W.wm_cache_alloc(c, 1 << 40, n, 4)
    fake = 1 << 41
    # fp32 caches and pages under 8 slots are not built
    c32 = cfg(dtype=W.WM_DT_F32)
    cache32 = W.wm_cache_alloc(c32, 1 << 40, W.wm_cache_bytes(c32, 4), 4)
    assert W.wm_prefill_attn(c32, cache32, 0, fake, fake, fake, 2, 8, 4, fake, None,
                             None) == W.WM_ERR_UNSUPPORTED
    c4 = cfg(page_size=4)
    cache4 = W.wm_cache_alloc(c4, 1 << 40, W.wm_cache_bytes(c4, 4), 4)
    assert W.wm_prefill_attn(c4, cache4, 0, fake, fake, fake, 2, 8, 4, fake, None,
                             None) == W.WM_ERR_UNSUPPORTED
    # layer out of range, NULL positions, misaligned output
    assert W.wm_prefill_attn(c, cache, c.L, fake, fake, fake, 2, 8, 4, fake, None,
                             None) == W.WM_ERR_INVALID_ARG
    assert W.wm_prefill_attn(c, cache, 0, fake, None, fake, 2, 8, 4, fake, None,
                             None) == W.WM_ERR_INVALID_ARG
    assert W.wm_prefill_attn(c, cache, 0, fake, fake, fake, 2, 8, 4, fake + 2, None,
                             None) == W.WM_ERR_INVALID_ARG
    # nothing to do is a no-op even with NULL buffers
    assert W.wm_prefill_attn(c, cache, 0, None, None, None, 0, 8, 4, None, None, None) == W.WM_OK
    assert W.wm_prefill_attn(c, cache, 0, None, None, None, 2, 0, 4, None, None, None) == W.WM_OK


def test_attention_plan_static_and_dynamic_split():
    # no_compression: 16 x 12 units of 2048 slots, 100 MB per launch -> static
    w = configs.get("no_compression")
    c = W.make_config(w.L, w.k, w.D, w.Hq, w.Hkv, w.d, w.p, w.page, w.dtype, w.chan_of_layer())
    max_pages = -(-(w.ctx + 1) // w.page)
    st = W.wm_decode_attn_plan(c, w.B, max_pages)
    assert st["chunk_stages"] == 0 and st["chunks"] == st["warps"] > 0
    dy = W.wm_decode_attn_plan(c, w.B, max_pages, W.WM_ATTN_DYNAMIC_SPLIT)
    assert dy["grid"] == st["grid"] and dy["chunk_stages"] >= 4
    assert dy["chunks"] > dy["warps"]  # warps take further chunks from the counter
    # the workspace query covers either split
    ws = W.wm_decode_attn_workspace(c, w.B, max_pages)
    rec = 4 * (w.d + 4)  # one partial record at G = 1 (d outputs, m, l, flag; 16-byte padded)
    assert ws >= 2 * dy["chunks"] * rec
    # a launch of over 2 GB (the long-context workload) splits dynamically anyway
    lw = configs.get("long128k")
    lc = W.make_config(lw.L, lw.k, lw.D, lw.Hq, lw.Hkv, lw.d, lw.p, lw.page, lw.dtype,
                       lw.chan_of_layer())
    big = W.wm_decode_attn_plan(lc, lw.B, -(-(lw.ctx + 1) // lw.page))
    assert big["chunk_stages"] > 0 and big["chunks"] > big["warps"]
    assert st["unit_ctas"] == 0 and dy["unit_ctas"] == 0 and big["unit_ctas"] == 0
    # the unit split: one cluster of C CTAs per (sequence, kv head) unit, C at
    # most 8 and no more SMs than the device has (units > SMs: C = 1)
    un = W.wm_decode_attn_plan(c, w.B, max_pages, W.WM_ATTN_UNIT_SPLIT)
    assert un["unit_ctas"] == 1 and un["grid"] == w.B * w.Hkv and un["chunk_stages"] == 0
    pw = configs.get("paper_k16")
    pc = W.make_config(pw.L, pw.k, pw.D, pw.Hq, pw.Hkv, pw.d, pw.p, pw.page, pw.dtype,
                       pw.chan_of_layer())
    pmax = -(-(pw.ctx + 1) // pw.page)
    pu = W.wm_decode_attn_plan(pc, pw.B, pmax, W.WM_ATTN_UNIT_SPLIT)
    units = pw.B * pw.Hkv
    assert 2 <= pu["unit_ctas"] <= 8 and pu["grid"] == units * pu["unit_ctas"]
    assert pu["warps"] == 4 * pu["grid"]  # d = 96, G = 2: 4 warps per CTA
    assert W.wm_decode_attn_plan(pc, 1, pmax, W.WM_ATTN_UNIT_SPLIT)["unit_ctas"] == 8
    with pytest.raises(W.WMError):
        W.wm_decode_attn_plan(c, w.B, max_pages, 8)  # unknown flag bit
    with pytest.raises(W.WMError):
        W.wm_decode_attn_plan(c, w.B, max_pages, W.WM_ATTN_DYNAMIC_SPLIT | W.WM_ATTN_UNIT_SPLIT)
    with pytest.raises(W.WMError):
        W.wm_decode_attn_plan(c, 0, max_pages)
