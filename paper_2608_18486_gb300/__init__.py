"""WhiteMatter decode hot path on GB300: Python binding of libwm.

``_lib`` mirrors the C ABI of include/wm.h entry point by entry point;
``session.DecodeSession`` owns the device memory a caller needs.  All
computation of the path runs in the CUDA kernels of libwm.so.
"""
from . import _lib  # noqa: F401
from ._lib import (WMError, make_config, wm_cache_alloc, wm_cache_bytes, wm_config_check,  # noqa: F401
                   wm_decode_attn, wm_decode_attn_workspace, wm_kv_mix, wm_kv_mix_workspace,
                   wm_status_string)
