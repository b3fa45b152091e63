"""Device-memory owner around the C ABI, for Python callers.

PyTorch provides device memory and streams only: a DecodeSession allocates
the cache buffer, the two workspaces and the status word once, and forwards
each call to libwm through the ctypes binding.  Nothing here computes any
part of the decode path.
"""
from __future__ import annotations

import ctypes

import torch

from . import _lib as W


def torch_dtype(dtype: str):
    return {"f32": torch.float32, "bf16": torch.bfloat16}[dtype]


class DecodeSession:
    def __init__(self, cfg: W.wm_config, B: int, num_pages: int, max_pages: int,
                 device: str | torch.device = "cuda:0"):
        rc = W.wm_config_check(cfg)
        if rc != W.WM_OK:
            raise W.WMError(rc, "wm_config_check")
        self.cfg = cfg
        self.B, self.num_pages, self.max_pages = int(B), int(num_pages), int(max_pages)
        self.device = torch.device(device)
        self.dtype = torch.float32 if cfg.dtype == W.WM_DT_F32 else torch.bfloat16
        nbytes = W.wm_cache_bytes(cfg, num_pages)
        if nbytes == 0:
            raise W.WMError(W.WM_ERR_INVALID_ARG, "wm_cache_bytes")
        self.cache_buf = torch.empty(nbytes, dtype=torch.uint8, device=self.device)
        self.cache = W.wm_cache_alloc(cfg, self.cache_buf, nbytes, num_pages)
        shape = (cfg.k, num_pages, cfg.Hkv, cfg.page_size, cfg.d)
        esz = 4 if cfg.dtype == W.WM_DT_F32 else 2
        n = cfg.k * num_pages * cfg.Hkv * cfg.page_size * cfg.d
        koff = self.cache.k_pool - self.cache_buf.data_ptr()
        voff = self.cache.v_pool - self.cache_buf.data_ptr()
        self.k_pool = self.cache_buf[koff:koff + n * esz].view(self.dtype).view(shape)
        self.v_pool = self.cache_buf[voff:voff + n * esz].view(self.dtype).view(shape)
        self.mix_ws_bytes = W.wm_kv_mix_workspace(cfg, B)
        self.attn_ws_bytes = W.wm_decode_attn_workspace(cfg, B, max_pages)
        self.mix_ws = torch.empty(self.mix_ws_bytes, dtype=torch.uint8, device=self.device)
        # the attention workspace holds arrival tickets that must start at zero
        self.attn_ws = torch.zeros(self.attn_ws_bytes, dtype=torch.uint8, device=self.device)
        self.status = torch.zeros(1, dtype=torch.int32, device=self.device)
        self._weights = None
        self._weight_refs = None

    # ------------------------------------------------------------------ setup
    def set_weights(self, pre_g, Wr, br, ch_g, Wkv, qk_g) -> None:
        """Per-branch sequences (index 0 = K, 1 = V) of device tensors."""
        self._weight_refs = (pre_g, Wr, br, ch_g, Wkv, qk_g)
        self._weights = W.mix_weights(pre_g, Wr, br, ch_g, Wkv, qk_g)

    @staticmethod
    def _stream(stream) -> ctypes.c_void_p:
        s = torch.cuda.current_stream() if stream is None else stream
        return ctypes.c_void_p(s.cuda_stream)

    # ------------------------------------------------------------------ calls
    def decode_attn(self, layer: int, q, page_table, seq_lens, out, B: int | None = None,
                    stream=None, inputs_ready: bool = False, dynamic_split: bool = False,
                    unit_split: bool = False) -> None:
        """inputs_ready: the previous work on the stream wrote no cache, page
        table, lengths or workspace (true for layers 1..L-1 of a decode step).
        dynamic_split: chunks handed out by a device counter whatever the
        launch size (WM_ATTN_DYNAMIC_SPLIT).  unit_split: one cluster of CTAs
        per (sequence, kv head) unit whatever the launch size
        (WM_ATTN_UNIT_SPLIT)."""
        B = self.B if B is None else B
        flags = (W.WM_ATTN_INPUTS_READY if inputs_ready else 0) | \
            (W.WM_ATTN_DYNAMIC_SPLIT if dynamic_split else 0) | \
            (W.WM_ATTN_UNIT_SPLIT if unit_split else 0)
        rc = W.wm_decode_attn_flags(self.cfg, self.cache, layer, q, page_table, seq_lens, B,
                                    self.max_pages, out, self.attn_ws, self.attn_ws_bytes, flags,
                                    self.status, self._stream(stream))
        if rc != W.WM_OK:
            raise W.WMError(rc, "wm_decode_attn_flags")

    def prefill_attn(self, layer: int, q, pos, page_table, out, stream=None) -> None:
        """Causal attention of query rows q [B][Tq][Hq][d] at token positions
        pos [B][Tq] over layer ``layer``'s channel (prefill / parallel passes)."""
        B, Tq = int(q.shape[0]), int(q.shape[1])
        rc = W.wm_prefill_attn(self.cfg, self.cache, layer, q, pos, page_table, B, Tq,
                               self.max_pages, out, self.status, self._stream(stream))
        if rc != W.WM_OK:
            raise W.WMError(rc, "wm_prefill_attn")

    def kv_mix(self, h, page_table, slot, B: int | None = None, stream=None) -> None:
        if self._weights is None:
            raise RuntimeError("set_weights() first")
        B = self.B if B is None else B
        rc = W.wm_kv_mix(self.cfg, self.cache, self._weights, h, page_table, slot, B,
                         self.max_pages, self.mix_ws, self.mix_ws_bytes, self.status,
                         self._stream(stream))
        if rc != W.WM_OK:
            raise W.WMError(rc, "wm_kv_mix")

    def read_status(self, reset: bool = True) -> int:
        v = int(self.status.item())
        if reset:
            self.status.zero_()
        return v
