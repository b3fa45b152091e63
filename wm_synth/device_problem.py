"""Put a seeded Problem on the device.

Small host-built tensors are copied; large spec'd tensors (pools, router and
projection weights, queries) are generated on the device by ``synth.cu`` from
the same counter-based streams the host uses, so that the oracle side can
regenerate any element without reading device memory.
"""
from __future__ import annotations

import numpy as np
import torch

from . import device
from .inputs import Problem


def _tdt(dtype: str):
    return torch.float32 if dtype == "f32" else torch.bfloat16


def host_to_device(arr: np.ndarray, dtype: str, dev) -> torch.Tensor:
    a = np.ascontiguousarray(arr)
    if dtype == "f32":
        return torch.from_numpy(a.astype(np.float32)).to(dev)
    return torch.from_numpy(a.view(np.int16)).to(dev).view(torch.bfloat16)


def spec_tensor(prob: Problem, name: str, dev) -> torch.Tensor:
    s = prob.specs[name]
    t = torch.empty(s.shape, dtype=_tdt(prob.w.dtype), device=dev)
    device.fill(t, prob.w.dtype, prob.seed, s.stream, s.std, s.mean)
    return t


class DeviceProblem:
    """Device tensors of one decode step; pools are filled in place."""

    def __init__(self, prob: Problem, k_pool: torch.Tensor, v_pool: torch.Tensor, dev="cuda:0",
                 fill_pools: bool = True):
        w = prob.w
        self.prob = prob
        if fill_pools:
            device.fill_spec(k_pool.view(-1), prob, "k_pool")
            device.fill_spec(v_pool.view(-1), prob, "v_pool")
        self.q = spec_tensor(prob, "q", dev)                      # [L][B][Hq][d]
        self.h = host_to_device(prob.host("h"), w.dtype, dev)     # [B][L][D]
        self.br = host_to_device(prob.host("br"), w.dtype, dev)   # [2][kL]
        self.pre_g = spec_tensor(prob, "pre_g", dev)
        self.ch_g = spec_tensor(prob, "ch_g", dev)
        self.qk_g = spec_tensor(prob, "qk_g", dev)
        self.Wr = spec_tensor(prob, "Wr", dev)
        self.Wkv = spec_tensor(prob, "Wkv", dev)
        self.page_table = torch.from_numpy(prob.page_table).to(dev)
        self.seq_lens = torch.from_numpy(prob.seq_lens).to(dev)
        # the new token of sequence b is written at slot seq_lens[b]
        self.slot = self.seq_lens.clone()

    def weights(self):
        return ((self.pre_g[0], self.pre_g[1]), (self.Wr[0], self.Wr[1]),
                (self.br[0], self.br[1]), (self.ch_g[0], self.ch_g[1]),
                (self.Wkv[0], self.Wkv[1]), self.qk_g)
