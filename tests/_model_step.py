"""A whole-model decode step around the library's path, for bench.py's model
mode and its parity test.

Random Qwen3-style decoder blocks (Sec. 4.1: RMSNorm, per-head QK-norm,
RoPE, SwiGLU MLP) in plain torch, with the library's decode attention in
place of each layer's attention and one pool after the stack (Sec. 3.2).  Per
layer l:  x = RMSNorm(h);  q = RoPE(RMSNorm_d(W_q x));  h += W_o attn_l(q);
h += W_d (silu(W_g x2) * (W_u x2)) with x2 = RMSNorm(h).  The states entering
the layers are stacked as H[b][l] for the pool.  The blocks are outside the
path; their weights and the step's input state come from the seeded input
generator, so a host reference can rebuild the whole step.
"""
from __future__ import annotations

import numpy as np
import torch
import torch.nn.functional as F

from wm_synth import device, gen

STREAM_WQ, STREAM_WO, STREAM_WG, STREAM_WU, STREAM_WD, STREAM_H0 = 50, 51, 52, 53, 54, 55


def block_specs(w, intermediate: int):
    """name -> (stream, shape, std) of the block weights and the input state."""
    I = intermediate
    return {"Wq": (STREAM_WQ, (w.L, w.Hq * w.d, w.D), w.D ** -0.5),
            "Wo": (STREAM_WO, (w.L, w.D, w.Hq * w.d), (w.Hq * w.d) ** -0.5),
            "Wg": (STREAM_WG, (w.L, I, w.D), w.D ** -0.5),
            "Wu": (STREAM_WU, (w.L, I, w.D), w.D ** -0.5),
            "Wd": (STREAM_WD, (w.L, w.D, I), I ** -0.5),
            "h0": (STREAM_H0, (w.B, w.D), 1.0)}


def host_block_tensor(w, seed: int, intermediate: int, name: str) -> np.ndarray:
    """The same tensor on the host, widened to float64."""
    stream, shape, std = block_specs(w, intermediate)[name]
    v = gen.values(w.dtype, seed, stream, 0, int(np.prod(shape)), float(np.float32(std)))
    return gen.to_f64(w.dtype, v).reshape(shape)


class ModelStep:
    def __init__(self, w, sess, dp, dev, intermediate: int = 0, seed: int = 0):
        self.w, self.sess, self.dp = w, sess, dp
        self.I = intermediate or 3 * w.D
        dt = sess.dtype
        self.t = {}
        for name, (stream, shape, std) in block_specs(w, self.I).items():
            t = torch.empty(shape, dtype=dt, device=dev)
            device.fill(t, w.dtype, seed, stream, float(np.float32(std)))
            self.t[name] = t
        # rotary angles of each sequence's new token (position seq_len - 1)
        pos = dp.seq_lens.to(torch.float64) - 1.0
        inv = w.rope_theta ** (-torch.arange(0, w.d // 2, device=dev, dtype=torch.float64) * 2.0 / w.d)
        ang = pos[:, None] * inv[None, :]
        self.cos = torch.cos(ang).float()[:, None, :]
        self.sin = torch.sin(ang).float()[:, None, :]
        self.H = torch.empty((w.B, w.L, w.D), dtype=dt, device=dev)
        self.q = torch.empty((w.L, w.B, w.Hq, w.d), dtype=dt, device=dev)
        self.out = torch.empty((w.L, w.B, w.Hq, w.d), dtype=dt, device=dev)

    @staticmethod
    def _rms(x, eps):
        xf = x.float()
        return xf * torch.rsqrt(xf.pow(2).mean(-1, keepdim=True) + eps)

    def step(self, stream, ev=None):
        """Enqueue one decode step on ``stream``; ev[l] = (start, end) events
        around layer l's attention (l < L) and the pool (l = L)."""
        w, sess, dp, t = self.w, self.sess, self.dp, self.t
        dt = sess.dtype
        h = t["h0"]
        for l in range(w.L):
            self.H[:, l] = h
            x = self._rms(h, w.eps_rms).to(dt)
            ql = self._rms((x @ t["Wq"][l].T).view(w.B, w.Hq, w.d), w.eps_qk)
            q1, q2 = ql[..., : w.d // 2], ql[..., w.d // 2:]
            self.q[l] = torch.cat([q1 * self.cos - q2 * self.sin, q2 * self.cos + q1 * self.sin],
                                  -1).to(dt)
            if ev is not None:
                ev[l][0].record(stream)
            # layer 0 follows the previous step's pool, which wrote the cache
            sess.decode_attn(l, self.q[l], dp.page_table, dp.seq_lens, self.out[l], stream=stream,
                             inputs_ready=l > 0)
            if ev is not None:
                ev[l][1].record(stream)
            h = h + self.out[l].view(w.B, -1) @ t["Wo"][l].T
            x2 = self._rms(h, w.eps_rms).to(dt)
            h = h + (F.silu(x2 @ t["Wg"][l].T) * (x2 @ t["Wu"][l].T)) @ t["Wd"][l].T
        if ev is not None:
            ev[w.L][0].record(stream)
        sess.kv_mix(self.H, dp.page_table, dp.slot, stream=stream)
        if ev is not None:
            ev[w.L][1].record(stream)
        return h
