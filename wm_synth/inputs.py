"""Seeded synthetic inputs of one decode step.

Every tensor is a pure function of ``(workload, seed)``: small tensors are
built here on the host; large ones (the KV pools, the router and projection
weights) are described by a :class:`TensorSpec` so that the GPU side can fill
them on the device (``synth.cu``) and the oracle side can regenerate any
element on the host, bit for bit, from the same counter-based stream.

The KV pools are filled in flat-index order; the element at flat index ``i``
of the K (or V) pool buffer is ``values(stream, i)``, whatever layout the
consumer gives those bytes.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

from . import gen
from .configs import Workload, pages_for

STREAM_H = 1
STREAM_PRE_G = 2
STREAM_CH_G = 4
STREAM_QK_G = 6
STREAM_WR = 10
STREAM_WKV = 20
STREAM_KPOOL = 30
STREAM_VPOOL = 31
STREAM_Q = 40
STREAM_Q_PREFILL = 41


@dataclass(frozen=True)
class TensorSpec:
    stream: int
    shape: tuple
    std: float
    mean: float = 0.0

    @property
    def count(self) -> int:
        return int(np.prod(self.shape))


@dataclass
class Problem:
    w: Workload
    seed: int
    seq_lens: np.ndarray          # int32 [B]: slots incl. dummy = the write slot
    page_table: np.ndarray        # int32 [B][max_pages], -1 where unused
    num_pages: int
    max_pages: int
    chan: list                    # channel read by each layer
    specs: dict = field(default_factory=dict)
    _cache: dict = field(default_factory=dict)

    # ------------------------------------------------------------------ specs
    def host(self, name: str) -> np.ndarray:
        """Full tensor in storage dtype (fp32 array or bf16 uint16 bits)."""
        if name in self._cache:
            return self._cache[name]
        if name == "h":
            a = self._hidden()
        elif name == "br":
            a = self._router_bias()
        else:
            s = self.specs[name]
            a = gen.values(self.w.dtype, self.seed, s.stream, 0, s.count, s.std,
                           s.mean).reshape(s.shape)
        self._cache[name] = a
        return a

    def at(self, name: str, index: np.ndarray) -> np.ndarray:
        """Elements of a spec'd tensor at flat indices (storage dtype)."""
        s = self.specs[name]
        return gen.values_at(self.w.dtype, self.seed, s.stream, index, s.std, s.mean)

    def rows(self, name: str, row0: int, nrows: int, row_len: int) -> np.ndarray:
        s = self.specs[name]
        return gen.values(self.w.dtype, self.seed, s.stream, row0 * row_len,
                          nrows * row_len, s.std, s.mean).reshape(nrows, row_len)

    # ------------------------------------------------------------- builders
    def _hidden(self) -> np.ndarray:
        w = self.w
        out = np.empty((w.B, w.L, w.D), dtype=np.float32 if w.dtype == "f32" else np.uint16)
        base = (np.arange(w.B, dtype=np.uint64)[:, None] * np.uint64(w.L * w.D)
                + np.arange(w.D, dtype=np.uint64)[None, :])
        for l in range(w.L):
            std = (1.0 + 0.1 * l) if w.layer_rms_scale else 1.0
            idx = base + np.uint64(l * w.D)
            out[:, l, :] = gen.values_at(w.dtype, self.seed, STREAM_H, idx, std)
        return out

    def _router_bias(self) -> np.ndarray:
        """Bias pattern of the router initialisation (Sec. 3.1, "Router
        initialization"): top for k=1, shifted identity for k=L, otherwise
        source layer l -> channel c(l).  Same pattern for both branches."""
        w = self.w
        b = np.zeros((w.k, w.L), dtype=np.float32)
        if w.k == 1:
            b[0, w.L - 1] = 1.0
        elif w.k == w.L:
            for j in range(w.k):
                b[j, min(j + 1, w.L - 1)] = 1.0
        else:
            for l, c in enumerate(self.chan):
                b[c, l] = 1.0
        b2 = np.stack([b.reshape(-1), b.reshape(-1)])
        return b2 if w.dtype == "f32" else gen.f32_to_bf16_bits(b2)

    def pool_elems(self) -> int:
        w = self.w
        return w.k * self.num_pages * w.Hkv * w.page * w.d


def make_problem(w: Workload, seed: int = 0, seq_lens=None) -> Problem:
    rng = np.random.Generator(np.random.PCG64(seed))
    if seq_lens is None:
        if w.ctx_lo > 0:
            seq_lens = rng.integers(w.ctx_lo, w.ctx + 1, size=w.B)
        else:
            seq_lens = np.full(w.B, w.ctx)
    seq_lens = np.asarray(seq_lens, dtype=np.int32)
    # pages hold slots 0..S_b inclusive (slot S_b receives the new token's KV)
    npg = np.array([pages_for(int(s) + 1, w.page) for s in seq_lens], dtype=np.int64)
    max_pages = int(npg.max()) if len(npg) else 1
    num_pages = int(npg.sum())
    phys = np.arange(num_pages, dtype=np.int32)
    if w.permute_pages:
        phys = rng.permutation(num_pages).astype(np.int32)
    pt = np.full((w.B, max_pages), -1, dtype=np.int32)
    o = 0
    for b in range(w.B):
        pt[b, :npg[b]] = phys[o:o + npg[b]]
        o += npg[b]
    chan = w.chan_of_layer()
    prob = Problem(w=w, seed=seed, seq_lens=seq_lens, page_table=pt,
                   num_pages=num_pages, max_pages=max_pages, chan=chan)
    g_std, g_mean = w.gain_std, 1.0
    pool_shape = (w.k, num_pages, w.Hkv, w.page, w.d)
    prob.specs = {
        "pre_g": TensorSpec(STREAM_PRE_G, (2, w.D), g_std, g_mean),
        "ch_g": TensorSpec(STREAM_CH_G, (2, w.k, w.D), g_std, g_mean),
        "qk_g": TensorSpec(STREAM_QK_G, (w.k, w.d), g_std, g_mean),
        "Wr": TensorSpec(STREAM_WR, (2, w.k * w.L, w.Lp * w.D), 1.0 / np.sqrt(w.Lp * w.D)),
        "Wkv": TensorSpec(STREAM_WKV, (2, w.k, w.Hkv * w.d, w.D), 1.0 / np.sqrt(w.D)),
        "k_pool": TensorSpec(STREAM_KPOOL, pool_shape, 1.0),
        "v_pool": TensorSpec(STREAM_VPOOL, pool_shape, 1.0),
        "q": TensorSpec(STREAM_Q, (w.L, w.B, w.Hq, w.d), w.q_scale),
    }
    return prob


def prefill_queries(w: Workload, seed: int, B: int, Tq: int) -> np.ndarray:
    """Query rows [B][Tq][Hq][d] of one prefill pass, stored in ``w.dtype``
    (same distribution as the decode queries)."""
    n = B * Tq * w.Hq * w.d
    return gen.values(w.dtype, seed, STREAM_Q_PREFILL, 0, n, w.q_scale).reshape(B, Tq, w.Hq, w.d)


def group_positions(T: int, g: int, q: int) -> np.ndarray:
    """Token positions of strided group q of g over a T-token prefill:
    {i : 0 <= i < T, i mod g = q} in increasing order (g = 1: all of them)."""
    return np.arange(q, T, g, dtype=np.int32)
