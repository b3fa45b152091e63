"""Synthetic decode workloads shaped like the ones the method is measured on.

Each workload fixes the model shape (L layers, k KV channels, width D, heads,
head dim), the decode batch, the cache context, the page size, the storage
dtype and the layer-to-channel map.  ``ctx`` counts cache slots per sequence
*including* the dummy slot 0, so a sequence holds ``ctx - 1`` past tokens and
the next token's KV is written to slot ``ctx``.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, replace


@dataclass(frozen=True)
class Workload:
    name: str
    L: int
    k: int
    D: int
    Hq: int
    Hkv: int
    d: int
    B: int
    ctx: int                 # slots per sequence incl. dummy (upper bound if ragged)
    page: int
    dtype: str               # "f32" or "bf16"
    chan_map: str            # "block": floor(l*k/L); "mod": l mod k
    ctx_lo: int = 0          # >0: ragged, lengths uniform in [ctx_lo, ctx]
    permute_pages: bool = False
    layer_rms_scale: bool = False   # h_l scaled by (1 + 0.1 l)
    p: int = 2               # router reads every p-th layer
    eps_rms: float = 1e-6
    eps_qk: float = 1e-6
    rope_theta: float = 1e6
    gain_std: float = 0.0    # 0: unit gains; >0: gains ~ N(1, gain_std^2)
    q_scale: float = 1.0     # 8.0 gives peaked attention

    @property
    def Lp(self) -> int:
        return -(-self.L // self.p)

    def chan_of_layer(self) -> list[int]:
        if self.chan_map == "block":
            return [(l * self.k) // self.L for l in range(self.L)]
        if self.chan_map == "mod":
            return [l % self.k for l in range(self.L)]
        raise ValueError(self.chan_map)

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)

    @property
    def elem_bytes(self) -> int:
        return 4 if self.dtype == "f32" else 2


WORKLOADS: dict[str, Workload] = {
    # L=4, k=2, c(l)=floor(l*k/L), D=256, 4 heads x 64, batch 2, context 128, fp32
    "tiny_f32": Workload("tiny_f32", L=4, k=2, D=256, Hq=4, Hkv=4, d=64, B=2,
                         ctx=128, page=16, dtype="f32", chan_map="block"),
    # L=12, k=12, D=768, 12 x 64, batch 16, context 2048, page 16, layer RMS 1+0.1l
    "no_compression": Workload("no_compression", L=12, k=12, D=768, Hq=12, Hkv=12,
                               d=64, B=16, ctx=2048, page=16, dtype="bf16",
                               chan_map="mod", layer_rms_scale=True),
    # L=24, k=12, c(l)=floor(l/2), D=1024, 16 x 64, batch 64, context 4096, permuted
    "compress50": Workload("compress50", L=24, k=12, D=1024, Hq=16, Hkv=16, d=64,
                           B=64, ctx=4096, page=16, dtype="bf16", chan_map="block",
                           permute_pages=True),
    # L=32, k=16, D=4096, 32 x 128, batch 32, ragged context U[4096, 8192], permuted
    "large": Workload("large", L=32, k=16, D=4096, Hq=32, Hkv=32, d=128, B=32,
                      ctx=8192, ctx_lo=4096, page=16, dtype="bf16", chan_map="mod",
                      permute_pages=True),
    # L=32, k=8, D=4096, 32 x 128, batch 8, page 64, context 32k / 64k / 128k
    "long32k": Workload("long32k", L=32, k=8, D=4096, Hq=32, Hkv=32, d=128, B=8,
                        ctx=32768, page=64, dtype="bf16", chan_map="mod",
                        permute_pages=True),
    "long64k": Workload("long64k", L=32, k=8, D=4096, Hq=32, Hkv=32, d=128, B=8,
                        ctx=65536, page=64, dtype="bf16", chan_map="mod",
                        permute_pages=True),
    "long128k": Workload("long128k", L=32, k=8, D=4096, Hq=32, Hkv=32, d=128, B=8,
                         ctx=131072, page=64, dtype="bf16", chan_map="mod",
                         permute_pages=True),
    # the paper's own model shape (Sec. 4.1): Qwen3 D=512, 6 query / 3 kv heads
    # of dimension 96, L=16; k=16 (full cache), k=8 (half cache) and k=1.
    # Decode batch 16 at the training length 2048 (the paper fixes no decode batch).
    "paper_k16": Workload("paper_k16", L=16, k=16, D=512, Hq=6, Hkv=3, d=96, B=16, ctx=2048,
                          page=16, dtype="bf16", chan_map="mod"),
    "paper_k8": Workload("paper_k8", L=16, k=8, D=512, Hq=6, Hkv=3, d=96, B=16, ctx=2048,
                         page=16, dtype="bf16", chan_map="mod"),
    "paper_k1": Workload("paper_k1", L=16, k=1, D=512, Hq=6, Hkv=3, d=96, B=16, ctx=2048,
                         page=16, dtype="bf16", chan_map="mod"),
}


def get(name: str) -> Workload:
    return WORKLOADS[name]


def kv_bytes_per_layer(w: Workload, seq_lens) -> int:
    """Bytes of K and V one decode-attention launch must read."""
    return int(sum(seq_lens)) * w.Hkv * w.d * 2 * w.elem_bytes


def attn_launch_bytes(w: Workload, seq_lens) -> int:
    """Algorithmic bytes of one attention launch: KV read + q read + out write."""
    qo = 2 * w.B * w.Hq * w.d * w.elem_bytes
    return kv_bytes_per_layer(w, seq_lens) + qo


def mix_bytes(w: Workload) -> int:
    """Algorithmic bytes of one pool evaluation (B tokens)."""
    e = w.elem_bytes
    h = w.B * w.L * w.D * e
    router = 2 * (w.k * w.L * w.Lp * w.D + w.k * w.L) * e
    proj = 2 * w.k * w.Hkv * w.d * w.D * e
    gains = (2 * w.D + 2 * w.k * w.D + w.k * w.d) * e
    write = w.B * w.k * 2 * w.Hkv * w.d * e
    return h + router + proj + gains + write


def step_bytes(w: Workload, seq_lens) -> int:
    return w.L * attn_launch_bytes(w, seq_lens) + mix_bytes(w)


def pages_for(slots: int, page: int) -> int:
    return int(math.ceil(slots / page))
