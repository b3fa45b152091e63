"""Decode attention on the dynamic split (Sec. 3.1 Step 3, dummy of Sec. 3.2),
every output row against the fp64 oracle.

Launches reading 2 GB of K/V or more cut the KV stream into about eight
chunks per warp and hand them out from a device counter; units crossing
chunk boundaries leave partial records that the piece completing the unit
merges.  Small launches take that path under WM_ATTN_DYNAMIC_SPLIT, so these
tests cover many chunk boundaries per unit on shapes the oracle checks in
full; whole full-size layers, where the path is taken by default, are
compared row by row in test_gpu_full_size.py.
"""
import numpy as np
import pytest
import torch

from paper_2608_18486_gb300 import _lib as W
from wm_synth import configs

from . import _harness as H

pytestmark = pytest.mark.gpu


def _free():
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def _run(sess, dp, layer, dynamic):
    w = dp.prob.w
    out = torch.full((w.B, w.Hq, w.d), float("nan"), dtype=sess.dtype, device=sess.device)
    sess.decode_attn(layer, dp.q[layer], dp.page_table, dp.seq_lens, out, dynamic_split=dynamic)
    return out


def _stages(w, lens):
    """Pipeline stages (8 KB of K+V, at most 32 slots) of all units of a launch."""
    row = 2 * w.d * w.elem_bytes
    slots = 1
    while slots * 2 * row <= 8192 and slots < 32:
        slots *= 2
    return w.Hkv * sum(-(-int(S) // slots) for S in lens)


RAGGED16 = [2048, 1, 33, 1500, 16, 17, 900, 2048, 2047, 1999, 64, 2048, 1024, 2048, 2000, 2048]


@pytest.mark.parametrize("name,overrides,lens,refill", [
    ("tiny_f32", dict(), None, False),                          # fewer chunks than warps
    ("no_compression", dict(), None, True),
    ("no_compression", dict(L=3, k=2, permute_pages=True), RAGGED16, True),
    ("paper_k16", dict(L=4, k=4), None, True),                  # GQA 6/3 heads of 96
    ("compress50", dict(B=8, L=2, k=2, Hq=64, Hkv=8),           # G = 8, ragged
     [4096, 3000, 129, 2, 4096, 4096, 4000, 3500], True),
])
def test_dynamic_split_every_row(name, overrides, lens, refill):
    w = configs.get(name).with_(**overrides)
    prob, sess, dp = H.setup(w, seq_lens=lens)
    plan = W.wm_decode_attn_plan(sess.cfg, w.B, prob.max_pages, W.WM_ATTN_DYNAMIC_SPLIT)
    assert plan["chunk_stages"] > 0, plan
    if refill:  # warps go back to the counter for further chunks
        assert _stages(w, prob.seq_lens) // plan["chunk_stages"] > plan["warps"], plan
    for layer in range(w.L):
        got = _run(sess, dp, layer, True)
        torch.cuda.synchronize()
        want = H.oracle_attn_full(prob, layer)
        err = H.rel_err(H.to_f64(got), want)
        assert err <= H.TOL[w.dtype], (layer, err)
        # the static split computes the same rows (another merge order)
        err_s = H.rel_err(H.to_f64(got), H.to_f64(_run(sess, dp, layer, False)))
        assert err_s <= H.TOL[w.dtype], (layer, err_s)
    assert sess.read_status() == 0
    _free()


def test_dynamic_split_repeated_launches_leave_no_stale_state():
    """Back-to-back dynamic launches on one workspace (the counter resets
    itself, tickets and flags are cleared by each merge) keep giving the
    oracle's rows, also when the batch shrinks between calls."""
    w = configs.get("no_compression").with_(L=2, k=2)
    prob, sess, dp = H.setup(w)
    want = H.oracle_attn_full(prob, 1)
    for B in (w.B, w.B, 5, w.B, 1):
        out = torch.full((B, w.Hq, w.d), float("nan"), dtype=sess.dtype, device=sess.device)
        sess.decode_attn(1, dp.q[1][:B], dp.page_table[:B], dp.seq_lens[:B], out, B=B,
                         dynamic_split=True)
        torch.cuda.synchronize()
        assert H.rel_err(H.to_f64(out), want[:B]) <= H.TOL[w.dtype], B
    assert sess.read_status() == 0
    _free()
