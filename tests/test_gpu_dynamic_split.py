"""Decode attention on the stream-K kernel's splits (Sec. 3.1 Step 3, dummy of
Sec. 3.2), every output row against the fp64 oracle.

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


def test_static_split_of_many_short_units_every_row():
    """More units than resident unit-split clusters (768 units of up to 512
    tokens, 50 MB): the default plan streams with the static split, one chunk
    per warp, units crossing chunk ends merged from partial records."""
    w = configs.get("no_compression").with_(B=64, L=2, k=2, ctx=512, ctx_lo=1, permute_pages=True)
    prob, sess, dp = H.setup(w)
    plan = W.wm_decode_attn_plan(sess.cfg, w.B, prob.max_pages)
    assert plan["unit_ctas"] == 0 and plan["chunk_stages"] == 0, plan
    for layer in range(w.L):
        got = _run(sess, dp, layer, False)
        torch.cuda.synchronize()
        err = H.rel_err(H.to_f64(got), H.oracle_attn_full(prob, layer))
        assert err <= H.TOL[w.dtype], (layer, err)
    assert sess.read_status() == 0
    _free()


def test_stream_k_edge_cases():
    """On the counter-driven split: slots past the length never reach the
    output, a dummy-only sequence returns the dummy's value, a bad page id or
    length sets WM_ERR_BOUNDS and a bad length zero-fills its rows."""
    w = configs.get("no_compression").with_(B=4, L=1, k=1)
    lens = [37, 16, 1000, 1]
    prob, sess, dp = H.setup(w, seq_lens=lens)
    base = _run(sess, dp, 0, True).clone()
    torch.cuda.synchronize()
    assert H.rel_err(H.to_f64(base), H.oracle_attn_full(prob, 0)) <= H.TOL[w.dtype]
    pg = int(prob.page_table[3, 0])
    assert torch.equal(base[3], sess.v_pool[0, pg, :, 0, :])
    for b, S in enumerate(lens):
        for i in range(int((prob.page_table[b] >= 0).sum())):
            lo = max(0, S - i * w.page)
            if lo < w.page:
                p = int(prob.page_table[b, i])
                sess.k_pool[:, p, :, lo:, :] = float("nan")
                sess.v_pool[:, p, :, lo:, :] = float("nan")
    assert torch.equal(_run(sess, dp, 0, True), base)
    assert sess.read_status() == 0
    dp.page_table[2, 3] = prob.num_pages + 5
    _run(sess, dp, 0, True)
    torch.cuda.synchronize()
    assert sess.read_status() == 4  # WM_ERR_BOUNDS
    dp.page_table[2, 3] = int(prob.page_table[2, 3])
    dp.seq_lens[1] = 0
    out = _run(sess, dp, 0, True)
    torch.cuda.synchronize()
    assert sess.read_status() == 4
    assert torch.count_nonzero(out[1].float()) == 0
    _free()
