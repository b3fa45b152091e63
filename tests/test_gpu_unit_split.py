"""Decode attention on the unit split (Sec. 3.1 Step 3, dummy of Sec. 3.2),
every output row against the fp64 oracle.

The unit split gives each (sequence, kv head) unit one cluster of C CTAs
whose warps stream equal shares of the unit and merge on chip.  The planner
takes it by default for small launches whose units fill the SMs (the paper's
model shape); WM_ATTN_UNIT_SPLIT forces it on any launch, so these tests run
it on every cluster size from 1 to 8, ragged and empty units, GQA up to 8
query heads per kv head, fp32 and bf16, pages smaller and larger than a
pipeline stage, and the length and page-id edge cases.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2608_18486_gb300 import _lib as W
from wm_synth import configs

from . import _harness as H

pytestmark = pytest.mark.gpu

RAGGED16 = [2048, 1, 33, 1500, 16, 17, 900, 2048, 2047, 1999, 64, 2048, 1024, 2048, 2000, 2048]


def _free():
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def _run(sess, dp, layer, unit, B=None):
    w = dp.prob.w
    B = w.B if B is None else B
    out = torch.full((B, w.Hq, w.d), float("nan"), dtype=sess.dtype, device=sess.device)
    sess.decode_attn(layer, dp.q[layer][:B], dp.page_table[:B], dp.seq_lens[:B], out, B=B,
                     unit_split=unit)
    return out


def _plan(sess, w, prob, flags=W.WM_ATTN_UNIT_SPLIT):
    return W.wm_decode_attn_plan(sess.cfg, w.B, prob.max_pages, flags)


@pytest.mark.parametrize("name,overrides,lens,ctas", [
    ("tiny_f32", dict(), None, 8),                                   # 8 units: clusters of 8
    ("no_compression", dict(), None, 1),                             # 192 units > SMs: C = 1
    ("no_compression", dict(L=3, k=2, permute_pages=True), RAGGED16, 1),
    ("paper_k16", dict(L=4, k=4), None, 3),                          # 6/3 heads of 96
    ("paper_k16", dict(L=2, k=2, B=5), [2048, 7, 1, 1000, 2049], 8),
    ("paper_k16", dict(L=2, k=2, permute_pages=True), RAGGED16, 3),
    ("compress50", dict(B=8, L=2, k=2, Hq=64, Hkv=8),                # G = 8, 64 units
     [4096, 3000, 129, 2, 4096, 4096, 4000, 3500], 2),
])
def test_unit_split_every_row(name, overrides, lens, ctas):
    w = configs.get(name).with_(**overrides)
    prob, sess, dp = H.setup(w, seq_lens=lens)
    plan = _plan(sess, w, prob)
    assert plan["unit_ctas"] == ctas and plan["grid"] == w.B * w.Hkv * ctas, plan
    for layer in range(w.L):
        got = _run(sess, dp, layer, True)
        torch.cuda.synchronize()
        want = H.oracle_attn_full(prob, layer)
        err = H.rel_err(H.to_f64(got), want)
        assert err <= H.TOL[w.dtype], (layer, err)
        # stream-K computes the same rows (another merge order)
        err_s = H.rel_err(H.to_f64(got), H.to_f64(_run(sess, dp, layer, False)))
        assert err_s <= H.TOL[w.dtype], (layer, err_s)
    assert sess.read_status() == 0
    _free()


@pytest.mark.parametrize("dtype,d,G,page", [
    ("bf16", 128, 1, 16), ("bf16", 64, 2, 1), ("bf16", 128, 4, 8), ("f32", 128, 1, 64),
    ("f32", 64, 8, 32), ("bf16", 64, 1, 128), ("bf16", 96, 2, 256), ("f32", 96, 4, 4)])
def test_unit_split_shapes_pages_ragged(dtype, d, G, page):
    """10 units, clusters of 8 CTAs (64 warps per unit): short units leave
    most warps without a stage."""
    Hkv = 2
    w = configs.Workload("t", L=3, k=2, D=64, Hq=Hkv * G, Hkv=Hkv, d=d, B=5, ctx=700,
                         ctx_lo=1, page=page, dtype=dtype, chan_map="mod", permute_pages=True)
    prob, sess, dp = H.setup(w, seed=3, seq_lens=[1, 2, 127, 700, 333])
    assert _plan(sess, w, prob)["unit_ctas"] == 8
    for layer in range(w.L):
        got = H.to_f64(_run(sess, dp, layer, True))
        want = H.oracle_attn_full(prob, layer)
        assert H.rel_err(got, want) <= H.TOL[dtype], (layer, H.rel_err(got, want))
    assert sess.read_status() == 0
    _free()


@pytest.mark.parametrize("name", ["paper_k16", "no_compression"])
def test_unit_split_edge_cases(name):
    """Slots past the length never reach the output (NaN there changes no
    bit); dummy-only sequences return the dummy's value; a bad page id or
    length sets WM_ERR_BOUNDS, and a bad length zero-fills its rows."""
    w = configs.get(name).with_(B=4, L=1, k=1)
    lens = [37, 16, 1000, 1]
    prob, sess, dp = H.setup(w, seq_lens=lens)
    base = _run(sess, dp, 0, True).clone()
    torch.cuda.synchronize()
    assert H.rel_err(H.to_f64(base), H.oracle_attn_full(prob, 0)) <= H.TOL[w.dtype]
    pg = int(prob.page_table[3, 0])
    assert torch.equal(base[3], sess.v_pool[0, pg, :, 0, :].repeat_interleave(w.Hq // w.Hkv, 0))
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
    assert torch.equal(out[0], base[0]) and torch.equal(out[2], base[2])
    _free()


def test_default_plan_takes_the_unit_split_only_where_it_keeps_the_warps():
    """Launches below 2 GB, or of one sequence, whose units fit resident
    clusters with at least 60% of the static grid's warps take the unit
    split; launches with more units than that, and launches of 2 GB or more
    over several sequences, stream."""
    for name, over, unit in (("paper_k16", {}, True), ("paper_k1", {}, True),
                             ("tiny_f32", {}, True), ("no_compression", {}, True),
                             ("compress50", {}, False), ("large", {}, False),
                             ("long32k", {}, False), ("long128k", {}, False),
                             ("long128k", dict(B=1), True), ("long128k", dict(B=2), False)):
        w = configs.get(name).with_(**over)
        c = H.config_of(w)
        max_pages = -(-(w.ctx + 1) // w.page)
        plan = W.wm_decode_attn_plan(c, w.B, max_pages)
        assert (plan["unit_ctas"] >= 1) == unit, (name, plan)
        if unit:
            static = W.wm_decode_attn_plan(c, w.B, max_pages, W.WM_ATTN_DYNAMIC_SPLIT)
            assert plan["grid"] == w.B * w.Hkv * plan["unit_ctas"], (name, plan)
            assert plan["warps"] >= 0.6 * static["warps"], (name, plan, static)


def test_unit_split_chain_and_graph_replay_over_changing_lengths():
    """At the paper's shape (unit split by default): layers chained with
    WM_ATTN_INPUTS_READY give the bits of plain launches, and one captured
    launch replayed while the lengths change gives the oracle's rows."""
    w = configs.get("paper_k16").with_(L=3, k=3)
    prob, sess, dp = H.setup(w)
    assert _plan(sess, w, prob, 0)["unit_ctas"] >= 2
    ref = [H.run_attn(sess, dp, l).clone() for l in range(w.L)]
    outs = torch.empty((w.L, w.B, w.Hq, w.d), dtype=sess.dtype, device="cuda")
    for _ in range(2):
        for l in range(w.L):
            sess.decode_attn(l, dp.q[l], dp.page_table, dp.seq_lens, outs[l], inputs_ready=l > 0)
    torch.cuda.synchronize()
    for l in range(w.L):
        assert torch.equal(outs[l], ref[l]), l
    lens = dp.seq_lens.clone()
    out = torch.empty((w.B, w.Hq, w.d), dtype=sess.dtype, device=sess.device)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        sess.decode_attn(1, dp.q[1], dp.page_table, lens, out)
    rng = np.random.default_rng(5)
    full = np.asarray(prob.seq_lens, np.int64)
    for S in (full, np.maximum(1, full // 3), rng.integers(1, full + 1), full - 17, full):
        lens.copy_(torch.as_tensor(S, dtype=torch.int32))
        out.fill_(float("nan"))
        g.replay()
        torch.cuda.synchronize()
        want = O.decode_attn(prob.host("q")[1], prob.host("k_pool"), prob.host("v_pool"),
                             prob.page_table, S.astype(np.int32), chan=prob.chan[1], Hq=w.Hq,
                             Hkv=w.Hkv, d=w.d, P=w.page, nthreads=8)
        assert H.rel_err(H.to_f64(out), want) <= H.TOL[w.dtype], S[:4]
    assert sess.read_status() == 0
    del g
    _free()
