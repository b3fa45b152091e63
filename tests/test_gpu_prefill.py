"""Causal prefill channel attention on the GPU (wm_prefill_attn) against the
fp64 oracle: Jacobi passes (every position) and cyclic Gauss-Seidel groups
(positions i mod g = q) of Sec. 3.3, with the dummy offset of Sec. 3.2."""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2608_18486_gb300 import _lib as W
from wm_synth import configs
from wm_synth.device_problem import host_to_device
from wm_synth.inputs import group_positions, prefill_queries

from . import _harness as H

pytestmark = pytest.mark.gpu


def _free():
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def _workload(d, G, page, T, B=2, Hkv=2, L=2, k=2, permute=True):
    return configs.Workload("prefill", L=L, k=k, D=64, Hq=Hkv * G, Hkv=Hkv, d=d, B=B, ctx=T,
                            page=page, dtype="bf16", chan_map="mod", permute_pages=permute)


def _run(sess, q_bits, pos, dp, layer):
    """One call: queries [B][Tq][Hq][d] (bf16 bits) at positions [B][Tq]."""
    dev = sess.device
    q = host_to_device(q_bits, "bf16", dev)
    pos_t = torch.from_numpy(np.ascontiguousarray(pos, dtype=np.int32)).to(dev)
    out = torch.full(q.shape, float("nan"), dtype=torch.bfloat16, device=dev)
    sess.prefill_attn(layer, q, pos_t, dp.page_table, out)
    torch.cuda.synchronize()
    return out


def _oracle(prob, q_bits, pos, layer, units=None):
    w = prob.w
    return O.prefill_attn(q_bits, prob.host("k_pool"), prob.host("v_pool"), prob.page_table, pos,
                          chan=prob.chan[layer], Hq=w.Hq, Hkv=w.Hkv, d=w.d, P=w.page,
                          units=units, nthreads=8)


def _oracle_units(prob, q_bits, pos, layer, units):
    """Sampled (b, r, hq) rows, each from only the pages its position reads."""
    w = prob.w
    chan = prob.chan[layer]
    e = np.arange(w.d, dtype=np.int64)
    s = np.arange(w.page, dtype=np.int64)
    res = []
    for b, r, hq in units:
        hkv = hq // (w.Hq // w.Hkv)
        i = int(pos[b, r])
        npg = i // w.page + 1
        pages = prob.page_table[b, :npg].astype(np.int64)
        base = ((chan * prob.num_pages + pages) * w.Hkv + hkv) * w.page
        idx = ((base[:, None] + s[None, :]) * w.d)[:, :, None] + e[None, None, :]
        kp = prob.at("k_pool", idx.reshape(-1)).reshape(1, npg, 1, w.page, w.d)
        vp = prob.at("v_pool", idx.reshape(-1)).reshape(1, npg, 1, w.page, w.d)
        pt = np.arange(npg, dtype=np.int32).reshape(1, npg)
        qr = np.ascontiguousarray(q_bits[b, r, hq]).reshape(1, 1, 1, w.d)
        res.append(O.prefill_attn(qr, kp, vp, pt, np.array([[i]], np.int32), chan=0, Hq=1,
                                  Hkv=1, d=w.d, P=w.page)[0, 0, 0])
    return np.stack(res)


@pytest.mark.parametrize("d,G,page,g", [
    (64, 1, 16, 1), (96, 2, 8, 8), (128, 1, 64, 8), (64, 4, 256, 3), (128, 2, 16, 1),
    (96, 1, 128, 2)])
def test_prefill_groups_match_oracle(d, G, page, g):
    T = 300  # three 128-row tiles, the last one ragged
    w = _workload(d, G, page, T)
    prob, sess, dp = H.setup(w, seed=5, seq_lens=[T, T])
    for layer in range(w.L):
        for q in sorted({0, g - 1}):
            pos = np.stack([group_positions(T, g, q)] * w.B)
            q_bits = prefill_queries(w, 11 + q + 7 * layer, w.B, pos.shape[1])
            got = H.to_f64(_run(sess, q_bits, pos, dp, layer))
            want = _oracle(prob, q_bits, pos, layer)
            err = H.rel_err(got, want)
            assert err <= H.TOL["bf16"], (layer, q, err)
    assert sess.read_status() == 0
    _free()


def test_prefill_rows_in_any_order_and_ragged_sequences():
    w = _workload(128, 1, 16, 700, B=3)
    lens = [700, 129, 1]
    prob, sess, dp = H.setup(w, seed=6, seq_lens=lens)
    rng = np.random.default_rng(0)
    Tq = 200
    pos = np.stack([rng.integers(0, S, Tq) for S in lens]).astype(np.int32)
    q_bits = prefill_queries(w, 21, w.B, Tq)
    got = H.to_f64(_run(sess, q_bits, pos, dp, 1))
    want = _oracle(prob, q_bits, pos, 1)
    assert H.rel_err(got, want) <= H.TOL["bf16"]
    assert sess.read_status() == 0
    _free()


def test_prefill_never_reads_slots_past_the_largest_position():
    """Slots past every query's position may hold anything: NaN there changes
    no bit of the output."""
    T, page = 250, 16
    w = _workload(64, 2, page, T)
    prob, sess, dp = H.setup(w, seed=7, seq_lens=[T, T])
    pos = np.stack([group_positions(T, 1, 0)] * w.B)
    q_bits = prefill_queries(w, 31, w.B, T)
    base = _run(sess, q_bits, pos, dp, 0)
    for b in range(w.B):
        for s in range(T, int(prob.page_table.shape[1]) * page):
            pg = int(prob.page_table[b, s // page])
            if pg >= 0:
                sess.k_pool[:, pg, :, s % page] = float("nan")
                sess.v_pool[:, pg, :, s % page] = float("nan")
    poisoned = _run(sess, q_bits, pos, dp, 0)
    assert torch.equal(base, poisoned)
    assert sess.read_status() == 0
    _free()


def test_prefill_page_permutation_is_bit_exact():
    T = 400
    w = _workload(128, 1, 16, T, B=2)
    pa, sa, da = H.setup(w.with_(permute_pages=False), seed=8, seq_lens=[T, T])
    pb, sb, db = H.setup(w.with_(permute_pages=True), seed=8, seq_lens=[T, T])
    for b in range(w.B):
        for i in range(pa.page_table.shape[1]):
            if pa.page_table[b, i] >= 0:
                sb.k_pool[:, pb.page_table[b, i]] = sa.k_pool[:, pa.page_table[b, i]]
                sb.v_pool[:, pb.page_table[b, i]] = sa.v_pool[:, pa.page_table[b, i]]
    pos = np.stack([group_positions(T, 8, 5)] * w.B)
    q_bits = prefill_queries(w, 41, w.B, pos.shape[1])
    assert torch.equal(_run(sa, q_bits, pos, da, 1), _run(sb, q_bits, pos, db, 1))
    _free()


def test_prefill_row_equals_decode_of_the_same_token():
    """Sec. 3.2: the token at position i decodes with i + 1 slots."""
    T = 260
    w = _workload(96, 2, 16, T, B=2)
    prob, sess, dp = H.setup(w, seed=9, seq_lens=[T, T])
    pos = np.array([[0, 127, 128, 259], [1, 200, 255, 64]], dtype=np.int32)
    q_bits = prefill_queries(w, 51, w.B, pos.shape[1])
    pre = _run(sess, q_bits, pos, dp, 0)
    for r in range(pos.shape[1]):
        qd = host_to_device(np.ascontiguousarray(q_bits[:, r]), "bf16", sess.device)
        lens = torch.from_numpy(pos[:, r] + 1).to(sess.device)
        out = torch.empty_like(qd)
        sess.decode_attn(0, qd, dp.page_table, lens, out)
        err = H.rel_err(H.to_f64(pre[:, r]), H.to_f64(out))
        assert err <= H.TOL["bf16"], (r, err)
    assert sess.read_status() == 0
    _free()


def test_prefill_bad_position_zero_row_and_status():
    T = 140
    w = _workload(64, 1, 16, T, B=2)
    prob, sess, dp = H.setup(w, seed=10, seq_lens=[T, T])
    pos = np.stack([group_positions(T, 1, 0)] * w.B)
    pos[1, 7] = prob.page_table.shape[1] * w.page  # one past the table
    pos[0, 3] = -1
    q_bits = prefill_queries(w, 61, w.B, T)
    got = _run(sess, q_bits, pos, dp, 0)
    assert sess.read_status() == W.WM_ERR_BOUNDS
    assert torch.all(got[1, 7] == 0) and torch.all(got[0, 3] == 0)
    ok = np.ones((w.B, T), bool)
    ok[1, 7] = ok[0, 3] = False
    units = [(b, r, h) for b in range(w.B) for r in range(T) for h in range(w.Hq) if ok[b, r]]
    want = _oracle(prob, q_bits, np.where(ok, pos, 0), 0, units=units)
    gotv = np.stack([H.to_f64(got[b, r, h]) for b, r, h in units])
    assert H.rel_err(gotv, want) <= H.TOL["bf16"]
    _free()


@pytest.mark.parametrize("name,T,g,q,rows", [
    ("paper_k8", 2048, 8, 3, None),       # the paper's shape, one Gauss-Seidel group
    ("large", 8192, 1, 0, 48),            # 32 heads of 128, a Jacobi pass over 8192 tokens
])
def test_prefill_full_size_sampled(name, T, g, q, rows):
    w = configs.get(name).with_(B=2, ctx=T, ctx_lo=0, L=2, k=2)
    prob, sess, dp = H.setup(w, seed=0, seq_lens=[T, T])
    pos = np.stack([group_positions(T, g, q)] * w.B)
    q_bits = prefill_queries(w, 71, w.B, pos.shape[1])
    got = _run(sess, q_bits, pos, dp, 1)
    rng = np.random.default_rng(1)
    if rows is None:
        units = None
        gotv = H.to_f64(got)
    else:
        rr = np.concatenate([[0, pos.shape[1] - 1], rng.integers(0, pos.shape[1], rows - 2)])
        units = [(int(rng.integers(w.B)), int(r), int(rng.integers(w.Hq))) for r in rr]
        gotv = np.stack([H.to_f64(got[b, r, h]) for b, r, h in units])
    want = _oracle(prob, q_bits, pos, 1) if units is None else \
        _oracle_units(prob, q_bits, pos, 1, units)
    assert H.rel_err(gotv, want) <= H.TOL["bf16"]
    assert sess.read_status() == 0
    del sess, dp
    _free()
