"""Oracle side of the GPU tests and of bench.py's CPU legs: the fp64 oracle
fed with inputs regenerated on the host from the seeded streams.

Imports only the oracle and the input generator, never the product library,
so the CPU baseline and the reference arm run none of the GPU path.
"""
from __future__ import annotations

import numpy as np

from oracle import oracle as O
from wm_synth import gen


def oracle_attn_full(prob, layer, nthreads=8) -> np.ndarray:
    w = prob.w
    return O.decode_attn(prob.host("q")[layer], prob.host("k_pool"), prob.host("v_pool"),
                         prob.page_table, prob.seq_lens, chan=prob.chan[layer], Hq=w.Hq,
                         Hkv=w.Hkv, d=w.d, P=w.page, nthreads=nthreads)


def oracle_attn_unit(prob, layer, b, hq) -> np.ndarray:
    """One (sequence, query head) of one layer, from only that sequence's pages."""
    w = prob.w
    hkv = hq // (w.Hq // w.Hkv)
    chan = prob.chan[layer]
    S = int(prob.seq_lens[b])
    npg = -(-S // w.page)
    pages = prob.page_table[b, :npg].astype(np.int64)
    s = np.arange(w.page, dtype=np.int64)
    e = np.arange(w.d, dtype=np.int64)
    # flat index of (chan, page, hkv, s, e) in the pool layout
    base = ((chan * prob.num_pages + pages) * w.Hkv + hkv) * w.page
    idx = ((base[:, None] + s[None, :]) * w.d)[:, :, None] + e[None, None, :]
    kp = prob.at("k_pool", idx.reshape(-1)).reshape(1, npg, 1, w.page, w.d)
    vp = prob.at("v_pool", idx.reshape(-1)).reshape(1, npg, 1, w.page, w.d)
    qi = ((layer * w.B + b) * w.Hq + hq) * w.d + e
    q = prob.at("q", qi).reshape(1, 1, w.d)
    pt = np.arange(npg, dtype=np.int32).reshape(1, npg)
    return O.decode_attn(q, kp, vp, pt, [S], chan=0, Hq=1, Hkv=1, d=w.d, P=w.page)[0, 0]


def oracle_attn_layer(prob, layer, seqs=None, nthreads=None) -> np.ndarray:
    """Every (sequence, query head) row of one layer: out[B][Hq][d] (rows of
    sequences not in ``seqs`` stay zero).  Each sequence's pages of channel
    c(layer) are regenerated on the host one sequence at a time, so host
    memory stays at one sequence's K and V even for the longest contexts."""
    import os
    w = prob.w
    chan = prob.chan[layer]
    nthreads = nthreads or len(os.sched_getaffinity(0))
    run = w.Hkv * w.page * w.d  # one page of one channel: all kv heads, contiguous
    q = prob.at("q", (layer * w.B * w.Hq * w.d + np.arange(w.B * w.Hq * w.d)).astype(np.uint64))
    q = q.reshape(w.B, w.Hq, w.d)
    ks, vs = prob.specs["k_pool"], prob.specs["v_pool"]
    out = np.zeros((w.B, w.Hq, w.d))
    for b in (range(w.B) if seqs is None else seqs):
        S = int(prob.seq_lens[b])
        npg = -(-S // w.page)
        pages = prob.page_table[b, :npg].astype(np.uint64)
        starts = (np.uint64(chan * prob.num_pages) + pages) * np.uint64(run)
        kp = gen.values_runs(w.dtype, prob.seed, ks.stream, starts, run, ks.std, ks.mean)
        vp = gen.values_runs(w.dtype, prob.seed, vs.stream, starts, run, vs.std, vs.mean)
        shape = (1, npg, w.Hkv, w.page, w.d)
        pt = np.arange(npg, dtype=np.int32).reshape(1, npg)
        out[b] = O.decode_attn(q[b:b + 1], kp.reshape(shape), vp.reshape(shape), pt, [S], chan=0,
                               Hq=w.Hq, Hkv=w.Hkv, d=w.d, P=w.page, nthreads=nthreads)[0]
        del kp, vp
    return out


def oracle_prefill_unit(prob, layer, b, pos, q_row) -> np.ndarray:
    """Causal prefill attention of one query row (token position ``pos`` of
    sequence b, query head given by ``q_row``'s head index), from only the
    pages it reads.  ``q_row`` is (hq, d storage-dtype values)."""
    w = prob.w
    hq, qv = q_row
    hkv = hq // (w.Hq // w.Hkv)
    chan = prob.chan[layer]
    npg = pos // w.page + 1
    pages = prob.page_table[b, :npg].astype(np.int64)
    s = np.arange(w.page, dtype=np.int64)
    e = np.arange(w.d, dtype=np.int64)
    base = ((chan * prob.num_pages + pages) * w.Hkv + hkv) * w.page
    idx = ((base[:, None] + s[None, :]) * w.d)[:, :, None] + e[None, None, :]
    kp = prob.at("k_pool", idx.reshape(-1)).reshape(1, npg, 1, w.page, w.d)
    vp = prob.at("v_pool", idx.reshape(-1)).reshape(1, npg, 1, w.page, w.d)
    pt = np.arange(npg, dtype=np.int32).reshape(1, npg)
    q = np.ascontiguousarray(qv).reshape(1, 1, 1, w.d)
    return O.prefill_attn(q, kp, vp, pt, np.array([[pos]], np.int32), chan=0, Hq=1, Hkv=1,
                          d=w.d, P=w.page)[0, 0, 0]


def oracle_mix_tokens(prob, tokens=None, chans=None):
    """K~ and V of the chosen tokens and channels: dict[(b, j)] -> (K[Hkv][d], V[Hkv][d])."""
    w = prob.w
    tokens = range(w.B) if tokens is None else tokens
    chans = range(w.k) if chans is None else chans
    h = prob.host("h")
    pre_g, br, ch_g, qk_g = (prob.host(n) for n in ("pre_g", "br", "ch_g", "qk_g"))
    Wr = prob.host("Wr")
    nout = w.Hkv * w.d
    Wj = {}
    for X in range(2):
        for j in chans:
            Wj[X, j] = prob.rows("Wkv", (X * w.k + j) * nout, nout, w.D)
    res = {}
    for b in tokens:
        hhat, alpha, _ = O.pool_route(h[b], pre_g, Wr, br, L=w.L, k=w.k, D=w.D, p=w.p,
                                      eps=w.eps_rms)
        pos = float(prob.seq_lens[b]) - 1.0
        for j in chans:
            outs = []
            for X in range(2):
                _, o, _ = O.pool_channel(hhat[X], alpha[X, j], ch_g[X, j], Wj[X, j], qk_g[j],
                                         is_key=(X == 0), pos=pos, Hkv=w.Hkv, d=w.d,
                                         eps=w.eps_rms, eps_qk=w.eps_qk, theta=w.rope_theta)
                outs.append(o.reshape(w.Hkv, w.d))
            res[b, j] = tuple(outs)
    return res
