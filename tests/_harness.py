"""Shared plumbing of the GPU parity tests.

Expected values come only from the fp64 oracle, fed with inputs regenerated
on the host from the seeded streams (never read back from the GPU path).
"""
from __future__ import annotations

import numpy as np
import torch

from oracle import oracle as O
from paper_2608_18486_gb300 import _lib as W
from paper_2608_18486_gb300.session import DecodeSession
from wm_synth import gen
from wm_synth.device_problem import DeviceProblem
from wm_synth.inputs import make_problem

TOL = {"f32": 1e-4, "bf16": 2e-2}


def config_of(w) -> W.wm_config:
    return W.make_config(w.L, w.k, w.D, w.Hq, w.Hkv, w.d, w.p, w.page, w.dtype,
                         w.chan_of_layer(), w.eps_rms, w.eps_qk, w.rope_theta)


def setup(w, seed=0, seq_lens=None, fill_pools=True):
    prob = make_problem(w, seed, seq_lens)
    sess = DecodeSession(config_of(w), w.B, prob.num_pages, prob.max_pages)
    dp = DeviceProblem(prob, sess.k_pool, sess.v_pool, fill_pools=fill_pools)
    sess.set_weights(*dp.weights())
    return prob, sess, dp


def to_f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().astype(np.float64)


def rel_err(got, want) -> float:
    got, want = np.asarray(got, np.float64), np.asarray(want, np.float64)
    return float(np.abs(got - want).max() / max(np.abs(want).max(), 1e-30))


def run_attn(sess, dp, layer) -> torch.Tensor:
    w = dp.prob.w
    out = torch.empty((w.B, w.Hq, w.d), dtype=sess.dtype, device=sess.device)
    sess.decode_attn(layer, dp.q[layer], dp.page_table, dp.seq_lens, out)
    return out


# ------------------------------------------------------------------ oracle side
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


def gpu_written_kv(sess, prob, b, j):
    """The K and V the GPU wrote for token b, channel j (slot seq_lens[b])."""
    w = prob.w
    s = int(prob.seq_lens[b])
    pg = int(prob.page_table[b, s // w.page])
    return (to_f64(sess.k_pool[j, pg, :, s % w.page, :]),
            to_f64(sess.v_pool[j, pg, :, s % w.page, :]))


def storage_to_f64(dtype, arr) -> np.ndarray:
    return gen.to_f64(dtype, arr)
