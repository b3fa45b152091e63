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
from ._oracle_side import (oracle_attn_full, oracle_attn_layer, oracle_attn_unit,  # noqa: E402,F401
                           oracle_mix_tokens, oracle_prefill_unit)


def gpu_written_kv(sess, prob, b, j):
    """The K and V the GPU wrote for token b, channel j (slot seq_lens[b])."""
    w = prob.w
    s = int(prob.seq_lens[b])
    pg = int(prob.page_table[b, s // w.page])
    return (to_f64(sess.k_pool[j, pg, :, s % w.page, :]),
            to_f64(sess.v_pool[j, pg, :, s % w.page, :]))


def storage_to_f64(dtype, arr) -> np.ndarray:
    return gen.to_f64(dtype, arr)
