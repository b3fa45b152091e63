"""The full-size workloads, every output against the fp64 oracle.

Decode attention (Sec. 3.1 Step 3, dummy of Sec. 3.2): one whole layer of
each of the full-size workloads -- 1.1 GB (static split) to 17.2 GB (the
counter-driven split) of K/V per launch, and one sequence of 131072 slots
(2.15 GB, the unit split) -- every (sequence, query head) row.
The pool (Sec. 3.1 Steps 1-2, appended as in Sec. 3.2): every token and
every channel of the key and value rows written.  The host regenerates only
what each comparison reads, a sequence's pages of one channel at a time.
"""
import os

import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2608_18486_gb300 import _lib as W
from wm_synth import configs

from . import _harness as H

pytestmark = pytest.mark.gpu

DYNAMIC_BYTES = 2.0e9  # launches reading this much K/V take the counter-driven split


def _free():
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


@pytest.mark.parametrize("name,layer,overrides", [
    ("compress50", 5, {}), ("large", 13, {}), ("long32k", 0, {}), ("long64k", 7, {}),
    ("long128k", 5, {}),
    ("long128k", 9, dict(B=1, k=2)),  # one sequence of 2.15 GB: the unit split, clusters of 8
])
def test_full_size_layer_every_row(name, layer, overrides):
    w = configs.get(name).with_(**overrides)
    prob, sess, dp = H.setup(w)
    plan = W.wm_decode_attn_plan(sess.cfg, w.B, prob.max_pages)
    kv_bytes = float(w.B) * w.Hkv * prob.max_pages * w.page * 2 * w.d * w.elem_bytes
    if w.B == 1:
        assert plan["unit_ctas"] >= 2 and plan["chunk_stages"] == 0, plan
    else:
        assert (plan["chunk_stages"] > 0) == (kv_bytes >= DYNAMIC_BYTES), plan
    out = H.run_attn(sess, dp, layer)
    torch.cuda.synchronize()
    assert sess.read_status() == 0
    got = H.to_f64(out)
    del sess, dp, out
    _free()
    want = H.oracle_attn_layer(prob, layer)
    assert np.abs(want).max() > 1e-4 and np.abs(got).max() > 1e-4  # a real comparison
    err_rows = np.abs(got - want).max(axis=2) / np.abs(want).max()
    assert float(err_rows.max()) <= H.TOL[w.dtype], np.unravel_index(err_rows.argmax(), err_rows.shape)


@pytest.mark.parametrize("name", ["compress50", "large", "long64k"])
def test_full_size_pool_every_token_and_channel(name):
    w = configs.get(name)
    prob, sess, dp = H.setup(w, fill_pools=False)
    sess.kv_mix(dp.h, dp.page_table, dp.slot)
    torch.cuda.synchronize()
    assert sess.read_status() == 0
    Kg = np.empty((w.B, w.k, w.Hkv, w.d))
    Vg = np.empty_like(Kg)
    for b in range(w.B):
        for j in range(w.k):
            Kg[b, j], Vg[b, j] = H.gpu_written_kv(sess, prob, b, j)
    del sess, dp
    _free()
    args = [prob.host(n) for n in ("pre_g", "Wr", "br", "ch_g", "Wkv", "qk_g")]
    pos = (prob.seq_lens - 1).astype(np.float64)
    K, V, _, _ = O.kv_mix(prob.host("h"), pos, *args, L=w.L, k=w.k, D=w.D, Hkv=w.Hkv, d=w.d,
                          p=w.p, eps=w.eps_rms, eps_qk=w.eps_qk, theta=w.rope_theta,
                          nthreads=len(os.sched_getaffinity(0)))
    assert H.rel_err(Kg, K) <= H.TOL[w.dtype] and H.rel_err(Vg, V) <= H.TOL[w.dtype], \
        (H.rel_err(Kg, K), H.rel_err(Vg, V))
