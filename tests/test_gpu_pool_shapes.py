"""The pool of a decode batch (Sec. 3.1 Steps 1-2, appended as in Sec. 3.2)
at the edges of its tiling: every written key and value against the fp64
oracle -- one projection row tile per channel up to eight, D of one k-block,
router inputs spanning several blocks per split, p = 1 and 3 with L not a
multiple of p, token counts that pad the MMA's N, GQA heads of 96, gains
off one, ragged slots on permuted pages -- and repeated and graph-replayed
pools writing the same bits."""
import pytest
import torch

from paper_2608_18486_gb300 import _lib as W
from wm_synth import configs

from . import _harness as H

pytestmark = pytest.mark.gpu


def _shape(name, **kw):
    base = dict(L=6, k=3, D=256, Hq=4, Hkv=4, d=64, B=8, ctx=100, page=16, dtype="bf16",
                chan_map="mod", ctx_lo=1, permute_pages=True)
    base.update(kw)
    return configs.Workload(name, **base)


CASES = [
    ("no_compression", configs.get("no_compression"), None),
    ("no_compression_B1", configs.get("no_compression").with_(B=1), None),
    ("no_compression_B17", configs.get("no_compression").with_(B=17, ctx_lo=2), None),
    ("no_compression_B24", configs.get("no_compression").with_(B=24, k=4, ctx_lo=2), None),
    ("paper_k16", configs.get("paper_k16"), None),
    ("paper_k1_gains", configs.get("paper_k1").with_(gain_std=0.1), None),
    ("R1_d128", _shape("R1_d128", Hq=2, Hkv=1, d=128), None),
    ("R8", _shape("R8", L=8, k=4, D=512, Hq=16, Hkv=16, p=1), None),
    ("p3_L7", _shape("p3_L7", L=7, k=5, D=320, p=3, gain_std=0.1), None),
    ("D64_R4", _shape("D64_R4", L=4, k=2, D=64, Hq=8, Hkv=8), None),
    ("G2_d96", _shape("G2_d96", L=5, k=5, D=384, Hq=8, Hkv=4, d=96, B=12), None),
]


@pytest.mark.parametrize("name,w,lens", CASES, ids=[c[0] for c in CASES])
def test_pool_matches_the_oracle(name, w, lens):
    prob, sess, dp = H.setup(w, seq_lens=lens)
    assert W.wm_kv_mix_launches(sess.cfg, w.B) == 4  # prenorm, router, mix, projection
    sess.kv_mix(dp.h, dp.page_table, dp.slot)
    torch.cuda.synchronize()
    assert sess.read_status() == 0
    want = H.oracle_mix_tokens(prob)
    errk = max(H.rel_err(H.gpu_written_kv(sess, prob, b, j)[0], want[b, j][0]) for b, j in want)
    errv = max(H.rel_err(H.gpu_written_kv(sess, prob, b, j)[1], want[b, j][1]) for b, j in want)
    assert errk <= H.TOL[w.dtype] and errv <= H.TOL[w.dtype], (errk, errv)
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def test_launch_counts():
    for name, B in (("large", 32), ("long128k", 8), ("compress50", 64), ("no_compression", 64)):
        w = configs.get(name)
        assert W.wm_kv_mix_launches(H.config_of(w), B) == 4, name
    assert W.wm_kv_mix_launches(H.config_of(configs.get("tiny_f32")), 2) == 5  # fp32
    assert W.wm_kv_mix_launches(H.config_of(configs.get("tiny_f32")), 0) == 0


def test_pool_twice_in_a_row_and_in_a_graph():
    """Back-to-back pools and a captured replay write the same bits."""
    w = configs.get("paper_k8")
    prob, sess, dp = H.setup(w)
    sess.kv_mix(dp.h, dp.page_table, dp.slot)
    torch.cuda.synchronize()
    k1, v1 = sess.k_pool.clone(), sess.v_pool.clone()
    sess.k_pool.zero_()
    sess.v_pool.zero_()
    s = torch.cuda.Stream()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        sess.kv_mix(dp.h, dp.page_table, dp.slot, stream=s)
    g.replay()
    g.replay()
    torch.cuda.synchronize()
    assert sess.read_status() == 0
    for b in range(w.B):
        for j in range(w.k):
            S = int(prob.seq_lens[b])
            pg = int(prob.page_table[b, S // w.page])
            assert torch.equal(sess.k_pool[j, pg, :, S % w.page], k1[j, pg, :, S % w.page])
            assert torch.equal(sess.v_pool[j, pg, :, S % w.page], v1[j, pg, :, S % w.page])
