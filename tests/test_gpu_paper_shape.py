"""The paper's own model shape (Sec. 4.1): D=512, 6 query / 3 kv heads of
d=96 (GQA groups of 2), L=16, k in {1, 8, 16} with the three router bias
initialisations of Sec. 3.1 (top, cyclic, shifted identity).  GPU path vs
the fp64 oracle, all layers and all tokens."""
import pytest
import torch

from wm_synth import configs

from . import _harness as H

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name,overrides", [
    ("paper_k8", dict()), ("paper_k16", dict()), ("paper_k1", dict()),
    ("paper_k8", dict(dtype="f32", B=4, ctx=300, permute_pages=True, gain_std=0.1)),
])
def test_paper_shape_attention_and_pool(name, overrides):
    w = configs.get(name).with_(**overrides)
    prob, sess, dp = H.setup(w)
    for layer in range(w.L):
        got = H.to_f64(H.run_attn(sess, dp, layer))
        want = H.oracle_attn_full(prob, layer)
        assert H.rel_err(got, want) <= H.TOL[w.dtype], (layer, H.rel_err(got, want))
    sess.kv_mix(dp.h, dp.page_table, dp.slot)
    torch.cuda.synchronize()
    assert sess.read_status() == 0
    want = H.oracle_mix_tokens(prob)
    for (b, j), (k, v) in want.items():
        gk, gv = H.gpu_written_kv(sess, prob, b, j)
        assert H.rel_err(gk, k) <= H.TOL[w.dtype], ("K", b, j, H.rel_err(gk, k))
        assert H.rel_err(gv, v) <= H.TOL[w.dtype], ("V", b, j, H.rel_err(gv, v))
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


@pytest.mark.parametrize("B,g", [(300, 8), (600, 16)])
def test_batched_pool_over_several_token_tiles(B, g):
    """The pool for a prefill-sized batch (Sec. 3.3: a Gauss-Seidel group of
    strided positions i = q (mod g) across sequences): more tokens than one
    tensor-core token tile (256), written to strided slots."""
    w = configs.get("paper_k8").with_(B=B, ctx=8 * g + 64, permute_pages=True)
    # token b sits at position q + g*t of its row: strided slots, distinct per row
    lens = [1 + (b % g) + g * ((b // g) % 8) for b in range(B)]
    prob, sess, dp = H.setup(w, seq_lens=lens, fill_pools=False)
    sess.kv_mix(dp.h, dp.page_table, dp.slot)
    torch.cuda.synchronize()
    assert sess.read_status() == 0
    tokens = [0, 1, 255, 256, 257, B - 1] + ([511, 512] if B > 512 else [])
    want = H.oracle_mix_tokens(prob, tokens=tokens, chans=(0, 3, 7))
    for (b, j), (k, v) in want.items():
        gk, gv = H.gpu_written_kv(sess, prob, b, j)
        assert H.rel_err(gk, k) <= H.TOL[w.dtype], ("K", b, j, H.rel_err(gk, k))
        assert H.rel_err(gv, v) <= H.TOL[w.dtype], ("V", b, j, H.rel_err(gv, v))
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


@pytest.mark.parametrize("dtype,D,B,L,k", [("f32", 256, 96, 4, 2), ("f32", 3072, 70, 4, 2),
                                           ("bf16", 4096, 64, 6, 3)])
def test_batched_pool_dtypes_and_widths(dtype, D, B, L, k):
    """The batched forms of the pool (64 tokens and up) in fp32 and bf16, at
    widths where a thread owns one or two 8-element vectors of D."""
    w = configs.Workload("pool", L=L, k=k, D=D, Hq=2, Hkv=2, d=64, B=B, ctx=40, page=16,
                         dtype=dtype, chan_map="mod", permute_pages=True, gain_std=0.1)
    prob, sess, dp = H.setup(w, fill_pools=False)
    sess.kv_mix(dp.h, dp.page_table, dp.slot)
    torch.cuda.synchronize()
    assert sess.read_status() == 0
    tokens = [0, 1, B // 2, B - 1]
    want = H.oracle_mix_tokens(prob, tokens=tokens)
    for (b, j), (kk, vv) in want.items():
        gk, gv = H.gpu_written_kv(sess, prob, b, j)
        assert H.rel_err(gk, kk) <= H.TOL[dtype], ("K", b, j, H.rel_err(gk, kk))
        assert H.rel_err(gv, vv) <= H.TOL[dtype], ("V", b, j, H.rel_err(gv, vv))
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
