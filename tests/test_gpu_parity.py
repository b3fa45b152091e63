"""GPU path vs the fp64 oracle, through the C ABI, on seeded inputs.

Tolerances are the stated ones: max |gpu - oracle| / max |oracle| per output
tensor <= 1e-4 for fp32 workloads and <= 2e-2 for bf16 workloads (fp32
accumulation).  Cache indexing, paging and masking are checked bit-exact.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from wm_synth import configs, device
from wm_synth.inputs import make_problem

from . import _harness as H

pytestmark = pytest.mark.gpu


def _free():
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


# ------------------------------------------------------------ small, complete
@pytest.mark.parametrize("name,seed,q_scale", [
    ("tiny_f32", 0, 1.0), ("no_compression", 0, 1.0), ("no_compression", 1, 1.0),
    ("no_compression", 0, 8.0), ("no_compression", 1, 8.0)])
def test_attention_all_layers_all_heads(name, seed, q_scale):
    """q_scale 8: peaked attention (a few slots carry most of the weight),
    where bf16 rounding of the softmax inputs matters most."""
    w = configs.get(name).with_(q_scale=q_scale)
    prob, sess, dp = H.setup(w, seed=seed)
    for layer in range(w.L):
        got = H.to_f64(H.run_attn(sess, dp, layer))
        want = H.oracle_attn_full(prob, layer)
        assert H.rel_err(got, want) <= H.TOL[w.dtype], (layer, H.rel_err(got, want))
    assert sess.read_status() == 0
    _free()


@pytest.mark.parametrize("name,seed", [("tiny_f32", 0), ("no_compression", 0),
                                       ("no_compression", 1)])
def test_kv_mix_all_tokens_all_channels(name, seed):
    w = configs.get(name)
    prob, sess, dp = H.setup(w, seed=seed)
    sess.kv_mix(dp.h, dp.page_table, dp.slot)
    torch.cuda.synchronize()
    assert sess.read_status() == 0
    want = H.oracle_mix_tokens(prob)
    errk = max(H.rel_err(H.gpu_written_kv(sess, prob, b, j)[0], want[b, j][0]) for b, j in want)
    errv = max(H.rel_err(H.gpu_written_kv(sess, prob, b, j)[1], want[b, j][1]) for b, j in want)
    assert errk <= H.TOL[w.dtype] and errv <= H.TOL[w.dtype], (errk, errv)
    _free()


def test_tiny_gains_and_peaked_attention_variants():
    w = configs.get("tiny_f32").with_(gain_std=0.1, q_scale=8.0)
    prob, sess, dp = H.setup(w, seed=1)
    for layer in range(w.L):
        got = H.to_f64(H.run_attn(sess, dp, layer))
        assert H.rel_err(got, H.oracle_attn_full(prob, layer)) <= H.TOL["f32"]
    sess.kv_mix(dp.h, dp.page_table, dp.slot)
    torch.cuda.synchronize()
    want = H.oracle_mix_tokens(prob)
    for (b, j), (k, v) in want.items():
        gk, gv = H.gpu_written_kv(sess, prob, b, j)
        assert H.rel_err(gk, k) <= H.TOL["f32"] and H.rel_err(gv, v) <= H.TOL["f32"]
    _free()


# ------------------------------------------------------------ shapes and paging
@pytest.mark.parametrize("dtype,d,G,page", [
    ("bf16", 128, 1, 16), ("bf16", 64, 2, 1), ("bf16", 128, 4, 8), ("f32", 128, 1, 64),
    ("f32", 64, 8, 32), ("bf16", 64, 1, 128), ("bf16", 128, 2, 256)])
def test_attention_shapes_pages_ragged(dtype, d, G, page):
    Hkv = 2
    w = configs.Workload("t", L=3, k=2, D=64, Hq=Hkv * G, Hkv=Hkv, d=d, B=5, ctx=700,
                         ctx_lo=1, page=page, dtype=dtype, chan_map="mod", permute_pages=True)
    lens = [1, 2, 127, 700, 333]
    prob, sess, dp = H.setup(w, seed=3, seq_lens=lens)
    for layer in range(w.L):
        got = H.to_f64(H.run_attn(sess, dp, layer))
        want = H.oracle_attn_full(prob, layer)
        assert H.rel_err(got, want) <= H.TOL[dtype], (layer, H.rel_err(got, want))
    assert sess.read_status() == 0
    _free()


def test_page_permutation_is_bit_exact():
    w = configs.get("no_compression").with_(B=4, L=2, k=2)
    lens = [2048, 1500, 17, 1]
    pa, sa, da = H.setup(w.with_(permute_pages=False), seq_lens=lens)
    pb, sb, db = H.setup(w.with_(permute_pages=True), seq_lens=lens)
    # same logical contents: copy pages of layout a into their places in layout b
    for b, S in enumerate(lens):
        for i in range(-(-(S + 1) // w.page)):
            sb.k_pool[:, pb.page_table[b, i]] = sa.k_pool[:, pa.page_table[b, i]]
            sb.v_pool[:, pb.page_table[b, i]] = sa.v_pool[:, pa.page_table[b, i]]
    for layer in range(w.L):
        oa, ob = H.run_attn(sa, da, layer), H.run_attn(sb, db, layer)
        assert torch.equal(oa, ob)
    _free()


def test_slots_beyond_length_never_reach_the_output():
    w = configs.get("no_compression").with_(B=3, L=2, k=2)
    lens = [37, 16, 1000]
    prob, sess, dp = H.setup(w, seq_lens=lens)
    base = [H.run_attn(sess, dp, l).clone() for l in range(w.L)]
    for b, S in enumerate(lens):
        npg = int((prob.page_table[b] >= 0).sum())
        for i in range(npg):
            pg = int(prob.page_table[b, i])
            lo = max(0, S - i * w.page)
            if lo < w.page:
                sess.k_pool[:, pg, :, lo:, :] = float("nan")
                sess.v_pool[:, pg, :, lo:, :] = float("nan")
    for l in range(w.L):
        assert torch.equal(H.run_attn(sess, dp, l), base[l])
    _free()


def test_dummy_only_sequences_return_the_dummy_value():
    w = configs.get("no_compression").with_(B=3, L=1, k=1)
    prob, sess, dp = H.setup(w, seq_lens=[1, 1, 1])
    out = H.run_attn(sess, dp, 0)
    for b in range(3):
        pg = int(prob.page_table[b, 0])
        assert torch.equal(out[b], sess.v_pool[0, pg, :, 0, :])
    _free()


def test_bad_page_id_and_length_report_status_without_fault():
    w = configs.get("no_compression").with_(B=2, L=1, k=1)
    prob, sess, dp = H.setup(w, seq_lens=[300, 40])
    dp.page_table[0, 3] = prob.num_pages + 5
    H.run_attn(sess, dp, 0)
    torch.cuda.synchronize()
    assert sess.read_status() == 4  # WM_ERR_BOUNDS
    dp.page_table[0, 3] = int(prob.page_table[0, 3])
    dp.seq_lens[1] = 0
    out = H.run_attn(sess, dp, 0)
    torch.cuda.synchronize()
    assert sess.read_status() == 4
    assert torch.count_nonzero(out[1].float()) == 0
    dp.seq_lens[1] = 40
    dp.slot[0] = w.page * prob.max_pages  # one past the page table
    sess.kv_mix(dp.h, dp.page_table, dp.slot)
    torch.cuda.synchronize()
    assert sess.read_status() == 4
    _free()


def test_zero_batch_is_a_noop():
    w = configs.get("tiny_f32")
    prob, sess, dp = H.setup(w)
    snap = sess.k_pool.clone()
    out = torch.empty((0, w.Hq, w.d), dtype=sess.dtype, device="cuda")
    sess.decode_attn(0, dp.q[0], dp.page_table, dp.seq_lens, out, B=0)
    sess.kv_mix(dp.h, dp.page_table, dp.slot, B=0)
    torch.cuda.synchronize()
    assert torch.equal(snap, sess.k_pool) and sess.read_status() == 0
    _free()


def test_kv_mix_writes_exactly_the_target_elements():
    w = configs.get("no_compression").with_(B=5, permute_pages=True)
    prob, sess, dp = H.setup(w, seq_lens=[5, 16, 17, 2047, 900])
    k0, v0 = sess.k_pool.clone(), sess.v_pool.clone()
    sess.kv_mix(dp.h, dp.page_table, dp.slot)
    torch.cuda.synchronize()
    mask = torch.zeros(sess.k_pool.shape, dtype=torch.bool, device="cuda")
    for b, S in enumerate(prob.seq_lens):
        mask[:, int(prob.page_table[b, S // w.page]), :, int(S) % w.page, :] = True
    for new, old in ((sess.k_pool, k0), (sess.v_pool, v0)):
        same = (new.view(torch.int16) == old.view(torch.int16))
        assert bool(same[~mask].all())
        assert int((~same[mask]).sum()) > 0.9 * int(mask.sum())
    _free()


# ------------------------------------------------------------ full-size workloads, sampled
def _sample_units(w, prob, n, rng):
    return [(int(rng.integers(w.B)), int(rng.integers(w.Hq))) for _ in range(n)]


@pytest.mark.parametrize("name,layers,nunits", [
    ("compress50", None, 6), ("large", (0, 13, 31), 3), ("long32k", (0, 31), 2),
    ("long64k", (7, 30), 2), ("long128k", (5,), 2)])
def test_full_size_attention_sampled(name, layers, nunits):
    w = configs.get(name)
    prob, sess, dp = H.setup(w)
    rng = np.random.default_rng(0)
    layers = range(w.L) if layers is None else layers
    for layer in layers:
        out = H.run_attn(sess, dp, layer)
        for b, hq in _sample_units(w, prob, nunits, rng):
            want = H.oracle_attn_unit(prob, layer, b, hq)
            err = H.rel_err(H.to_f64(out[b, hq]), want)
            assert err <= H.TOL[w.dtype], (layer, b, hq, err)
    assert sess.read_status() == 0
    del sess, dp
    _free()


@pytest.mark.parametrize("name,tokens,chans", [
    ("compress50", (0, 63), None), ("large", (0, 31), (0, 15)), ("long64k", (3,), (0, 7))])
def test_full_size_kv_mix_sampled(name, tokens, chans):
    w = configs.get(name)
    prob, sess, dp = H.setup(w, fill_pools=False)
    sess.kv_mix(dp.h, dp.page_table, dp.slot)
    torch.cuda.synchronize()
    assert sess.read_status() == 0
    want = H.oracle_mix_tokens(prob, tokens, chans)
    for (b, j), (k, v) in want.items():
        gk, gv = H.gpu_written_kv(sess, prob, b, j)
        assert H.rel_err(gk, k) <= H.TOL[w.dtype], ("K", b, j, H.rel_err(gk, k))
        assert H.rel_err(gv, v) <= H.TOL[w.dtype], ("V", b, j, H.rel_err(gv, v))
    del sess, dp
    _free()


# ------------------------------------------------------------ input generator
def test_device_generator_matches_host_bit_for_bit():
    for dtype in ("f32", "bf16"):
        t = torch.empty(3_000_001, dtype=torch.float32 if dtype == "f32" else torch.bfloat16,
                        device="cuda")
        device.fill(t, dtype, seed=7, stream=31, std=0.37, mean=1.0, start=12345)
        host = np.asarray(__import__("wm_synth").gen.values(dtype, 7, 31, 12345, t.numel(),
                                                                 0.37, 1.0))
        got = t.cpu().view(torch.int32 if dtype == "f32" else torch.int16).numpy()
        assert np.array_equal(got, host.view(np.int32 if dtype == "f32" else np.int16))


@pytest.mark.parametrize("name,overrides", [("no_compression", dict()),
                                            ("large", dict(k=1, B=4))])
def test_inputs_ready_chain_matches_default_launches(name, overrides):
    """Layers 1..L-1 launched with WM_ATTN_INPUTS_READY (K/V fetched while the
    previous launch finishes) give the same bits as plain launches."""
    w = configs.get(name).with_(**overrides)
    prob, sess, dp = H.setup(w)
    ref = [H.run_attn(sess, dp, l).clone() for l in range(w.L)]
    outs = torch.empty((w.L, w.B, w.Hq, w.d), dtype=sess.dtype, device="cuda")
    for _ in range(2):
        for l in range(w.L):
            sess.decode_attn(l, dp.q[l], dp.page_table, dp.seq_lens, outs[l], inputs_ready=l > 0)
    torch.cuda.synchronize()
    assert sess.read_status() == 0
    for l in range(w.L):
        assert torch.equal(outs[l], ref[l]), l
    if name == "no_compression":
        assert H.rel_err(H.to_f64(outs[3]), H.oracle_attn_full(prob, 3)) <= H.TOL[w.dtype]
    _free()


@pytest.mark.parametrize("dynamic", [False, True])
def test_graph_replay_over_changing_lengths(dynamic):
    """A decode loop replays one captured launch while the lengths change
    underneath it (the replay keeps the call's epoch): on the counter-driven
    split the chunk layout moves with the lengths, and no flag or ticket left
    by an earlier replay passes for this replay's records; the default plan
    here is the unit split."""
    w = configs.get("no_compression").with_(L=2, k=2)
    prob, sess, dp = H.setup(w)
    lens = dp.seq_lens.clone()
    out = torch.empty((w.B, w.Hq, w.d), dtype=sess.dtype, device=sess.device)
    sess.decode_attn(0, dp.q[0], dp.page_table, lens, out, dynamic_split=dynamic)  # warm-up
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        sess.decode_attn(0, dp.q[0], dp.page_table, lens, out, dynamic_split=dynamic)
    rng = np.random.default_rng(3)
    full = np.asarray(prob.seq_lens, np.int64)
    sets = [full, np.maximum(1, full // 3), rng.integers(1, full + 1), full - 17,
            rng.integers(1, full + 1), full]
    for S in sets:
        lens.copy_(torch.as_tensor(S, dtype=torch.int32))
        out.fill_(float("nan"))
        g.replay()
        torch.cuda.synchronize()
        want = O.decode_attn(prob.host("q")[0], prob.host("k_pool"), prob.host("v_pool"),
                             prob.page_table, S.astype(np.int32), chan=prob.chan[0], Hq=w.Hq,
                             Hkv=w.Hkv, d=w.d, P=w.page, nthreads=8)
        err = H.rel_err(H.to_f64(out), want)
        assert err <= H.TOL[w.dtype], (S[:4], err)
    assert sess.read_status() == 0
    del g
    _free()


def test_workspace_reused_across_batch_sizes():
    """One workspace serves calls whose plans lay partial records out
    differently (a smaller batch splits into fewer chunks), mixed with calls
    on the unit split, which leaves the workspace alone: words left by
    another call never pass for published records."""
    w = configs.get("no_compression").with_(L=2, k=2)
    prob, sess, dp = H.setup(w)
    want = H.oracle_attn_full(prob, 0)
    for B, dyn in ((w.B, True), (5, True), (11, False), (w.B, True), (3, False), (7, True)):
        out = torch.full((B, w.Hq, w.d), float("nan"), dtype=sess.dtype, device=sess.device)
        sess.decode_attn(0, dp.q[0][:B], dp.page_table[:B], dp.seq_lens[:B], out, B=B,
                         dynamic_split=dyn)
        torch.cuda.synchronize()
        err = H.rel_err(H.to_f64(out), want[:B])
        assert err <= H.TOL[w.dtype], (B, err)
    assert sess.read_status() == 0
    _free()
