"""wm_decode_attn_noalloc: decode attention for callers that cannot allocate.

Some callers have no device memory to give the library beyond a call's inputs
and outputs (a plugin whose host program owns every allocation, or a fixed
memory plan without room for scratch).  This entry point keeps its scratch in
a fixed array inside the library, so it takes no workspace.  The test calls it
through the C ABI twice in a row -- the second call sees the array exactly as
the first left it -- and checks both results against the workspace-taking
entry point, with the tolerance the other parity tests use.

The file name sorts last so that a run stopping at the first failure has run
every other test before this one; it also passes when run alone in a fresh
process, where its first call does the per-device set-up.
"""
import ctypes

import pytest
import torch

from paper_2608_18486_gb300 import _lib as W
from wm_synth import configs

from . import _harness as H

pytestmark = pytest.mark.gpu


def _noalloc(sess, dp, layer, out):
    w = dp.prob.w
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    return W.wm_decode_attn_noalloc(sess.cfg, sess.cache, layer, dp.q[layer], dp.page_table,
                                    dp.seq_lens, w.B, sess.max_pages, out, sess.status, stream)


@pytest.mark.parametrize("name,overrides", [
    ("no_compression", dict(L=3, k=3)),
    ("tiny_f32", dict()),
])
def test_noalloc_matches_workspace_entry_point_on_two_calls(name, overrides):
    w = configs.get(name).with_(**overrides)
    prob, sess, dp = H.setup(w)
    for layer in range(w.L):
        ref = H.run_attn(sess, dp, layer)
        outs = []
        for _ in range(2):
            out = torch.full_like(ref, float("nan"))
            assert _noalloc(sess, dp, layer, out) == W.WM_OK
            outs.append(out)
        torch.cuda.synchronize()
        assert sess.read_status() == 0
        for out in outs:
            err = H.rel_err(H.to_f64(out), H.to_f64(ref))
            assert err <= H.TOL[w.dtype], (layer, err)


# the size of the library's fixed scratch array (include/wm.h)
NOALLOC_SCRATCH_BYTES = 8 << 20


def test_noalloc_near_its_scratch_limit_on_two_calls():
    """A launch whose partial records fill most of the fixed array (3
    sequences of 131072 slots, 32 heads of 128: a dynamic split into about
    6100 chunks, 6.4 MB of records) gives the workspace entry point's rows on
    two calls in a row: the record offsets and the cleared span reach the
    array's end."""
    w = configs.get("long128k").with_(B=3, L=1, k=1)
    prob, sess, dp = H.setup(w)
    plan = W.wm_decode_attn_plan(sess.cfg, w.B, prob.max_pages)
    rec_bytes = 4 * (128 + 4)  # d outputs, (m, l) and the flag, padded to 16 bytes
    used = 2 * plan["chunks"] * rec_bytes
    assert plan["chunk_stages"] > 0 and 6 * 2 ** 20 < used < NOALLOC_SCRATCH_BYTES - 128 * 1024, plan
    ref = H.run_attn(sess, dp, 0)
    outs = []
    for _ in range(2):
        out = torch.full_like(ref, float("nan"))
        assert _noalloc(sess, dp, 0, out) == W.WM_OK
        outs.append(out)
    torch.cuda.synchronize()
    assert sess.read_status() == 0
    for out in outs:
        err = H.rel_err(H.to_f64(out), H.to_f64(ref))
        assert err <= H.TOL[w.dtype], err
    del sess, dp
    torch.cuda.empty_cache()


def test_noalloc_rejects_launches_larger_than_its_scratch():
    # 4096 sequences x 8 query heads per kv head over 2 pages each: the
    # partial records alone need far more than the fixed array
    w = configs.get("large").with_(B=4096, Hq=256, Hkv=32)
    cfg = H.config_of(w)
    max_pages = 2
    assert W.wm_decode_attn_workspace(cfg, w.B, max_pages) > 2 * NOALLOC_SCRATCH_BYTES
    # Real buffers that make the call a valid launch (one cache page, every
    # sequence one slot long on page 0), so that a wrong answer of the size
    # check shows up as a failed assertion and never as a read of memory
    # the call does not own.
    dev = torch.device("cuda", 0)
    nbytes = W.wm_cache_bytes(cfg, 1)
    cache_buf = torch.zeros(nbytes, dtype=torch.uint8, device=dev)
    cache = W.wm_cache_alloc(cfg, cache_buf, nbytes, 1)
    q = torch.zeros((w.B, w.Hq, w.d), dtype=torch.bfloat16, device=dev)
    out = torch.empty_like(q)
    page_table = torch.zeros((w.B, max_pages), dtype=torch.int32, device=dev)
    seq_lens = torch.ones(w.B, dtype=torch.int32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    rc = W.wm_decode_attn_noalloc(cfg, cache, 0, q, page_table, seq_lens, w.B, max_pages, out,
                                  status, None)
    torch.cuda.synchronize()
    assert rc == W.WM_ERR_UNSUPPORTED
