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


def test_noalloc_rejects_launches_larger_than_its_scratch():
    # 4096 sequences x 8 query heads per kv head need more than the fixed array
    w = configs.get("large").with_(B=4096, Hq=256, Hkv=32)
    cfg = H.config_of(w)
    nbytes = W.wm_cache_bytes(cfg, 1)
    cache = W.wm_cache_alloc(cfg, 1 << 40, nbytes, 1)  # a layout only; never touched
    fake = 1 << 41
    rc = W.wm_decode_attn_noalloc(cfg, cache, 0, fake, fake, fake, w.B, 1, fake, None, None)
    assert rc == W.WM_ERR_UNSUPPORTED
