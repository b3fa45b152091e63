"""Failure detection without a GPU fault.

Every pipeline wait in libwm is bounded: a wait that runs out makes the
kernel report WM_ERR_TIMEOUT in the status word and return.  The self-test
kernel waits on a barrier that nothing completes (a short limit), and the
test checks the status and that the context still runs the decode path.
Bad indices are turned into WM_ERR_BOUNDS by the kernels' own checks
(test_gpu_parity.py).  Nothing here traps, faults or hangs the GPU.
"""
import ctypes
import time

import pytest
import torch

from paper_2608_18486_gb300 import _lib as W
from wm_synth import configs

from . import _harness as H


def test_selftest_rejects_bad_arguments_on_the_host():
    assert W.wm_selftest_bounded_wait(None, 1000, None) == W.WM_ERR_INVALID_ARG
    assert W.wm_selftest_bounded_wait(1 << 40, 0, None) == W.WM_ERR_INVALID_ARG
    assert W.wm_selftest_bounded_wait(1 << 40, 3_000_000, None) == W.WM_ERR_INVALID_ARG


@pytest.mark.gpu
def test_a_wait_that_runs_out_reports_timeout_and_the_context_stays_usable():
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    t0 = time.time()
    assert W.wm_selftest_bounded_wait(status, 20_000, stream) == W.WM_OK  # 20 ms limit
    torch.cuda.synchronize()
    assert time.time() - t0 < 10.0
    assert int(status.item()) == W.WM_ERR_TIMEOUT
    # the decode path still runs and still matches the oracle
    w = configs.get("tiny_f32")
    prob, sess, dp = H.setup(w)
    got = H.to_f64(H.run_attn(sess, dp, 0))
    assert H.rel_err(got, H.oracle_attn_full(prob, 0)) <= H.TOL["f32"]
    assert sess.read_status() == 0
