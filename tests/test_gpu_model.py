"""The whole-model decode step (random Qwen3-style blocks around the
library's attention and pool, Sec. 4.1 / Sec. 3.2) on the GPU.

* The step runs through bench.py's model mode and leaves no status set.
* Inside the step -- eager and replayed from a captured CUDA graph, with the
  attention launches chained by programmatic dependent launch -- every
  library output (the L attention outputs and the appended cache rows of
  every channel) equals the fp64 oracle run on the inputs those calls got.
* For the fp32 workload the whole step is also rebuilt on the host in fp64
  from the seeded block weights (blocks in numpy, attention and pool by the
  oracle), and the GPU step's outputs match it.
"""
import json
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

from oracle import oracle as O
from wm_synth import configs

from . import _harness as H
from ._model_step import ModelStep, host_block_tensor

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("workload", ["paper_k8", "tiny_f32"])
def test_model_mode_runs(workload):
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--mode", "model",
                        "--workload", workload, "--steps", "3", "--warmup", "3"],
                       cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    line = json.loads([l for l in r.stdout.splitlines() if l.startswith("{")][-1])
    assert line["value"] > 0 and line["config"]["mode"] == "model"
    assert 0.0 < line["whitematter_share"] < 1.0


def _storage(w, x64):
    """float64 values -> the storage dtype the oracle reads (fp32 or bf16 bits)."""
    from wm_synth import gen
    x = np.asarray(x64, np.float32)
    return x if w.dtype == "f32" else gen.f32_to_bf16_bits(x)


def _device_storage(w, t):
    a = t.detach().cpu()
    return a.numpy() if w.dtype == "f32" else a.view(torch.int16).numpy().view(np.uint16)


def _run_steps(w, graph: bool):
    prob, sess, dp = H.setup(w)
    model = ModelStep(w, sess, dp, sess.device)
    stream = torch.cuda.Stream(sess.device)
    with torch.cuda.stream(stream):
        model.step(stream)
    torch.cuda.synchronize()
    if graph:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for _ in range(2):
                model.step(stream)
        model.out.fill_(float("nan"))
        with torch.cuda.stream(stream):
            g.replay()
        torch.cuda.synchronize()
    assert sess.read_status() == 0
    return prob, sess, dp, model


def _written_rows(sess, prob):
    w = prob.w
    K = np.empty((w.B, w.k, w.Hkv, w.d))
    V = np.empty_like(K)
    for b in range(w.B):
        for j in range(w.k):
            K[b, j], V[b, j] = H.gpu_written_kv(sess, prob, b, j)
    return K, V


def _oracle_pool(prob, Hstates):
    w = prob.w
    args = [prob.host(n) for n in ("pre_g", "Wr", "br", "ch_g", "Wkv", "qk_g")]
    pos = (prob.seq_lens - 1).astype(np.float64)
    K, V, _, _ = O.kv_mix(Hstates, pos, *args, L=w.L, k=w.k, D=w.D, Hkv=w.Hkv, d=w.d, p=w.p,
                          eps=w.eps_rms, eps_qk=w.eps_qk, theta=w.rope_theta, nthreads=8)
    return K, V


@pytest.mark.parametrize("name,graph", [("tiny_f32", False), ("tiny_f32", True),
                                        ("paper_k8", False), ("paper_k8", True)])
def test_library_outputs_inside_the_model_step_match_the_oracle(name, graph):
    w = configs.get(name)
    prob, sess, dp, model = _run_steps(w, graph)
    tol = H.TOL[w.dtype]
    q = _device_storage(w, model.q)          # the queries the attention calls got
    kp, vp = prob.host("k_pool"), prob.host("v_pool")
    for l in range(w.L):
        want = O.decode_attn(q[l], kp, vp, prob.page_table, prob.seq_lens, chan=prob.chan[l],
                             Hq=w.Hq, Hkv=w.Hkv, d=w.d, P=w.page, nthreads=8)
        err = H.rel_err(H.to_f64(model.out[l]), want)
        assert err <= tol, (l, err)
    Kw, Vw = _oracle_pool(prob, _device_storage(w, model.H))  # the states the pool got
    Kg, Vg = _written_rows(sess, prob)
    assert H.rel_err(Kg, Kw) <= tol and H.rel_err(Vg, Vw) <= tol


def test_whole_step_matches_an_fp64_host_rebuild():
    w = configs.get("tiny_f32")
    prob, sess, dp, model = _run_steps(w, graph=True)
    I = model.I
    T = {n: host_block_tensor(w, 0, I, n) for n in ("Wq", "Wo", "Wg", "Wu", "Wd", "h0")}

    def rms(x, eps):
        return x / np.sqrt((x * x).mean(-1, keepdims=True) + eps)

    pos = prob.seq_lens.astype(np.float64) - 1.0
    inv = w.rope_theta ** (-np.arange(w.d // 2) * 2.0 / w.d)
    cos, sin = np.cos(pos[:, None] * inv)[:, None, :], np.sin(pos[:, None] * inv)[:, None, :]
    kp, vp = prob.host("k_pool"), prob.host("v_pool")
    h = T["h0"].copy()
    Hs = np.empty((w.B, w.L, w.D))
    for l in range(w.L):
        Hs[:, l] = h
        ql = rms((rms(h, w.eps_rms) @ T["Wq"][l].T).reshape(w.B, w.Hq, w.d), w.eps_qk)
        q1, q2 = ql[..., : w.d // 2], ql[..., w.d // 2:]
        ql = np.concatenate([q1 * cos - q2 * sin, q2 * cos + q1 * sin], -1)
        o = O.decode_attn(_storage(w, ql), kp, vp, prob.page_table, prob.seq_lens,
                          chan=prob.chan[l], Hq=w.Hq, Hkv=w.Hkv, d=w.d, P=w.page, nthreads=8)
        err = H.rel_err(H.to_f64(model.out[l]), o)
        assert err <= H.TOL[w.dtype], (l, err)
        h = h + o.reshape(w.B, -1) @ T["Wo"][l].T
        x2 = rms(h, w.eps_rms)
        g = x2 @ T["Wg"][l].T
        h = h + ((g / (1.0 + np.exp(-g))) * (x2 @ T["Wu"][l].T)) @ T["Wd"][l].T
    Kw, Vw = _oracle_pool(prob, _storage(w, Hs))
    Kg, Vg = _written_rows(sess, prob)
    assert H.rel_err(Kg, Kw) <= H.TOL[w.dtype] and H.rel_err(Vg, Vw) <= H.TOL[w.dtype]
