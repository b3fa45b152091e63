"""Decode-step throughput of the WhiteMatter hot path on GB300.

One step = L calls of wm_decode_attn (layer l reads channel c(l) of the
paged k-channel cache) + one wm_kv_mix (the cross-layer KV pool for the B
new tokens), i.e. B decoded tokens.  Prints one JSON line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   # the fp64 CPU oracle, timed on host cores

Multi-GPU runs (torchrun) are data-parallel replicas: each rank decodes its
own batch of sequences (weak scaling) with no collective on the data path;
only the timing barrier and the max over ranks use torch.distributed.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "decode tokens/s per step (mix+channel attention) at 1 GB300; HBM GB/s vs peak"
# The largest single-GPU workload: B=8 sequences of 131072 slots, L=32 layers of
# 32 heads x 128 over k=8 channels (137 GB of cache, 17.2 GB read per layer).
DEFAULT_WORKLOAD = "long128k"
# Timed work the default step count aims at (--steps overrides it).
TARGET_TIMED_S = 2.0
FALLBACK_HBM_GBS = 6800.0


# ---------------------------------------------------------------- helpers
def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def measured_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def kernel_source_hash() -> str:
    h = hashlib.sha256()
    for f in ("attn.cu", "attn_kernel.cuh", "attn_bf16.cu", "attn_unit.cuh", "attn_unit_bf16.cu",
              "common.cuh", "internal.h", "wm_api.cu"):
        with open(os.path.join(ROOT, "paper_2608_18486_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def attn_kernel_name(cfg, w, prob) -> str:
    """The decode-attention kernel the library's planner picks for this launch."""
    from paper_2608_18486_gb300 import _lib as W
    plan = W.wm_decode_attn_plan(cfg, w.B, prob.max_pages)
    return "decode_attn_unit_kernel" if plan["unit_ctas"] > 0 else "decode_attn_kernel"


def ncu_traffic(workload: str):
    """DRAM bytes per attention launch from the committed ncu summary, if it
    was taken on the current kernel source; else None."""
    path = os.path.join(ROOT, "profiles", "decode_attn_traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)
        e = d.get(workload)
        if e and e.get("kernel_hash") == kernel_source_hash():
            return float(e["dram_bytes_per_launch"])
    except Exception:
        pass
    return None


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while running."""

    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.proc = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "50", "-i", gpu_id], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                text=True)
        except Exception:
            self.proc = None

    def stop(self, t0: float, t1: float):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            return None
        rows = []
        for line in out.strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                ts = time.mktime(time.strptime(parts[0].split(".")[0], "%Y/%m/%d %H:%M:%S"))
                ts += float("0." + parts[0].split(".")[1]) if "." in parts[0] else 0.0
                rows.append((ts, float(parts[1]), float(parts[2]), parts[5:9]))
            except Exception:
                continue
        if not rows:
            return None
        inside = [r for r in rows if t0 - 0.25 <= r[0] <= t1 + 0.05] or rows[-3:]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in inside for i, v in enumerate(r[3]) if v == "Active"})
        return {"sm_mhz": statistics.median(r[1] for r in inside),
                "sm_max_mhz": max(r[2] for r in inside), "reasons": reasons,
                "samples": len(inside)}


def rank_problem(w, rank: int):
    """The batch of sequences replica `rank` decodes: its own seeded problem
    (own cache contents, lengths and page table), so ranks share nothing."""
    from wm_synth.inputs import make_problem
    return make_problem(w, seed=rank)


def max_over_ranks(values, world: int, device=None):
    """Element-wise max of per-rank timings (the job is as slow as its
    slowest replica); a no-op for one rank."""
    import torch
    import torch.distributed as dist
    t = torch.tensor(list(values), dtype=torch.float64, device=device)
    if world > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(x) for x in t]


def default_steps(w) -> int:
    """Timed steps worth about TARGET_TIMED_S at the measured HBM rate."""
    from wm_synth import configs as C
    from wm_synth.inputs import make_problem
    peak, _ = measured_peak()
    lens = make_problem(w, seed=0).seq_lens if w.ctx_lo else [w.ctx] * w.B
    est = C.step_bytes(w, lens) / (0.8 * peak * 1e9)
    return int(min(200, max(10, round(TARGET_TIMED_S / max(est, 1e-6)))))


# ---------------------------------------------------------------- CPU oracle timing
def oracle_step_estimate(prob, budget_s: float = 4.0, nthreads: int | None = None):
    """Time the fp64 oracle on a bounded sample of one decode step and
    extrapolate to a full step (L attention layers + the pool for B tokens).
    Returns (seconds per full step, cores used, sample description)."""
    import numpy as np
    from oracle import oracle as O
    w = prob.w
    cores = nthreads or len(os.sched_getaffinity(0))
    # attention: one layer, a prefix of the (b, hq) units, scaled by slots read
    units_all = [(b, hq) for b in range(w.B) for hq in range(w.Hq)]
    q = prob.host("q")[0]
    kp = prob.host("k_pool") if prob.pool_elems() <= (1 << 28) else None
    t_attn, slots_done, units_done = 0.0, 0, 0
    if kp is not None:
        vp = prob.host("v_pool")
        step = max(1, cores)
        i = 0
        while i < len(units_all) and t_attn < budget_s / 2:
            u = units_all[i:i + step]
            t = time.perf_counter()
            O.decode_attn(q, kp, vp, prob.page_table, prob.seq_lens, chan=prob.chan[0], Hq=w.Hq,
                          Hkv=w.Hkv, d=w.d, P=w.page, units=u, nthreads=cores)
            t_attn += time.perf_counter() - t
            slots_done += sum(int(prob.seq_lens[b]) for b, _ in u)
            units_done += len(u)
            i += step
    else:
        from tests import _oracle_side as H  # per-unit regeneration for pools too big for host RAM
        i = 0
        while i < len(units_all) and t_attn < budget_s / 2:
            b, hq = units_all[i]
            t = time.perf_counter()
            H.oracle_attn_unit(prob, 0, b, hq)
            t_attn += time.perf_counter() - t
            slots_done += int(prob.seq_lens[b])
            units_done += 1
            i += 1
    slots_total = int(sum(int(s) for s in prob.seq_lens)) * w.Hq
    attn_step = w.L * t_attn * slots_total / max(slots_done, 1)
    # the pool: whole tokens until the budget is spent
    h = prob.host("h")
    args = [prob.host(n) for n in ("pre_g", "Wr", "br", "ch_g", "Wkv", "qk_g")] \
        if w.D * w.D * w.k <= (1 << 27) else None
    t_mix, tok = 0.0, 0
    if args is not None:
        while tok < w.B and t_mix < budget_s / 2:
            # one token first (a wide model's pool costs seconds per token
            # group), then groups of one token per core while time is left
            n = 1 if tok == 0 else min(cores, w.B - tok)
            pos = (prob.seq_lens[tok:tok + n] - 1).astype(np.float64)
            t = time.perf_counter()
            O.kv_mix(h[tok:tok + n], pos, *args, L=w.L, k=w.k, D=w.D, Hkv=w.Hkv, d=w.d, p=w.p,
                     eps=w.eps_rms, eps_qk=w.eps_qk, theta=w.rope_theta, nthreads=cores)
            t_mix += time.perf_counter() - t
            tok += n
    mix_step = t_mix * w.B / tok if tok else 0.0
    sample = (f"layer 0 attention for {units_done} of {len(units_all)} (sequence, head) units "
              f"({slots_done} slot reads), extrapolated by slots x {w.L} layers; pool for "
              f"{tok} of {w.B} tokens, extrapolated by tokens")
    return attn_step + mix_step, cores, sample


def oracle_prefill_estimate(prob, T: int, g: int, budget_s: float = 4.0):
    """Time the fp64 oracle on a bounded sample of query rows of a prefill
    pass and extrapolate by work (a row at position i reads i + 1 slots) to
    every row, head and layer.  Returns (seconds per pass, cores, sample)."""
    import numpy as np
    from tests import _oracle_side as H
    from wm_synth import gen
    from wm_synth.inputs import STREAM_Q_PREFILL
    w = prob.w
    rng = np.random.default_rng(0)
    t_used, work, rows = 0.0, 0, 0
    while t_used < budget_s:
        b, pos, hq = int(rng.integers(w.B)), int(rng.integers(T)), int(rng.integers(w.Hq))
        qv = gen.values(w.dtype, 0, STREAM_Q_PREFILL, rows * w.d, w.d, w.q_scale)
        t = time.perf_counter()
        H.oracle_prefill_unit(prob, 0, b, pos, (hq, qv))
        t_used += time.perf_counter() - t
        work += pos + 1
        rows += 1
    total = w.L * w.B * w.Hq * T * (T + 1) / 2.0
    sample = (f"{rows} query rows at random positions (one head, layer 0; {work} slot reads), "
              f"extrapolated by slots read to {w.L} layers x {w.B} sequences x {w.Hq} heads "
              f"x {T} positions")
    return t_used * total / max(work, 1), 1, sample


def oracle_pool_estimate(prob, budget_s: float = 4.0, nthreads: int | None = None):
    """Time the fp64 oracle's pool on whole tokens until the budget is spent
    and extrapolate to B tokens.  Returns (seconds per pool, cores, sample)."""
    import numpy as np
    from oracle import oracle as O
    w = prob.w
    cores = nthreads or len(os.sched_getaffinity(0))
    args = [prob.host(n) for n in ("pre_g", "Wr", "br", "ch_g", "Wkv", "qk_g")]
    hall = prob.host("h")
    t_mix, tok = 0.0, 0
    while tok < w.B and t_mix < budget_s:
        n = min(cores, w.B - tok)
        h = hall[tok:tok + n]
        pos = (prob.seq_lens[tok:tok + n] - 1).astype(np.float64)
        t = time.perf_counter()
        O.kv_mix(h, pos, *args, L=w.L, k=w.k, D=w.D, Hkv=w.Hkv, d=w.d, p=w.p, eps=w.eps_rms,
                 eps_qk=w.eps_qk, theta=w.rope_theta, nthreads=cores)
        t_mix += time.perf_counter() - t
        tok += n
    return t_mix * w.B / max(tok, 1), cores, f"pool for {tok} of {w.B} tokens, extrapolated by tokens"


# ---------------------------------------------------------------- arms
REF_TOTAL_S = 120.0  # oracle seconds a whole --impl reference run may spend


def run_reference(args, w):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    from wm_synth.inputs import make_problem
    prob = make_problem(w, seed=0)
    full, walls = [], []
    cores, sample = None, ""
    # Every step is a bounded sample of one decode step (some attention units
    # of one layer and some tokens of the pool), timed as it runs; together
    # the steps stay within about REF_TOTAL_S of oracle time whatever --steps
    # asks for.  ms_per_step is the time of the sample actually run; value is
    # tokens/s of a whole step, extrapolated from that sample by the work it
    # covered (stated in cpu_baseline.sample).
    per_step = min(args.ref_budget, REF_TOTAL_S / max(1, args.warmup + args.steps))
    for i in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        t, cores, sample = oracle_step_estimate(prob, budget_s=per_step)
        wall = time.perf_counter() - t0
        if i >= args.warmup:
            full.append(t)
            walls.append(wall)
    step_s = statistics.median(full)
    value = w.B / step_s
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": statistics.median(walls) * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": config_dict(w, world),
            "extrapolated": {"ms_per_full_step": step_s * 1e3,
                             "note": "each timed step ran the bounded sample in cpu_baseline.sample; "
                                     "value is B tokens over the full step extrapolated from it"},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores,
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def config_dict(w, world):
    return {"workload": w.name, "L": w.L, "k": w.k, "D": w.D, "Hq": w.Hq, "Hkv": w.Hkv,
            "d": w.d, "batch_per_gpu": w.B, "global_batch": w.B * world,
            "context": w.ctx if not w.ctx_lo else f"U[{w.ctx_lo},{w.ctx}]", "page": w.page,
            "p": w.p, "channel_map": w.chan_map,
            "l2": "inputs larger than L2: each step reads every channel once (> 129 MB)",
            "parallelism": f"replicas x{world} (batch-sharded, no collective)",
            "launch": "timed steps captured once as a CUDA graph (programmatic dependent launch between kernels), replayed"}


def run_gpu(args, w):
    import numpy as np
    import torch
    import torch.distributed as dist

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1 and not dist.is_initialized():
        dist.init_process_group("nccl", device_id=dev)

    from paper_2608_18486_gb300 import _lib as W
    from paper_2608_18486_gb300 import make_config
    from paper_2608_18486_gb300.session import DecodeSession
    from wm_synth import configs as C
    from wm_synth.device_problem import DeviceProblem

    prob = rank_problem(w, rank)  # each replica decodes its own sequences
    cfg = make_config(w.L, w.k, w.D, w.Hq, w.Hkv, w.d, w.p, w.page, w.dtype, w.chan_of_layer(),
                      w.eps_rms, w.eps_qk, w.rope_theta)
    sess = DecodeSession(cfg, w.B, prob.num_pages, prob.max_pages, dev)
    dp = DeviceProblem(prob, sess.k_pool, sess.v_pool, dev)
    sess.set_weights(*dp.weights())
    stream = torch.cuda.Stream(dev)
    outs = torch.empty((w.L, w.B, w.Hq, w.d), dtype=sess.dtype, device=dev)
    torch.cuda.synchronize()

    def step(ev_attn=None):
        if ev_attn is not None:
            ev_attn[0].record(stream)
        for layer in range(w.L):
            # layers after the first read nothing the previous launch wrote but q
            sess.decode_attn(layer, dp.q[layer], dp.page_table, dp.seq_lens, outs[layer],
                             stream=stream, inputs_ready=layer > 0)
        if ev_attn is not None:
            ev_attn[1].record(stream)
        sess.kv_mix(dp.h, dp.page_table, dp.slot, stream=stream)

    def barrier():
        torch.cuda.synchronize(dev)
        if world > 1:
            dist.barrier()

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            step()
    barrier()
    if sess.read_status() != 0:
        raise RuntimeError("device status set during warm-up")

    # The timed steps run as one CUDA graph (captured after the eager warm-up,
    # replayed once untimed): the launch path then costs nothing on the host
    # and programmatic dependent launch chains every kernel.  Timing events
    # are graph nodes when this torch supports external events; otherwise the
    # attention and the pool of each step are separate graphs with events
    # between their replays.
    def new_event(external):
        if external:
            return torch.cuda.Event(enable_timing=True, external=True)
        return torch.cuda.Event(enable_timing=True)

    try:
        new_event(True)
        external = True
    except TypeError:
        external = False
    K = args.steps
    ev = [(new_event(external), new_event(external)) for _ in range(K)]
    if external:
        g_all = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g_all, stream=stream):
            for i in range(K):
                step(ev[i])

        def timed_region():
            g_all.replay()
    else:
        g_attn, g_mix = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
        with torch.cuda.graph(g_attn, stream=stream):
            for layer in range(w.L):
                sess.decode_attn(layer, dp.q[layer], dp.page_table, dp.seq_lens, outs[layer],
                                 stream=stream, inputs_ready=layer > 0)
        with torch.cuda.graph(g_mix, stream=stream):
            sess.kv_mix(dp.h, dp.page_table, dp.slot, stream=stream)

        def timed_region():
            for i in range(K):
                ev[i][0].record(stream)
                g_attn.replay()
                ev[i][1].record(stream)
                g_mix.replay()
    with torch.cuda.stream(stream):
        timed_region()  # untimed: uploads the graph(s)
    barrier()

    gpu_uuid = str(getattr(torch.cuda.get_device_properties(dev), "uuid", "") or local)
    if gpu_uuid and not gpu_uuid.startswith("GPU-") and len(gpu_uuid) > 8:
        gpu_uuid = "GPU-" + gpu_uuid
    sampler = ClockSampler(gpu_uuid) if rank == 0 else None
    time.sleep(0.3 if sampler else 0)
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    t0 = time.time()
    with torch.cuda.stream(stream):
        start.record(stream)
        timed_region()
        end.record(stream)
    barrier()
    t1 = time.time()
    clocks = sampler.stop(t0, t1) if sampler else None
    status = sess.read_status()
    if status != 0:
        raise RuntimeError(f"device status {status} during the timed region")
    ms = start.elapsed_time(end)
    attn_ms = sum(a.elapsed_time(b) for a, b in ev)
    ms, attn_ms = max_over_ranks([ms, attn_ms], world, dev)

    # ---- end to end through the public API with pinned host buffers: every
    # step copies its queries and hidden states in and all attention outputs
    # out; the K steps are one captured graph as above
    q_host = torch.empty(dp.q.shape, dtype=dp.q.dtype, pin_memory=True)
    q_host.copy_(dp.q)
    h_host = torch.empty(dp.h.shape, dtype=dp.h.dtype, pin_memory=True)
    h_host.copy_(dp.h)
    out_host = torch.empty(outs.shape, dtype=outs.dtype, pin_memory=True)
    e2e_steps = max(1, args.steps)

    def e2e_step():
        dp.q.copy_(q_host, non_blocking=True)
        dp.h.copy_(h_host, non_blocking=True)
        step()
        out_host.copy_(outs, non_blocking=True)

    g_e2e = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_e2e, stream=stream):
        for _ in range(e2e_steps):
            e2e_step()
    with torch.cuda.stream(stream):
        g_e2e.replay()
    barrier()
    e_start, e_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e_start.record(stream)
        g_e2e.replay()
        e_end.record(stream)
    barrier()
    e2e_ms = max_over_ranks([e_start.elapsed_time(e_end)], world, dev)[0]

    if rank == 0:
        tokens = w.B * world * args.steps
        value = tokens / (ms / 1e3)
        launch_bytes = C.attn_launch_bytes(w, prob.seq_lens)
        attn_launch_s = attn_ms / 1e3 / (args.steps * w.L)
        achieved = launch_bytes / attn_launch_s / 1e9
        peak, peak_kind = measured_peak()
        traffic = ncu_traffic(w.name)
        step_bytes = C.step_bytes(w, prob.seq_lens)
        cpu_s, cores, sample = oracle_step_estimate(prob, budget_s=args.ref_budget)
        line = {
            "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": w.dtype,
            "data": "synthetic", "config": config_dict(w, world),
            "roofline": {"bound": "hbm", "kernel": attn_kernel_name(cfg, w, prob), "achieved": achieved,
                         "peak": peak, "peak_kind": peak_kind, "unit": "GB/s",
                         "frac": achieved / peak, "traffic": traffic,
                         "algorithmic_bytes_per_launch": launch_bytes,
                         "avg_launch_us": attn_launch_s * 1e6},
            "step_hbm_gbs": step_bytes / (ms / 1e3 / args.steps) / 1e9,
            "attn_share_of_step": attn_ms / ms,
            "cpu_baseline": {"value": w.B / cpu_s, "unit": "tokens/s", "cores": cores,
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": w.B * world * e2e_steps / (e2e_ms / 1e3), "unit": "tokens/s",
                    "h2d_bytes_per_step": int(dp.q.numel() * dp.q.element_size()
                                              + dp.h.numel() * dp.h.element_size()),
                    "d2h_bytes_per_step": int(outs.numel() * outs.element_size())},
            "clocks": clocks,
            "gpu_launches": args.steps * (w.L + W.wm_kv_mix_launches(cfg, w.B)),
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


def run_model(args, w):
    """Whole-model decode step: random Qwen3-style blocks (Sec. 4.1) around the
    WhiteMatter path (tests/_model_step.py).  Per layer l: x = RMSNorm(h);
    q = RoPE(QKNorm(W_q x)); h += W_o * attention over channel c(l)
    (wm_decode_attn); h += SwiGLU MLP of RMSNorm(h).  The L states entering
    the layers then go through the pool (wm_kv_mix), as in Sec. 3.2.  The
    blocks are plain torch (cuBLAS GEMMs): they are outside the path and only
    give the path its real neighbours.  Prints one JSON line: whole-model
    tokens/s and the WhiteMatter share."""
    import torch
    from paper_2608_18486_gb300 import make_config
    from paper_2608_18486_gb300.session import DecodeSession
    from tests._model_step import ModelStep
    from wm_synth.device_problem import DeviceProblem

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    prob = rank_problem(w, 0)
    cfg = make_config(w.L, w.k, w.D, w.Hq, w.Hkv, w.d, w.p, w.page, w.dtype, w.chan_of_layer(),
                      w.eps_rms, w.eps_qk, w.rope_theta)
    sess = DecodeSession(cfg, w.B, prob.num_pages, prob.max_pages, dev)
    dp = DeviceProblem(prob, sess.k_pool, sess.v_pool, dev)
    sess.set_weights(*dp.weights())
    model = ModelStep(w, sess, dp, dev, args.intermediate)
    stream = torch.cuda.Stream(dev)

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            model.step(stream)
    torch.cuda.synchronize()
    K = args.steps
    evs = [[(torch.cuda.Event(enable_timing=True, external=True),
             torch.cuda.Event(enable_timing=True, external=True)) for _ in range(w.L + 1)]
           for _ in range(K)]
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        for i in range(K):
            model.step(stream, evs[i])
    with torch.cuda.stream(stream):
        graph.replay()
    torch.cuda.synchronize()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        start.record(stream)
        graph.replay()
        end.record(stream)
    torch.cuda.synchronize()
    if sess.read_status() != 0:
        raise RuntimeError("device status set during the model steps")
    ms = start.elapsed_time(end)
    attn_ms = sum(e[l][0].elapsed_time(e[l][1]) for e in evs for l in range(w.L))
    mix_ms = sum(e[w.L][0].elapsed_time(e[w.L][1]) for e in evs)
    line = {"metric": "whole-model decode tokens/s (random Qwen3-style blocks around the path)",
            "value": w.B * K / (ms / 1e3), "unit": "tokens/s", "n_gpus": 1, "steps": K,
            "warmup": args.warmup, "ms_per_step": ms / K, "higher_is_better": True,
            "dtype": w.dtype, "data": "synthetic",
            "config": dict(config_dict(w, 1), intermediate=model.I, mode="model"),
            "whitematter_share": (attn_ms + mix_ms) / ms,
            "attn_ms_per_step": attn_ms / K, "pool_ms_per_step": mix_ms / K}
    print(json.dumps(line), flush=True)


def gpu_uuid_of(dev, fallback):
    import torch
    u = str(getattr(torch.cuda.get_device_properties(dev), "uuid", "") or fallback)
    if u and not u.startswith("GPU-") and len(u) > 8:
        u = "GPU-" + u
    return u


def run_prefill(args, w):
    """One prefill pass of causal channel attention over every layer (Sec. 3.2
    dummy offset; Sec. 3.3 passes): for each layer, each of the g strided
    Gauss-Seidel groups {i mod g = q} of the T-token prompt (g = 1: one Jacobi
    pass) attends over its layer's channel.  The cache holds the dummy and T
    tokens per sequence.  Prints one JSON line: prompt tokens/s of the pass and
    the kernel's useful TFLOP/s (causal FLOPs only) against the measured bf16
    tensor peak."""
    import numpy as np
    import torch
    from paper_2608_18486_gb300 import make_config
    from paper_2608_18486_gb300.session import DecodeSession
    from wm_synth import device as wdev
    from wm_synth.device_problem import DeviceProblem
    from wm_synth.inputs import STREAM_Q_PREFILL, group_positions, make_problem

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    T, g = w.ctx, args.groups
    prob = make_problem(w, seed=0, seq_lens=[T] * w.B)
    cfg = make_config(w.L, w.k, w.D, w.Hq, w.Hkv, w.d, w.p, w.page, w.dtype, w.chan_of_layer(),
                      w.eps_rms, w.eps_qk, w.rope_theta)
    sess = DecodeSession(cfg, w.B, prob.num_pages, prob.max_pages, dev)
    dp = DeviceProblem(prob, sess.k_pool, sess.v_pool, dev)
    groups = []
    start_idx = 0
    for q in range(g):
        pos = torch.from_numpy(np.stack([group_positions(T, g, q)] * w.B)).to(dev)
        Tq = pos.shape[1]
        qt = torch.empty((w.B, Tq, w.Hq, w.d), dtype=sess.dtype, device=dev)
        wdev.fill(qt, w.dtype, 0, STREAM_Q_PREFILL, w.q_scale, 0.0, start=start_idx)
        start_idx += qt.numel()
        groups.append((qt, pos, torch.empty_like(qt)))
    stream = torch.cuda.Stream(dev)

    def step():
        for layer in range(w.L):
            for qt, pos, out in groups:
                sess.prefill_attn(layer, qt, pos, dp.page_table, out, stream=stream)

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            step()
    torch.cuda.synchronize()
    if sess.read_status() != 0:
        raise RuntimeError("device status set during warm-up")
    K = args.steps
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        for _ in range(K):
            step()
    with torch.cuda.stream(stream):
        graph.replay()
    torch.cuda.synchronize()
    sampler = ClockSampler(gpu_uuid_of(dev, "0"))
    time.sleep(0.3)
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0 = time.time()
    with torch.cuda.stream(stream):
        start.record(stream)
        graph.replay()
        end.record(stream)
    torch.cuda.synchronize()
    t1 = time.time()
    clocks = sampler.stop(t0, t1)
    if sess.read_status() != 0:
        raise RuntimeError("device status set during the timed region")
    ms = start.elapsed_time(end) / K
    flops = w.L * w.B * w.Hq * 4.0 * w.d * (T * (T + 1) / 2.0)  # sum over positions of pos + 1
    tflops = flops / (ms * 1e-3) / 1e12
    peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    peak = float(peaks["bf16_tflops_sustained"])
    line = {"metric": "prefill attention tokens/s (one pass over all layers; causal channel attention)",
            "value": w.B * T / (ms * 1e-3), "unit": "tokens/s", "n_gpus": 1, "steps": K,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "dtype": "bf16",
            "data": "synthetic",
            "config": dict(config_dict(w, 1), mode="prefill", prompt_tokens=T, groups=g,
                           launches_per_step=w.L * g),
            "roofline": {"bound": "tensor", "achieved": tflops, "peak": peak, "unit": "TFLOP/s",
                         "frac": tflops / peak, "peak_kind": "measured sustained bf16",
                         "flops_per_step": flops},
            "clocks": clocks, "gpu_launches": K * w.L * g}
    t_cpu, cores, sample = oracle_prefill_estimate(prob, T, g, budget_s=args.ref_budget)
    line["cpu_baseline"] = {"value": w.B * T / t_cpu, "unit": "tokens/s", "cores": cores,
                            "kind": "oracle", "sample": sample}
    print(json.dumps(line), flush=True)


def sess_launches(sess, B):
    from paper_2608_18486_gb300 import _lib as W
    return W.wm_kv_mix_launches(sess.cfg, B)


def run_pool(args, w):
    """The cross-layer KV pool (Sec. 3.1 Steps 1-2) over the B tokens of one
    batched evaluation: a prefill group of Sec. 3.3 hands the pool |G_q| x
    sequences tokens at once, and at that size the router and projection are
    real tensor-core GEMMs.  Prints one JSON line: pooled tokens/s and the
    contraction FLOP/s (router + K/V projections) against the measured bf16
    tensor peak."""
    import torch
    from paper_2608_18486_gb300 import make_config
    from paper_2608_18486_gb300.session import DecodeSession
    from wm_synth.device_problem import DeviceProblem
    from wm_synth.inputs import make_problem

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    prob = make_problem(w, seed=0)
    cfg = make_config(w.L, w.k, w.D, w.Hq, w.Hkv, w.d, w.p, w.page, w.dtype, w.chan_of_layer(),
                      w.eps_rms, w.eps_qk, w.rope_theta)
    sess = DecodeSession(cfg, w.B, prob.num_pages, prob.max_pages, dev)
    dp = DeviceProblem(prob, sess.k_pool, sess.v_pool, dev)
    sess.set_weights(*dp.weights())
    stream = torch.cuda.Stream(dev)

    def step():
        sess.kv_mix(dp.h, dp.page_table, dp.slot, stream=stream)

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            step()
    torch.cuda.synchronize()
    if sess.read_status() != 0:
        raise RuntimeError("device status set during warm-up")
    K = args.steps
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        for _ in range(K):
            step()
    with torch.cuda.stream(stream):
        graph.replay()
    torch.cuda.synchronize()
    sampler = ClockSampler(gpu_uuid_of(dev, "0"))
    time.sleep(0.3)
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0 = time.time()
    with torch.cuda.stream(stream):
        start.record(stream)
        graph.replay()
        end.record(stream)
    torch.cuda.synchronize()
    t1 = time.time()
    clocks = sampler.stop(t0, t1)
    if sess.read_status() != 0:
        raise RuntimeError("device status set during the timed region")
    ms = start.elapsed_time(end) / K
    # two branches: router kL x L'D and k projections of Hkv*d x D, 2 FLOP per MAC
    flops = 2.0 * 2.0 * w.B * (w.k * w.L * w.Lp * w.D + w.k * w.Hkv * w.d * w.D)
    tflops = flops / (ms * 1e-3) / 1e12
    peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    peak = float(peaks["bf16_tflops_sustained"])
    from wm_synth import configs as wcfg
    line = {"metric": "batched pool tokens/s (router + K/V projections + cache write, one evaluation)",
            "value": w.B / (ms * 1e-3), "unit": "tokens/s", "n_gpus": 1, "steps": K,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "dtype": w.dtype,
            "data": "synthetic", "config": dict(config_dict(w, 1), mode="pool", tokens=w.B),
            "roofline": {"bound": "tensor", "achieved": tflops, "peak": peak, "unit": "TFLOP/s",
                         "frac": tflops / peak, "peak_kind": "measured sustained bf16",
                         "flops_per_step": flops, "bytes_per_step": wcfg.mix_bytes(w)},
            "clocks": clocks, "gpu_launches": K * sess_launches(sess, w.B)}
    t_cpu, cores, sample = oracle_pool_estimate(prob, budget_s=args.ref_budget)
    line["cpu_baseline"] = {"value": w.B / t_cpu, "unit": "tokens/s", "cores": cores,
                            "kind": "oracle", "sample": sample}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None,
                    help="timed steps (default: about TARGET_TIMED_S of work, 10..200)")
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--mode", default="path", choices=["path", "model", "prefill", "pool"],
                    help="path: the WhiteMatter decode hot path (default); model: a whole-model "
                         "decode step; prefill: causal channel attention of a prefill pass; "
                         "pool: one batched pool evaluation over B tokens")
    ap.add_argument("--groups", type=int, default=8,
                    help="--mode prefill: strided Gauss-Seidel groups (1: a Jacobi pass)")
    ap.add_argument("--intermediate", type=int, default=0,
                    help="MLP width for --mode model (default 3*D)")
    ap.add_argument("--ref-budget", type=float, default=4.0,
                    help="seconds of oracle time per reference/CPU-baseline sample")
    ap.add_argument("--set", action="append", default=[], metavar="FIELD=VALUE",
                    help="override a workload field, e.g. --set k=1 (smaller cache for profiling)")
    args = ap.parse_args()
    from wm_synth import configs
    w = configs.get(args.workload)
    for kv in args.set:
        key, val = kv.split("=", 1)
        cur = getattr(w, key)
        w = w.with_(**{key: type(cur)(val) if not isinstance(cur, bool) else val == "1"})
    if args.set:
        w = w.with_(name=w.name + "[" + ",".join(args.set) + "]")
    if args.warmup < 3 and args.impl != "reference":
        args.warmup = 3
    if args.steps is None:
        args.steps = default_steps(w)
    if args.impl == "reference":
        run_reference(args, w)
    elif args.mode == "model":
        run_model(args, w)
    elif args.mode == "prefill":
        run_prefill(args, w)
    elif args.mode == "pool":
        run_pool(args, w)
    else:
        run_gpu(args, w)


if __name__ == "__main__":
    main()
