"""Multi-rank host logic of bench.py on CPU (gloo, world size 2).

The decode path shards by sequence: each replica decodes its own batch with
no data exchange, and torch.distributed carries only the timing barrier and
the max over ranks.  These tests run that host logic as two gloo ranks.
"""
import os
import socket

import numpy as np
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        from wm_synth import configs
        r, w, _ = bench.dist_env()
        assert (r, w) == (rank, world)
        wl = configs.get("large").with_(B=4)
        prob = bench.rank_problem(wl, rank)
        # rank-specific timings; every rank must see the same maximum
        mx = bench.max_over_ranks([10.0 + rank, 5.0 - rank], world)
        q.put((rank, prob.seq_lens.tolist(), prob.page_table[:, :3].tolist(), mx))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_shard_by_sequence_and_take_the_max_time():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, lens0, pt0, mx0), (r1, lens1, pt1, mx1) = res
    assert mx0 == mx1 == [11.0, 5.0]
    # replicas decode different sequences (own seeds), with no shared state
    assert lens0 != lens1 or pt0 != pt1


def test_reference_arm_runs_on_rank_zero_only(capsys):
    import bench
    from wm_synth import configs
    os.environ["RANK"], os.environ["WORLD_SIZE"] = "1", "2"
    try:
        class A:
            steps, warmup, ref_budget = 1, 0, 0.1
        bench.run_reference(A, configs.get("tiny_f32"))
        assert capsys.readouterr().out == ""
    finally:
        os.environ.pop("RANK")
        os.environ.pop("WORLD_SIZE")
    assert np.isfinite(bench.max_over_ranks([1.5], 1)[0])
