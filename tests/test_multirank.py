"""The multi-rank host logic of bench.py on CPU ranks (gloo, world size 2): process
group set-up from the torchrun environment, the timing barrier, the max over ranks and
the whole-job rate, and the reference arm's rank-0-only rule."""
import os
import socket

import pytest
import torch
import torch.multiprocessing as mp


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import bench
    import torch.distributed as dist
    r, w, local = bench.dist_init(world)
    assert (r, w, local) == (rank, world, rank)
    assert dist.get_backend() == "gloo"
    bench.barrier(w)
    # per-rank timings: the job is as slow as its slowest rank
    mine = 10.0 + 5.0 * rank
    slowest = bench.max_over_ranks(mine, w)
    rate = bench.whole_job_rate(1000, 4, w, slowest)
    out.put((rank, slowest, rate))
    dist.destroy_process_group()


@pytest.mark.skipif(torch.cuda.is_available(), reason="CPU ranks only")
def test_two_cpu_ranks_barrier_max_and_rate():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=5) for _ in range(world))
    for rank, slowest, rate in res:
        assert slowest == 15.0
        assert rate == pytest.approx(1000 * 4 * 2 / 0.015)


def test_whole_job_rate_is_weak_scaling():
    import bench
    one = bench.whole_job_rate(100, 10, 1, 2.0)
    four = bench.whole_job_rate(100, 10, 4, 2.0)
    assert four == pytest.approx(4 * one)


def test_reference_arm_runs_on_rank_zero_only(capsys, monkeypatch):
    import bench
    monkeypatch.setenv("RANK", "1")

    class A:
        workload, ref_frames, steps, warmup, gpus = "tiny", 4, 1, 0, 2
    bench.run_reference(A())
    assert capsys.readouterr().out == ""
