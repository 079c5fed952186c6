"""The multi-rank host logic of bench.py on CPU (gloo, world size 2).

The path has no cross-rank exchange: each rank runs its own replica of the
cache (weak scaling), and the only collectives are the timing barrier and the
max over ranks of the step time.  These run here with the gloo backend; the
reference arm leaves every rank but rank 0 without work.
"""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, times, q):
    import torch.distributed as dist
    import bench
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        dist.barrier()
        slowest = bench.max_over_ranks(times[rank], dist, "cpu")
        q.put((rank, slowest, bench.whole_job_gbs(world, 1e9, slowest)))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_and_whole_job_value():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    times = [0.75, 1.25]  # ms per step on rank 0 and rank 1
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, times, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    # both ranks see the slower rank's time; the job moves 2 x 1 GB in 1.25 ms
    assert [o[1] for o in out] == [1.25, 1.25]
    assert out[0][2] == pytest.approx(2 * 1e9 / 1.25e-3 / 1e9)


def test_single_rank_is_unchanged():
    import bench
    assert bench.max_over_ranks(3.5, None, "cpu") == 3.5
    assert bench.whole_job_gbs(1, 2e9, 1.0) == pytest.approx(2000.0)


def test_reference_arm_other_ranks_do_no_work(monkeypatch, capsys):
    import bench
    monkeypatch.setenv("RANK", "1")
    args = bench.parse_args_from(["--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "0"])
    assert bench.run_reference(args) == 0
    assert capsys.readouterr().out == ""
