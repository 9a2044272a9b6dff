"""The multi-rank path of the benchmark on CPU (gloo, world size 2): each
rank resolves its own gradient set (the buckets are independent units,
Section 3.2), so the only cross-rank step is the timing reduction -- the
slowest rank's time and the sum of all ranks' bytes -- and the reference arm
runs on rank 0 alone."""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    import torch
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms = [10.0, 12.5][rank]
    nbytes = [4e9, 6e9][rank]
    got = bench.reduce_over_ranks(ms, nbytes, torch.device("cpu"))
    ws, r, local = bench._dist()
    q.put((rank, got, (ws, r, local)))
    dist.barrier()
    dist.destroy_process_group()


@pytest.mark.timeout(120)
def test_reduce_over_ranks_gloo_world2():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=100) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, (ms, gbs), dist_env in res:
        assert ms == 12.5                                   # slowest rank
        assert abs(gbs - 10e9 / 12.5e-3 / 1e9) < 1e-9       # all ranks' bytes
        assert dist_env == (2, rank, rank)


def test_reduce_over_ranks_single_process():
    import torch
    sys.path.insert(0, ROOT)
    import bench
    ms, gbs = bench.reduce_over_ranks(20.0, 8e9, torch.device("cpu"))
    assert ms == 20.0 and abs(gbs - 400.0) < 1e-9


def test_reference_arm_other_ranks_exit_without_work(monkeypatch, capsys):
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")

    class A:
        workload = "tiny"
        warmup = 3
        steps = 1
        gpus = 2

    bench.run_reference(A())       # returns at once on rank 1
    assert capsys.readouterr().out == ""
