"""The multi-GPU path of the benchmark on CPU: N independent replicas (one
batch of requests per rank, no collective on the data path) report the
slowest rank's time and the sets all ranks scored. Two gloo ranks stand in for
two GPUs; the reference arm runs on rank 0 only."""
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    # rank r took (r + 1) * 10 ms for 5 steps of 16 requests; e2e 20 ms per step
    out = bench.aggregate(10.0 * (rank + 1), 20.0 + rank, 16, 5, world)
    q.put((rank, out))
    dist.barrier()
    dist.destroy_process_group()


def test_replicas_report_slowest_rank_and_whole_job_throughput():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    world, port = 2, _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = dict(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r in range(world):
        total_ms, e2e_ms, ms_per_step, value, e2e_value = res[r]
        assert total_ms == 20.0 and e2e_ms == 21.0           # max over ranks
        assert ms_per_step == pytest.approx(4.0)
        assert value == pytest.approx(2 * 16 / 4e-3)        # all ranks' sets / slowest time
        assert e2e_value == pytest.approx(2 * 16 / 21e-3)


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    total_ms, e2e_ms, ms_per_step, value, _ = bench.aggregate(8.0, 9.0, 16, 4, 1)
    assert (total_ms, ms_per_step, value) == (8.0, 2.0, pytest.approx(8000.0))


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("RANK", "1")

    class Args:
        workload = "tiny"
        R = 0
        ref_sample = 1
        steps = 1
        warmup = 3
    bench.run_reference(Args())
    assert capsys.readouterr().out == ""   # the other ranks print nothing and do no work
