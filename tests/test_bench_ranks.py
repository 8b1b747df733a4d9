"""The multi-rank host logic of bench.py on two gloo ranks (CPU).

The pass does not shard: under torchrun each rank compresses its own request
on its own GPU, with no collective on the data path.  What the ranks share is
the measurement: the job's time is the slowest rank's (an all-reduce MAX of
the timed region), the value counts every rank's tokens, and the reference
arm runs on rank 0 alone.
"""
import socket
import types

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, times, q):
    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank,
                            world_size=world)
    try:
        ms = bench.max_over_ranks(times[rank], dist, "cpu")
        q.put((rank, ms, bench.whole_job_rate(world, 131072, 5, ms / 1e3)))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_ranks_report_the_slowest_rank_and_count_both_requests():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    times = [120.0, 180.0]
    ps = [ctx.Process(target=_rank, args=(r, 2, port, times, q)) for r in range(2)]
    for p in ps:
        p.start()
    out = sorted(q.get(timeout=180) for _ in range(2))
    for p in ps:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r for r, _, _ in out] == [0, 1]
    for _, ms, value in out:
        assert ms == 180.0
        assert value == pytest.approx(2 * 131072 * 5 / 0.180)


def test_one_rank_needs_no_process_group():
    import bench
    assert bench.max_over_ranks(42.5, None, "cpu") == 42.5
    assert bench.whole_job_rate(1, 1000, 4, 2.0) == 2000.0


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    import bench
    monkeypatch.setenv("RANK", "1")
    args = types.SimpleNamespace(warmup=3, steps=1, ratio=32.0, ref_tokens=256, gpus=2)
    bench.run_reference(args, None)          # returns before touching the workload
    assert capsys.readouterr().out == ""
