"""The multi-process path of bench.py on the CPU (the step does not shard, so N GPUs run N
replicas): two gloo ranks reduce their step times to the slowest rank's, the job value counts
every replica's samples over that time, and the reference arm's other ranks exit without
output."""
import os
import socket
import types

import pytest
import torch.multiprocessing as mp

import bench


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import torch.distributed as dist
    import bench as b
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        assert b.rank_env() == (world, rank, rank)
        # rank 0 is slower on the first and third value, rank 1 on none of them
        mine = [3.0 - rank, 5.0 - 2 * rank, 1.25 + 0.5 * (1 - rank)]
        out[rank] = b.max_over_ranks(dist, mine, "cpu")
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_reduce_to_the_slowest_rank():
    world, port = 2, _free_port()
    with mp.Manager() as manager:
        out = manager.dict()
        mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    assert res[0] == res[1] == [3.0, 5.0, 1.75]
    # every replica's 32 samples over the slowest replica's 3 ms step
    assert bench.job_value(world, 32, res[0][0]) == pytest.approx(2 * 32 / 0.003)


def test_single_process_defaults(monkeypatch):
    for k in ("WORLD_SIZE", "RANK", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)
    assert bench.rank_env() == (1, 0, 0)
    assert bench.max_over_ranks(None, [1, 2.5], "cpu") == [1.0, 2.5]
    assert bench.job_value(1, 32, 2.0) == pytest.approx(16000.0)


def test_reference_arm_other_ranks_exit_quietly(monkeypatch, capsys):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    args = types.SimpleNamespace(config="base", steps=3, warmup=1, gpus=2)
    assert bench.reference_main(args) == 0
    assert capsys.readouterr().out == ""
