"""Multi-rank host logic of bench.py on CPU (gloo, world_size 2).

The layer does not shard: `bench.py --gpus N` runs N independent replicas and
only aggregates timings across ranks (max of the per-rank times, sum of the
work).  These checks run that aggregation over a real process group on the
CPU, and check that the reference arm prints only on rank 0.
"""

import os
import socket
import sys

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ws, r, local = bench.dist_env()
    assert (ws, r, local) == (world, rank, rank)
    t_max = bench.max_over_ranks(1.0 + rank, ws)
    w_sum = bench.sum_over_ranks(10.0 * (rank + 1), ws)
    out[rank] = (t_max, w_sum)
    dist.barrier()
    dist.destroy_process_group()


def test_rank_aggregation_gloo():
    world = 2
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    for rank in range(world):
        t_max, w_sum = res[rank]
        assert t_max == 2.0          # the slowest rank decides the time
        assert w_sum == 30.0         # the work of all ranks counts


def test_single_rank_aggregation_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(3.5, 1) == 3.5
    assert bench.sum_over_ranks(7.0, 1) == 7.0


def test_reference_arm_prints_on_rank_zero_only(monkeypatch, capsys):
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("RANK", "1")
    assert bench.main(["--impl", "reference", "--gpus", "2", "--steps", "3", "--warmup", "3"]) == 0
    assert capsys.readouterr().out == ""


def test_warmup_must_be_at_least_three():
    sys.path.insert(0, ROOT)
    import bench
    with pytest.raises(SystemExit):
        bench.main(["--warmup", "2"])
