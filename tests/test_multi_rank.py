"""The N > 1 host path of bench.py on CPU: two gloo ranks draw disjoint
sequences, take the slowest rank's time and report whole-job throughput.
The ranks exchange nothing but that one timing value."""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    from paper_2608_26112_gb300 import synth
    wl = synth.make_workload("tiny", seed=bench.rank_seed(0, rank), with_strong=False)
    t_local = 1.0 + 0.5 * rank                      # this rank's timed-region seconds
    bench.barrier(world)
    t_max = bench.max_over_ranks(t_local, world)
    out[rank] = dict(t_max=t_max, value=bench.job_throughput(world, 100, t_max),
                     q_sum=float(np.asarray(wl["q"], dtype=np.float64).sum()),
                     parent=wl["parent"].tolist())
    dist.destroy_process_group()


@pytest.mark.timeout(120)
def test_two_gloo_ranks_weak_scaling():
    world = 2
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_rank_main, args=(world, _free_port(), out), nprocs=world, join=True)
        res = dict(out)
    assert sorted(res) == [0, 1]
    # the job time is the slowest rank's; throughput counts both ranks' steps
    assert res[0]["t_max"] == res[1]["t_max"] == 1.5
    assert res[0]["value"] == pytest.approx(2 * 100 / 1.5)
    # the ranks work on different sequences
    assert res[0]["q_sum"] != res[1]["q_sum"]


def test_single_rank_is_identity():
    import bench
    assert bench.max_over_ranks(2.5, 1) == 2.5
    assert bench.job_throughput(1, 10, 2.0) == 5.0
    assert bench.rank_seed(7, 0) == 7 and bench.rank_seed(7, 3) == 3007
