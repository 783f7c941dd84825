"""The multi-replica path of the benchmark (one process per GPU, no collective on the
data path) on the CPU: two gloo ranks check the barrier, the max-over-ranks timing and
the whole-job throughput arithmetic, and that each rank's replica draws its own sample."""

import os
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _worker(rank, world, port, out):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import torch.distributed as dist

    import bench
    from paper_2608_09231_gb300 import configs, synth
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ws, r, local = bench._dist()
    bench.replica_barrier(ws)
    ms_local = 100.0 + 50.0 * r           # the slower replica decides the job's time
    ms = bench.max_over_ranks(ms_local, ws)
    cfg = configs.get_config("tiny")
    x = synth.make_inputs(cfg, sample_seed=r)["x"]
    out[r] = (ws, r, local, ms, bench.job_seconds_per_sample(ms, ws), float(x[0, 0]))
    dist.destroy_process_group()


@pytest.mark.parametrize("world", [2])
def test_two_gloo_replicas(world):
    port = 29500 + (os.getpid() % 2000)
    with mp.get_context("spawn").Manager() as m:
        out = m.dict()
        mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    assert sorted(res) == list(range(world))
    for r, (ws, rank, local, ms, sps, _) in res.items():
        assert (ws, rank, local) == (world, r, r)
        assert ms == 150.0                       # max over ranks
        assert sps == 150.0 / 1e3 / world        # two samples per slowest step
    assert res[0][5] != res[1][5]                # independent samples per replica


def test_single_process_path():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(3.5, 1) == 3.5
    assert bench.job_seconds_per_sample(1200.0, 1) == 1.2
