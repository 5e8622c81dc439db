"""The multi-GPU path of bench.py is replicas only (every rank trains its own
batch, no data-path collective). Its host logic, on CPU with two gloo ranks:
each rank draws a different batch, the job's step time is the slowest
rank's, and the throughput counts every rank's samples."""

import importlib.util
import os
import socket

import numpy as np
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    m = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(m)
    return m


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    import torch
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        bench = _bench()
        from paper_2607_14672_gb300 import configs
        assert bench.dist_env() == (rank, world, rank)
        cfg = configs.config2(batch=8)
        t0, lab = bench.rank_batch(cfg, rank)
        digest = torch.tensor([float(np.nansum(np.where(np.isfinite(t0), t0, 0.0))), float(lab.sum())])
        all_d = [torch.zeros(2) for _ in range(world)]
        dist.all_gather(all_d, digest)
        ms = 1.0 + rank                     # rank 1 is the slower one
        job_ms = bench.max_over_ranks(ms, world)
        value = bench.job_throughput(world, cfg["batch"], job_ms)
        out[rank] = (all_d[0].tolist(), all_d[1].tolist(), job_ms, value)
    finally:
        dist.destroy_process_group()


def test_two_replicas_on_gloo():
    world, port = 2, _free_port()
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    assert set(res) == {0, 1}
    for r in (0, 1):
        d0, d1, job_ms, value = res[r]
        assert d0 != d1                     # different batches per rank
        assert job_ms == 2.0                # the slowest rank's time
        assert value == 2 * 8 / (2.0 / 1000.0)
    assert res[0][:2] == res[1][:2]         # every rank saw the same gathered digests
