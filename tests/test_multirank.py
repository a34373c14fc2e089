"""The multi-GPU path of bench.py on CPU: two gloo ranks run the timing
aggregation (max over ranks, whole-job throughput) and draw distinct,
reproducible batches, with no collective on the data path."""
import os
import socket

import numpy as np
import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    from workloads import make_workload
    ms = 100.0 + 25.0 * rank                     # each rank's own elapsed time
    agg = bench.max_over_ranks(ms, world, torch.device("cpu"))
    w = make_workload("tiny", with_tensors=False, seed=bench.rank_seed(None, rank, world))
    out[rank] = (agg, bench.job_throughput(512, world, 10, agg), int(w.tokens[:64].sum()))
    dist.barrier()
    dist.destroy_process_group()


def test_two_ranks_aggregate_and_shard():
    world = 2
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_worker, args=(world, _free_port(), out), nprocs=world, join=True)
    (a0, v0, s0), (a1, v1, s1) = out[0], out[1]
    assert a0 == a1 == 125.0                      # slowest rank
    assert v0 == v1 == pytest.approx(2 * 512 * 10 / 0.125)
    assert s0 != s1                               # each rank draws its own batch


def test_single_rank_is_identity():
    import bench
    assert bench.max_over_ranks(42.0, 1) == 42.0
    assert bench.rank_seed(None, 0, 1) is None
    assert bench.job_throughput(65536, 1, 10, 1000.0) == pytest.approx(655360.0)


def test_cpu_baseline_reports_the_blas_threads(monkeypatch):
    """cpu_baseline's `cores` is the thread count numpy's BLAS gets: the host
    cores, capped by a thread-count variable such as the OMP_NUM_THREADS=1 that
    torchrun gives every rank."""
    import bench
    for k in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
        monkeypatch.delenv(k, raising=False)
    n = os.cpu_count() or 1
    assert bench.blas_threads() == n
    monkeypatch.setenv("OMP_NUM_THREADS", "1")
    assert bench.blas_threads() == 1
    monkeypatch.setenv("OPENBLAS_NUM_THREADS", str(n + 7))
    assert bench.blas_threads() == n
