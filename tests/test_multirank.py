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


def _vp_worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import paper_2607_21653_gb300 as molt
    from oracle import molt_oracle as O
    rng = np.random.default_rng(5)                     # the same problem on every rank
    T, H, V = 40, 12, 301
    h = rng.standard_normal((T, H))
    W = rng.standard_normal((V, H)) * 0.5
    x = rng.integers(0, V, T)
    a, e = molt.vocab_shard_bounds(V, world)[rank]
    rows = np.arange(T)
    local = torch.from_numpy(O.shard_partials(h, W[a:e], x, a, rows).astype(np.float32))
    parts = molt.gather_shard_partials(local)
    lse, logp, ent = O.merge_shard_partials(parts.double().numpy())
    coef = rng.standard_normal(T) * 0.01
    term = torch.from_numpy(O.shard_dhidden(h, W[a:e], x, a, lse, coef, rows))
    dh = molt.sum_dhidden(term)
    out[rank] = (parts.numpy(), lse, logp, ent, dh.numpy(), h, W, x, coef)
    dist.barrier()
    dist.destroy_process_group()


def test_vocab_parallel_exchange_two_ranks():
    """The host exchange of the vocabulary-parallel step on two gloo ranks:
    each rank's shard statistics gathered in rank order merge into the whole
    row's lse / logp / entropy (fp32 statistics, as the library exchanges
    them), and the ranks' dhidden terms sum to the full-vocabulary dhidden."""
    from oracle import molt_oracle as O
    world = 2
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_vp_worker, args=(world, _free_port(), out), nprocs=world, join=True)
    parts0, lse0, lp0, ent0, dh0, h, W, x, coef = out[0]
    parts1, lse1, lp1, ent1, dh1 = out[1][:5]
    np.testing.assert_array_equal(parts0, parts1)             # every rank holds the same stack
    assert parts0.shape == (2, 40, 4)
    np.testing.assert_array_equal(lse0, lse1)
    lse, lp, ent = O.full_forward_rows(h, W, x, np.arange(40))
    np.testing.assert_allclose(lse0, lse, atol=1e-5)
    np.testing.assert_allclose(lp0, lp, atol=1e-5)
    np.testing.assert_allclose(ent0, ent, atol=1e-5)
    np.testing.assert_array_equal(dh0, dh1)
    full_dh = O.shard_dhidden(h, W, x, 0, lse0, coef, np.arange(40))
    np.testing.assert_allclose(dh0, full_dh, rtol=1e-9, atol=1e-12)
