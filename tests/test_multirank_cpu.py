"""The benchmark's multi-rank host logic on CPU with the gloo backend (world size 2): the
max-over-ranks timing reduction, the barrier and the weak-scaling aggregate. No GPU and no
data-path collective are involved: ranks score independent batches."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms = [120.0, 150.0][rank]  # rank 1 is the slower one
    bench.barrier(world)
    ms_max = bench.max_over_ranks(ms, world)
    value = bench.aggregate(2048, 10, world, ms_max)
    q.put((rank, ms_max, value))
    bench.barrier(world)
    dist.destroy_process_group()


def test_max_over_ranks_and_weak_scaling_aggregate():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(2))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, ms_max, value in res:
        assert ms_max == 150.0
        assert value == pytest.approx(2048 * 10 * 2 / 0.150)


def test_single_rank_is_identity():
    import bench
    assert bench.max_over_ranks(3.5, 1) == 3.5
    assert bench.aggregate(100, 4, 1, 200.0) == pytest.approx(2000.0)


def _moments_worker(rank, world, port, q):
    """Each rank holds one shard of an advantage batch, computes its (n, mean, M2), and the
    library's all-reduce merges them; every rank must get the whole batch's moments."""
    import numpy as np
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from paper_2309_00754_gb300 import hydra as H
    rng = np.random.default_rng(11)
    adv = rng.normal(0.5, 1.7, (6, 9))
    lengths = np.array([9, 3, 0, 7, 9, 1])
    rows = slice(0, 2) if rank == 0 else slice(2, 6)
    a, ln = adv[rows], lengths[rows]
    v = a[np.arange(9)[None, :] < ln[:, None]]
    mine = torch.tensor([len(v), v.mean(), ((v - v.mean()) ** 2).sum()], dtype=torch.float64)
    H.all_reduce_adv_moments(mine)
    q.put((rank, mine.tolist()))
    dist.barrier()
    dist.destroy_process_group()


def test_all_reduce_adv_moments_gloo():
    import numpy as np
    import oracle.hydra_oracle as O
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_moments_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(2))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    rng = np.random.default_rng(11)
    adv = rng.normal(0.5, 1.7, (6, 9))
    lengths = np.array([9, 3, 0, 7, 9, 1])
    z = np.zeros_like(adv)
    ref = O.ppo_loss(z, z, adv, z, z, lengths)
    assert res[0][1] == res[1][1]  # the same bits on every rank
    n, mean, m2 = res[0][1]
    assert n == ref["n"]
    assert abs(mean - ref["adv_mean"]) < 1e-13
    assert abs(np.sqrt(m2 / n) - ref["adv_std"]) < 1e-13


def test_blas_thread_control_sets_and_restores():
    # the CPU baseline's single-thread leg drives numpy's OpenBLAS through its own setter
    import bench
    ctl = bench.blas_thread_control()
    if ctl is None:
        pytest.skip("numpy is not linked against an OpenBLAS with a thread setter here")
    get, set_ = ctl
    prev = get()
    try:
        set_(1)
        assert get() == 1
    finally:
        set_(prev)
    assert get() == prev
