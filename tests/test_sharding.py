"""Scenario sharding over ranks, checked on the CPU with two gloo processes.

Each rank composes its own contiguous slice of one scenario batch (here with the
CPU oracle, as no GPU is needed to check the rank logic); rank 0 gathers the
results, which must equal the composition of the whole batch in one process.
"""
import os
import socket

import numpy as np
import pytest

from paper_2412_12487_gb300 import sharding as SH
from paper_2412_12487_gb300 import workloads as W

N_TOTAL = 7


def _free_port():
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _batch():
    c = W.config("tiny")
    c = W.GPTConfig(**{**c.__dict__, "fixed_scenario": False})
    g = W.build_gpt_graph(c)
    return g, W.make_scenarios(g, c, n_scen=N_TOTAL)


def _worker(rank, world, port, out_path):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    import torch.distributed as dist
    import oracle
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        g, full = _batch()
        s0, s1 = SH.shard_bounds(N_TOTAL, world, rank)
        res = oracle.compose(g, SH.slice_scenarios(full, s0, s1), refine_passes=1)
        mk = SH.gather_scenarios(res.makespan, N_TOTAL)
        fin = SH.gather_scenarios(res.finish, N_TOTAL)
        ov = SH.gather_scenarios(res.overlapped, N_TOTAL)
        t = SH.max_over_ranks([float(rank), 10.0 - rank, float(s1 - s0)])
        if rank == 0:
            np.savez(out_path, mk=mk, fin=fin, ov=ov, t=np.array(t))
        else:
            assert mk is None and fin is None
    finally:
        dist.destroy_process_group()


def test_shard_bounds_partition_the_batch():
    for n in (0, 1, 5, 7, 1024, 1025):
        for world in (1, 2, 3, 8):
            b = [SH.shard_bounds(n, world, r) for r in range(world)]
            assert b[0][0] == 0 and b[-1][1] == n
            assert all(b[r][1] == b[r + 1][0] for r in range(world - 1))
            sizes = [e - s for s, e in b]
            assert max(sizes) - min(sizes) <= 1
    with pytest.raises(ValueError):
        SH.shard_bounds(4, 2, 2)


def test_slice_scenarios_takes_columns():
    g, full = _batch()
    part = SH.slice_scenarios(full, 2, 5)
    assert part.n_scen == 3
    assert np.array_equal(part.dur, full.dur[:, 2:5])
    assert np.array_equal(part.slowdown, full.slowdown[:, 2:5])
    assert np.array_equal(part.bw_inter, full.bw_inter[2:5])


def test_two_gloo_ranks_compose_their_slices_and_gather(tmp_path):
    import torch.multiprocessing as mp
    import oracle
    oracle.build()
    out = str(tmp_path / "rank0.npz")
    mp.start_processes(_worker, args=(2, _free_port(), out), nprocs=2, join=True, start_method="spawn")
    got = np.load(out)
    g, full = _batch()
    want = oracle.compose(g, full, refine_passes=1)
    assert np.array_equal(got["mk"], want.makespan)
    assert np.array_equal(got["fin"], want.finish)
    assert np.array_equal(got["ov"], want.overlapped)
    # max over ranks: [1, 10, 4] from ranks holding 4 and 3 scenarios
    assert got["t"].tolist() == [1.0, 10.0, 4.0]


def _gpu_worker(rank, world, port, out_path):
    # the same rank logic with each rank composing its slice through the library on
    # cuda:0 (independent compositions, one context per process)
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    import torch.distributed as dist
    from paper_2412_12487_gb300 import Echo
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        g, full = _batch()
        s0, s1 = SH.shard_bounds(N_TOTAL, world, rank)
        with Echo(0) as e:
            e.load_graph(g)
            e.load_scenarios(SH.slice_scenarios(full, s0, s1))
            e.estimate_collectives()
            e.compose(refine_passes=1)
            st, fn = e.read_times()
            mk = e.read_makespan()
            ov = e.read_overlap()
        mk = SH.gather_scenarios(mk, N_TOTAL)
        fin = SH.gather_scenarios(fn, N_TOTAL)
        sta = SH.gather_scenarios(st, N_TOTAL)
        ov = SH.gather_scenarios(ov, N_TOTAL)
        if rank == 0:
            np.savez(out_path, mk=mk, fin=fin, st=sta, ov=ov)
    finally:
        dist.destroy_process_group()


@pytest.mark.gpu
def test_two_gloo_ranks_compose_their_slices_through_the_library(tmp_path):
    import torch.multiprocessing as mp
    import oracle
    oracle.build()
    out = str(tmp_path / "rank0.npz")
    mp.start_processes(_gpu_worker, args=(2, _free_port(), out), nprocs=2, join=True, start_method="spawn")
    got = np.load(out)
    g, full = _batch()
    want = oracle.compose(g, full, refine_passes=1)
    assert np.array_equal(got["mk"], want.makespan)
    assert np.array_equal(got["fin"], want.finish)
    assert np.array_equal(got["st"], want.start)
    assert np.array_equal(got["ov"], want.overlapped)
