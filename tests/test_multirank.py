"""Multi-GPU logic of the benchmark on CPU ranks (gloo, world size 2): every rank plans its own
supergraph of the same shape (the paper gives each core its own supergraph), the whole-job
figures are the slowest rank's time and the sum of all ranks' node-steps, and the data-parallel
gradient exchange leaves every rank with the mean of all ranks' gradients.  No GPU is used."""
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


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    from paper_1906_11786_gb300 import _binding as L
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        graphs, c = bench.workload("packed64", rank)
        # same workload shape on every rank, different graphs
        sig = torch.tensor([len(graphs), sum(g.n_nodes for g in graphs), c["S"], c["P"], c["H"]],
                           dtype=torch.float64)
        lo, hi = sig.clone(), sig.clone()
        dist.all_reduce(lo, op=dist.ReduceOp.MIN)
        dist.all_reduce(hi, op=dist.ReduceOp.MAX)
        edges = torch.tensor([float(sum(g.n_edges for g in graphs))], dtype=torch.float64)
        e_lo, e_hi = edges.clone(), edges.clone()
        dist.all_reduce(e_lo, op=dist.ReduceOp.MIN)
        dist.all_reduce(e_hi, op=dist.ReduceOp.MAX)
        plan = L.band_plan(graphs[:4], c["P"], c["S"])
        units = plan.info()["n_real"] * c["T"]
        ms = 10.0 + rank
        ms_max, units_sum = bench.reduce_over_ranks(dist, ms, float(units), device="cpu")
        u_all = torch.tensor([float(units)], dtype=torch.float64)
        gathered = [torch.zeros(1, dtype=torch.float64) for _ in range(world)]
        dist.all_gather(gathered, u_all)
        out[rank] = (bool(torch.equal(lo, hi)), float(e_lo.item()) != float(e_hi.item()),
                     ms_max, units_sum, float(sum(x.item() for x in gathered)))
    finally:
        dist.destroy_process_group()


@pytest.mark.timeout(300)
def test_two_cpu_ranks_plan_own_supergraphs_and_aggregate():
    world = 2
    port = _free_port()
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    mp.start_processes(_worker, args=(world, port, out), nprocs=world, start_method="spawn")
    for r in range(world):
        same_shape, different_graphs, ms_max, units_sum, units_expected = out[r]
        assert same_shape and different_graphs
        assert ms_max == 10.0 + world - 1
        assert units_sum == units_expected


def _grad_worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank r's gradients are r + 1 + 0.5 k on element k; the mean over ranks is known exactly
        flat = torch.arange(12, dtype=torch.float32) * 0.5 + (rank + 1)
        view = flat[4:10].view(2, 3)  # gradients live as views of the flat buffer
        bench.allreduce_grads(dist, flat)
        out[rank] = (flat.tolist(), view.tolist())
    finally:
        dist.destroy_process_group()


@pytest.mark.timeout(300)
def test_data_parallel_gradient_mean_over_cpu_ranks():
    world = 2
    port = _free_port()
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    mp.start_processes(_grad_worker, args=(world, port, out), nprocs=world, start_method="spawn")
    mean_offset = sum(r + 1 for r in range(world)) / world
    expect = [0.5 * k + mean_offset for k in range(12)]
    for r in range(world):
        flat, view = out[r]
        assert flat == pytest.approx(expect, abs=0)
        assert view == [expect[4:7], expect[7:10]]


def test_single_process_gradients_untouched():
    import bench
    flat = torch.arange(5, dtype=torch.float32)
    bench.allreduce_grads(None, flat)
    assert flat.tolist() == [0.0, 1.0, 2.0, 3.0, 4.0]
