"""Multi-GPU logic of the benchmark on CPU ranks (gloo, world size 2): every rank plans its own
supergraph of the same shape (the paper gives each core its own supergraph), the whole-job
figures are the slowest rank's time and the sum of all ranks' node-steps, and the data-parallel
gradient exchange leaves every rank with the mean of all ranks' gradients, which equals the
gradient of the union of the ranks' graphs divided by the number of ranks.  The block-row split
of one supergraph exchanges halos and sums dW, db.  No GPU is used."""
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


def _split_worker(rank, world, port, out):
    """One rank of a block-row split: plans the whole supergraph, takes its part, fills its own
    rows of E and dY, exchanges the halo rows with its neighbour, propagates its part forward and
    backward with the oracle on its local tiles, sums dW and db over the ranks."""
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import numpy as np

    import oracle
    from paper_1906_11786_gb300 import _binding as L
    from paper_1906_11786_gb300 import halo, synth
    from test_plan_abi import edges_from_masks
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        P, S, H = 8, 64, 16
        gs = synth.gen_batch(10, 100, 500, 4, True, 32, 20, 2.0, 808)
        n = sum(g.n_nodes for g in gs)
        cap = -(-(-(-n // S)) // 2) * 2
        full = L.band_plan(gs, P, S, cap)
        N = full.info()["n_pad"]
        rng = np.random.default_rng(1)
        E = rng.standard_normal((N, H)); dY = rng.standard_normal((N, H))
        prm = synth.gen_params(P, H, 2)
        sub, inf = L.plan_partition(full, world, rank)
        r0, nl, ob, oe = inf["row0"], inf["n_local"], inf["own_begin"], inf["own_end"]
        El = torch.zeros((nl, H), dtype=torch.float64)
        El[ob:oe] = torch.from_numpy(E[r0 + ob:r0 + oe])
        halo.exchange(El, inf, rank, world)
        dYl = torch.zeros((nl, H), dtype=torch.float64)
        dYl[ob:oe] = torch.from_numpy(dY[r0 + ob:r0 + oe])
        halo.exchange(dYl, inf, rank, world)
        # the halo rows now hold the neighbours' rows of the full arrays
        halo_ok = bool(np.array_equal(El.numpy(), E[r0:r0 + nl]) and
                       np.array_equal(dYl.numpy(), dY[r0:r0 + nl]))
        fe = edges_from_masks(sub.export(L.BG_EXPORT_MASKS), S)
        Yl = oracle.propagate_fwd(nl, P, H, *fe, El.numpy(), prm["W"], prm["b"])
        te = edges_from_masks(sub.export(L.BG_EXPORT_MASKS_T), S, transposed=True)
        dEl, dWl, dbl = oracle.propagate_bwd(nl, P, H, *te, El.numpy(), prm["W"], dYl.numpy())
        dW_t, db_t = torch.from_numpy(dWl), torch.from_numpy(dbl)
        halo.allreduce_sum([dW_t, db_t])
        # the whole plan, on every rank, for comparison
        ge = edges_from_masks(full.export(L.BG_EXPORT_MASKS), S)
        Y = oracle.propagate_fwd(N, P, H, *ge, E, prm["W"], prm["b"])
        dE, dW, db = oracle.propagate_bwd(N, P, H, *ge, E, prm["W"], dY)
        own = slice(r0 + ob, r0 + oe)
        out[rank] = (halo_ok,
                     float(np.max(np.abs(Yl[ob:oe] - Y[own]))),
                     float(np.max(np.abs(Yl[:ob])) if ob else 0.0) + float(np.max(np.abs(Yl[oe:])) if oe < nl else 0.0),
                     float(np.max(np.abs(dEl[ob:oe] - dE[own]))),
                     float(np.max(np.abs(dW_t.numpy() - dW))), float(np.max(np.abs(db_t.numpy() - db))),
                     oe - ob)
    finally:
        dist.destroy_process_group()


@pytest.mark.timeout(300)
def test_block_row_split_two_ranks_matches_the_whole_plan():
    """The block-row split (bg_plan_partition) on two gloo ranks with halo.exchange: each rank's
    own rows of Y and dE equal the whole plan's, its halo rows of Y are 0, and the all-reduced
    dW, db equal the whole plan's (fp64 oracle arithmetic on both sides)."""
    world = 2
    port = _free_port()
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    mp.start_processes(_split_worker, args=(world, port, out), nprocs=world, start_method="spawn")
    rows = 0
    for r in range(world):
        halo_ok, eY, eYhalo, edE, edW, edb, own = out[r]
        assert halo_ok
        assert eY < 1e-12 and eYhalo == 0.0 and edE < 1e-12
        assert edW < 1e-9 and edb < 1e-9
        rows += own
    assert rows > 0



DP_P, DP_S, DP_H, DP_T = 4, 64, 8, 2


def _dp_grads(graphs, seeds):
    """Oracle GGNN forward + backward (T = 2) over one supergraph of `graphs`, nothing dropped,
    graph i's states and incoming gradient drawn from seeds[i] in its original node order: the
    parameter gradients as one flat fp64 vector."""
    import numpy as np

    import oracle
    from paper_1906_11786_gb300 import synth
    P, S, H, T = DP_P, DP_S, DP_H, DP_T
    lay = oracle.layout(graphs, P, S)
    assert lay.n_dropped == 0 and lay.n_packed == len(graphs)
    E_orig = np.concatenate([synth.gen_states(g.n_nodes, H, s) for g, s in zip(graphs, seeds)])
    dET_orig = np.concatenate([synth.gen_states(g.n_nodes, H, s + 7)
                               for g, s in zip(graphs, seeds)])
    N, gi = lay.n_pad, lay.gather_index()
    E0 = np.zeros((N, H)); E0[:lay.n_real] = E_orig[gi]
    dET = np.zeros((N, H)); dET[:lay.n_real] = dET_orig[gi]
    prm = synth.gen_params(P, H, 4242)
    edges = (lay.kept_dst, lay.kept_src, lay.kept_type)
    Es, Ys = oracle.ggnn_fwd(N, P, H, T, lay.n_real, *edges, E0, prm)
    g = oracle.ggnn_bwd(N, P, H, T, lay.n_real, *edges, prm, Es, Ys, dET)
    return np.concatenate([g[k].ravel() for k in ("dW", "db", "dW_ih", "dW_hh", "db_ih", "db_hh")])


def _dp_graphs(rank):
    from paper_1906_11786_gb300 import synth
    gs = synth.gen_batch(3, 30, 60, 2, True, 6, 6, 1.0, 900 + rank)
    return gs, [1000 * (rank + 1) + 31 * i for i in range(len(gs))]


def _dp_worker(rank, world, port, out):
    """One data-parallel rank: its own supergraph's gradients (the oracle standing in for the
    device step on CPU), then the benchmark's gradient exchange."""
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        own = _dp_grads(*_dp_graphs(rank))
        flat = torch.from_numpy(own.copy())
        bench.allreduce_grads(dist, flat)
        out[rank] = (own.tolist(), flat.tolist())
    finally:
        dist.destroy_process_group()


@pytest.mark.timeout(300)
def test_data_parallel_mean_equals_the_union_batch_gradient():
    """The synchronous data-parallel step (each rank its own supergraph, as the paper trains on
    several cores; gradients averaged by the exchange) equals one step over the union of the
    ranks' graphs with its gradient divided by the number of ranks: the graphs share no edge, so
    their gradient contributions add.  fp64 oracle arithmetic throughout; gloo ranks."""
    import numpy as np
    world = 2
    port = _free_port()
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    mp.start_processes(_dp_worker, args=(world, port, out), nprocs=world, start_method="spawn")
    parts = [_dp_graphs(r) for r in range(world)]
    union = _dp_grads([g for gs, _ in parts for g in gs], [s for _, ss in parts for s in ss])
    own = [np.array(out[r][0]) for r in range(world)]
    assert np.max(np.abs(own[0] - own[1])) > 1e-3  # the ranks' supergraphs differ
    for r in range(world):
        got = np.array(out[r][1])
        np.testing.assert_allclose(got, (own[0] + own[1]) / world, rtol=0, atol=1e-12)
        np.testing.assert_allclose(got, union / world, rtol=1e-10,
                                   atol=1e-10 * np.max(np.abs(union)))
