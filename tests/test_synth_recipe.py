"""The synthetic inputs follow their stated recipe: per workload the graph sizes, block size,
number of edge types, and per graph the edge families in the latent (pre-relabelling) order -- a
chain i -> i+1, a tree edge from each node to a parent at most `tree_win` before it, short-range
families of about lam * n edges at offsets of at most `max_off`, each family mirrored by a reverse
type, no duplicate (src, dst, type) and no self-loop -- and two calls give identical bytes."""
import numpy as np
import pytest

from paper_1906_11786_gb300 import synth


def _check_graph(g, F, reverse, max_off, tree_win, lam):
    n = g.n_nodes
    P = 2 * F if reverse else F
    assert g.n_types == P
    assert g.src.dtype == np.int32 and g.dst.dtype == np.int32 and g.etype.dtype == np.int32
    assert g.src.min() >= 0 and g.src.max() < n and g.dst.min() >= 0 and g.dst.max() < n
    assert np.all(g.src != g.dst)
    relabel = g.meta["latent_relabel"]
    assert sorted(relabel.tolist()) == list(range(n))
    latent = np.empty(n, np.int64)
    latent[relabel] = np.arange(n)  # latent position of each relabelled node
    ls, ld, t = latent[g.src], latent[g.dst], g.etype
    key = (t.astype(np.int64) * n + ls) * n + ld
    assert len(np.unique(key)) == len(key), "duplicate (src, dst, type)"
    # chain: exactly i -> i + 1 for every i
    c = t == 0
    assert np.array_equal(np.sort(ls[c]), np.arange(n - 1)) and np.all(ld[c] == ls[c] + 1)
    # tree: every node but the first sends one edge to a parent within tree_win before it
    r = t == 1
    assert np.array_equal(np.sort(ls[r]), np.arange(1, n))
    assert np.all(ld[r] < ls[r]) and np.all(ls[r] - ld[r] <= tree_win)
    m = int(round(lam * n))
    for f in range(2, F):
        e = t == f
        off = np.abs(ld[e] - ls[e])
        assert off.min() >= 1 and off.max() <= max_off
        # round(lam n) draws, minus the duplicates removed (a few percent at most here)
        assert 0.9 * m <= e.sum() <= m
    if reverse:
        for f in range(F):
            fwd = set(zip(ls[t == f].tolist(), ld[t == f].tolist()))
            back = set(zip(ld[t == f + F].tolist(), ls[t == f + F].tolist()))
            assert fwd == back, f"type {f + F} does not mirror type {f}"


@pytest.mark.parametrize("name", ["single512", "packed64", "single20k", "sweep131k", "train100k"])
def test_workload_follows_its_recipe(name):
    c = synth.WORKLOADS[name]
    gs = synth.workload_graphs(name)
    kind = c["sizes"][0]
    sizes = [g.n_nodes for g in gs]
    if kind == "fixed":
        assert sizes == list(c["sizes"][1])
    elif kind == "uniform":
        _, count, lo, hi = c["sizes"]
        assert len(sizes) == count and min(sizes) >= lo and max(sizes) <= hi
    else:  # fill: graphs until one past the capacity
        _, cap, lo, hi = c["sizes"]
        assert min(sizes) >= lo and max(sizes) <= hi
        assert sum(sizes) > cap and sum(sizes[:-1]) <= cap
    S = c["S"]
    for g in gs[:12]:
        _check_graph(g, c["F"], c["reverse"], c["max_off"] or S // 2, c["tree_win"] or S // 2,
                     c["lam"])
    again = synth.workload_graphs(name)
    for a, b in zip(gs[:4], again[:4]):
        assert a.src.tobytes() == b.src.tobytes() and a.etype.tobytes() == b.etype.tobytes()


def test_block_size_sweep_scales_the_edge_reach():
    """sweep131k at block size S draws its short-range offsets and tree windows up to S / 2."""
    for S in (32, 512):
        g = synth.workload_graphs("sweep131k", S=S, scale=0.02)[0]
        c = synth.WORKLOADS["sweep131k"]
        _check_graph(g, c["F"], c["reverse"], S // 2, S // 2, c["lam"])


def test_states_and_parameters_are_seeded_and_shaped():
    a, b = synth.gen_states(100, 16, 3), synth.gen_states(100, 16, 3)
    assert a.shape == (100, 16) and a.tobytes() == b.tobytes()
    assert abs(a.mean()) < 0.1 and abs(a.std() - 1) < 0.1
    p = synth.gen_params(5, 16, 7)
    assert p["W"].shape == (5, 16, 16) and p["b"].shape == (5, 16)
    assert p["W_ih"].shape == (48, 16) and p["W_hh"].shape == (48, 16)
    assert p["b_ih"].shape == (48,) and p["b_hh"].shape == (48,) and p["w_out"].shape == (16,)
    assert np.max(np.abs(p["b"])) <= 0.1 and np.max(np.abs(p["b_ih"])) <= 0.1
    # Xavier-uniform bound of the GRU weights: sqrt(6 / (fan_in + fan_out)) with fan_in = H
    bound = np.sqrt(6.0 / (16 + 48))
    assert np.max(np.abs(p["W_ih"])) <= bound and np.max(np.abs(p["W_ih"])) > 0.8 * bound
