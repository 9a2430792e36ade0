"""Seeded synthetic inputs shaped like program graphs (Section 4 "Data", Appendix A.1).

The VarMisuse graphs the paper trains on are not available, so program-shaped graphs are generated
from a latent order: a token chain, an AST-like tree, and short-range "semantic" edges, each family
with a reverse type, then randomly relabelled so that a bandwidth-reducing ordering has to recover
the band (Section 3.1).  This module only draws random numbers and shapes them into graphs and
parameter tensors; it holds none of the method's arithmetic and is the one module that both the
CUDA path and the CPU oracle take inputs from.

Every array is produced by numpy's PCG64 generator from an integer seed, so two calls with the same
arguments return identical bytes.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

__all__ = [
    "Graph", "gen_graph", "gen_batch", "gen_states", "gen_params", "WORKLOADS", "workload_graphs",
    "graph_seed", "hub_graph", "with_self_loops", "gen_candidates",
]


@dataclass
class Graph:
    """One directed multi-type graph: edge e goes src[e] -> dst[e] with type etype[e]."""

    n_nodes: int
    src: np.ndarray
    dst: np.ndarray
    etype: np.ndarray
    n_types: int = 0
    meta: dict = field(default_factory=dict)

    @property
    def n_edges(self) -> int:
        return int(self.src.shape[0])


def graph_seed(workload: str, graph_index: int) -> int:
    """Seed of graph `graph_index` of the named workload."""
    return WORKLOADS[workload]["seed"] + 17 * graph_index


def gen_graph(n: int, n_families: int, reverse: bool, max_off: int, tree_win: int, lam: float,
              seed: int) -> Graph:
    """Program-shaped graph with `n` nodes.

    Types: 0 = chain i->i+1; 1 = tree i->parent with parent uniform in [max(0,i-tree_win), i-1];
    2..F-1 = round(lam*n) edges each from a uniform source to source +- uniform[1,max_off]
    (offset and sign redrawn while the target falls outside [0,n)).  Duplicates (same src, dst,
    type) are removed.  With `reverse`, type f+F carries every type-f edge reversed.  Finally node
    ids are relabelled by a uniform random permutation.
    """
    if n < 1:
        raise ValueError("n must be >= 1")
    rng = np.random.default_rng(seed)
    srcs, dsts, types = [], [], []
    # chain
    if n >= 2:
        s = np.arange(n - 1, dtype=np.int64)
        srcs.append(s); dsts.append(s + 1); types.append(np.zeros(n - 1, np.int64))
    # tree
    if n_families >= 2 and n >= 2:
        i = np.arange(1, n, dtype=np.int64)
        lo = np.maximum(0, i - tree_win)
        span = i - lo
        parent = lo + np.floor(rng.random(n - 1) * span).astype(np.int64)
        parent = np.minimum(parent, i - 1)
        srcs.append(i); dsts.append(parent); types.append(np.ones(n - 1, np.int64))
    # short-range semantic families
    m = int(round(lam * n))
    for f in range(2, n_families):
        if m == 0 or n < 2:
            continue
        s = rng.integers(0, n, size=m, dtype=np.int64)
        off = rng.integers(1, max_off + 1, size=m, dtype=np.int64)
        sign = np.where(rng.random(m) < 0.5, -1, 1)
        t = s + sign * off
        bad = (t < 0) | (t >= n)
        while bad.any():
            k = int(bad.sum())
            off[bad] = rng.integers(1, max_off + 1, size=k, dtype=np.int64)
            sign[bad] = np.where(rng.random(k) < 0.5, -1, 1)
            t = s + sign * off
            bad = (t < 0) | (t >= n)
        srcs.append(s); dsts.append(t); types.append(np.full(m, f, np.int64))
    if srcs:
        src = np.concatenate(srcs); dst = np.concatenate(dsts); et = np.concatenate(types)
    else:
        src = np.zeros(0, np.int64); dst = np.zeros(0, np.int64); et = np.zeros(0, np.int64)
    # dedupe (src, dst, type)
    key = (et * n + src) * n + dst
    _, first = np.unique(key, return_index=True)
    first.sort()
    src, dst, et = src[first], dst[first], et[first]
    n_types = n_families
    if reverse:
        src, dst, et = (np.concatenate([src, dst]), np.concatenate([dst, src]),
                        np.concatenate([et, et + n_families]))
        n_types = 2 * n_families
    relabel = rng.permutation(n).astype(np.int64)
    src, dst = relabel[src], relabel[dst]
    return Graph(n, src.astype(np.int32), dst.astype(np.int32), et.astype(np.int32), n_types,
                 {"latent_relabel": relabel.astype(np.int32)})


# Workloads: sizes follow the paper's program graphs (Section 4: up to ~20k nodes per graph,
# P = 22 edge types; Appendix A.1: 70,272-node supergraphs at S = 128) with P = 20.  `seed` is the
# base of the workload's random streams (graph sizes, and graph g from seed + 17 g).
WORKLOADS = {
    "single512": dict(seed=2906, sizes=("fixed", [512]), F=4, reverse=False, max_off=48,
                      tree_win=32, lam=1.0, S=64, H=64, T=1, dtype="f32", gru=False),
    "packed64": dict(seed=3906, sizes=("uniform", 64, 200, 2000), F=10, reverse=True, max_off=96,
                     tree_win=64, lam=3.0, S=128, H=64, T=8, dtype="bf16", gru=True),
    "single20k": dict(seed=4906, sizes=("fixed", [20000]), F=10, reverse=True, max_off=200,
                      tree_win=133, lam=3.0, S=256, H=128, T=8, dtype="bf16", gru=True),
    "sweep131k": dict(seed=5906, sizes=("fill", 131072, 200, 2000), F=10, reverse=True,
                      max_off=None, tree_win=None, lam=3.0, S=128, H=64, T=1, dtype="bf16",
                      gru=False),
    "train100k": dict(seed=6906, sizes=("fill", 100000, 200, 5000), F=10, reverse=True, max_off=96,
                      tree_win=64, lam=3.0, S=128, H=64, T=8, dtype="bf16", gru=True, train=True),
}
for _name, _w in WORKLOADS.items():
    _w["name"] = _name


def _sizes(workload: str, spec) -> list[int]:
    kind = spec[0]
    if kind == "fixed":
        return list(spec[1])
    rng = np.random.default_rng(WORKLOADS[workload]["seed"])
    if kind == "uniform":
        _, count, lo, hi = spec
        return [int(x) for x in rng.integers(lo, hi + 1, size=count)]
    if kind == "fill":
        _, cap, lo, hi = spec
        out, tot = [], 0
        while True:
            x = int(rng.integers(lo, hi + 1))
            out.append(x)
            tot += x
            if tot > cap:  # one past capacity, so the packer stops at the first graph that does not fit
                return out
    raise ValueError(kind)


def workload_graphs(workload: str, S: int | None = None, scale: float = 1.0, **over) -> list[Graph]:
    """Graphs of the named workload.  `S` overrides the block size (the sweep sets max_off =
    tree_win = S/2); `scale` < 1 keeps only a leading fraction of the graph list (small parity
    cases)."""
    c = dict(WORKLOADS[workload]); c.update(over)
    S = S or c["S"]
    max_off = c["max_off"] if c["max_off"] is not None else max(1, S // 2)
    tree_win = c["tree_win"] if c["tree_win"] is not None else max(1, S // 2)
    sizes = _sizes(workload, c["sizes"])
    if scale < 1.0:
        sizes = sizes[:max(1, int(round(len(sizes) * scale)))]
    return [gen_graph(n, c["F"], c["reverse"], max_off, tree_win, c["lam"], graph_seed(workload, g))
            for g, n in enumerate(sizes)]


def gen_batch(count: int, n_lo: int, n_hi: int, n_families: int, reverse: bool, max_off: int,
              tree_win: int, lam: float, seed: int) -> list[Graph]:
    """`count` graphs with node counts uniform in [n_lo, n_hi] (small test batches)."""
    rng = np.random.default_rng(seed)
    sizes = rng.integers(n_lo, n_hi + 1, size=count)
    return [gen_graph(int(n), n_families, reverse, max_off, tree_win, lam, seed * 7919 + 13 * g)
            for g, n in enumerate(sizes)]


def hub_graph(n_leaves: int, n_types: int, seed: int, lam: float = 1.0) -> Graph:
    """A program-shaped graph with one hub: a chain (type 1) over n_leaves + 1 nodes, every node
    also sending a type-0 edge to node 0 (in-degree n_leaves of one type, as a much-used variable
    or a shared declaration would receive), plus round(lam n) short-range edges of types
    2..n_types-1 at offsets up to 8; then a uniform random relabelling."""
    n = n_leaves + 1
    rng = np.random.default_rng(seed)
    src = [np.arange(1, n), np.arange(n - 1)]
    dst = [np.zeros(n - 1, np.int64), np.arange(1, n)]
    et = [np.zeros(n - 1, np.int64), np.ones(n - 1, np.int64)]
    m = int(round(lam * n)) if n_types > 2 else 0
    if m:
        s = rng.integers(0, n, size=m)
        t = np.clip(s + rng.integers(-8, 9, size=m), 0, n - 1)
        src.append(s); dst.append(t); et.append(rng.integers(2, n_types, size=m))
    src, dst, et = (np.concatenate(x).astype(np.int64) for x in (src, dst, et))
    key = (et * n + src) * n + dst
    _, first = np.unique(key, return_index=True)
    first.sort()
    relabel = rng.permutation(n)
    return Graph(n, relabel[src[first]].astype(np.int32), relabel[dst[first]].astype(np.int32),
                 et[first].astype(np.int32), n_types)


def with_self_loops(g: Graph, frac: float, n_types: int, seed: int) -> Graph:
    """`g` plus a self-loop u -> u of a uniform type on a uniform random `frac` of its nodes."""
    rng = np.random.default_rng(seed)
    k = int(round(frac * g.n_nodes))
    u = rng.choice(g.n_nodes, size=k, replace=False).astype(np.int32)
    t = rng.integers(0, n_types, size=k).astype(np.int32)
    return Graph(g.n_nodes, np.concatenate([g.src, u]), np.concatenate([g.dst, u]),
                 np.concatenate([g.etype, t]), max(g.n_types, n_types), dict(g.meta))


def gen_candidates(g: Graph, k: int, seed: int) -> np.ndarray:
    """k distinct candidate nodes of `g` drawn uniformly (the synthetic stand-in for the
    VarMisuse hole's type-correct in-scope variables, Section 4 "Data"), ascending."""
    rng = np.random.default_rng(seed)
    return np.sort(rng.choice(g.n_nodes, size=min(k, g.n_nodes), replace=False)).astype(np.int32)


def gen_states(n: int, H: int, seed: int) -> np.ndarray:
    """Initial node states E(0) ~ N(0, 1), float64 [n, H]."""
    return np.random.default_rng(seed).standard_normal((n, H))


def _xavier(rng, shape, fan_in, fan_out):
    a = np.sqrt(6.0 / (fan_in + fan_out))
    return rng.uniform(-a, a, size=shape)


def gen_params(P: int, H: int, seed: int, bias_scale: float = 0.1,
               mean_in_degree: float = 1.0) -> dict:
    """Edge-type transforms W [P, H, H] (message = state @ W[p]), per-type bias b [P, H],
    GRU weights W_ih, W_hh [3H, H] (gate rows r, z, n) and biases b_ih, b_hh [3H], readout
    w_out [H].  Weights Xavier-uniform, biases uniform in +-bias_scale.  All float64.

    Incoming messages are summed (Appendix D), so the message layer's fan-in is H times the mean
    in-degree: W's Xavier bound uses fan_in = H * mean_in_degree (1.0 gives the plain H x H
    bound)."""
    rng = np.random.default_rng(seed)
    return {
        "W": _xavier(rng, (P, H, H), H * max(mean_in_degree, 1.0), H),
        "b": rng.uniform(-bias_scale, bias_scale, size=(P, H)),
        "W_ih": _xavier(rng, (3 * H, H), H, 3 * H),
        "W_hh": _xavier(rng, (3 * H, H), H, 3 * H),
        "b_ih": rng.uniform(-bias_scale, bias_scale, size=(3 * H,)),
        "b_hh": rng.uniform(-bias_scale, bias_scale, size=(3 * H,)),
        "w_out": _xavier(rng, (H,), H, 1),
    }
