"""Pins of the CPU oracle to things other than itself (no GPU needed).

Each test checks the oracle against what the paper and the mathematics fix: hand-worked examples
(tests/golden), a brute-force dense N x N adjacency product, the block-diagonal special case
(Eq. 2) as a batched matmul, Algorithm 1 restated with einsum on the oracle's exported tiles,
permutation equivariance, finite differences, torch.nn.GRUCell / torch.optim.Adam / autograd,
the bandwidth and RCM properties, and the coverage rule after Eq. 3.
"""
import itertools
import json
import os

import numpy as np
import pytest
import torch

import oracle
from paper_1906_11786_gb300 import synth

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _graph(n, edges, types=None, P=1):
    e = np.asarray(edges, np.int32).reshape(-1, 2)
    t = np.zeros(len(e), np.int32) if types is None else np.asarray(types, np.int32)
    return synth.Graph(n, e[:, 0].copy(), e[:, 1].copy(), t, P)


def _dense_A(N, P, src, dst, typ, keep=None):
    """Dense 0/1 adjacency per type, straight from the definition a_vu = 1 iff edge u -> v
    (Section 2), optionally restricted by a boolean keep(v, u)."""
    A = np.zeros((P, N, N))
    for u, v, p in zip(src, dst, typ):
        if keep is None or keep(v, u):
            A[p, v, u] = 1.0
    return A


def _dense_propagate(A, E, W, b):
    At = torch.from_numpy(A)
    Et = torch.from_numpy(E)
    Y = torch.zeros_like(Et)
    for p in range(A.shape[0]):
        Y += At[p] @ Et @ torch.from_numpy(W[p])
        Y += (At[p] @ torch.ones(E.shape[0], 1, dtype=torch.float64)) @ torch.from_numpy(b[p])[None]
    return Y.numpy()


# ---------------------------------------------------------------------------- golden / hand-worked


def test_golden_propagate_tiny():
    g = json.load(open(os.path.join(GOLD, "propagate_tiny.json")))
    e = np.array(g["edges_src_dst_type"])
    N, P, H = g["N"], g["P"], g["H"]
    Y = oracle.propagate_fwd(N, P, H, e[:, 1], e[:, 0], e[:, 2], np.array(g["E"], float),
                             np.array(g["W"], float), np.array(g["b"], float))
    np.testing.assert_array_equal(Y, np.array(g["Y"], float))
    dE, dW, db = oracle.propagate_bwd(N, P, H, e[:, 1], e[:, 0], e[:, 2], np.array(g["E"], float),
                                      np.array(g["W"], float), np.array(g["dY"], float))
    np.testing.assert_array_equal(dE, np.array(g["dE"], float))
    np.testing.assert_array_equal(dW, np.array(g["dW"], float))
    np.testing.assert_array_equal(db, np.array(g["db"], float))


def test_golden_rcm_tiny():
    g = json.load(open(os.path.join(GOLD, "rcm_tiny.json")))
    for c in g["cases"]:
        e = np.array(c["edges"], np.int32)
        perm = oracle.rcm(c["n"], e[:, 0], e[:, 1])
        assert perm.tolist() == c["perm"], c["name"]
        pos = np.argsort(perm)
        assert oracle.bandwidth(c["n"], e[:, 0], e[:, 1]) == c["bw_before"]
        assert oracle.bandwidth(c["n"], e[:, 0], e[:, 1], pos) == c["bw_after"]


# ---------------------------------------------------------------------------- propagation


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_propagate_matches_dense_bruteforce(seed):
    """All edges kept (one block covers the graph): scatter-add == sum_p A_p (E W_p + 1 b_p^T)."""
    rng = np.random.default_rng(seed)
    N, P, H = 37, 3, 5
    g = synth.gen_graph(N, 3, False, 9, 6, 1.0, 100 + seed)
    g.etype = (g.etype % P).astype(np.int32)
    L = oracle.layout([g], P, 64, flags=0)
    assert L.K == 1 and L.n_dropped == 0
    E = rng.standard_normal((64, H)); E[N:] = 0
    W = rng.standard_normal((P, H, H)); b = rng.standard_normal((P, H))
    Y = oracle.propagate_fwd(64, P, H, L.kept_dst, L.kept_src, L.kept_type, E, W, b)
    A = _dense_A(64, P, g.src, g.dst, g.etype)
    np.testing.assert_allclose(Y, _dense_propagate(A, E, W, b), rtol=1e-12, atol=1e-12)


def test_propagate_band_restricted_matches_masked_dense():
    """With S < bandwidth, the oracle equals the dense product restricted to the block-tridiagonal
    cover |floor(i/S) - floor(j/S)| <= 1 (Eq. 3 and the coverage rule after it)."""
    rng = np.random.default_rng(5)
    N, P, H, S = 64, 4, 4, 8
    g = synth.gen_graph(N, 2, True, 30, 20, 1.5, 77)
    L = oracle.layout([g], P, S, flags=0)
    assert L.n_dropped > 0 and L.n_kept > 0
    E = rng.standard_normal((N, H)); W = rng.standard_normal((P, H, H)); b = rng.standard_normal((P, H))
    Y = oracle.propagate_fwd(N, P, H, L.kept_dst, L.kept_src, L.kept_type, E, W, b)
    A = _dense_A(N, P, g.src, g.dst, g.etype, keep=lambda v, u: abs(v // S - u // S) <= 1)
    np.testing.assert_allclose(Y, _dense_propagate(A, E, W, b), rtol=1e-12, atol=1e-12)


def test_block_diagonal_special_case_is_bmm():
    """Eq. 2: with only within-block edges, A E = reshape(BMM([C_1..C_K], reshape(E,[K,S,H])))."""
    rng = np.random.default_rng(3)
    K, S, H = 5, 8, 6
    src, dst = [], []
    for k in range(K):
        for _ in range(20):
            src.append(k * S + rng.integers(S)); dst.append(k * S + rng.integers(S))
    g = _graph(K * S, list(zip(src, dst)))
    L = oracle.layout([g], 1, S, flags=0)
    assert L.n_dropped == 0
    E = rng.standard_normal((K * S, H))
    W = np.eye(H)[None]; b = np.zeros((1, H))
    Y = oracle.propagate_fwd(K * S, 1, H, L.kept_dst, L.kept_src, L.kept_type, E, W, b)
    C = torch.zeros(K, S, S, dtype=torch.float64)
    for u, v in set(zip(src, dst)):
        C[v // S, v % S, u % S] = 1.0
    ref = torch.bmm(C, torch.from_numpy(E).reshape(K, S, H)).reshape(K * S, H)
    np.testing.assert_allclose(Y, ref.numpy(), rtol=1e-12, atol=1e-12)


def test_algorithm1_einsum_on_exported_tiles_equals_scatter():
    """Algorithm 1 restated with numpy einsum (aggregate first, then the [P*H, H] edge weights) on
    the oracle's exported tiles, with the super-diagonal line reading block k+1 (Eq. 3) and the
    types interleaved along z = s*P + p, equals the oracle's scatter-add (no bias)."""
    rng = np.random.default_rng(11)
    P, H, S = 3, 4, 16
    gs = synth.gen_batch(4, 20, 40, 3, False, 12, 8, 1.0, 9)
    L = oracle.layout(gs, P, S)
    K, N = L.K, L.K * S
    bits = np.unpackbits(L.masks, axis=-1, bitorder="little").astype(np.float64)  # [K,3,P,S,S]
    # Cks/Uks/Lks with rows z = s*P + p
    Cks = bits[:, 1].transpose(0, 2, 1, 3).reshape(K, S * P, S)
    Uks = bits[:-1, 2].transpose(0, 2, 1, 3).reshape(K - 1, S * P, S)  # row k reads block k+1
    Lks = bits[1:, 0].transpose(0, 2, 1, 3).reshape(K - 1, S * P, S)   # row k reads block k-1
    E = rng.standard_normal((N, H)); W = rng.standard_normal((P, H, H))
    Eks = E.reshape(K, S, H)
    pre = np.einsum("kzs,ksh->kzh", Cks, Eks)
    pre[0:K - 1] += np.einsum("kzs,ksh->kzh", Uks, Eks[1:K])
    pre[1:K] += np.einsum("kzs,ksh->kzh", Lks, Eks[0:K - 1])
    pre = pre.reshape(K, S, P * H)
    Y1 = np.einsum("ksy,yh->ksh", pre, W.reshape(P * H, H)).reshape(N, H)
    Y = oracle.propagate_fwd(N, P, H, L.kept_dst, L.kept_src, L.kept_type, E, W, np.zeros((P, H)))
    np.testing.assert_allclose(Y, Y1, rtol=1e-11, atol=1e-11)


def test_single_block_reduces_to_dense_matmul():
    """K = 1: the band op is one dense product sum_p A_p E W_p (torch.matmul, fp64)."""
    rng = np.random.default_rng(4)
    N, P, H = 32, 4, 8
    g = synth.gen_graph(N, 2, True, 5, 4, 2.0, 5)
    L = oracle.layout([g], P, 32, flags=0)
    assert L.K == 1
    E = rng.standard_normal((N, H)); W = rng.standard_normal((P, H, H))
    Y = oracle.propagate_fwd(N, P, H, L.kept_dst, L.kept_src, L.kept_type, E, W, np.zeros((P, H)))
    A = torch.from_numpy(np.unpackbits(L.masks[0, 1], axis=-1, bitorder="little").astype(np.float64))
    ref = sum(torch.matmul(torch.matmul(A[p], torch.from_numpy(E)), torch.from_numpy(W[p]))
              for p in range(P))
    np.testing.assert_allclose(Y, ref.numpy(), rtol=1e-12, atol=1e-12)


def test_permutation_equivariance_exact_sparse():
    """Relabelling nodes by pi and propagating equals propagating and relabelling (Section 3.1)."""
    rng = np.random.default_rng(8)
    N, P, H = 50, 3, 4
    g = synth.gen_graph(N, 3, False, 10, 6, 1.0, 31)
    E = rng.standard_normal((N, H)); W = rng.standard_normal((P, H, H)); b = rng.standard_normal((P, H))
    Y = oracle.propagate_fwd(N, P, H, g.dst, g.src, g.etype, E, W, b)
    pi = rng.permutation(N)  # new id of old node v is pi[v]
    Ep = np.zeros_like(E); Ep[pi] = E
    Yp = oracle.propagate_fwd(N, P, H, pi[g.dst], pi[g.src], g.etype, Ep, W, b)
    np.testing.assert_allclose(Yp[pi], Y, rtol=1e-12, atol=1e-12)


def test_messages_are_summed_not_averaged():
    """Appendix D: a node with two identical in-messages gets twice the message."""
    W = np.eye(2)[None]; b = np.zeros((1, 2)); E = np.array([[1.0, 2.0], [1.0, 2.0], [0, 0]])
    Y = oracle.propagate_fwd(3, 1, 2, [2, 2], [0, 1], [0, 0], E, W, b)
    np.testing.assert_array_equal(Y[2], [2.0, 4.0])


# ---------------------------------------------------------------------------- backward


def _fd(f, x, eps=1e-6):
    g = np.zeros_like(x)
    it = np.nditer(x, flags=["multi_index"])
    for _ in it:
        i = it.multi_index
        old = x[i]
        x[i] = old + eps; fp = f()
        x[i] = old - eps; fm = f()
        x[i] = old
        g[i] = (fp - fm) / (2 * eps)
    return g


def test_propagate_bwd_finite_differences_and_adjoint():
    rng = np.random.default_rng(12)
    N, P, H = 12, 4, 3
    g = synth.gen_graph(N, 2, True, 4, 3, 1.0, 3)
    E = rng.standard_normal((N, H)); W = rng.standard_normal((P, H, H)); b = rng.standard_normal((P, H))
    G = rng.standard_normal((N, H))
    args = (N, P, H, g.dst, g.src, g.etype)
    f = lambda: float((oracle.propagate_fwd(*args, E, W, b) * G).sum())  # noqa: E731
    dE, dW, db = oracle.propagate_bwd(*args, E, W, G)
    np.testing.assert_allclose(dE, _fd(f, E), rtol=1e-6, atol=1e-7)
    np.testing.assert_allclose(dW, _fd(f, W), rtol=1e-6, atol=1e-7)
    np.testing.assert_allclose(db, _fd(f, b), rtol=1e-6, atol=1e-7)
    # adjoint: <G, A M> = <A^T G, M> with M = E W (b = 0) gives <G, Y> = <dE, E> for linear Y(E)
    Y0 = oracle.propagate_fwd(*args, E, W, np.zeros((P, H)))
    np.testing.assert_allclose((G * Y0).sum(), (dE * E).sum(), rtol=1e-12)


def _torch_gru(X, Hs, prm):
    H = X.shape[1]
    cell = torch.nn.GRUCell(H, H).double()
    with torch.no_grad():
        cell.weight_ih.copy_(torch.from_numpy(prm["W_ih"]))
        cell.weight_hh.copy_(torch.from_numpy(prm["W_hh"]))
        cell.bias_ih.copy_(torch.from_numpy(prm["b_ih"]))
        cell.bias_hh.copy_(torch.from_numpy(prm["b_hh"]))
    return cell


def test_gru_matches_torch_grucell_fwd_and_bwd():
    """Reading c4: the oracle GRU is torch.nn.GRUCell (input = messages, hidden = state)."""
    rng = np.random.default_rng(13)
    N, H = 9, 6
    prm = synth.gen_params(1, H, 21, bias_scale=0.5)
    X = rng.standard_normal((N, H)); Hs = rng.standard_normal((N, H)); G = rng.standard_normal((N, H))
    cell = _torch_gru(X, Hs, prm)
    Xt = torch.from_numpy(X).requires_grad_(); Ht = torch.from_numpy(Hs).requires_grad_()
    out = cell(Xt, Ht)
    (out * torch.from_numpy(G)).sum().backward()
    ours = oracle.gru_fwd(X, Hs, prm["W_ih"], prm["W_hh"], prm["b_ih"], prm["b_hh"])
    np.testing.assert_allclose(ours, out.detach().numpy(), rtol=1e-12, atol=1e-13)
    dX, dH, dWi, dWh, dbi, dbh = oracle.gru_bwd(X, Hs, prm["W_ih"], prm["W_hh"], prm["b_ih"],
                                                prm["b_hh"], G)
    np.testing.assert_allclose(dX, Xt.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(dH, Ht.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(dWi, cell.weight_ih.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(dWh, cell.weight_hh.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(dbi, cell.bias_ih.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(dbh, cell.bias_hh.grad.numpy(), rtol=1e-10, atol=1e-12)


def test_gru_padding_rows_are_zero():
    rng = np.random.default_rng(1)
    prm = synth.gen_params(1, 4, 2, bias_scale=0.5)
    X = rng.standard_normal((6, 4)); Hs = rng.standard_normal((6, 4))
    out = oracle.gru_fwd(X, Hs, prm["W_ih"], prm["W_hh"], prm["b_ih"], prm["b_hh"], n_real=4)
    assert np.all(out[4:] == 0) and np.all(out[:4] != 0)


def test_ggnn_bwd_finite_differences():
    """Whole T = 2 GGNN (propagate + GRU) backward against central differences."""
    rng = np.random.default_rng(14)
    N, P, H, T = 10, 4, 3, 2
    g = synth.gen_graph(N, 2, True, 4, 3, 1.0, 9)
    prm = synth.gen_params(P, H, 5, bias_scale=0.3)
    E0 = rng.standard_normal((N, H)); G = rng.standard_normal((N, H))
    n_real = N - 2  # two padding rows
    args = (N, P, H, T, n_real, g.dst, g.src, g.etype)

    def f():
        Es, _ = oracle.ggnn_fwd(*args, E0, prm)
        return float((Es[T] * G).sum())

    Es, Ys = oracle.ggnn_fwd(*args, E0, prm)
    out = oracle.ggnn_bwd(*args, prm, Es, Ys, G)
    np.testing.assert_allclose(out["dE0"], _fd(f, E0), rtol=1e-6, atol=1e-8)
    for k, gk in [("W", "dW"), ("b", "db"), ("W_ih", "dW_ih"), ("W_hh", "dW_hh"),
                  ("b_ih", "db_ih"), ("b_hh", "db_hh")]:
        np.testing.assert_allclose(out[gk], _fd(f, prm[k]), rtol=1e-6, atol=1e-8, err_msg=k)



def _ggnn(N, P, H, T, g_dst, g_src, g_typ, E0, G, prm):
    args = (N, P, H, T, N, g_dst, g_src, g_typ)
    Es, Ys = oracle.ggnn_fwd(*args, E0, prm)
    return Es[T], oracle.ggnn_bwd(*args, prm, Es, Ys, G)


def test_ggnn_relabelling_and_disjoint_graphs():
    """T = 3 GGNN steps over the exact edge list: relabelling the nodes relabels E(T) and dE(0)
    and leaves every parameter gradient unchanged (Eq. 1 has no node order); a union of two graphs
    that share no edge gives each graph's own E(T) and dE(0), and parameter gradients that are the
    sum of the two graphs' (they share only the parameters)."""
    rng = np.random.default_rng(21)
    P, H, T = 3, 4, 3
    prm = synth.gen_params(P, H, 8, bias_scale=0.3)
    keys = ("dW", "db", "dW_ih", "dW_hh", "db_ih", "db_hh")
    a = synth.gen_graph(25, 3, False, 6, 4, 1.0, 41)
    E0 = rng.standard_normal((25, H)); G = rng.standard_normal((25, H))
    ET, gr = _ggnn(25, P, H, T, a.dst, a.src, a.etype, E0, G, prm)
    pi = rng.permutation(25)  # node v becomes pi[v]
    Ep = np.zeros_like(E0); Ep[pi] = E0
    Gp = np.zeros_like(G); Gp[pi] = G
    ETp, grp = _ggnn(25, P, H, T, pi[a.dst], pi[a.src], a.etype, Ep, Gp, prm)
    np.testing.assert_allclose(ETp[pi], ET, rtol=0, atol=1e-12)
    np.testing.assert_allclose(grp["dE0"][pi], gr["dE0"], rtol=0, atol=1e-12)
    for k in keys:
        np.testing.assert_allclose(grp[k], gr[k], rtol=1e-12, atol=1e-12, err_msg=k)
    b = synth.gen_graph(17, 3, False, 6, 4, 1.0, 42)
    Eb = rng.standard_normal((17, H)); Gb = rng.standard_normal((17, H))
    ETb, grb = _ggnn(17, P, H, T, b.dst, b.src, b.etype, Eb, Gb, prm)
    ETu, gru = _ggnn(42, P, H, T, np.concatenate([a.dst, b.dst + 25]),
                     np.concatenate([a.src, b.src + 25]), np.concatenate([a.etype, b.etype]),
                     np.concatenate([E0, Eb]), np.concatenate([G, Gb]), prm)
    np.testing.assert_allclose(ETu, np.concatenate([ET, ETb]), rtol=0, atol=1e-12)
    np.testing.assert_allclose(gru["dE0"], np.concatenate([gr["dE0"], grb["dE0"]]), rtol=0,
                               atol=1e-12)
    for k in keys:
        np.testing.assert_allclose(gru[k], gr[k] + grb[k], rtol=1e-12, atol=1e-12, err_msg=k)

def test_readout_loss_matches_autograd():
    rng = np.random.default_rng(15)
    N, H = 20, 5
    E = rng.standard_normal((N, H)); w = rng.standard_normal(H); y = rng.standard_normal(3)
    off = np.array([0, 7, 12], np.int32); cnt = np.array([7, 5, 6], np.int32)
    loss, dE, dw = oracle.readout_loss(E, off, cnt, w, y)
    Et = torch.from_numpy(E).requires_grad_(); wt = torch.from_numpy(w).requires_grad_()
    L = 0
    for o, c, yy in zip(off, cnt, y):
        L = L + 0.5 * (Et[o:o + c].mean(0) @ wt - yy) ** 2
    L.backward()
    assert abs(loss - L.item()) < 1e-12
    np.testing.assert_allclose(dE, Et.grad.numpy(), rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(dw, wt.grad.numpy(), rtol=1e-12, atol=1e-14)


def test_adam_matches_torch_optim():
    rng = np.random.default_rng(16)
    p0 = rng.standard_normal(17); grads = [rng.standard_normal(17) for _ in range(3)]
    pt = torch.from_numpy(p0.copy()).requires_grad_()
    opt = torch.optim.Adam([pt], lr=1e-2, betas=(0.9, 0.999), eps=1e-8)
    p, m, v = p0.copy(), np.zeros(17), np.zeros(17)
    for t, g in enumerate(grads, 1):
        pt.grad = torch.from_numpy(g.copy())
        opt.step()
        p, m, v = oracle.adam(p, m, v, g, 1e-2, 0.9, 0.999, 1e-8, t)
    np.testing.assert_allclose(p, pt.detach().numpy(), rtol=1e-12, atol=1e-14)


# ---------------------------------------------------------------------------- bandwidth and RCM


def _bw_bruteforce(n, src, dst):
    best = None
    for perm in itertools.permutations(range(n)):
        pos = np.array(perm)
        b = int(np.max(np.abs(pos[src] - pos[dst]))) if len(src) else 0
        best = b if best is None else min(best, b)
    return best


def test_bandwidth_definition():
    # a_ij = 0 whenever |i - j| > B: edges at distances 1 and 4 give B = 4; no edges give 0
    assert oracle.bandwidth(6, [0, 1], [1, 5]) == 4
    assert oracle.bandwidth(3, np.zeros(0, np.int32), np.zeros(0, np.int32)) == 0
    assert oracle.bandwidth(3, [2], [2]) == 0


@pytest.mark.parametrize("seed", range(6))
def test_rcm_path_and_cycle_and_complete(seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(5, 40))
    lab = rng.permutation(n)
    src, dst = lab[:-1], lab[1:]
    perm = oracle.rcm(n, src, dst)
    assert sorted(perm.tolist()) == list(range(n))
    assert oracle.bandwidth(n, src, dst, np.argsort(perm)) == 1
    cs, cd = lab, np.roll(lab, 1)
    assert oracle.bandwidth(n, cs, cd, np.argsort(oracle.rcm(n, cs, cd))) == 2
    m = 7
    a, b = np.triu_indices(m, 1)
    assert oracle.bandwidth(m, a, b, np.argsort(oracle.rcm(m, a, b))) == m - 1


def test_rcm_disconnected_union_takes_max_of_parts():
    rng = np.random.default_rng(3)
    lab = rng.permutation(30)
    path = list(zip(lab[:14], lab[1:15]))
    cyc = list(zip(lab[15:], np.roll(lab[15:], 1)))
    e = np.array(path + cyc)
    perm = oracle.rcm(30, e[:, 0], e[:, 1])
    assert oracle.bandwidth(30, e[:, 0], e[:, 1], np.argsort(perm)) == 2


@pytest.mark.parametrize("seed", range(8))
def test_rcm_never_worse_than_input_and_not_below_optimum(seed):
    rng = np.random.default_rng(100 + seed)
    n = 7
    m = int(rng.integers(4, 12))
    src = rng.integers(0, n, m); dst = rng.integers(0, n, m)
    perm = oracle.rcm(n, src, dst, keep_if_better=True)
    assert sorted(perm.tolist()) == list(range(n))
    bw = oracle.bandwidth(n, src, dst, np.argsort(perm))
    assert bw <= oracle.bandwidth(n, src, dst)
    assert bw >= _bw_bruteforce(n, src, dst)


def test_rcm_recovers_band_of_program_graphs():
    for name in ("single512", "single20k"):
        g = synth.workload_graphs(name)[0]
        perm = oracle.rcm(g.n_nodes, g.src, g.dst)
        before = oracle.bandwidth(g.n_nodes, g.src, g.dst)
        after = oracle.bandwidth(g.n_nodes, g.src, g.dst, np.argsort(perm))
        assert after < before // 4


# ---------------------------------------------------------------------------- layout


def test_coverage_rule_after_eq3():
    """|i-j| < S always kept; S <= |i-j| < 2S kept iff the blocks are adjacent; >= 2S dropped."""
    S = 8
    cases = [((0, 7), True), ((0, 8), True), ((0, 15), True), ((0, 16), False), ((7, 8), True),
             ((7, 16), False), ((8, 23), True), ((8, 24), False), ((24, 31), True), ((31, 24), True)]
    e = [c[0] for c in cases]
    g = _graph(32, e)
    L = oracle.layout([g], 1, S, flags=0)
    kept = set(zip(L.kept_src.tolist(), L.kept_dst.tolist()))
    for (u, v), want in cases:
        assert ((u, v) in kept) == want, (u, v)
    assert L.n_kept + L.n_dropped == L.n_unique == len(set(e))


def test_layout_masks_agree_with_kept_edges_and_packing_rule():
    gs = synth.gen_batch(9, 30, 90, 4, True, 10, 8, 1.0, 4)
    P, S = 8, 32
    cap = 12  # 384 positions: not all graphs fit
    L = oracle.layout(gs, P, S, capacity_blocks=cap)
    assert L.K == cap
    # packing: contiguous in input order, stop at the first that does not fit
    pos = 0
    for g, n in enumerate(L.n_nodes):
        if pos + n <= cap * S and (g == 0 or L.offset[g - 1] >= 0):
            assert L.offset[g] == pos
            pos += n
        else:
            assert L.offset[g] == -1
    assert L.n_real == pos
    bits = np.unpackbits(L.masks, axis=-1, bitorder="little")  # [K,3,P,S,S]
    assert int(bits.sum()) == L.n_kept
    k, d, p, r, c = np.nonzero(bits)
    got = set(zip((k * S + r).tolist(), ((k + d - 1) * S + c).tolist(), p.tolist()))
    want = set(zip(L.kept_dst.tolist(), L.kept_src.tolist(), L.kept_type.tolist()))
    assert got == want
    assert not bits[0, 0].any() and not bits[-1, 2].any()



def test_batch_without_nodes_is_one_padding_block():
    """Reading c9: K = ceil(sum n / S), at least one block; graphs with no nodes are packed at the
    current offset and take no positions."""
    e = np.zeros(0, np.int32)
    empty = synth.Graph(0, e, e, e, 2)
    lay = oracle.layout([empty, empty], 2, 32)
    assert lay.K == 1 and lay.n_packed == 2 and lay.n_real == 0 and lay.offset.tolist() == [0, 0]
    assert lay.n_kept == 0 and not lay.masks.any()
    g = _graph(40, [(0, 1), (1, 2)], P=2)
    lay = oracle.layout([g, empty, g], 2, 32)
    assert lay.K == 3 and lay.offset.tolist() == [0, 40, 40] and lay.n_real == 80

def test_duplicate_edges_count_once():
    g = _graph(4, [(0, 1), (0, 1), (0, 1), (2, 3)])
    L = oracle.layout([g], 1, 8, flags=0)
    assert L.n_unique == 2 and L.n_kept == 2
    Y = oracle.propagate_fwd(8, 1, 1, L.kept_dst, L.kept_src, L.kept_type, np.ones((8, 1)),
                             np.ones((1, 1, 1)), np.zeros((1, 1)))
    assert Y[1, 0] == 1.0


def test_invalid_input_is_rejected():
    g = _graph(3, [(0, 5)])
    with pytest.raises(ValueError):
        oracle.layout([g], 1, 8)
    g = _graph(3, [(0, 1)], types=[3])
    with pytest.raises(ValueError):
        oracle.layout([g], 2, 8)


# ------------------------------------------------------------------------ multi-threaded variant


def test_parallel_oracle_equals_the_oracle_to_the_last_bit():
    """The pull-based multi-threaded oracle (the CPU baseline on all host cores) adds every sum's
    terms in the single-threaded oracle's order, so its outputs are identical to the last bit:
    propagation forward and backward, and a T = 2 GGNN step forward and backward, with 4 threads
    on a packed batch with self-loops and a hub."""
    gs = synth.gen_batch(5, 50, 300, 4, True, 20, 12, 2.0, 404)
    gs = [synth.with_self_loops(g, 0.1, 8, 5 + i) for i, g in enumerate(gs)]
    gs.append(synth.hub_graph(150, 8, 9))
    lay = oracle.layout(gs, 8, 64)
    N, P, H, T = lay.n_pad, 8, 12, 2
    e = (lay.kept_dst, lay.kept_src, lay.kept_type)
    rng = np.random.default_rng(3)
    E = np.zeros((N, H)); E[:lay.n_real] = rng.standard_normal((lay.n_real, H))
    prm = synth.gen_params(P, H, 4)
    dY = rng.standard_normal((N, H))
    np.testing.assert_array_equal(oracle.par_propagate_fwd(N, P, H, *e, E, prm["W"], prm["b"], 4),
                                  oracle.propagate_fwd(N, P, H, *e, E, prm["W"], prm["b"]))
    for a, b in zip(oracle.par_propagate_bwd(N, P, H, *e, E, prm["W"], dY, 4),
                    oracle.propagate_bwd(N, P, H, *e, E, prm["W"], dY)):
        np.testing.assert_array_equal(a, b)
    Es, Ys = oracle.ggnn_fwd(N, P, H, T, lay.n_real, *e, E, prm)
    Es2, Ys2 = oracle.par_ggnn_fwd(N, P, H, T, lay.n_real, *e, E, prm, 4)
    np.testing.assert_array_equal(Es2, Es)
    np.testing.assert_array_equal(Ys2, Ys)
    r = oracle.ggnn_bwd(N, P, H, T, lay.n_real, *e, prm, Es, Ys, dY)
    r2 = oracle.par_ggnn_bwd(N, P, H, T, lay.n_real, *e, prm, Es, Ys, dY, 4)
    for k in r:
        np.testing.assert_array_equal(r2[k], r[k], err_msg=k)
    assert oracle.par_max_threads() >= 1



@pytest.mark.parametrize("seed", range(6))
def test_parallel_oracle_equals_the_oracle_on_unsorted_edge_lists(seed):
    """The same on raw edge lists in arbitrary order, with repeated edges and self-loops and thread
    counts from 1 to 7: the pull-based gather visits each target's and each source's edges in
    list order, as the scatter does."""
    rng = np.random.default_rng(600 + seed)
    N, P, H, T = int(rng.integers(5, 80)), int(rng.integers(1, 5)), int(rng.integers(1, 9)), 2
    m = int(rng.integers(0, 6 * N))
    e = (rng.integers(0, N, m), rng.integers(0, N, m), rng.integers(0, P, m))
    threads = int(rng.integers(1, 8))
    E = rng.standard_normal((N, H)); dY = rng.standard_normal((N, H))
    prm = synth.gen_params(P, H, 9 + seed)
    np.testing.assert_array_equal(
        oracle.par_propagate_fwd(N, P, H, *e, E, prm["W"], prm["b"], threads),
        oracle.propagate_fwd(N, P, H, *e, E, prm["W"], prm["b"]))
    for a, b in zip(oracle.par_propagate_bwd(N, P, H, *e, E, prm["W"], dY, threads),
                    oracle.propagate_bwd(N, P, H, *e, E, prm["W"], dY)):
        np.testing.assert_array_equal(a, b)
    n_real = N - int(rng.integers(0, 3))
    Es, Ys = oracle.ggnn_fwd(N, P, H, T, n_real, *e, E, prm)
    Es2, Ys2 = oracle.par_ggnn_fwd(N, P, H, T, n_real, *e, E, prm, threads)
    np.testing.assert_array_equal(Es2, Es)
    r = oracle.ggnn_bwd(N, P, H, T, n_real, *e, prm, Es, Ys, dY)
    r2 = oracle.par_ggnn_bwd(N, P, H, T, n_real, *e, prm, Es, Ys, dY, threads)
    for k in r:
        np.testing.assert_array_equal(r2[k], r[k], err_msg=k)

# ------------------------------------------------------------------------ reachability (Section 4)


@pytest.mark.parametrize("seed", [0, 1, 2, 3])
def test_reach_matches_all_pairs_shortest_paths(seed):
    """Brute force: directed shortest-path lengths by Floyd-Warshall on a small random graph; a
    node is kept iff its distance to the nearest candidate is at most T."""
    rng = np.random.default_rng(seed)
    n = 25
    m = 45
    src = rng.integers(0, n, m).astype(np.int32)
    dst = rng.integers(0, n, m).astype(np.int32)
    cand = np.unique(rng.integers(0, n, 3)).astype(np.int32)
    D = np.full((n, n), np.inf)
    np.fill_diagonal(D, 0)
    D[src, dst] = np.minimum(D[src, dst], 1)
    for k in range(n):
        D = np.minimum(D, D[:, [k]] + D[[k], :])
    for T in (0, 1, 2, 3, 6):
        want = D[:, cand].min(axis=1) <= T
        np.testing.assert_array_equal(oracle.reach(n, src, dst, cand, T), want)


def test_reach_on_a_chain_keeps_the_last_T_plus_one_nodes():
    """Chain 0 -> 1 -> ... -> n-1 with the last node the only candidate: exactly the T + 1 nodes
    n-1-T .. n-1 reach it within T steps; reversing the edges keeps only the candidate's
    successors-side nodes (none here)."""
    n = 40
    src = np.arange(n - 1, dtype=np.int32)
    dst = src + 1
    for T in (0, 1, 5, 8):
        keep = oracle.reach(n, src, dst, [n - 1], T)
        assert keep.sum() == T + 1 and keep[n - 1 - T:].all()
        rev = oracle.reach(n, dst, src, [n - 1], T)
        assert rev.sum() == 1 and rev[n - 1]


def test_reach_filter_leaves_candidate_states_unchanged():
    """The reason the preprocessing is lossless (Section 4): after T GGNN steps the candidates'
    states on the reduced graph equal those on the full graph (fp64, up to summation order)."""
    g = synth.gen_graph(300, 4, True, 12, 8, 1.0, 21)
    cand = synth.gen_candidates(g, 4, 5)
    T, H, P = 3, 8, 8
    node_map, nk, s2, d2, t2 = oracle.reach_filter(g, cand, T)
    assert 0 < nk < g.n_nodes
    prm = synth.gen_params(P, H, 6)
    E = synth.gen_states(g.n_nodes, H, 7)
    Es, _ = oracle.ggnn_fwd(g.n_nodes, P, H, T, g.n_nodes, g.dst, g.src, g.etype, E, prm)
    keep = node_map >= 0
    Er, _ = oracle.ggnn_fwd(nk, P, H, T, nk, d2, s2, t2, E[keep], prm)
    np.testing.assert_allclose(Er[T][node_map[cand]], Es[T][cand], rtol=1e-12, atol=1e-12)
    # and a node the preprocessing dropped would have changed nothing: perturbing it leaves the
    # candidates' final states as they were
    dropped = np.flatnonzero(~keep)[0]
    E2 = E.copy(); E2[dropped] += 10.0
    Es2, _ = oracle.ggnn_fwd(g.n_nodes, P, H, T, g.n_nodes, g.dst, g.src, g.etype, E2, prm)
    np.testing.assert_array_equal(Es2[T][cand], Es[T][cand])


# ------------------------------------------------------------------------ supernodes (Section 6)


def _star_chain(n_leaves, seed):
    """A chain over n_leaves + 1 nodes plus a hub (node 0) that every node sends a type-0 edge to
    and that sends a type-2 edge back to every node, relabelled at random."""
    g = synth.hub_graph(n_leaves, 3, seed, lam=0.0)
    hub = int(np.bincount(g.dst[g.etype == 0]).argmax())
    back = g.src[g.etype == 0]
    return synth.Graph(g.n_nodes, np.concatenate([g.src, np.full(len(back), hub, np.int32)]),
                       np.concatenate([g.dst, back]),
                       np.concatenate([g.etype, np.full(len(back), 2, np.int32)]), 3), hub


def test_supernode_selection_rule_and_positions():
    """Degrees are distinct neighbours over all types and both directions; nodes at or above the
    threshold become supernodes, highest degree first, ties by lower id, at most max_super; they
    take the graph's first positions in that order."""
    # node 0: 5 neighbours, node 1: 4, node 2: 4, others fewer; node 0 -> node 0 self-loop ignored
    src = np.array([0, 0, 0, 0, 0, 1, 1, 1, 2, 2, 2, 0, 7], np.int32)
    dst = np.array([1, 2, 3, 4, 5, 6, 7, 8, 6, 7, 8, 0, 2], np.int32)
    g = synth.Graph(9, src, dst, np.zeros(13, np.int32), 1)
    F = oracle.FLAG_RCM | oracle.FLAG_KEEP_IF_BETTER | oracle.FLAG_SUPERNODES
    lay = oracle.layout([g], 1, 32, flags=F, super_min_degree=4, max_super=8)
    assert list(lay.perm[:3]) == [0, 1, 2] and lay.is_super[:3].all() and not lay.is_super[3:].any()
    lay = oracle.layout([g], 1, 32, flags=F, super_min_degree=4, max_super=2)
    assert list(lay.perm[:2]) == [0, 1] and lay.is_super.sum() == 2
    lay = oracle.layout([g], 1, 32, flags=F, super_min_degree=6, max_super=8)
    plain = oracle.layout([g], 1, 32)
    assert not lay.is_super.any() and np.array_equal(lay.perm, plain.perm)


def test_supernodes_keep_every_hub_edge_and_restore_a_narrow_band():
    """A hub connected both ways to 300 chain nodes: without supernodes RCM cannot give a band
    narrower than about half the graph and the cover at S = 32 drops most hub edges; as a
    supernode the hub takes position 0, the rest is a chain of bandwidth 1, and nothing is
    dropped, so the band propagation equals dense brute force over all edges (Eq. 1)."""
    g, hub = _star_chain(300, 3)
    plain = oracle.layout([g], 3, 32)
    assert plain.n_dropped > 300 and plain.bw_after_max > 100
    F = oracle.FLAG_RCM | oracle.FLAG_KEEP_IF_BETTER | oracle.FLAG_SUPERNODES
    lay = oracle.layout([g], 3, 32, flags=F, super_min_degree=64, max_super=4)
    assert lay.perm[0] == hub and lay.is_super.sum() == 1
    assert lay.n_dropped == 0 and lay.bw_after_max == 1
    assert lay.kept_super.sum() == np.sum((g.src == hub) | (g.dst == hub))  # 300 in, 301 out
    # the band masks hold exactly the kept edges without a supernode end
    bits = np.unpackbits(lay.masks, bitorder="little").sum()
    assert bits == lay.n_kept - lay.kept_super.sum()
    H, P = 6, 3
    rng = np.random.default_rng(1)
    E = np.zeros((lay.n_pad, H)); E[:lay.n_real] = rng.standard_normal((lay.n_real, H))
    prm = synth.gen_params(P, H, 2)
    Y = oracle.propagate_fwd(lay.n_pad, P, H, lay.kept_dst, lay.kept_src, lay.kept_type, E,
                             prm["W"], prm["b"])
    pos = np.empty(g.n_nodes, np.int64); pos[lay.perm] = np.arange(g.n_nodes)
    A = np.zeros((P, lay.n_pad, lay.n_pad))
    A[g.etype, pos[g.dst], pos[g.src]] = 1.0
    want = sum(A[p] @ (E @ prm["W"][p]) + A[p].sum(1, keepdims=True) * prm["b"][p] for p in range(P))
    np.testing.assert_allclose(Y, want, rtol=1e-12, atol=1e-12)
