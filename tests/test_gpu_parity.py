"""GPU parity: the CUDA path, called through the C ABI, against the CPU oracle on the same seeded
inputs.  Tolerances (max-abs error over the reference's max-abs value, per tensor): 1e-4 for the
fp32 path, 2e-2 for the bf16 path (bf16 states/weights, fp32 accumulation); layout work is
bit-exact."""
import numpy as np
import pytest
import torch

import oracle
from paper_1906_11786_gb300 import _binding as L
from paper_1906_11786_gb300 import synth

from gpu_common import TOL, Case, assert_close, ensure_built, f32_dev, quantize, rel_err

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    ensure_built()
    torch.manual_seed(0)


def _tc_shape(c: Case) -> bool:
    """Shapes the fused tensor-core band kernels carry: bf16, P <= 32, whole 128-row tiles,
    H in {32, 64, 128} at S in {32, 64, 128, 256, 512}, H = 256 at S in {32, 64, 128}."""
    return (c.dtype == "bf16" and c.P <= 32 and c.N % 128 == 0 and
            ((c.H in (32, 64, 128) and c.S in (32, 64, 128, 256, 512)) or
             (c.H == 256 and c.S in (32, 64, 128))))


def _cap_whole_tiles(gs, S):
    """Capacity (blocks) that makes the padded size a whole number of 128-row tiles."""
    n = sum(g.n_nodes for g in gs)
    per_tile = max(1, 128 // S)
    blocks = -(-n // S)
    return -(-blocks // per_tile) * per_tile


def _expect_path(c: Case):
    """The fused tensor-core kernels must carry every shape they support."""
    assert L.band_uses_tensor_cores(c.plan, c.dtype, c.H) == _tc_shape(c)


def _fwd(c: Case, with_bias=True):
    _expect_path(c)
    Y = torch.empty((c.N, c.H), dtype=torch.float32, device="cuda")
    L.band_propagate_fwd(c.plan, c.dtype, c.H, c.E_band_dev, c.dprm["W"],
                         c.dprm["b"] if with_bias else None, Y, c.ws(L.BG_OP_PROPAGATE_FWD))
    torch.cuda.synchronize()
    L.check_device()
    ref = oracle.propagate_fwd(c.N, c.P, c.H, *c.edges, c.E_band, c.prm["W"],
                               c.prm["b"] if with_bias else None)
    return Y.cpu().numpy(), ref


def _bwd(c: Case, seed=7):
    dY = quantize(np.random.default_rng(seed).standard_normal((c.N, c.H)), "f32")
    dY[c.n_real:] = 0
    dE = torch.empty((c.N, c.H), dtype=torch.float32, device="cuda")
    dW = torch.empty((c.P, c.H, c.H), dtype=torch.float32, device="cuda")
    db = torch.empty((c.P, c.H), dtype=torch.float32, device="cuda")
    L.band_propagate_bwd(c.plan, c.dtype, c.H, c.E_band_dev, c.dprm["W"], f32_dev(dY), dE, dW, db,
                         c.ws(L.BG_OP_PROPAGATE_BWD))
    torch.cuda.synchronize()
    L.check_device()
    ref = oracle.propagate_bwd(c.N, c.P, c.H, *c.edges, c.E_band, c.prm["W"], dY)
    return (dE.cpu().numpy(), dW.cpu().numpy(), db.cpu().numpy()), ref


# ------------------------------------------------------------------------------------ layout


def test_pack_unpack_bit_exact():
    c = Case(synth.workload_graphs("packed64", scale=0.1), 20, 128, 64, "bf16", seed=3)
    got = c.E_band_dev.float().cpu().numpy()
    np.testing.assert_array_equal(got, c.E_band)
    back = torch.zeros_like(c.E_orig_dev)
    L.unpack_states(c.plan, c.dtype, c.H, c.E_band_dev, back)
    np.testing.assert_array_equal(back.float().cpu().numpy(), c.E_orig)


# ------------------------------------------------------------------------------------ propagate


def test_propagate_fp32_single512():
    """Single 512-node graph, 4 types, S = 64, H = 64, fp32, fwd + bwd."""
    c = Case(synth.workload_graphs("single512"), 4, 64, 64, "f32", seed=11)
    Y, ref = _fwd(c)
    assert_close(Y, ref, TOL["f32"], "")
    got, ref = _bwd(c)
    for g, r, name in zip(got, ref, ("dE", "dW", "db")):
        assert_close(g, r, TOL["f32"], name)


@pytest.mark.parametrize("S,H,whole", [(128, 64, 0), (64, 64, 1), (32, 32, 0), (256, 128, 0),
                                       (128, 256, 0), (256, 64, 1), (32, 64, 1), (64, 64, 0),
                                       (128, 128, 0), (64, 128, 1), (32, 128, 1),
                                       (64, 256, 1), (32, 256, 1), (128, 96, 0),
                                       (128, 32, 0), (64, 32, 1), (256, 32, 0),
                                       (512, 64, 0), (512, 32, 0), (512, 128, 0)])
def test_propagate_bf16_packed_batch(S, H, whole):
    """Several graphs packed into several block-rows with a ragged tail (`whole`: capacity padded
    to whole 128-row tiles, as the tensor-core kernels need below S = 128)."""
    gs = synth.gen_batch(7, 60, 400, 10, True, S // 2, S // 3, 2.0, 100 + S + H)
    c = Case(gs, 20, S, H, "bf16", seed=S + H, cap=_cap_whole_tiles(gs, S) if whole else 0)
    assert c.info["K"] >= 3 and c.n_real % S != 0
    Y, ref = _fwd(c)
    assert_close(Y, ref, TOL["bf16"], "")
    assert np.all(Y[c.n_real:] == 0)
    got, ref = _bwd(c)
    for g, r, name in zip(got, ref, ("dE", "dW", "db")):
        assert_close(g, r, TOL["bf16"], name)


def test_propagate_bf16_no_bias_and_single_block():
    g = synth.gen_graph(100, 4, True, 20, 10, 1.0, 5)
    c = Case([g], 8, 128, 64, "bf16", seed=2)
    assert c.info["K"] == 1
    Y, ref = _fwd(c, with_bias=False)
    assert_close(Y, ref, TOL["bf16"], "")


def test_propagate_graph_without_edges():
    g = synth.Graph(70, np.zeros(0, np.int32), np.zeros(0, np.int32), np.zeros(0, np.int32), 2)
    c = Case([g], 2, 32, 32, "f32")
    Y, ref = _fwd(c)
    assert np.all(Y == 0) and np.all(ref == 0)


def test_propagate_bf16_dropped_edges_single20k_shape():
    """Wide band: S = 256 < bandwidth, so some edges are dropped (coverage rule)."""
    g = synth.gen_graph(3000, 10, True, 200, 133, 3.0, 17)
    c = Case([g], 20, 256, 128, "bf16", seed=5)
    Y, ref = _fwd(c)
    assert_close(Y, ref, TOL["bf16"], "")


# ------------------------------------------------------------------------------------ GGNN


def _ggnn(c: Case, T, seed=3):
    saved = torch.empty(L.ggnn_saved_bytes(c.plan, c.dtype, c.H, T), dtype=torch.uint8,
                        device="cuda")
    ET = torch.empty_like(c.E_band_dev)
    L.ggnn_step(c.plan, c.dtype, c.H, T, c.dprm, c.E_band_dev, ET, saved, c.ws(L.BG_OP_GGNN_FWD, T))
    dET = quantize(np.random.default_rng(seed).standard_normal((c.N, c.H)), "f32")
    dE0 = torch.empty((c.N, c.H), dtype=torch.float32, device="cuda")
    grads = dict(dW=torch.empty((c.P, c.H, c.H), device="cuda"),
                 db=torch.empty((c.P, c.H), device="cuda"),
                 dW_ih=torch.empty((3 * c.H, c.H), device="cuda"),
                 dW_hh=torch.empty((3 * c.H, c.H), device="cuda"),
                 db_ih=torch.empty(3 * c.H, device="cuda"),
                 db_hh=torch.empty(3 * c.H, device="cuda"))
    L.ggnn_step_bwd(c.plan, c.dtype, c.H, T, c.dprm, saved, f32_dev(dET), dE0, grads,
                    c.ws(L.BG_OP_GGNN_BWD, T))
    torch.cuda.synchronize()
    L.check_device()
    Es, Ys = oracle.ggnn_fwd(c.N, c.P, c.H, T, c.n_real, *c.edges, c.E_band, c.prm)
    ref = oracle.ggnn_bwd(c.N, c.P, c.H, T, c.n_real, *c.edges, c.prm, Es, Ys, dET)
    return ET.float().cpu().numpy(), Es[T], {k: v.cpu().numpy() for k, v in grads.items()}, \
        dE0.cpu().numpy(), ref


@pytest.mark.parametrize("dtype,T,S,H,whole", [("f32", 2, 64, 64, 0), ("bf16", 3, 64, 64, 0),
                                               ("bf16", 2, 128, 128, 0), ("bf16", 2, 32, 32, 0),
                                               ("bf16", 2, 128, 256, 0), ("bf16", 2, 256, 64, 1),
                                               ("bf16", 2, 256, 128, 0), ("bf16", 3, 64, 128, 1),
                                               ("bf16", 2, 32, 128, 0), ("bf16", 2, 128, 32, 0),
                                               ("bf16", 3, 64, 64, 1), ("bf16", 2, 32, 64, 1),
                                               ("bf16", 3, 64, 32, 1)])
def test_ggnn_fwd_bwd(dtype, T, S, H, whole):
    """Every kernel family of the GGNN step: SIMT (fp32), tensor-core GEMMs around the SIMT band
    sums (ragged tiles: H = 32 at S = 32, and H = 128 at S = 32), the band kernel with the GEMM
    GRU (H = 256), fused band and GRU kernels at H = 32 (S = 64, 128), H = 64 (S = 32, 64, 256) and
    H = 128 (S = 64, 128, 256; weights streamed through the GRU kernels' piece ring)."""
    gs = synth.gen_batch(5, 60, 300, 10, True, max(8, S // 2), max(8, S // 3), 2.0, 41)
    c = Case(gs, 20, S, H, dtype, seed=9, cap=_cap_whole_tiles(gs, S) if whole else 0)
    assert L.band_uses_tensor_cores(c.plan, c.dtype, c.H) == _tc_shape(c)
    ET, ref_ET, grads, dE0, ref = _ggnn(c, T)
    tol = TOL[dtype]
    assert_close(ET, ref_ET, tol, "")
    assert np.all(ET[c.n_real:] == 0)
    assert_close(dE0, ref["dE0"], tol, "")
    for k, v in grads.items():
        assert_close(v, ref[k], tol, k)


def test_ggnn_packed64_shape_T8_reduced_batch():
    """The packed64 workload's shapes (P = 20, S = 128, H = 64, bf16, T = 8) on an 8-graph batch."""
    c = Case(synth.workload_graphs("packed64", scale=0.125), 20, 128, 64, "bf16", seed=2)
    ET, ref_ET, grads, dE0, ref = _ggnn(c, 8)
    assert_close(ET, ref_ET, TOL["bf16"], "")
    assert_close(dE0, ref["dE0"], TOL["bf16"], "")
    for k, v in grads.items():
        assert_close(v, ref[k], TOL["bf16"], k)


# ------------------------------------------------------------------------------------ readout, Adam


def test_readout_loss_and_adam():
    c = Case(synth.gen_batch(6, 50, 200, 3, True, 20, 10, 1.0, 8), 6, 64, 64, "bf16", seed=4)
    n_g = c.info["n_packed"]
    target = np.random.default_rng(1).standard_normal(n_g)
    loss = torch.zeros(4, device="cuda")
    dET = torch.empty((c.N, c.H), device="cuda")
    dw = torch.empty(c.H, device="cuda")
    L.readout_loss(c.plan, c.dtype, c.H, c.E_band_dev, c.dprm["w_out"], f32_dev(target), loss, dET,
                   dw, c.ws(L.BG_OP_READOUT))
    torch.cuda.synchronize()
    off, cnt = c.ref.graph_segments()
    rl, rdE, rdw = oracle.readout_loss(c.E_band, off, cnt, c.prm["w_out"], target)
    assert abs(loss[0].item() - rl) / abs(rl) < 1e-4
    assert rel_err(dET.cpu().numpy(), rdE) < 1e-4
    assert rel_err(dw.cpu().numpy(), rdw) < 1e-4
    # Adam on the edge weights: fp32 master, bf16 working copy
    rng = np.random.default_rng(2)
    p0 = rng.standard_normal(1000); g = rng.standard_normal(1000)
    master = f32_dev(p0); work = master.to(torch.bfloat16)
    m = torch.zeros_like(master); v = torch.zeros_like(master)
    rp, rm, rv = p0, np.zeros(1000), np.zeros(1000)
    for t in (1, 2):
        L.adam_step(master, work, m, v, f32_dev(g), 1e-3, 0.9, 0.999, 1e-8, t)
        rp, rm, rv = oracle.adam(rp, rm, rv, quantize(g, "f32"), 1e-3, 0.9, 0.999, 1e-8, t)
    torch.cuda.synchronize()
    assert rel_err(master.cpu().numpy(), rp) < 1e-5
    assert rel_err(work.float().cpu().numpy(), rp) < 1e-2


# ------------------------------------------------------------------------------------ full size


def _full_size_propagation(c: Case, seed: int, n_rows: int = 400, types=(0, 7, 13)):
    """One forward and one backward propagation through the C ABI on a full-size plan (the
    benchmark's launches), checked on outputs the oracle computes one by one:
      Y on sampled rows, from the kept edges into those rows (Eq. 1, Eq. 3);
      dE on the same rows, from a compacted problem holding the rows and the targets of their
      out-edges (dE[u] = sum_p (sum over edges u -> v of type p of dY[v]) W_p^T needs nothing else);
      dW_p and db_p for sampled types p, from the edges of those types over all nodes.
    Padding rows must come back as exact zeros in Y and dE."""
    assert L.band_uses_tensor_cores(c.plan, c.dtype, c.H)
    Y = torch.empty((c.N, c.H), dtype=torch.float32, device="cuda")
    L.band_propagate_fwd(c.plan, c.dtype, c.H, c.E_band_dev, c.dprm["W"], c.dprm["b"], Y,
                         c.ws(L.BG_OP_PROPAGATE_FWD))
    dY = quantize(np.random.default_rng(seed).standard_normal((c.N, c.H)), "f32")
    dY[c.n_real:] = 0
    dE = torch.empty((c.N, c.H), dtype=torch.float32, device="cuda")
    dW = torch.empty((c.P, c.H, c.H), dtype=torch.float32, device="cuda")
    db = torch.empty((c.P, c.H), dtype=torch.float32, device="cuda")
    L.band_propagate_bwd(c.plan, c.dtype, c.H, c.E_band_dev, c.dprm["W"], f32_dev(dY), dE, dW, db,
                         c.ws(L.BG_OP_PROPAGATE_BWD))
    torch.cuda.synchronize()
    L.check_device()
    Y, dE, dW, db = (x.cpu().numpy() for x in (Y, dE, dW, db))
    assert np.all(Y[c.n_real:] == 0) and np.all(dE[c.n_real:] == 0)

    rows = np.unique(np.concatenate([np.random.default_rng(seed + 1).integers(0, c.n_real, n_rows),
                                     [0, c.n_real - 1]]))
    d, s, t = c.edges
    sel = np.isin(d, rows)
    ref = oracle.propagate_fwd(c.N, c.P, c.H, d[sel], s[sel], t[sel], c.E_band, c.prm["W"],
                               c.prm["b"])
    assert_close(Y[rows], ref[rows], TOL["bf16"], "Y")

    out = np.isin(s, rows)
    nodes = np.unique(np.concatenate([rows, d[out]]))
    new = np.full(c.N, -1, np.int64)
    new[nodes] = np.arange(len(nodes))
    ref_dE, _, _ = oracle.propagate_bwd(len(nodes), c.P, c.H, new[d[out]], new[s[out]], t[out],
                                        c.E_band[nodes], c.prm["W"], dY[nodes])
    assert_close(dE[rows], ref_dE[new[rows]], TOL["bf16"], "dE")

    types = np.asarray(types)
    tmap = np.full(c.P, -1, np.int64)
    tmap[types] = np.arange(len(types))
    ts = tmap[t] >= 0
    _, ref_dW, ref_db = oracle.propagate_bwd(c.N, len(types), c.H, d[ts], s[ts], tmap[t[ts]],
                                             c.E_band, c.prm["W"][types], dY)
    assert_close(dW[types], ref_dW, TOL["bf16"], "dW")
    assert_close(db[types], ref_db, TOL["bf16"], "db")


def test_full_size_packed64_propagate_sampled_rows():
    """The packed64 workload at full size (64 graphs, ~72k nodes, 566 tiles, P = 20, S = 128, H = 64, bf16):
    one forward and backward propagation, every tile whole."""
    _full_size_propagation(Case(synth.workload_graphs("packed64"), 20, 128, 64, "bf16", seed=21), 41)


def test_full_size_single20k_propagate_sampled_rows():
    """The single20k workload at full size (one 20,000-node graph, S = 256, H = 128, 158 tiles): on a GPU with a
    few SMs fewer than tiles, a whole round of tiles runs as whole tiles and the few tiles left are
    split over several CTAs (partial sums and the fix-up kernel), the schedule the benchmark runs."""
    c = Case(synth.workload_graphs("single20k"), 20, 256, 128, "bf16", seed=43)
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    tiles = c.N // 128
    assert tiles > sms and tiles % sms < sms // 2
    _full_size_propagation(c, 47)


@pytest.mark.parametrize("S", [32, 256, 512])
def test_full_size_sweep131k_propagate_sampled_rows(S):
    """The block-size sweep at full size (131,072 positions, P = 20, H = 64, max offset S / 2):
    S = 32 (four block-rows per tile), S = 256 (six window chunks) and S = 512 (32-column state
    slices over a twelve-chunk window), with the sweep's capacity of 131,072 / S blocks."""
    c = Case(synth.workload_graphs("sweep131k", S=S), 20, S, 64, "bf16", seed=50 + S, cap=-(-131072 // S))
    assert c.N == 131072
    _full_size_propagation(c, 53 + S)


def _full_size_ggnn_sampled_graphs(c: Case, T: int, pick, seed: int):
    """Runs T GGNN steps forward and backward on the whole plan (the benchmark's launches) with a
    dE(T) that is zero outside the graphs `pick`, and checks them against the oracle run on those
    graphs alone.

    Graphs share no edge, so (Eq. 1 and Eq. 2 act per graph) E(T) of a graph depends on that graph
    alone, and a dE(T) that is zero outside a few sampled graphs leaves dE(0) zero outside them and
    makes every parameter gradient a sum over the sampled graphs only.  The oracle therefore runs on
    the sampled graphs, compacted, and is compared with the full-size launch on E(T) of the sampled
    rows, on all of dE(0) and on all six parameter gradients."""
    assert L.band_uses_tensor_cores(c.plan, c.dtype, c.H)
    saved = torch.empty(L.ggnn_saved_bytes(c.plan, c.dtype, c.H, T), dtype=torch.uint8,
                        device="cuda")
    ET = torch.empty_like(c.E_band_dev)
    L.ggnn_step(c.plan, c.dtype, c.H, T, c.dprm, c.E_band_dev, ET, saved, c.ws(L.BG_OP_GGNN_FWD, T))
    off, cnt = c.ref.graph_segments()
    rows = np.concatenate([np.arange(off[g], off[g] + cnt[g]) for g in pick])
    dET = np.zeros((c.N, c.H))
    dET[rows] = quantize(np.random.default_rng(seed).standard_normal((len(rows), c.H)), "f32")
    dE0 = torch.empty((c.N, c.H), dtype=torch.float32, device="cuda")
    grads = dict(dW=torch.empty((c.P, c.H, c.H), device="cuda"),
                 db=torch.empty((c.P, c.H), device="cuda"),
                 dW_ih=torch.empty((3 * c.H, c.H), device="cuda"),
                 dW_hh=torch.empty((3 * c.H, c.H), device="cuda"),
                 db_ih=torch.empty(3 * c.H, device="cuda"),
                 db_hh=torch.empty(3 * c.H, device="cuda"))
    L.ggnn_step_bwd(c.plan, c.dtype, c.H, T, c.dprm, saved, f32_dev(dET), dE0, grads,
                    c.ws(L.BG_OP_GGNN_BWD, T))
    torch.cuda.synchronize()
    L.check_device()

    # compact sub-problem: the sampled graphs' rows, renumbered 0..m-1, with their edges
    m = len(rows)
    new = np.full(c.N, -1, np.int64)
    new[rows] = np.arange(m)
    e_dst, e_src, e_type = c.edges
    sel = new[e_dst] >= 0
    assert np.all(new[e_src[sel]] >= 0)
    sub = (new[e_dst[sel]], new[e_src[sel]], e_type[sel])
    Es, Ys = oracle.ggnn_fwd(m, c.P, c.H, T, m, *sub, c.E_band[rows], c.prm)
    ref = oracle.ggnn_bwd(m, c.P, c.H, T, m, *sub, c.prm, Es, Ys, dET[rows])

    got_ET = ET.float().cpu().numpy()
    assert_close(got_ET[rows], Es[T], TOL["bf16"], "")
    got_dE0 = dE0.cpu().numpy()
    assert_close(got_dE0[rows], ref["dE0"], TOL["bf16"], "")
    rest = np.ones(c.N, bool)
    rest[rows] = False
    assert np.all(got_dE0[rest] == 0.0)
    for k, v in grads.items():
        assert_close(v.cpu().numpy(), ref[k], TOL["bf16"], k)
    return ET


def test_full_size_packed64_ggnn_T8_fwd_bwd_sampled_graphs():
    """The benchmark workload end to end: packed64 at full size (64 graphs, ~72k nodes, P = 20,
    S = 128, H = 64, bf16, T = 8) through the fused tensor-core path, forward + backward."""
    c = Case(synth.workload_graphs("packed64"), 20, 128, 64, "bf16", seed=23)
    off, _ = c.ref.graph_segments()
    _full_size_ggnn_sampled_graphs(c, 8, np.random.default_rng(5).choice(len(off), 4, replace=False),
                                   31)


@pytest.mark.parametrize("H", [32, 128, 256])
def test_full_size_train100k_ggnn_T8_fwd_bwd_sampled_graphs(H):
    """The train100k batch at full size with the benchmark's capacity (100,000 positions rounded up to
    whole blocks: 782 tiles, P = 20, S = 128, bf16, T = 8), forward + backward against the oracle on
    a few of the smaller graphs: H = 32 (32-column band products, resident-weight GRU kernels),
    H = 128 (64-column state passes, GRU weights streamed), H = 256 (four state passes, the GRU on
    tensor-core GEMMs); H = 64 runs at full size as packed64.  On a 152-SM GB300 the band kernels
    run five whole rounds of tiles and split the 22-tile tail four ways.  The training step's mean-pool readout and loss are checked over the whole batch on the E(T) the
    launch produced."""
    cap = -(-synth.WORKLOADS["train100k"]["sizes"][1] // 128)
    c = Case(synth.workload_graphs("train100k"), 20, 128, H, "bf16", seed=29, cap=cap)
    assert c.N == cap * 128
    off, cnt = c.ref.graph_segments()
    if H <= 128:
        pick = np.random.default_rng(7).choice(np.flatnonzero(cnt <= 1500), 3, replace=False)
    else:
        pick = np.argsort(cnt, kind="stable")[:2]  # the oracle's cost grows with H^2
    ET = _full_size_ggnn_sampled_graphs(c, 8, pick, 37)
    target = np.random.default_rng(11).standard_normal(len(off))
    loss = torch.zeros(4, device="cuda")
    dET = torch.empty((c.N, c.H), device="cuda")
    dw = torch.empty(c.H, device="cuda")
    L.readout_loss(c.plan, c.dtype, c.H, ET, c.dprm["w_out"], f32_dev(target), loss, dET, dw,
                   c.ws(L.BG_OP_READOUT))
    torch.cuda.synchronize()
    L.check_device()
    rl, rdE, rdw = oracle.readout_loss(ET.float().cpu().numpy().astype(np.float64), off, cnt,
                                       c.prm["w_out"], target)
    assert abs(loss[0].item() - rl) / abs(rl) < 1e-4
    assert rel_err(dET.cpu().numpy(), rdE) < 1e-4
    assert rel_err(dw.cpu().numpy(), rdw) < 1e-4


# ------------------------------------------------------------------------------------ failure path
def test_device_wait_timeout_is_reported_and_the_context_survives():
    """A bounded device wait that is never satisfied gives up after its poll cap, the status word
    carries BG_ETIMEOUT with the wait's site to the host, the word is cleared, and the context
    still runs and checks clean work (no fault, no hang: the wait returns by itself)."""
    L.selftest_device_wait()
    with pytest.raises(L.BandGGNNError) as err:
        L.check_device()
    assert "BG_ETIMEOUT" in str(err.value) and "901" in str(err.value)
    L.check_device()  # cleared
    g = synth.gen_graph(300, 4, True, 20, 10, 1.0, 11)
    c = Case([g], 8, 128, 64, "bf16", seed=4)
    Y, ref = _fwd(c)
    assert_close(Y, ref, TOL["bf16"], "")

