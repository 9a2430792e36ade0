"""The C-ABI library on the CPU: it loads, exports every declared symbol, and its host planner
(RCM, packing, band tiles) is bit-exact against the oracle's independent implementation."""
import ctypes

import numpy as np
import pytest

import oracle
from paper_1906_11786_gb300 import _binding as L
from paper_1906_11786_gb300 import build as B
from paper_1906_11786_gb300 import synth


@pytest.fixture(scope="module", autouse=True)
def built():
    B.build()
    L.load()


def test_every_declared_symbol_is_exported():
    lib = ctypes.CDLL(L.LIB_PATH)
    names = L.declared_symbols()
    assert len(names) >= 20
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing


def _compare(graphs, P, S, cap=0, flags=L.BG_RCM | L.BG_KEEP_IF_BETTER):
    plan = L.band_plan(graphs, P, S, cap, flags)
    ref = oracle.layout(graphs, P, S, cap, flags=flags)
    info = plan.info()
    assert info["K"] == ref.K and info["n_pad"] == ref.K * S
    assert info["n_packed"] == ref.n_packed and info["n_real"] == ref.n_real
    assert info["n_edges_unique"] == ref.n_unique
    assert info["n_kept"] == ref.n_kept and info["n_dropped"] == ref.n_dropped
    assert info["bw_before_max"] == ref.bw_before_max and info["bw_after_max"] == ref.bw_after_max
    np.testing.assert_array_equal(plan.export(L.BG_EXPORT_PERM), ref.perm)
    np.testing.assert_array_equal(plan.export(L.BG_EXPORT_OFFSETS), ref.offset)
    bw = plan.export(L.BG_EXPORT_BW)
    np.testing.assert_array_equal(bw[0], ref.bw_before)
    np.testing.assert_array_equal(bw[1], ref.bw_after)
    masks = plan.export(L.BG_EXPORT_MASKS)
    assert masks.tobytes() == ref.masks.tobytes()
    # transposed orientation: (j, e, p, c, i) set  <=>  forward (j+e-1, 2-e, p, i, c) set;
    # checked on every block-row of small plans and on a seeded sample of block-rows otherwise
    K = ref.K
    mT = plan.export(L.BG_EXPORT_MASKS_T)
    rows = range(K) if K * P * S * S <= 4_000_000 else \
        sorted(set(np.random.default_rng(0).integers(0, K, 12).tolist()) | {0, K - 1})
    for j in rows:
        tb = np.unpackbits(mT[j], axis=-1, bitorder="little")            # [3,P,S,S]
        for e in range(3):
            k = j + e - 1
            if 0 <= k < K:
                fb = np.unpackbits(ref.masks[k, 2 - e], axis=-1, bitorder="little")
                np.testing.assert_array_equal(tb[e], fb.transpose(0, 2, 1))
            else:
                assert not tb[e].any()
    np.testing.assert_array_equal(plan.export(L.BG_EXPORT_GATHER), ref.gather_index())
    return plan, ref


def test_planner_bit_exact_single512():
    _compare(synth.workload_graphs("single512"), 4, 64)


def test_planner_bit_exact_packed64():
    _compare(synth.workload_graphs("packed64"), 20, 128)


def test_planner_bit_exact_single20k():
    _compare(synth.workload_graphs("single20k"), 20, 256)


@pytest.mark.parametrize("S", [32, 128, 512])
def test_planner_bit_exact_self_loops_and_hubs(S):
    """Self-loops (reading c6: allowed, on the diagonal tile) and a hub node with more in-edges
    of one type than the block size: the planner stays bit-exact against the oracle."""
    gs = synth.gen_batch(4, 50, 2 * S, 5, True, max(2, S // 2), max(2, S // 3), 1.5, 900 + S)
    gs = [synth.with_self_loops(g, 0.2, 10, 31 + i) for i, g in enumerate(gs)]
    gs.insert(2, synth.with_self_loops(synth.hub_graph(S + 40, 10, 5 + S), 0.1, 10, 3))
    plan, ref = _compare(gs, 10, S)
    loops = sum(int(np.sum(g.src == g.dst)) for g in gs)
    assert loops > 0 and ref.n_kept > 0


@pytest.mark.parametrize("S", [32, 64, 128, 256, 512])
def test_planner_bit_exact_sweep131k_capacity(S):
    gs = synth.workload_graphs("sweep131k", S=S, scale=0.25)
    cap = max(1, (sum(g.n_nodes for g in gs) - 300) // S)  # the last graphs do not fit
    plan, ref = _compare(gs, 20, S, cap)
    assert ref.n_packed < len(gs)


def test_planner_bit_exact_train100k():
    """The train100k graphs (200 .. 5000 nodes, the largest RCM inputs of any workload), full batch."""
    _compare(synth.workload_graphs("train100k"), 20, 128)


def test_planner_without_rcm_and_without_keep():
    gs = synth.gen_batch(5, 40, 90, 3, True, 12, 8, 1.0, 3)
    _compare(gs, 6, 32, flags=0)
    _compare(gs, 6, 32, flags=L.BG_RCM)


def test_planner_tiny_golden_rcm():
    import json
    import os
    g = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "rcm_tiny.json")))
    for c in g["cases"]:
        e = np.array(c["edges"], np.int32)
        gr = synth.Graph(c["n"], e[:, 0].copy(), e[:, 1].copy(), np.zeros(len(e), np.int32), 1)
        plan = L.band_plan([gr], 1, 32)
        assert plan.export(L.BG_EXPORT_PERM).tolist() == c["perm"], c["name"]


def test_flop_counts():
    plan = L.band_plan(synth.workload_graphs("single512"), 4, 64)
    i = plan.info()
    K, S, P, H = i["K"], 64, 4, 64
    assert plan.flops(H, L.BG_FLOPS_BAND) == 2 * (3 * K - 2) * P * S * S * H
    assert plan.flops(H, L.BG_FLOPS_XFORM) == 2 * K * S * P * H * H
    assert plan.flops(H, L.BG_FLOPS_NNZ) == 2 * H * i["n_kept"]


@pytest.mark.parametrize("bad", ["id", "type", "S", "P", "capacity"])
def test_invalid_inputs_return_einval_or_ecapacity(bad):
    g = synth.gen_graph(50, 2, False, 5, 4, 1.0, 1)
    P, S, cap = 2, 32, 0
    if bad == "id":
        g.dst = g.dst.copy(); g.dst[3] = 50
    elif bad == "type":
        g.etype = g.etype.copy(); g.etype[0] = 2
    elif bad == "S":
        S = 48
    elif bad == "P":
        P = 0
    elif bad == "capacity":
        cap = 1
    with pytest.raises(L.BandGGNNError) as ei:
        L.band_plan([g], P, S, cap)
    assert ei.value.code == (-2 if bad == "capacity" else -1)
    assert L.load().bg_last_error().decode()


def test_device_calls_require_upload():
    import torch
    plan = L.band_plan(synth.workload_graphs("single512"), 4, 64)
    x = torch.zeros(16)
    # a plan that was never uploaded is rejected before any CUDA call
    rc = L.load().bg_band_propagate_fwd(plan.handle, 0, 64, x.data_ptr(), x.data_ptr(), None,
                                        x.data_ptr(), x.data_ptr(), 64, None)
    assert rc == -7


def test_workspace_and_saved_sizes_are_positive():
    plan = L.band_plan(synth.workload_graphs("single512"), 4, 64)
    for op in (L.BG_OP_PROPAGATE_FWD, L.BG_OP_PROPAGATE_BWD, L.BG_OP_READOUT):
        assert L.workspace_bytes(plan, "f32", 64, op) > 0
    for op in (L.BG_OP_GGNN_FWD, L.BG_OP_GGNN_BWD):
        assert L.ggnn_workspace_bytes(plan, "f32", 64, 8, op) > 0
    assert L.ggnn_saved_bytes(plan, "bf16", 64, 8) >= 9 * 512 * 64 * 2 + 8 * 512 * 64 * 4


def _probe_binary(tmp_path_factory):
    """Compiles tests/tiles_probe.cpp against the in-tree library (g++, host code only)."""
    import os
    import shutil
    import subprocess
    gxx = shutil.which("g++")
    if gxx is None:
        pytest.skip("g++ not available")
    here = os.path.dirname(os.path.abspath(__file__))
    root = os.path.dirname(here)
    pkg = os.path.dirname(L.LIB_PATH)
    exe = str(tmp_path_factory.mktemp("probe") / "tiles_probe")
    subprocess.run([gxx, "-O1", "-std=c++17", "-I", os.path.join(root, "include"), "-I",
                    os.path.join(pkg, "csrc"), os.path.join(here, "tiles_probe.cpp"), "-L", pkg,
                    "-lbandggnn", f"-Wl,-rpath,{pkg}", "-lpthread", "-o", exe], check=True)
    return exe


def _interleave(w):
    """Column 2j of a 32-column word to bit j, column 2j+1 to bit 16+j (the bf16-pair expansion
    order of the tensor-core kernels' A operand)."""
    w = w.astype(np.uint64)
    out = np.zeros_like(w)
    for j in range(16):
        out |= ((w >> np.uint64(2 * j)) & np.uint64(1)) << np.uint64(j)
        out |= ((w >> np.uint64(2 * j + 1)) & np.uint64(1)) << np.uint64(16 + j)
    return out.astype(np.uint32)


@pytest.mark.parametrize("S,hub", [(32, 0), (64, 0), (128, 0), (256, 0), (512, 0), (256, 1),
                                   (512, 1)])
def test_tensor_core_upload_layout_from_the_bit_tiles(S, hub, tmp_path_factory, tmp_path):
    """The host-built operands of the tensor-core band kernels, rebuilt from the plan's bit tiles
    (themselves bit-exact against the oracle): for each 128-row tile and type, C1 window chunks
    of 128 columns starting one block before the tile's block-row, 4 interleaved words per row,
    zero outside the row's three block diagonals; the transposed orientation likewise from the
    transposed tiles; and per row and type the in-degree over the three diagonals as bf16."""
    exe = _probe_binary(tmp_path_factory)
    P = 6
    gs = synth.gen_batch(5, 40, 3 * S, 6, False, max(2, S // 2), max(2, S // 3), 1.5, 300 + S)
    if hub:  # in-degrees above 256: the table switches to fp16
        gs.insert(1, synth.hub_graph(S + S // 4, 2, 7 + S))
    max_deg = _check_upload(exe, gs, P, S, tmp_path)
    assert (max_deg > 256) == bool(hub)


def _check_upload(exe, gs, P, S, tmp_path):
    """Runs the probe on `gs` (padded with an edgeless graph to whole 128-row tiles) and checks
    the tensor-core operands it writes against the ones rebuilt here from its bit tiles."""
    n = sum(g.n_nodes for g in gs)
    K0 = -(-n // S)
    if K0 * S % 128:  # whole 128-row tiles, as the tensor-core path requires: pad with a graph
        gs.append(synth.Graph(128 * (-(-K0 * S // 128)) - n, np.zeros(0, np.int32),
                              np.zeros(0, np.int32), np.zeros(0, np.int32), P))
    blob = [np.int32(len(gs)).tobytes()]
    for g in gs:
        blob += [np.int32(g.n_nodes).tobytes(), np.int64(g.n_edges).tobytes(),
                 np.asarray(g.src, np.int32).tobytes(), np.asarray(g.dst, np.int32).tobytes(),
                 np.asarray(g.etype, np.int32).tobytes()]
    (tmp_path / "in.bin").write_bytes(b"".join(blob))
    C1 = 2 if S <= 64 else 3 * S // 128
    import subprocess
    subprocess.run([exe, str(tmp_path / "in.bin"), str(tmp_path / "out.bin"), str(P), str(S),
                    str(C1)], check=True)
    raw = (tmp_path / "out.bin").read_bytes()
    K, max_deg = np.frombuffer(raw[:8], np.int32)
    nm, nI, nTI, nd = np.frombuffer(raw[8:40], np.int64)
    o = 40
    masks = np.frombuffer(raw[o:o + 4 * nm], np.uint32); o += 4 * nm
    masksT = np.frombuffer(raw[o:o + 4 * nm], np.uint32); o += 4 * nm
    mI = np.frombuffer(raw[o:o + 4 * nI], np.uint32); o += 4 * nI
    mTI = np.frombuffer(raw[o:o + 4 * nTI], np.uint32); o += 4 * nTI
    deg = np.frombuffer(raw[o:o + 2 * nd], np.uint16)
    W32 = S // 32
    N = int(K) * S
    T = N // 128
    assert N % 128 == 0 and nI == T * P * C1 * 128 * 4 and nd == N * 64
    for tiles, got in ((masks, mI), (masksT, mTI)):
        tiles = tiles.reshape(int(K), 3, P, S, W32)
        exp = np.zeros((T, P, C1, 128, 4), np.uint32)
        for t in range(T):
            R = 128 * t + np.arange(128)
            kr = R // S
            ws = (128 * t // S) * S - S
            for j in range(C1):
                for w in range(4):
                    c = ws + 128 * j + 32 * w
                    if not 0 <= c < N:
                        continue
                    d = c // S - kr + 1
                    ok = (d >= 0) & (d <= 2)
                    words = tiles[kr[ok], d[ok], :, R[ok] % S, (c % S) // 32]   # [rows, P]
                    exp[t, :, j, np.flatnonzero(ok), w] = _interleave(words)  # [rows, P]
        np.testing.assert_array_equal(got.reshape(T, P, C1, 128, 4), exp)
    bits = np.unpackbits(masks.reshape(int(K), 3, P, S, W32).view(np.uint8), axis=-1)
    cnt = bits.reshape(int(K), 3, P, S, -1).sum(axis=(1, 4))                    # [K, P, S]
    if cnt.max() > 256:  # a hub: fp16 integers (exact up to 2048)
        enc = cnt.astype(np.float16).view(np.uint16)
    else:
        enc = (cnt.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    exp_deg = np.zeros((N, 64), np.uint16)
    exp_deg[:, :P] = enc.transpose(0, 2, 1).reshape(N, P)
    exp_deg[:, 32:32 + P] = exp_deg[:, :P]
    np.testing.assert_array_equal(deg.reshape(N, 64), exp_deg)
    assert max_deg == cnt.max()
    return int(max_deg)


@pytest.mark.parametrize("T", [0, 1, 3, 8])
def test_reach_filter_bit_exact_against_the_oracle(T):
    """Reachability preprocessing (Section 4): the library's kept nodes, renumbering and kept
    edges equal the oracle's, on program-shaped graphs with seeded candidates, at several T."""
    for i, g in enumerate(synth.gen_batch(6, 50, 1500, 10, True, 96, 64, 3.0, 77 + T)):
        cand = synth.gen_candidates(g, 5, 100 + i)
        got = L.reach_filter(g, cand, T)
        want = oracle.reach_filter(g, cand, T)
        np.testing.assert_array_equal(got[0], want[0])
        assert got[1] == want[1]
        for a, b in zip(got[2:], want[2:]):
            np.testing.assert_array_equal(a, b)
    with pytest.raises(L.BandGGNNError):
        L.reach_filter(g, [g.n_nodes], T)


def _hub_batch(S, seed):
    """Program-shaped graphs with hubs: two hub graphs (one node sending to and receiving from
    every other node) among ordinary ones."""
    gs = synth.gen_batch(4, 100, max(3 * S, 300), 5, True, max(2, S // 2), max(2, S // 3), 1.5,
                         seed)
    for i, k in ((1, 3 * S), (3, S + 7)):
        h = synth.hub_graph(k, 10, seed + i, lam=1.0)
        hub = int(np.bincount(h.dst[h.etype == 0]).argmax())
        back = h.src[h.etype == 0]
        gs.insert(i, synth.Graph(h.n_nodes, np.concatenate([h.src, np.full(len(back), hub, np.int32)]),
                                 np.concatenate([h.dst, back]),
                                 np.concatenate([h.etype, np.full(len(back), 5, np.int32)]), 10))
    return gs


@pytest.mark.parametrize("S,min_deg,max_sup", [(32, 64, 4), (128, 100, 2), (512, 40, 8),
                                               (64, 1000000, 4)])
def test_planner_bit_exact_with_supernodes(S, min_deg, max_sup):
    """Supernodes (Section 6): the library's positions, band tiles, counts and supernode edge
    list equal the oracle's independent layout; every edge with a supernode end is kept, and the
    band masks hold the other kept edges only."""
    gs = _hub_batch(S, 60 + S)
    F = L.BG_RCM | L.BG_KEEP_IF_BETTER | L.BG_SUPERNODES
    plan = L.band_plan(gs, 10, S, 0, F, min_deg, max_sup)
    ref = oracle.layout(gs, 10, S, flags=F, super_min_degree=min_deg, max_super=max_sup)
    info = plan.info()
    for k in ("K", "n_packed", "n_real"):
        assert info[k] == getattr(ref, k)
    assert info["n_kept"] == ref.n_kept and info["n_dropped"] == ref.n_dropped
    assert info["bw_after_max"] == ref.bw_after_max and info["n_edges_unique"] == ref.n_unique
    np.testing.assert_array_equal(plan.export(L.BG_EXPORT_PERM), ref.perm)
    assert plan.export(L.BG_EXPORT_MASKS).tobytes() == ref.masks.tobytes()
    sup = plan.export(L.BG_EXPORT_SUPER_EDGES)
    want = np.stack([ref.kept_dst, ref.kept_src, ref.kept_type], 1)[ref.kept_super]
    np.testing.assert_array_equal(sup, want)
    assert info["n_super_edges"] == len(want) and info["n_super"] == ref.is_super.sum()
    counts = plan.export(L.BG_EXPORT_SUPER_COUNT)
    assert counts.sum() >= info["n_super"]
    if min_deg < 1000:
        assert info["n_super"] > 0 and len(want) > 0
        plain = L.band_plan(gs, 10, S)
        assert plain.info()["n_dropped"] > info["n_dropped"]
    else:
        assert info["n_super"] == 0 and len(want) == 0


def edges_from_masks(m, S, transposed=False):
    """(dst, src, type) of the set bits of exported forward (or transposed) band masks."""
    bits = np.unpackbits(m, axis=-1, bitorder="little")
    k, d, p, r, c = np.nonzero(bits)
    a, b = k.astype(np.int64) * S + r, (k.astype(np.int64) + d - 1) * S + c
    return (b, a, p) if transposed else (a, b, p)


@pytest.mark.parametrize("S,n_parts", [(32, 2), (128, 3), (256, 2), (64, 5)])
def test_partition_tiles_rows_and_halos(S, n_parts):
    """Block-row split (Eq. 3): the parts own contiguous ranges of whole units (max(128, S) rows)
    covering the supergraph; each local plan spans its range plus one unit of halo per side; its forward
    tiles hold exactly the kept edges whose target it owns and its transposed tiles those whose
    source it owns, in local positions."""
    gs = synth.gen_batch(8, 100, 600, 4, True, max(2, S // 2), max(2, S // 3), 1.5, 5 + S)
    full = _check_partition(gs, 8, S, n_parts)
    with pytest.raises(L.BandGGNNError):
        L.plan_partition(full, 0, 0)
    sup = L.band_plan([synth.hub_graph(300, 8, 1)], 8, S, 0,
                      L.BG_RCM | L.BG_KEEP_IF_BETTER | L.BG_SUPERNODES, 100, 1)
    with pytest.raises(L.BandGGNNError):
        L.plan_partition(sup, 2, 0)


def _check_partition(gs, P, S, n_parts):
    """Plans `gs` at whole 128-row tiles, splits the plan into n_parts and checks every part
    (own ranges, halos, local forward and transposed tiles, real rows); returns the plan."""
    n = sum(g.n_nodes for g in gs)
    unit = max(1, 128 // S)
    cap = -(-(-(-n // S)) // unit) * unit
    full = L.band_plan(gs, P, S, cap)
    fi = full.info()
    d, s_, t = edges_from_masks(full.export(L.BG_EXPORT_MASKS), S)
    pos_all = []
    for part in range(n_parts):
        sub, inf = L.plan_partition(full, n_parts, part)
        si = sub.info()
        assert si["n_pad"] == inf["n_local"] and inf["n_local"] % 128 == 0
        assert inf["halo_lo"] == inf["own_begin"] and inf["halo_hi"] == inf["n_local"] - inf["own_end"]
        assert inf["halo_lo"] == (0 if part == 0 else max(S, 128))
        assert inf["halo_hi"] == (0 if part == n_parts - 1 else max(S, 128))
        own = np.arange(inf["own_begin"], inf["own_end"]) + inf["row0"]
        pos_all.append(own)
        r0 = inf["row0"]
        ld, ls, lt = edges_from_masks(sub.export(L.BG_EXPORT_MASKS), S)
        sel = np.isin(d, own)
        got = sorted(zip((ld + r0).tolist(), (ls + r0).tolist(), lt.tolist()))
        assert got == sorted(zip(d[sel].tolist(), s_[sel].tolist(), t[sel].tolist()))
        ld, ls, lt = edges_from_masks(sub.export(L.BG_EXPORT_MASKS_T), S, transposed=True)
        sel = np.isin(s_, own)
        got = sorted(zip((ld + r0).tolist(), (ls + r0).tolist(), lt.tolist()))
        assert got == sorted(zip(d[sel].tolist(), s_[sel].tolist(), t[sel].tolist()))
        assert si["n_real"] == max(0, min(inf["n_local"], fi["n_real"] - r0))
    pos_all = np.concatenate(pos_all)
    np.testing.assert_array_equal(pos_all, np.arange(fi["n_pad"]))
    return full


def _random_graph(rng, n, P):
    """Arbitrary (not program-shaped) typed edges: uniform pairs, a dense clump, duplicates,
    self-loops and isolated nodes."""
    m = int(rng.integers(0, 4 * n + 1)) if n else 0
    src = rng.integers(0, max(n, 1), m)
    dst = rng.integers(0, max(n, 1), m)
    if n >= 8 and rng.random() < 0.5:  # a dense clump of 8 nodes somewhere in the graph
        c = rng.choice(n, 8, replace=False)
        a, b = np.meshgrid(c, c)
        src, dst = np.concatenate([src, a.ravel()]), np.concatenate([dst, b.ravel()])
    if len(src) and rng.random() < 0.5:  # duplicates
        k = rng.integers(0, len(src), len(src) // 4 + 1)
        src, dst = np.concatenate([src, src[k]]), np.concatenate([dst, dst[k]])
    typ = rng.integers(0, P, len(src))
    return synth.Graph(n, src.astype(np.int32), dst.astype(np.int32), typ.astype(np.int32), P)


@pytest.mark.parametrize("seed", range(48))
def test_planner_bit_exact_on_arbitrary_graphs(seed):
    """Random batches of arbitrary graphs (0 to 400 nodes, up to 4n random typed edges plus dense
    clumps, duplicates and self-loops), every block size, random capacities (the batch may not
    fit) and every ordering flag: the planner stays bit-exact against the oracle."""
    rng = np.random.default_rng(7000 + seed)
    P = int(rng.integers(1, 7))
    S = int(rng.choice([32, 64, 128, 256, 512]))
    sizes = [0 if rng.random() < 0.1 else int(rng.integers(1, 401))
             for _ in range(int(rng.integers(1, 7)))]
    gs = [_random_graph(rng, n, P) for n in sizes]
    total = sum(g.n_nodes for g in gs)
    cap = 0 if rng.random() < 0.5 else int(rng.integers(1, max(1, -(-total // S)) + 1))
    if cap and gs[0].n_nodes > cap * S:
        cap = max(1, -(-gs[0].n_nodes // S))  # at least the first graph fits
    flags = [0, L.BG_RCM, L.BG_RCM | L.BG_KEEP_IF_BETTER][int(rng.integers(0, 3))]
    _compare(gs, P, S, cap, flags)


def test_planner_bit_exact_on_batches_without_nodes():
    e = np.zeros(0, np.int32)
    empty = synth.Graph(0, e, e, e, 3)
    plan, ref = _compare([empty], 3, 64)
    assert ref.K == 1 and ref.n_real == 0
    _compare([empty, synth.gen_graph(70, 3, False, 6, 4, 1.0, 2), empty], 3, 32)


@pytest.mark.parametrize("seed", range(24))
def test_reach_filter_bit_exact_on_arbitrary_graphs(seed):
    """Reachability preprocessing on arbitrary graphs (duplicates, self-loops, isolated nodes,
    repeated candidates, T from 0 to 6): the library's kept nodes, renumbering and kept edges
    equal the oracle's."""
    rng = np.random.default_rng(8100 + seed)
    g = _random_graph(rng, int(rng.integers(1, 301)), int(rng.integers(1, 5)))
    cand = rng.integers(0, g.n_nodes, int(rng.integers(1, 6))).astype(np.int32)
    T = int(rng.integers(0, 7))
    got = L.reach_filter(g, cand, T)
    want = oracle.reach_filter(g, cand, T)
    np.testing.assert_array_equal(got[0], want[0])
    assert got[1] == want[1]
    for a, b in zip(got[2:], want[2:]):
        np.testing.assert_array_equal(a, b)


@pytest.mark.parametrize("seed", range(24))
def test_planner_bit_exact_with_supernodes_on_arbitrary_graphs(seed):
    """Supernodes on arbitrary graphs with random thresholds and caps (including none found and
    more candidates than the cap): positions, band tiles, counts and the supernode edge list equal
    the oracle's."""
    rng = np.random.default_rng(8200 + seed)
    P = int(rng.integers(1, 6))
    S = int(rng.choice([32, 64, 128, 256, 512]))
    gs = [_random_graph(rng, int(rng.integers(0, 301)), P) for _ in range(int(rng.integers(1, 5)))]
    min_deg = int(rng.integers(1, 40))
    max_sup = int(rng.integers(0, 6))
    F = L.BG_RCM | L.BG_KEEP_IF_BETTER | L.BG_SUPERNODES
    plan = L.band_plan(gs, P, S, 0, F, min_deg, max_sup)
    ref = oracle.layout(gs, P, S, flags=F, super_min_degree=min_deg, max_super=max_sup)
    info = plan.info()
    for k in ("K", "n_packed", "n_real"):
        assert info[k] == getattr(ref, k)
    assert info["n_kept"] == ref.n_kept and info["n_dropped"] == ref.n_dropped
    assert info["bw_after_max"] == ref.bw_after_max and info["n_edges_unique"] == ref.n_unique
    np.testing.assert_array_equal(plan.export(L.BG_EXPORT_PERM), ref.perm)
    np.testing.assert_array_equal(plan.export(L.BG_EXPORT_OFFSETS), ref.offset)
    assert plan.export(L.BG_EXPORT_MASKS).tobytes() == ref.masks.tobytes()
    sup = plan.export(L.BG_EXPORT_SUPER_EDGES)
    want = np.stack([ref.kept_dst, ref.kept_src, ref.kept_type], 1)[ref.kept_super]
    np.testing.assert_array_equal(sup.reshape(-1, 3), want.reshape(-1, 3))
    assert info["n_super_edges"] == len(want) and info["n_super"] == ref.is_super.sum()


@pytest.mark.parametrize("seed", range(12))
def test_tensor_core_upload_layout_on_arbitrary_graphs(seed, tmp_path_factory, tmp_path):
    """The tensor-core operands on arbitrary graphs (dropped edges, duplicates, self-loops, dense
    clumps), every block size."""
    rng = np.random.default_rng(8300 + seed)
    P = int(rng.integers(1, 7))
    S = int(rng.choice([32, 64, 128, 256, 512]))
    gs = [_random_graph(rng, int(rng.integers(1, 401)), P) for _ in range(int(rng.integers(1, 5)))]
    _check_upload(_probe_binary(tmp_path_factory), gs, P, S, tmp_path)


@pytest.mark.parametrize("seed", range(16))
def test_partition_on_arbitrary_graphs(seed):
    """The block-row split on arbitrary graphs (dropped edges, duplicates, self-loops), every block
    size, from two parts up to one part per unit of max(128, S) rows."""
    rng = np.random.default_rng(8400 + seed)
    P = int(rng.integers(1, 7))
    S = int(rng.choice([32, 64, 128, 256, 512]))
    gs = [_random_graph(rng, int(rng.integers(1, 401)), P) for _ in range(int(rng.integers(2, 7)))]
    n = sum(g.n_nodes for g in gs)
    rows = max(128, S)  # the partition's unit: a 128-row tile, or one block-row when S > 128
    if -(-n // rows) < 2:
        gs.append(_random_graph(rng, rows, P))
        n += rows
    units = -(-n // rows)
    _check_partition(gs, P, S, int(rng.integers(2, min(units, 6) + 1)))


def _header_prototypes():
    """(return type, [argument types]) of every function the C header declares."""
    import re
    src = open(L.HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    src = re.sub(r"//[^\n]*", "", src)
    out = {}
    for m in re.finditer(r"([A-Za-z_][\w\s\*]*?)\s*\b(bg_\w+)\s*\(([^;{]*?)\)\s*;", src):
        ret, name, args = m.group(1).strip(), m.group(2), m.group(3).strip()
        ret = ret.split("\n")[-1].strip()
        params = [] if args in ("", "void") else [a.strip() for a in args.split(",")]
        # drop the parameter name: the type is everything before the last identifier
        types = [re.sub(r"\s*\b\w+$", "", a) if not a.endswith("*") else a for a in params]
        out[name] = (ret, types)
    return out


def _ctype_of(ctype: str):
    t = " ".join(ctype.replace("const ", "").split())
    if "*" in t:
        return "char_p" if t.replace(" ", "") == "char*" else "pointer"
    return {"int": ctypes.c_int, "int32_t": ctypes.c_int32, "uint32_t": ctypes.c_uint32,
            "int64_t": ctypes.c_int64, "size_t": ctypes.c_size_t, "float": ctypes.c_float,
            "double": ctypes.c_double, "bg_dtype": ctypes.c_int, "void": None}[t]


def test_binding_signatures_match_the_header():
    """Every function the header declares is bound with the same number of arguments and
    matching types (pointer, 32/64-bit integer, size, float, double) and return type: a
    mismatch would hand the library shifted or truncated arguments."""
    lib = L.load()
    protos = _header_prototypes()
    assert set(protos) == set(L.declared_symbols())
    for name, (ret, args) in protos.items():
        fn = getattr(lib, name)
        assert fn.argtypes is not None, f"{name} has no bound signature"
        assert len(fn.argtypes) == len(args), (name, len(fn.argtypes), args)
        for i, (a, b) in enumerate(zip(args, fn.argtypes)):
            want = _ctype_of(a)
            if want == "pointer":
                assert b in (ctypes.c_void_p, ctypes.c_char_p), (name, i, a, b)
            else:
                assert b is want or ctypes.sizeof(b) == ctypes.sizeof(want) and \
                    (b in (ctypes.c_float, ctypes.c_double)) == (want in (ctypes.c_float,
                                                                          ctypes.c_double)), \
                    (name, i, a, b)
        want = _ctype_of(ret)
        if want == "pointer":
            assert fn.restype == ctypes.c_void_p, (name, ret)
        elif want == "char_p":
            assert fn.restype == ctypes.c_char_p, (name, ret)
        elif want is None:
            assert fn.restype is None, (name, ret)
        else:
            assert fn.restype is want or ctypes.sizeof(fn.restype) == ctypes.sizeof(want), \
                (name, ret, fn.restype)


def test_binding_structs_match_the_c_layout(tmp_path):
    """The ctypes structures of the binding have the header's fields in its order, at the offsets
    and total size the C compiler gives them (a small C program compiled against the header
    prints them)."""
    import re
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    src = re.sub(r"/\*.*?\*/", "", open(L.HEADER).read(), flags=re.S)
    structs = {}
    for m in re.finditer(r"typedef struct (bg_\w+) \{(.*?)\} \1;", src, flags=re.S):
        fields = re.findall(r"(\w+)\s*;", m.group(2))
        structs[m.group(1)] = fields
    assert set(structs) == {"bg_graph", "bg_info", "bg_plan_opts", "bg_part_info", "bg_params",
                            "bg_grads"}
    lines = ['#include <stddef.h>', '#include <stdio.h>', '#include "bandggnn.h"', "int main(void) {"]
    for s, fields in structs.items():
        lines.append(f'  printf("{s} . %zu\\n", sizeof({s}));')
        for f in fields:
            lines.append(f'  printf("{s} {f} %zu\\n", offsetof({s}, {f}));')
    lines += ["  return 0;", "}"]
    (tmp_path / "layout.c").write_text("\n".join(lines))
    exe = str(tmp_path / "layout")
    import os
    inc = os.path.dirname(L.HEADER)
    subprocess.run([cc, "-std=c99", "-I", inc, str(tmp_path / "layout.c"), "-o", exe], check=True)
    got = {}
    for line in subprocess.run([exe], capture_output=True, text=True, check=True).stdout.split("\n"):
        if line:
            s, f, v = line.split()
            got[(s, f)] = int(v)
    for s, fields in structs.items():
        cls = getattr(L, s)
        assert [f for f, _ in cls._fields_] == fields, s
        assert ctypes.sizeof(cls) == got[(s, ".")], s
        for f in fields:
            assert getattr(cls, f).offset == got[(s, f)], (s, f)


def test_binding_constants_match_the_header():
    """Every constant of the header (status codes, flags, dtype values, export, op and kernel ids)
    has the same value in the binding; the status names cover every code."""
    import re
    src = re.sub(r"/\*.*?\*/", "", open(L.HEADER).read(), flags=re.S)
    consts = {m.group(1): int(m.group(2))
              for m in re.finditer(r"#define (BG_\w+)\s+\(?(-?\d+)u?\)?", src)}
    for m in re.finditer(r"(BG_\w+)\s*=\s*(-?\d+)", src):
        consts[m.group(1)] = int(m.group(2))
    assert len(consts) >= 30
    status = {k: v for k, v in consts.items() if k in ("BG_OK",) or k.startswith("BG_E") and
              not k.startswith("BG_EXPORT")}
    assert {v: k for k, v in status.items()} == L.STATUS
    missing = []
    for k, v in consts.items():
        if k in status or k == "BG_KID_COUNT":
            continue
        if not hasattr(L, k):
            missing.append(k)
        else:
            assert getattr(L, k) == v, (k, getattr(L, k), v)
    assert not missing, missing
