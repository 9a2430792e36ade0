"""CPU oracle for band-GGNN propagation -- TEST INFRASTRUCTURE ONLY.

Plain fp64 C++ (oracle.cpp) behind ctypes.  Only the tests, the smoke check and the benchmark's
CPU-baseline leg may import this package; the CUDA library never does, and the oracle imports
nothing from the library.  Inputs come from `paper_1906_11786_gb300.synth`, which draws random
numbers only.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.cpp")
_SRC_PAR = os.path.join(_HERE, "oracle_par.cpp")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

_i32p = np.ctypeslib.ndpointer(np.int32, flags="C_CONTIGUOUS")
_i64p = np.ctypeslib.ndpointer(np.int64, flags="C_CONTIGUOUS")
_f64p = np.ctypeslib.ndpointer(np.float64, flags="C_CONTIGUOUS")
_u8p = np.ctypeslib.ndpointer(np.uint8, flags="C_CONTIGUOUS")


def build(force: bool = False) -> str:
    """Compile oracle.cpp and its multi-threaded variant oracle_par.cpp into liboracle.so (g++ -O2,
    portable flags only; no floating-point contraction, so that both files evaluate every
    expression exactly as written on every host; OpenMP when the compiler has it)."""
    with _lock:
        newest = max(os.path.getmtime(_SRC), os.path.getmtime(_SRC_PAR))
        if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < newest:
            tmp = _LIB + f".tmp{os.getpid()}"
            base = ["g++", "-O2", "-std=c++17", "-ffp-contract=off", "-shared", "-fPIC", "-o", tmp,
                    _SRC, _SRC_PAR]
            if subprocess.call(base + ["-fopenmp"], stderr=subprocess.DEVNULL) != 0:
                subprocess.check_call(base)
            os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is not None:
        return _lib
    build()
    lib = ctypes.CDLL(_LIB)
    c = ctypes
    opt = lambda t: t  # noqa: E731  (nullable pointers are passed as None through c_void_p)
    lib.orc_bandwidth.restype = c.c_int64
    lib.orc_bandwidth.argtypes = [c.c_int32, c.c_int64, _i32p, _i32p, c.c_void_p]
    lib.orc_rcm.restype = c.c_int
    lib.orc_rcm.argtypes = [c.c_int32, c.c_int64, _i32p, _i32p, c.c_int, _i32p]
    lib.orc_reach.restype = c.c_int32
    lib.orc_reach.argtypes = [c.c_int32, c.c_int64, _i32p, _i32p, _i32p, c.c_int32, c.c_int32, _u8p]
    lib.orc_num_blocks.restype = c.c_int32
    lib.orc_num_blocks.argtypes = [c.c_int32, _i32p, c.c_int32, c.c_int32]
    lib.orc_layout.restype = c.c_int
    lib.orc_layout.argtypes = [c.c_int32, _i32p, _i64p, _i32p, _i32p, _i32p, c.c_int32, c.c_int32,
                               c.c_int32, c.c_int32, _i32p, _i32p, _i64p, c.c_void_p, c.c_void_p,
                               c.c_void_p, c.c_void_p, _i64p, _i64p, c.c_int32, c.c_int32,
                               c.c_void_p, c.c_void_p]
    lib.orc_propagate_fwd.restype = None
    lib.orc_propagate_fwd.argtypes = [c.c_int32] * 3 + [c.c_int64, _i32p, _i32p, _i32p, _f64p,
                                                         _f64p, c.c_void_p, _f64p]
    lib.orc_propagate_bwd.restype = None
    lib.orc_propagate_bwd.argtypes = [c.c_int32] * 3 + [c.c_int64, _i32p, _i32p, _i32p, _f64p,
                                                         _f64p, _f64p, _f64p, _f64p, c.c_void_p]
    lib.orc_gru_fwd.restype = None
    lib.orc_gru_fwd.argtypes = [c.c_int32] * 3 + [_f64p] * 7
    lib.orc_gru_bwd.restype = None
    lib.orc_gru_bwd.argtypes = [c.c_int32] * 3 + [_f64p] * 13
    lib.orc_ggnn_fwd.restype = None
    lib.orc_ggnn_fwd.argtypes = [c.c_int32] * 5 + [c.c_int64, _i32p, _i32p, _i32p] + [_f64p] * 8
    lib.orc_ggnn_bwd.restype = None
    lib.orc_ggnn_bwd.argtypes = ([c.c_int32] * 5 + [c.c_int64, _i32p, _i32p, _i32p] + [_f64p] * 16)
    lib.orc_readout_loss.restype = None
    lib.orc_readout_loss.argtypes = [c.c_int32] * 3 + [_i32p, _i32p, _f64p, _f64p, _f64p, _f64p,
                                                        _f64p, _f64p]
    lib.orc_par_propagate_fwd.restype = None
    lib.orc_par_propagate_fwd.argtypes = ([c.c_int32] * 3 + [c.c_int64, _i32p, _i32p, _i32p, _f64p,
                                          _f64p, c.c_void_p, _f64p, c.c_int32])
    lib.orc_par_propagate_bwd.restype = None
    lib.orc_par_propagate_bwd.argtypes = ([c.c_int32] * 3 + [c.c_int64, _i32p, _i32p, _i32p, _f64p,
                                          _f64p, _f64p, _f64p, _f64p, c.c_void_p, c.c_int32])
    lib.orc_par_ggnn_fwd.restype = None
    lib.orc_par_ggnn_fwd.argtypes = ([c.c_int32] * 5 + [c.c_int64, _i32p, _i32p, _i32p] +
                                     [_f64p] * 8 + [c.c_int32])
    lib.orc_par_ggnn_bwd.restype = None
    lib.orc_par_ggnn_bwd.argtypes = ([c.c_int32] * 5 + [c.c_int64, _i32p, _i32p, _i32p] +
                                     [_f64p] * 16 + [c.c_int32])
    lib.orc_par_max_threads.restype = c.c_int32
    lib.orc_par_max_threads.argtypes = []
    lib.orc_adam.restype = None
    lib.orc_adam.argtypes = [c.c_int64, _f64p, _f64p, _f64p, _f64p, c.c_double, c.c_double,
                             c.c_double, c.c_double, c.c_int32]
    del opt
    _lib = lib
    return lib


def _i32(a):
    return np.ascontiguousarray(a, dtype=np.int32)


def _f64(a):
    return np.ascontiguousarray(a, dtype=np.float64)


# ---------------------------------------------------------------------------------------------
# ordering and layout


def bandwidth(n, src, dst, pos=None) -> int:
    """Bandwidth of the adjacency with node v at position pos[v] (identity if None)."""
    lib = _load()
    src, dst = _i32(src), _i32(dst)
    p = None if pos is None else _i32(pos)
    return int(lib.orc_bandwidth(n, src.shape[0], src, dst,
                                 None if p is None else p.ctypes.data_as(ctypes.c_void_p)))


def rcm(n, src, dst, keep_if_better=True) -> np.ndarray:
    """Reverse Cuthill-McKee order: perm[new] = old."""
    lib = _load()
    perm = np.zeros(n, np.int32)
    src, dst = _i32(src), _i32(dst)
    if lib.orc_rcm(n, src.shape[0], src, dst, int(bool(keep_if_better)), perm):
        raise ValueError("invalid graph")
    return perm


def reach(n, src, dst, candidates, T) -> np.ndarray:
    """Reachability preprocessing (Section 4): bool [n], True for nodes from which a candidate is
    reachable along at most T edges."""
    lib = _load()
    keep = np.zeros(n, np.uint8)
    src, dst, cand = _i32(src), _i32(dst), _i32(candidates)
    if lib.orc_reach(n, src.shape[0], src, dst, cand, cand.shape[0], T, keep) < 0:
        raise ValueError("invalid graph or candidates")
    return keep.astype(bool)


def reach_filter(graph, candidates, T):
    """The graph reduced to its kept nodes (renumbered in ascending old id) and the edges between
    them (input order): (node_map [n] new id or -1, n_kept, src, dst, etype)."""
    keep = reach(graph.n_nodes, graph.src, graph.dst, candidates, T)
    node_map = np.full(graph.n_nodes, -1, np.int32)
    node_map[keep] = np.arange(int(keep.sum()), dtype=np.int32)
    ek = keep[graph.src] & keep[graph.dst]
    return (node_map, int(keep.sum()), node_map[graph.src[ek]], node_map[graph.dst[ek]],
            np.asarray(graph.etype)[ek].astype(np.int32))


FLAG_RCM = 1
FLAG_KEEP_IF_BETTER = 2
FLAG_SUPERNODES = 4


@dataclass
class Layout:
    K: int
    S: int
    P: int
    n_packed: int
    n_real: int
    n_unique: int
    n_kept: int
    n_dropped: int
    bw_before_max: int
    bw_after_max: int
    perm: np.ndarray        # concatenated per-graph perm[new] = old
    offset: np.ndarray      # per graph, -1 if not packed
    masks: np.ndarray       # uint8 [K, 3, P, S, S/8]
    kept_dst: np.ndarray
    kept_src: np.ndarray
    kept_type: np.ndarray
    bw_before: np.ndarray
    bw_after: np.ndarray
    n_nodes: np.ndarray
    kept_super: np.ndarray = None  # bool per kept edge: has a supernode end
    is_super: np.ndarray = None    # bool per position: a supernode

    @property
    def n_pad(self) -> int:
        return self.K * self.S

    def gather_index(self) -> np.ndarray:
        """For each packed position q < n_real, the row of the concatenated original state array."""
        node_off = np.concatenate([[0], np.cumsum(self.n_nodes)])
        out = np.zeros(self.n_real, np.int64)
        for g in range(len(self.n_nodes)):
            o = self.offset[g]
            if o < 0:
                continue
            n = self.n_nodes[g]
            out[o:o + n] = node_off[g] + self.perm[node_off[g]:node_off[g] + n]
        return out

    def graph_segments(self):
        """(offset, count) of every packed graph."""
        sel = self.offset >= 0
        return self.offset[sel].astype(np.int32), self.n_nodes[sel].astype(np.int32)


def layout(graphs, P, S, capacity_blocks=0, flags=FLAG_RCM | FLAG_KEEP_IF_BETTER,
           with_masks=True, super_min_degree=0, max_super=0) -> Layout:
    """Supergraph layout of `graphs` (objects with n_nodes, src, dst, etype); with
    FLAG_SUPERNODES, nodes of at least super_min_degree distinct neighbours (at most max_super per
    graph) become supernodes."""
    lib = _load()
    n_nodes = _i32([g.n_nodes for g in graphs])
    counts = np.array([g.n_edges for g in graphs], np.int64)
    edge_off = np.concatenate([[0], np.cumsum(counts)]).astype(np.int64)
    src = _i32(np.concatenate([g.src for g in graphs]) if graphs else [])
    dst = _i32(np.concatenate([g.dst for g in graphs]) if graphs else [])
    et = _i32(np.concatenate([g.etype for g in graphs]) if graphs else [])
    K = int(lib.orc_num_blocks(len(graphs), n_nodes, S, capacity_blocks))
    perm = np.zeros(int(n_nodes.sum()), np.int32)
    offset = np.zeros(len(graphs), np.int32)
    info = np.zeros(8, np.int64)
    m = int(edge_off[-1])
    masks = np.zeros((K, 3, P, S, S // 8), np.uint8) if with_masks else None
    kd, ks, kt = (np.zeros(max(m, 1), np.int32) for _ in range(3))
    bwb = np.zeros(len(graphs), np.int64)
    bwa = np.zeros(len(graphs), np.int64)
    ksup = np.zeros(max(m, 1), np.uint8)
    isup = np.zeros(max(K * S, 1), np.uint8)
    vp = lambda a: None if a is None else a.ctypes.data_as(ctypes.c_void_p)  # noqa: E731
    rc = lib.orc_layout(len(graphs), n_nodes, edge_off, src, dst, et, P, S, capacity_blocks, flags,
                        perm, offset, info, vp(masks), vp(kd), vp(ks), vp(kt), bwb, bwa,
                        super_min_degree, max_super, vp(ksup), vp(isup))
    if rc:
        raise ValueError("invalid graphs for layout")
    nk = int(info[4])
    return Layout(K=int(info[0]), S=S, P=P, n_packed=int(info[1]), n_real=int(info[2]),
                  n_unique=int(info[3]), n_kept=nk, n_dropped=int(info[5]),
                  bw_before_max=int(info[6]), bw_after_max=int(info[7]), perm=perm, offset=offset,
                  masks=masks, kept_dst=kd[:nk].copy(), kept_src=ks[:nk].copy(),
                  kept_type=kt[:nk].copy(), bw_before=bwb, bw_after=bwa, n_nodes=n_nodes,
                  kept_super=ksup[:nk].astype(bool), is_super=isup[:K * S].astype(bool))


# ---------------------------------------------------------------------------------------------
# propagation, GRU, GGNN


def propagate_fwd(N, P, H, e_dst, e_src, e_type, E, W, b=None) -> np.ndarray:
    lib = _load()
    e_dst, e_src, e_type = _i32(e_dst), _i32(e_src), _i32(e_type)
    E, W = _f64(E), _f64(W)
    bb = None if b is None else _f64(b)
    Y = np.zeros((N, H))
    lib.orc_propagate_fwd(N, P, H, e_dst.shape[0], e_dst, e_src, e_type, E, W,
                          None if bb is None else bb.ctypes.data_as(ctypes.c_void_p), Y)
    return Y


def propagate_bwd(N, P, H, e_dst, e_src, e_type, E, W, dY):
    lib = _load()
    e_dst, e_src, e_type = _i32(e_dst), _i32(e_src), _i32(e_type)
    dE = np.zeros((N, H)); dW = np.zeros((P, H, H)); db = np.zeros((P, H))
    lib.orc_propagate_bwd(N, P, H, e_dst.shape[0], e_dst, e_src, e_type, _f64(E), _f64(W),
                          _f64(dY), dE, dW, db.ctypes.data_as(ctypes.c_void_p))
    return dE, dW, db


def gru_fwd(X, Hs, W_ih, W_hh, b_ih, b_hh, n_real=None):
    lib = _load()
    N, H = X.shape
    out = np.zeros((N, H))
    lib.orc_gru_fwd(N, H, N if n_real is None else n_real, _f64(X), _f64(Hs), _f64(W_ih),
                    _f64(W_hh), _f64(b_ih), _f64(b_hh), out)
    return out


def gru_bwd(X, Hs, W_ih, W_hh, b_ih, b_hh, dHn, n_real=None):
    lib = _load()
    N, H = X.shape
    dX = np.zeros((N, H)); dH = np.zeros((N, H))
    dWi = np.zeros((3 * H, H)); dWh = np.zeros((3 * H, H)); dbi = np.zeros(3 * H)
    dbh = np.zeros(3 * H)
    lib.orc_gru_bwd(N, H, N if n_real is None else n_real, _f64(X), _f64(Hs), _f64(W_ih),
                    _f64(W_hh), _f64(b_ih), _f64(b_hh), _f64(dHn), dX, dH, dWi, dWh, dbi, dbh)
    return dX, dH, dWi, dWh, dbi, dbh


def ggnn_fwd(N, P, H, T, n_real, e_dst, e_src, e_type, E0, prm):
    """Returns (Es [T+1,N,H], Ys [T,N,H])."""
    lib = _load()
    Es = np.zeros((T + 1, N, H)); Es[0] = E0
    Ys = np.zeros((max(T, 1), N, H))
    e_dst, e_src, e_type = _i32(e_dst), _i32(e_src), _i32(e_type)
    lib.orc_ggnn_fwd(N, P, H, T, n_real, e_dst.shape[0], e_dst, e_src, e_type, _f64(prm["W"]),
                     _f64(prm["b"]), _f64(prm["W_ih"]), _f64(prm["W_hh"]), _f64(prm["b_ih"]),
                     _f64(prm["b_hh"]), Es, Ys)
    return Es, Ys


def ggnn_bwd(N, P, H, T, n_real, e_dst, e_src, e_type, prm, Es, Ys, dET):
    """Returns dict(dE0, dW, db, dW_ih, dW_hh, db_ih, db_hh)."""
    lib = _load()
    e_dst, e_src, e_type = _i32(e_dst), _i32(e_src), _i32(e_type)
    out = dict(dE0=np.zeros((N, H)), dW=np.zeros((P, H, H)), db=np.zeros((P, H)),
               dW_ih=np.zeros((3 * H, H)), dW_hh=np.zeros((3 * H, H)), db_ih=np.zeros(3 * H),
               db_hh=np.zeros(3 * H))
    lib.orc_ggnn_bwd(N, P, H, T, n_real, e_dst.shape[0], e_dst, e_src, e_type, _f64(prm["W"]),
                     _f64(prm["b"]), _f64(prm["W_ih"]), _f64(prm["W_hh"]), _f64(prm["b_ih"]),
                     _f64(prm["b_hh"]), _f64(Es), _f64(Ys), _f64(dET), out["dE0"], out["dW"],
                     out["db"], out["dW_ih"], out["dW_hh"], out["db_ih"], out["db_hh"])
    return out


def readout_loss(E, offset, count, w_out, target):
    """Returns (loss, dE, dw_out)."""
    lib = _load()
    N, H = E.shape
    loss = np.zeros(1); dE = np.zeros((N, H)); dw = np.zeros(H)
    offset, count = _i32(offset), _i32(count)
    lib.orc_readout_loss(N, H, offset.shape[0], offset, count, _f64(E), _f64(w_out), _f64(target),
                         loss, dE, dw)
    return float(loss[0]), dE, dw


def adam(param, m, v, grad, lr, b1, b2, eps, t):
    """One Adam step; returns new (param, m, v) copies."""
    lib = _load()
    p, mm, vv = _f64(param).copy(), _f64(m).copy(), _f64(v).copy()
    lib.orc_adam(p.size, p, mm, vv, _f64(grad), lr, b1, b2, eps, t)
    return p, mm, vv


# ---------------------------------------------------------------------------------------------
# multi-threaded pull-based variant (CPU baseline on all host cores; equal to the last bit to the
# functions above)


def par_max_threads() -> int:
    """Threads the multi-threaded variant uses by default (1 when built without OpenMP)."""
    return int(_load().orc_par_max_threads())


def par_propagate_fwd(N, P, H, e_dst, e_src, e_type, E, W, b=None, threads=0) -> np.ndarray:
    lib = _load()
    e_dst, e_src, e_type = _i32(e_dst), _i32(e_src), _i32(e_type)
    bb = None if b is None else _f64(b)
    Y = np.zeros((N, H))
    lib.orc_par_propagate_fwd(N, P, H, e_dst.shape[0], e_dst, e_src, e_type, _f64(E), _f64(W),
                              None if bb is None else bb.ctypes.data_as(ctypes.c_void_p), Y,
                              threads)
    return Y


def par_propagate_bwd(N, P, H, e_dst, e_src, e_type, E, W, dY, threads=0):
    lib = _load()
    e_dst, e_src, e_type = _i32(e_dst), _i32(e_src), _i32(e_type)
    dE = np.zeros((N, H)); dW = np.zeros((P, H, H)); db = np.zeros((P, H))
    lib.orc_par_propagate_bwd(N, P, H, e_dst.shape[0], e_dst, e_src, e_type, _f64(E), _f64(W),
                              _f64(dY), dE, dW, db.ctypes.data_as(ctypes.c_void_p), threads)
    return dE, dW, db


def par_ggnn_fwd(N, P, H, T, n_real, e_dst, e_src, e_type, E0, prm, threads=0):
    lib = _load()
    Es = np.zeros((T + 1, N, H)); Es[0] = E0
    Ys = np.zeros((max(T, 1), N, H))
    e_dst, e_src, e_type = _i32(e_dst), _i32(e_src), _i32(e_type)
    lib.orc_par_ggnn_fwd(N, P, H, T, n_real, e_dst.shape[0], e_dst, e_src, e_type, _f64(prm["W"]),
                         _f64(prm["b"]), _f64(prm["W_ih"]), _f64(prm["W_hh"]), _f64(prm["b_ih"]),
                         _f64(prm["b_hh"]), Es, Ys, threads)
    return Es, Ys


def par_ggnn_bwd(N, P, H, T, n_real, e_dst, e_src, e_type, prm, Es, Ys, dET, threads=0):
    lib = _load()
    e_dst, e_src, e_type = _i32(e_dst), _i32(e_src), _i32(e_type)
    out = dict(dE0=np.zeros((N, H)), dW=np.zeros((P, H, H)), db=np.zeros((P, H)),
               dW_ih=np.zeros((3 * H, H)), dW_hh=np.zeros((3 * H, H)), db_ih=np.zeros(3 * H),
               db_hh=np.zeros(3 * H))
    lib.orc_par_ggnn_bwd(N, P, H, T, n_real, e_dst.shape[0], e_dst, e_src, e_type, _f64(prm["W"]),
                         _f64(prm["b"]), _f64(prm["W_ih"]), _f64(prm["W_hh"]), _f64(prm["b_ih"]),
                         _f64(prm["b_hh"]), _f64(Es), _f64(Ys), _f64(dET), out["dE0"], out["dW"],
                         out["db"], out["dW_ih"], out["dW_hh"], out["db_ih"], out["db_hh"],
                         threads)
    return out
