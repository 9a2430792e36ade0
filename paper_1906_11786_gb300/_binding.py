"""ctypes binding of libbandggnn.so (include/bandggnn.h): argument marshalling only.

Every function here forwards to the C entry point of the same name.  Device arrays are torch
CUDA tensors (their data pointers are passed); streams default to torch's current stream.  A
non-zero status raises BandGGNNError with the library's message.  Loading fails loudly when the
compiled library is missing: there is no fallback implementation.
"""
from __future__ import annotations

import ctypes
import os
import re

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libbandggnn.so")
HEADER = os.path.join(os.path.dirname(_PKG), "include", "bandggnn.h")

BG_F32, BG_BF16 = 0, 1
BG_RCM, BG_KEEP_IF_BETTER, BG_SUPERNODES = 1, 2, 4
BG_ACCUM = 1
BG_FLOPS_BAND, BG_FLOPS_XFORM, BG_FLOPS_GRU, BG_FLOPS_NNZ = 0, 1, 2, 3
(BG_EXPORT_PERM, BG_EXPORT_OFFSETS, BG_EXPORT_MASKS, BG_EXPORT_MASKS_T, BG_EXPORT_BW,
 BG_EXPORT_GATHER, BG_EXPORT_SUPER_EDGES, BG_EXPORT_SUPER_COUNT) = range(8)
BG_OP_PROPAGATE_FWD, BG_OP_PROPAGATE_BWD, BG_OP_GGNN_FWD, BG_OP_GGNN_BWD, BG_OP_READOUT = range(5)
BG_KID_BAND_FWD, BG_KID_BAND_BWD, BG_KID_GRU_FWD, BG_KID_GRU_BWD, BG_KID_DW = range(5)
STATUS = {0: "BG_OK", -1: "BG_EINVAL", -2: "BG_ECAPACITY", -3: "BG_ENOMEM", -4: "BG_ECUDA",
          -5: "BG_ETIMEOUT", -6: "BG_EDEVICE", -7: "BG_ESTATE"}


class BandGGNNError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"{STATUS.get(code, code)}: {msg}")
        self.code = code


class bg_graph(ctypes.Structure):
    _fields_ = [("n_nodes", ctypes.c_int32), ("n_edges", ctypes.c_int64),
                ("src", ctypes.c_void_p), ("dst", ctypes.c_void_p), ("etype", ctypes.c_void_p)]


class bg_info(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("K", "S", "P", "n_graphs", "n_packed", "n_real",
                                              "n_pad")] + \
               [(n, ctypes.c_int64) for n in ("n_edges_in", "n_edges_unique", "n_kept",
                                              "n_dropped", "bw_before_max", "bw_after_max")] + \
               [("n_super", ctypes.c_int32), ("n_super_edges", ctypes.c_int64)]


class bg_plan_opts(ctypes.Structure):
    _fields_ = [("flags", ctypes.c_uint32), ("supernode_min_degree", ctypes.c_int32),
                ("max_supernodes", ctypes.c_int32)]


class bg_part_info(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("row0", "n_local", "own_begin", "own_end", "halo_lo",
                                              "halo_hi")]


class bg_params(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in ("W", "b", "W_ih", "W_hh", "b_ih", "b_hh")]


class bg_grads(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in ("dW", "db", "dW_ih", "dW_hh", "db_ih", "db_hh")]


_lib = None


def load(path: str = LIB_PATH):
    """Load the compiled library (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise ImportError(f"{path} is missing: build it with `python -m paper_1906_11786_gb300.build`"
                          " (the CUDA library is required; there is no fallback)")
    lib = ctypes.CDLL(path)
    c = ctypes
    vp, i32, i64, sz, f32 = c.c_void_p, c.c_int32, c.c_int64, c.c_size_t, c.c_float
    sig = {
        "bg_band_plan": (c.c_int, [vp, i32, i32, i32, i32, c.c_uint32, vp]),
        "bg_band_plan_opts": (c.c_int, [vp, i32, i32, i32, i32, vp, vp]),
        "bg_plan_free": (None, [vp]),
        "bg_plan_info": (c.c_int, [vp, vp]),
        "bg_plan_flops": (c.c_double, [vp, i32, i32]),
        "bg_plan_export_bytes": (sz, [vp, i32]),
        "bg_plan_export": (c.c_int, [vp, i32, vp, sz]),
        "bg_plan_upload": (c.c_int, [vp, vp]),
        "bg_pack_states": (c.c_int, [vp, c.c_int, i32, vp, vp, vp]),
        "bg_unpack_states": (c.c_int, [vp, c.c_int, i32, vp, vp, vp]),
        "bg_workspace_bytes": (sz, [vp, c.c_int, i32, i32]),
        "bg_band_propagate_fwd": (c.c_int, [vp, c.c_int, i32, vp, vp, vp, vp, vp, sz, vp]),
        "bg_band_propagate_fwd_noalloc": (c.c_int, [vp, c.c_int, i32, vp, vp, vp, vp, vp]),
        "bg_band_propagate_bwd": (c.c_int, [vp, c.c_int, i32, vp, vp, vp, vp, vp, vp, c.c_uint32,
                                            vp, sz, vp]),
        "bg_ggnn_saved_bytes": (sz, [vp, c.c_int, i32, i32]),
        "bg_ggnn_workspace_bytes": (sz, [vp, c.c_int, i32, i32, i32]),
        "bg_ggnn_step": (c.c_int, [vp, c.c_int, i32, i32, vp, vp, vp, vp, sz, vp, sz, vp]),
        "bg_ggnn_step_bwd": (c.c_int, [vp, c.c_int, i32, i32, vp, vp, sz, vp, vp, vp, c.c_uint32,
                                       vp, sz, vp]),
        "bg_readout_loss": (c.c_int, [vp, c.c_int, i32, vp, vp, vp, vp, vp, vp, vp, sz, vp]),
        "bg_adam_step": (c.c_int, [i64, vp, vp, c.c_int, vp, vp, vp, f32, f32, f32, f32, i32, vp]),
        "bg_last_error": (c.c_char_p, []),
        "bg_check_device": (c.c_int, [vp]),
        "bg_selftest_device_wait": (c.c_int, [vp]),
        "bg_profile_enable": (c.c_int, [i32]),
        "bg_profile_read": (c.c_int, [i32, vp, vp, i32]),
        "bg_launch_count": (i64, []),
        "bg_band_uses_tensor_cores": (c.c_int, [vp, c.c_int, i32]),
        "bg_reach_filter": (c.c_int, [vp, vp, i32, i32, vp, vp, vp, vp, vp, vp]),
        "bg_plan_partition": (c.c_int, [vp, i32, i32, vp, vp]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def declared_symbols(header: str = HEADER) -> list[str]:
    """Names of the functions include/bandggnn.h declares."""
    text = open(header).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(bg_[a-z0-9_]+)\s*\(", text)))


def _check(rc):
    if rc != 0:
        raise BandGGNNError(rc, load().bg_last_error().decode())


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    if not t.is_contiguous():
        raise ValueError("tensor must be contiguous")
    return t.data_ptr()


def _dev_ptr(t, name):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    return _ptr(t)


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def dtype_code(dt) -> int:
    import torch
    if dt in (BG_F32, BG_BF16):
        return dt
    if dt in (torch.float32, "f32", "fp32", "float32"):
        return BG_F32
    if dt in (torch.bfloat16, "bf16", "bfloat16"):
        return BG_BF16
    raise ValueError(f"unsupported dtype {dt}")


# --------------------------------------------------------------------------------- plan


class Plan:
    """Owns a bg_plan*; frees it on close/deletion."""

    def __init__(self, handle, n_types):
        self._h = handle
        self.P = n_types

    @property
    def handle(self):
        if not self._h:
            raise ValueError("plan is closed")
        return self._h

    def close(self):
        if self._h:
            load().bg_plan_free(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def info(self) -> dict:
        out = bg_info()
        _check(load().bg_plan_info(self.handle, ctypes.byref(out)))
        return {f: getattr(out, f) for f, _ in bg_info._fields_}

    def flops(self, H, which) -> float:
        return float(load().bg_plan_flops(self.handle, H, which))

    def export(self, which) -> np.ndarray:
        lib = load()
        n = lib.bg_plan_export_bytes(self.handle, which)
        buf = np.zeros(max(n, 1), np.uint8)
        _check(lib.bg_plan_export(self.handle, which, buf.ctypes.data, n))
        buf = buf[:n]
        if which in (BG_EXPORT_PERM, BG_EXPORT_OFFSETS, BG_EXPORT_GATHER, BG_EXPORT_SUPER_COUNT):
            return buf.view(np.int32)
        if which == BG_EXPORT_SUPER_EDGES:
            return buf.view(np.int32).reshape(-1, 3)
        if which == BG_EXPORT_BW:
            return buf.view(np.int64).reshape(2, -1)
        i = self.info()
        return buf.reshape(i["K"], 3, i["P"], i["S"], i["S"] // 8)

    def upload(self, stream=None):
        _check(load().bg_plan_upload(self.handle, _stream(stream)))


def band_plan(graphs, n_types, block_S, capacity_blocks=0, flags=BG_RCM | BG_KEEP_IF_BETTER,
              supernode_min_degree=0, max_supernodes=0) -> Plan:
    """bg_band_plan (bg_band_plan_opts with BG_SUPERNODES) on a list of objects with n_nodes, src,
    dst, etype (int32 arrays)."""
    lib = load()
    keep = []
    arr = (bg_graph * len(graphs))()
    for i, g in enumerate(graphs):
        s = np.ascontiguousarray(g.src, np.int32)
        d = np.ascontiguousarray(g.dst, np.int32)
        t = np.ascontiguousarray(g.etype, np.int32)
        keep += [s, d, t]
        arr[i] = bg_graph(int(g.n_nodes), int(s.shape[0]), s.ctypes.data, d.ctypes.data,
                          t.ctypes.data)
    h = ctypes.c_void_p()
    if flags & BG_SUPERNODES:
        opts = bg_plan_opts(flags, supernode_min_degree, max_supernodes)
        _check(lib.bg_band_plan_opts(arr, len(graphs), n_types, block_S, capacity_blocks,
                                     ctypes.byref(opts), ctypes.byref(h)))
    else:
        _check(lib.bg_band_plan(arr, len(graphs), n_types, block_S, capacity_blocks, flags,
                                ctypes.byref(h)))
    return Plan(h.value, n_types)


def plan_partition(plan, n_parts, part):
    """bg_plan_partition: (local Plan, info dict) of part `part` of a block-row split."""
    h = ctypes.c_void_p()
    info = bg_part_info()
    _check(load().bg_plan_partition(plan.handle, n_parts, part, ctypes.byref(h), ctypes.byref(info)))
    return Plan(h.value, plan.P), {f: getattr(info, f) for f, _ in bg_part_info._fields_}


def reach_filter(graph, candidates, T):
    """bg_reach_filter: (node_map [n] new id or -1, n_kept, src, dst, etype) of the graph reduced
    to the nodes that reach a candidate within T steps."""
    lib = load()
    s = np.ascontiguousarray(graph.src, np.int32)
    d = np.ascontiguousarray(graph.dst, np.int32)
    t = np.ascontiguousarray(graph.etype, np.int32)
    cand = np.ascontiguousarray(candidates, np.int32)
    g = bg_graph(int(graph.n_nodes), int(s.shape[0]), s.ctypes.data, d.ctypes.data, t.ctypes.data)
    node_map = np.zeros(max(graph.n_nodes, 1), np.int32)
    so, do, to = (np.zeros(max(s.shape[0], 1), np.int32) for _ in range(3))
    nn, ne = ctypes.c_int32(), ctypes.c_int64()
    _check(lib.bg_reach_filter(ctypes.byref(g), cand.ctypes.data, cand.shape[0], T,
                               node_map.ctypes.data, ctypes.byref(nn), ctypes.byref(ne),
                               so.ctypes.data, do.ctypes.data, to.ctypes.data))
    m = ne.value
    return node_map[:graph.n_nodes], nn.value, so[:m].copy(), do[:m].copy(), to[:m].copy()


# --------------------------------------------------------------------------------- device calls


def workspace_bytes(plan, dtype, H, op) -> int:
    return int(load().bg_workspace_bytes(plan.handle, dtype_code(dtype), H, op))


def ggnn_workspace_bytes(plan, dtype, H, T, op) -> int:
    return int(load().bg_ggnn_workspace_bytes(plan.handle, dtype_code(dtype), H, T, op))


def ggnn_saved_bytes(plan, dtype, H, T) -> int:
    return int(load().bg_ggnn_saved_bytes(plan.handle, dtype_code(dtype), H, T))


def pack_states(plan, dtype, H, E_orig, E_band, stream=None):
    _check(load().bg_pack_states(plan.handle, dtype_code(dtype), H, _dev_ptr(E_orig, "E_orig"),
                                 _dev_ptr(E_band, "E_band"), _stream(stream)))


def unpack_states(plan, dtype, H, E_band, E_orig, stream=None):
    _check(load().bg_unpack_states(plan.handle, dtype_code(dtype), H, _dev_ptr(E_band, "E_band"),
                                   _dev_ptr(E_orig, "E_orig"), _stream(stream)))


def band_propagate_fwd(plan, dtype, H, E, W, b, Y, ws, stream=None):
    _check(load().bg_band_propagate_fwd(plan.handle, dtype_code(dtype), H, _dev_ptr(E, "E"),
                                        _dev_ptr(W, "W"), _dev_ptr(b, "b"), _dev_ptr(Y, "Y"),
                                        _dev_ptr(ws, "ws"), ws.numel() * ws.element_size(),
                                        _stream(stream)))


def band_propagate_fwd_noalloc(plan, dtype, H, E, W, b, Y, stream=None):
    _check(load().bg_band_propagate_fwd_noalloc(plan.handle, dtype_code(dtype), H, _dev_ptr(E, "E"),
                                                _dev_ptr(W, "W"), _dev_ptr(b, "b"),
                                                _dev_ptr(Y, "Y"), _stream(stream)))


def band_propagate_bwd(plan, dtype, H, E, W, dY, dE, dW, db, ws, flags=0, stream=None):
    _check(load().bg_band_propagate_bwd(plan.handle, dtype_code(dtype), H, _dev_ptr(E, "E"),
                                        _dev_ptr(W, "W"), _dev_ptr(dY, "dY"), _dev_ptr(dE, "dE"),
                                        _dev_ptr(dW, "dW"), _dev_ptr(db, "db"), flags,
                                        _dev_ptr(ws, "ws"), ws.numel() * ws.element_size(),
                                        _stream(stream)))


def _params(prm):
    return bg_params(*[_dev_ptr(prm.get(k), k) for k in ("W", "b", "W_ih", "W_hh", "b_ih", "b_hh")])


def _grads(gr):
    return bg_grads(*[_dev_ptr(gr.get(k), k) for k in ("dW", "db", "dW_ih", "dW_hh", "db_ih",
                                                       "db_hh")])


def ggnn_step(plan, dtype, H, T, prm, E0, ET, saved, ws, stream=None):
    p = _params(prm)
    _check(load().bg_ggnn_step(plan.handle, dtype_code(dtype), H, T, ctypes.byref(p),
                               _dev_ptr(E0, "E0"), _dev_ptr(ET, "ET"), _dev_ptr(saved, "saved"),
                               saved.numel() * saved.element_size(), _dev_ptr(ws, "ws"),
                               ws.numel() * ws.element_size(), _stream(stream)))


def ggnn_step_bwd(plan, dtype, H, T, prm, saved, dET, dE0, grads, ws, flags=0, stream=None):
    p = _params(prm)
    g = _grads(grads)
    _check(load().bg_ggnn_step_bwd(plan.handle, dtype_code(dtype), H, T, ctypes.byref(p),
                                   _dev_ptr(saved, "saved"), saved.numel() * saved.element_size(),
                                   _dev_ptr(dET, "dET"), _dev_ptr(dE0, "dE0"), ctypes.byref(g),
                                   flags, _dev_ptr(ws, "ws"), ws.numel() * ws.element_size(),
                                   _stream(stream)))


def readout_loss(plan, dtype, H, ET, w_out, target, loss, dET, dw_out, ws, stream=None):
    _check(load().bg_readout_loss(plan.handle, dtype_code(dtype), H, _dev_ptr(ET, "ET"),
                                  _dev_ptr(w_out, "w_out"), _dev_ptr(target, "target"),
                                  _dev_ptr(loss, "loss"), _dev_ptr(dET, "dET"),
                                  _dev_ptr(dw_out, "dw_out"), _dev_ptr(ws, "ws"),
                                  ws.numel() * ws.element_size(), _stream(stream)))


def adam_step(master, working, m, v, grad, lr, beta1, beta2, eps, step, stream=None):
    wdt = BG_BF16 if (working is not None and working.element_size() == 2) else BG_F32
    _check(load().bg_adam_step(master.numel(), _dev_ptr(master, "master"),
                               _dev_ptr(working, "working"), wdt, _dev_ptr(m, "m"),
                               _dev_ptr(v, "v"), _dev_ptr(grad, "grad"), lr, beta1, beta2, eps,
                               step, _stream(stream)))


def check_device(stream=None):
    _check(load().bg_check_device(_stream(stream)))


def selftest_device_wait(stream=None):
    """Launch the failure-path self test (a bounded wait that gives up); check_device() then
    raises BG_ETIMEOUT."""
    _check(load().bg_selftest_device_wait(_stream(stream)))


def profile_enable(on: bool):
    _check(load().bg_profile_enable(1 if on else 0))


def profile_read(kid, reset=False):
    ms = ctypes.c_double()
    n = ctypes.c_int64()
    _check(load().bg_profile_read(kid, ctypes.byref(ms), ctypes.byref(n), 1 if reset else 0))
    return ms.value, n.value


def band_uses_tensor_cores(plan, dtype, H) -> bool:
    rc = load().bg_band_uses_tensor_cores(plan.handle, dtype_code(dtype), H)
    if rc < 0:
        _check(rc)
    return rc == 1


def launch_count() -> int:
    return int(load().bg_launch_count())
