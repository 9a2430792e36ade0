"""Shared set-up of the GPU parity tests: seeded inputs, device copies, oracle references and the
parity measure (max-abs error relative to the reference's max-abs value, per tensor)."""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_1906_11786_gb300 import _binding as L
from paper_1906_11786_gb300 import build as B
from paper_1906_11786_gb300 import synth

TOL = {"f32": 1e-4, "bf16": 2e-2}


def ensure_built():
    B.build()
    L.load()


def rel_err(got, ref) -> float:
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    return float(np.max(np.abs(got - ref)) / max(float(np.max(np.abs(ref))), 1e-30))


def med_rel_err(got, ref) -> float:
    """Element-wise median relative error |g - o| / |o| over the entries with |o| > 1e-3 max|o|
    (reading c14's second measure: an error confined to small entries, such as the rows of
    low-degree nodes, is under-weighted by the max-norm measure)."""
    got = np.asarray(got, np.float64).ravel()
    ref = np.asarray(ref, np.float64).ravel()
    big = np.abs(ref) > 1e-3 * max(float(np.max(np.abs(ref))), 1e-30)
    if not big.any():
        return 0.0
    return float(np.median(np.abs(got[big] - ref[big]) / np.abs(ref[big])))


def assert_close(got, ref, tol: float, what: str = ""):
    """Both parity measures of reading c14 under the same tolerance: the max-abs error over the
    reference's max-abs value, and the element-wise median relative error."""
    e_inf, e_med = rel_err(got, ref), med_rel_err(got, ref)
    assert e_inf < tol and e_med < tol, \
        f"{what}: max-norm rel {e_inf:.3e}, median rel {e_med:.3e}, tolerance {tol:g}"


def quantize(x: np.ndarray, dtype: str) -> np.ndarray:
    """Round to the device dtype and back to float64 (both sides then start from equal values)."""
    if dtype == "bf16":
        return torch.from_numpy(np.asarray(x, np.float32)).to(torch.bfloat16).double().numpy()
    return np.asarray(x, np.float32).astype(np.float64)


def to_dev(x: np.ndarray, dtype: str) -> torch.Tensor:
    t = torch.from_numpy(np.ascontiguousarray(x, np.float32))
    if dtype == "bf16":
        t = t.to(torch.bfloat16)
    return t.cuda()


def f32_dev(x) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).cuda()


class Case:
    """A planned, uploaded supergraph with packed device states and the oracle's view of it."""

    def __init__(self, graphs, P, S, H, dtype, seed=0, cap=0, plain_xavier=False, sup=None):
        self.P, self.S, self.H, self.dtype = P, S, H, dtype
        if sup:  # (supernode_min_degree, max_supernodes)
            F = L.BG_RCM | L.BG_KEEP_IF_BETTER | L.BG_SUPERNODES
            self.plan = L.band_plan(graphs, P, S, cap, F, *sup)
            self.ref = oracle.layout(graphs, P, S, cap, flags=F, super_min_degree=sup[0],
                                     max_super=sup[1])
        else:
            self.plan = L.band_plan(graphs, P, S, cap)
            self.ref = oracle.layout(graphs, P, S, cap)
        self.plan.upload()
        info = self.plan.info()
        self.info = info
        self.N = info["n_pad"]
        self.n_real = info["n_real"]
        n_all = sum(g.n_nodes for g in graphs)
        E_orig = quantize(synth.gen_states(n_all, H, seed), dtype)
        self.E_orig = E_orig
        self.E_orig_dev = to_dev(E_orig, dtype)
        self.E_band_dev = torch.empty((self.N, H), dtype=self.E_orig_dev.dtype, device="cuda")
        L.pack_states(self.plan, dtype, H, self.E_orig_dev, self.E_band_dev)
        gi = self.ref.gather_index()
        self.E_band = np.zeros((self.N, H))
        self.E_band[: self.n_real] = E_orig[gi]
        # plain_xavier: the H x H Xavier bound for W_p, as the workloads state it; otherwise the
        # message layer's fan-in H x mean in-degree (reading r1, for the T = 8 recurrences)
        prm = synth.gen_params(P, H, seed + 1, mean_in_degree=1.0 if plain_xavier else
                               self.ref.n_kept / max(self.ref.n_real, 1))
        for k in ("W", "W_ih", "W_hh"):
            prm[k] = quantize(prm[k], dtype)
        for k in ("b", "b_ih", "b_hh", "w_out"):
            prm[k] = quantize(prm[k], "f32")
        self.prm = prm
        self.dprm = {k: (to_dev(v, dtype) if k in ("W", "W_ih", "W_hh") else f32_dev(v))
                     for k, v in prm.items()}
        self.edges = (self.ref.kept_dst, self.ref.kept_src, self.ref.kept_type)

    def ws(self, op, T=1):
        if op in (L.BG_OP_GGNN_FWD, L.BG_OP_GGNN_BWD):
            n = L.ggnn_workspace_bytes(self.plan, self.dtype, self.H, T, op)
        else:
            n = L.workspace_bytes(self.plan, self.dtype, self.H, op)
        return torch.empty(n, dtype=torch.uint8, device="cuda")
