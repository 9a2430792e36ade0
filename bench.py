"""Benchmark: band-GGNN forward + backward on GB300 (arXiv 1906.11786 hot path).

One step = one pass of the whole hot path over one supergraph: T GGNN steps forward (band
propagation + GRU) and their backward (GRU backward + transposed-band propagation, all parameter
gradients); the training workload adds the mean-pool readout, loss and Adam.  Metric: node-steps
per second = real (non-padding) nodes x T / step time.  Default workload: 64 program-shaped graphs
(~72k nodes) packed at S = 128, P = 20 edge types, H = 64, bf16, T = 8.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload packed64] [--impl ours|reference]

Under torchrun every rank plans its own supergraph (different seeds; the paper gives each core its
own supergraph: weak scaling); the step's one collective is the mean of the ranks' gradients after
the backward (the paper's synchronous data-parallel update); rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "node-steps/s (fwd+bwd)"
WORKLOAD_NAMES = ("single512", "packed64", "single20k", "sweep131k", "train100k")


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return {"hbm_gbs": d["hbm_gbs"], "bf16": d["bf16_tflops"],
                "bf16_sustained": d["bf16_tflops_sustained"],
                "sm_max_mhz": d.get("sm_max_mhz", 2070.0), "src": "measured"}
    return {"hbm_gbs": 6800.0, "bf16": 1900.0, "bf16_sustained": 1700.0, "sm_max_mhz": 2070.0,
            "src": "fallback"}


def _profiled_traffic(kernel: str, workload: str):
    """DRAM bytes per launch of `kernel` from the committed ncu summary of `workload`, or None when
    there is none or the kernel's source changed since it was captured."""
    import hashlib
    path = os.path.join(ROOT, "profiles", f"k_band_tc_{kernel}_{workload}.md")
    if not os.path.exists(path):
        return None
    vals = {}
    for line in open(path):
        if ":" in line and line.split(":")[0] in ("dram_bytes_per_launch", "source_sha256_16"):
            k, v = line.split(":", 1)
            vals[k.strip()] = v.strip()
    m = hashlib.sha256()
    for f in ("band_tc.cu", "tc_util.cuh"):
        m.update(open(os.path.join(ROOT, "paper_1906_11786_gb300", "csrc", f), "rb").read())
    if vals.get("source_sha256_16") != m.hexdigest()[:16] or "dram_bytes_per_launch" not in vals:
        return None
    return int(vals["dram_bytes_per_launch"])


def _flops(L, plan, H):
    """FLOPs of one forward pass over the plan: band-dense (all tiles of Eq. 3 as dense products),
    edge-type transforms, GRU gates, and the useful count (one H-vector add per kept edge)."""
    f = {k: plan.flops(H, c) for k, c in (("band_dense", L.BG_FLOPS_BAND),
                                         ("xform", L.BG_FLOPS_XFORM), ("gru", L.BG_FLOPS_GRU),
                                         ("nnz", L.BG_FLOPS_NNZ))}
    f["nnz_over_band_dense"] = f["nnz"] / f["band_dense"] if f["band_dense"] else 0.0
    return f


def _host():
    """The host cores the CPU baseline ran on: machine, core count, CPU model as /proc reports it."""
    import platform
    model = ""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.lower().startswith("model name:"):
                model = line.split(":", 1)[1].strip()
                break
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        for line in open("/proc/cpuinfo") if not model else ():
            key = line.split(":")[0].strip().lower()
            if key in ("model name", "cpu part", "cpu implementer") and not model:
                model = line.split(":", 1)[1].strip()
    except OSError:
        pass
    return {"machine": platform.machine(), "nproc": os.cpu_count(), "cpu_model": model}


def _dist():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


class Clocks:
    """Samples nvidia-smi clocks and throttle reasons every 50 ms from before the warm-up to the
    end of the end-to-end run (the timed steps, then a profiled pass of at least two seconds under
    the same load); marks bracket the timed steps."""

    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []
        self.marks = {}

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.perf_counter(), line.strip()))

    def mark(self, tag: str):
        self.marks[tag] = time.perf_counter()

    def __exit__(self, *a):
        if self.proc:
            time.sleep(0.1)  # the sample in flight
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, timed, mx, reasons = [], [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        t0, t1 = self.marks.get("timed_start"), self.marks.get("timed_end")
        for t, ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 8:
                continue
            try:
                v = float(f[0])
                mx = float(f[1])
            except ValueError:
                continue
            sm.append(v)
            if t0 is not None and t1 is not None and t0 <= t <= t1 + 0.05:
                timed.append(v)
            for n, r in zip(names, f[4:8]):
                if r.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm), "samples_timed": len(timed),
                "sm_mhz_timed": statistics.median(timed) if timed else None,
                "window": "warm-up, the timed steps, the profiled pass (>= 2 s) and the "
                          "end-to-end run, every 50 ms"}


# --------------------------------------------------------------------------------- workload


def workload(name: str, rank: int, S=None, H=None):
    from paper_1906_11786_gb300 import synth
    c = dict(synth.WORKLOADS[name])
    S = S or c["S"]
    H = H or c["H"]
    if rank == 0:
        graphs = synth.workload_graphs(name, S=S)
    else:  # every rank gets its own supergraph of the same shape
        graphs = synth.workload_graphs(name, S=S)
        graphs = [synth.gen_graph(g.n_nodes, c["F"], c["reverse"],
                                  c["max_off"] or S // 2, c["tree_win"] or S // 2, c["lam"],
                                  synth.graph_seed(name, i) + 7919 * rank)
                  for i, g in enumerate(graphs)]
    P = 2 * c["F"] if c["reverse"] else c["F"]
    cap = 0
    if c["sizes"][0] == "fill":
        cap = -(-c["sizes"][1] // S)
    return graphs, dict(c, S=S, H=H, P=P, cap=cap)


def reduce_over_ranks(dist, ms: float, units: float, device="cuda"):
    """Whole-job aggregation: the slowest rank's time and the node-steps of all ranks."""
    if dist is None:
        return ms, units
    import torch
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    u = torch.tensor([units], dtype=torch.float64, device=device)
    dist.all_reduce(u, op=dist.ReduceOp.SUM)
    return float(t.item()), float(u.item())


def allreduce_grads(dist, flat):
    """Data-parallel gradient exchange, the one collective of a step with N > 1: every rank's
    gradients (one flat buffer) replaced in place by their mean over the ranks, as in the paper's
    synchronous data-parallel training (one supergraph per core, Section 4.2)."""
    if dist is None or dist.get_world_size() == 1:
        return
    dist.all_reduce(flat, op=dist.ReduceOp.SUM)
    flat.mul_(1.0 / dist.get_world_size())


class OursStep:
    """Device buffers and one fwd+bwd step through the C ABI."""

    def __init__(self, graphs, c, seed=0, dist=None):
        import torch

        from paper_1906_11786_gb300 import _binding as L
        from paper_1906_11786_gb300 import synth
        self.L, self.torch = L, torch
        self.c = c
        P, S, H, T = c["P"], c["S"], c["H"], c["T"]
        self.dt = c["dtype"]
        tdt = torch.bfloat16 if self.dt == "bf16" else torch.float32
        t0 = time.perf_counter()
        self.plan = L.band_plan(graphs, P, S, c["cap"])
        self.plan_ms = (time.perf_counter() - t0) * 1e3
        t0 = time.perf_counter()
        self.plan.upload()
        torch.cuda.synchronize()
        self.upload_ms = (time.perf_counter() - t0) * 1e3
        self.info = self.plan.info()
        N, n_real = self.info["n_pad"], self.info["n_real"]
        self.N, self.n_real = N, n_real
        n_all = sum(g.n_nodes for g in graphs)
        self.n_all = n_all
        E = torch.from_numpy(synth.gen_states(n_all, H, seed).astype(np.float32)).to(tdt)
        self.E_orig_host = E.pin_memory()
        self.E_orig_dev = E.cuda()
        self.E0 = torch.empty((N, H), dtype=tdt, device="cuda")
        L.pack_states(self.plan, self.dt, H, self.E_orig_dev, self.E0)
        prm = synth.gen_params(P, H, seed + 1,
                               mean_in_degree=self.info["n_kept"] / max(n_real, 1))
        self.prm = {}
        for k, v in prm.items():
            t = torch.from_numpy(np.asarray(v, np.float32))
            self.prm[k] = (t.to(tdt) if k in ("W", "W_ih", "W_hh") else t).cuda()
        dET = np.random.default_rng(seed + 2).standard_normal((N, H)).astype(np.float32)
        dET[n_real:] = 0
        self.dET = torch.from_numpy(dET).cuda()
        self.dET_host = torch.from_numpy(dET).pin_memory()
        # every gradient is a view of one flat buffer: one all-reduce per step for N > 1
        shapes = (("dW", (P, H, H)), ("db", (P, H)), ("dW_ih", (3 * H, H)), ("dW_hh", (3 * H, H)),
                  ("db_ih", (3 * H,)), ("db_hh", (3 * H,)), ("dw_out", (H,)))
        self.gflat = torch.zeros(sum(int(np.prod(sh)) for _, sh in shapes), device="cuda")
        views, o = {}, 0
        for k, sh in shapes:
            n = int(np.prod(sh))
            views[k] = self.gflat[o:o + n].view(sh)
            o += n
        self.dw_out = views.pop("dw_out")
        self.grads = views
        self.dist = dist
        self.grads_host = {k: torch.empty(v.shape, pin_memory=True) for k, v in self.grads.items()}
        self.dE0 = torch.empty((N, H), device="cuda")
        self.dE0_orig = torch.zeros((n_all, H), device="cuda")
        self.dE0_host = torch.empty((n_all, H), pin_memory=True)
        self.Y = torch.empty((N, H), device="cuda")
        self.train = bool(c.get("train"))
        if c["gru"]:
            self.saved = torch.empty(L.ggnn_saved_bytes(self.plan, self.dt, H, T), dtype=torch.uint8,
                                     device="cuda")
            self.ws_f = torch.empty(L.ggnn_workspace_bytes(self.plan, self.dt, H, T, L.BG_OP_GGNN_FWD),
                                    dtype=torch.uint8, device="cuda")
            self.ws_b = torch.empty(L.ggnn_workspace_bytes(self.plan, self.dt, H, T, L.BG_OP_GGNN_BWD),
                                    dtype=torch.uint8, device="cuda")
            self.ET = torch.empty((N, H), dtype=tdt, device="cuda")
        else:
            self.ws_f = torch.empty(L.workspace_bytes(self.plan, self.dt, H, L.BG_OP_PROPAGATE_FWD),
                                    dtype=torch.uint8, device="cuda")
            self.ws_b = torch.empty(L.workspace_bytes(self.plan, self.dt, H, L.BG_OP_PROPAGATE_BWD),
                                    dtype=torch.uint8, device="cuda")
        if self.train:
            n_g = self.info["n_packed"]
            self.target = torch.from_numpy(
                np.random.default_rng(seed + 3).standard_normal(n_g).astype(np.float32)).cuda()
            self.loss = torch.zeros(4, device="cuda")
            self.ws_r = torch.empty(L.workspace_bytes(self.plan, self.dt, H, L.BG_OP_READOUT),
                                    dtype=torch.uint8, device="cuda")
            names = ["W", "b", "W_ih", "W_hh", "b_ih", "b_hh", "w_out"]
            self.opt = {}
            for k in names:
                master = torch.from_numpy(np.asarray(prm[k], np.float32)).cuda().reshape(-1)
                self.opt[k] = (master, torch.zeros_like(master), torch.zeros_like(master))
            self.adam_t = 0

    def step(self, E0=None, dET=None):
        L, c = self.L, self.c
        H, T = c["H"], c["T"]
        E0 = self.E0 if E0 is None else E0
        dET = self.dET if dET is None else dET
        if not c["gru"]:
            L.band_propagate_fwd(self.plan, self.dt, H, E0, self.prm["W"], self.prm["b"], self.Y,
                                 self.ws_f)
            L.band_propagate_bwd(self.plan, self.dt, H, E0, self.prm["W"], dET, self.dE0,
                                 self.grads["dW"], self.grads["db"], self.ws_b)
            allreduce_grads(self.dist, self.gflat)
            return
        L.ggnn_step(self.plan, self.dt, H, T, self.prm, E0, self.ET, self.saved, self.ws_f)
        if self.train:
            L.readout_loss(self.plan, self.dt, H, self.ET, self.prm["w_out"], self.target,
                           self.loss, self.dET, self.dw_out, self.ws_r)
            dET = self.dET
        L.ggnn_step_bwd(self.plan, self.dt, H, T, self.prm, self.saved, dET, self.dE0, self.grads,
                        self.ws_b)
        allreduce_grads(self.dist, self.gflat)
        if self.train:
            self.adam_t += 1
            gmap = dict(self.grads, w_out=self.dw_out)
            for k, (master, m, v) in self.opt.items():
                g = gmap["d" + k] if k != "w_out" else gmap["w_out"]
                work = self.prm[k].reshape(-1)
                L.adam_step(master, work if work.dtype != self.torch.float32 else work, m, v,
                            g.reshape(-1), 1e-3, 0.9, 0.999, 1e-8, self.adam_t)

    def e2e_run(self, steps, stream):
        """`steps` steps of the user's call sequence with host buffers, timed on `stream`: every step
        copies its inputs from pinned host memory (H2D), packs, runs fwd+bwd, unpacks and reads its
        results back (D2H).  As in a training loop with prefetching, the copies run on their own
        stream with double buffers: step k+1's inputs go up and step k's results come down while
        step k computes.  Returns (ms per step, H2D bytes per step, D2H bytes per step)."""
        torch, L, c = self.torch, self.L, self.c
        H = c["H"]
        if not hasattr(self, "e_cs"):
            self.e_cs = torch.cuda.Stream()
            self.e_in = [self.E_orig_dev, torch.empty_like(self.E_orig_dev)]
            self.e_dET = [torch.empty_like(self.dET), torch.empty_like(self.dET)]
            self.e_out = [self.dE0_orig, torch.empty_like(self.dE0_orig)]
            self.e_out_host = [self.dE0_host, torch.empty(self.dE0_host.shape, pin_memory=True)]
            self.e_gdev = [torch.empty_like(self.gflat), torch.empty_like(self.gflat)]
            self.e_ghost = [torch.empty(self.gflat.shape, pin_memory=True) for _ in range(2)]
            self.e_h2d = [torch.cuda.Event(), torch.cuda.Event()]
            self.e_comp = [torch.cuda.Event(), torch.cuda.Event()]
        cs = self.e_cs
        t0, t1, fin = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True),
                       torch.cuda.Event())

        def h2d(k):
            b = k % 2
            with torch.cuda.stream(cs):
                self.e_in[b].copy_(self.E_orig_host, non_blocking=True)
                self.e_dET[b].copy_(self.dET_host, non_blocking=True)
            self.e_h2d[b].record(cs)

        t0.record(stream)
        cs.wait_event(t0)
        h2d(0)
        for k in range(steps):
            b, nb = k % 2, (k + 1) % 2
            if k + 1 < steps:
                if k >= 1:
                    cs.wait_event(self.e_comp[nb])  # step k-1 is done with buffer set nb
                h2d(k + 1)
            stream.wait_event(self.e_h2d[b])  # also orders step k-2's reads of set b before this
            L.pack_states(self.plan, self.dt, H, self.e_in[b], self.E0)
            self.step(dET=self.e_dET[b])
            L.unpack_states(self.plan, "f32", H, self.dE0, self.e_out[b])
            self.e_gdev[b].copy_(self.gflat, non_blocking=True)
            self.e_comp[b].record(stream)
            cs.wait_event(self.e_comp[b])
            with torch.cuda.stream(cs):
                self.e_out_host[b].copy_(self.e_out[b], non_blocking=True)
                self.e_ghost[b].copy_(self.e_gdev[b], non_blocking=True)
        fin.record(cs)
        stream.wait_event(fin)
        t1.record(stream)
        torch.cuda.synchronize()
        bi = self.E_orig_host.numel() * self.E_orig_host.element_size() + self.dET_host.numel() * 4
        bo = self.dE0_host.numel() * 4 + self.gflat.numel() * 4
        return t0.elapsed_time(t1) / steps, bi, bo


# --------------------------------------------------------------------------------- CPU oracle


def oracle_sample(name: str, c, budget_s: float = 15.0, parallel: bool = False,
                  smallest_first: bool = False, graphs=None):
    """The oracle as it stands on a bounded sample of the workload: fp64 forward + backward of the
    workload's step (T GGNN steps with the GRU, or one propagation), timed without the layout
    (the GPU number excludes the plan too).  Single-threaded: one graph at a time, leading graphs
    first (or smallest first); parallel: the pull-based multi-threaded oracle on all host cores,
    on supergraphs of eight graphs at a time.  A problem larger than the rest of the budget allows
    (at the per-node cost measured so far, or before the first measurement at 1e9 multiply-adds
    per second and thread) is cut to a prefix of its band positions: the subgraph the first m
    positions induce, nodes of the same degree mix.  The graphs are taken in turn (again from the
    first when the list ends) until the budget is spent.  Returns (node-steps/s, sample
    description)."""
    import oracle
    from paper_1906_11786_gb300 import synth
    graphs = graphs if graphs is not None else synth.workload_graphs(name, S=c["S"])
    P, S, H, T = c["P"], c["S"], c["H"], c["T"]
    order = sorted(range(len(graphs)), key=lambda i: graphs[i].n_nodes) if smallest_first \
        else list(range(len(graphs)))
    group = 8 if parallel else 1
    threads = oracle.par_max_threads() if parallel else 1
    done_nodes, spent, used, cut = 0, 0.0, 0, 0
    rng = np.random.default_rng(0)
    n_chunks = -(-len(order) // group)
    for it in range(1 << 20):
        i0 = (it % n_chunks) * group
        chunk = [graphs[i] for i in order[i0:i0 + group]]
        lay = oracle.layout(chunk, P, S, with_masks=False)
        N, n_real = lay.n_pad, lay.n_real
        d, s_, t_ = lay.kept_dst, lay.kept_src, lay.kept_type
        if done_nodes == 0:  # before any measurement: about 1e9 multiply-adds per second
            cap = int(budget_s * 1e9 * max(1, threads // 2) / (6.0 * T * (P + 6) * H * H))
        else:
            cap = int((budget_s - spent) / (spent / done_nodes))
        cap = max(32, cap)
        if n_real > cap:
            keep = (d < cap) & (s_ < cap)
            d, s_, t_ = d[keep], s_[keep], t_[keep]
            N = n_real = cap
            cut += 1
        E0 = np.zeros((N, H)); E0[:n_real] = rng.standard_normal((n_real, H))
        dY = rng.standard_normal((N, H))
        e = (d, s_, t_)
        prm = synth.gen_params(P, H, 1, mean_in_degree=lay.n_kept / max(lay.n_real, 1))
        t0 = time.perf_counter()
        if c["gru"] and parallel:
            Es, Ys = oracle.par_ggnn_fwd(N, P, H, T, n_real, *e, E0, prm, threads)
            oracle.par_ggnn_bwd(N, P, H, T, n_real, *e, prm, Es, Ys, dY, threads)
        elif c["gru"]:
            Es, Ys = oracle.ggnn_fwd(N, P, H, T, n_real, *e, E0, prm)
            oracle.ggnn_bwd(N, P, H, T, n_real, *e, prm, Es, Ys, dY)
        elif parallel:
            oracle.par_propagate_fwd(N, P, H, *e, E0, prm["W"], prm["b"], threads)
            oracle.par_propagate_bwd(N, P, H, *e, E0, prm["W"], dY, threads)
        else:
            oracle.propagate_fwd(N, P, H, *e, E0, prm["W"], prm["b"])
            oracle.propagate_bwd(N, P, H, *e, E0, prm["W"], dY)
        spent += time.perf_counter() - t0
        done_nodes += n_real
        used += len(chunk)
        if spent > 0.95 * budget_s:
            break
    value = done_nodes * T / spent
    desc = {"graphs": used, "nodes": done_nodes, "seconds": spent, "threads": threads,
            "kind": "parallel" if parallel else "single",
            "text": (f"{'smallest' if smallest_first else 'leading'} graphs, {used} taken "
                     + (f"({cut} cut to a prefix of band positions) " if cut else "")
                     + f"({done_nodes} nodes) of the same workload, fwd+bwd, {spent:.1f}s of "
                     + (f"pull-based fp64 on {threads} host threads" if parallel
                        else "single-threaded fp64") + ", layout not timed")}
    return value, desc


# --------------------------------------------------------------------------------- main


def fixed_config(name, graphs, c, world, n_packed, n_real, n_pad, K):
    """The workload's identity, the same for both arms: what ran, not how fast.  `l2` states
    whether one step's working set (the band's bit tiles in both orientations and the states and
    saved activations, estimated from the shapes) exceeds the 129 MB L2 or is timed L2-resident."""
    tiles = 2 * K * 3 * c["P"] * c["S"] * c["S"] // 8
    acts = (2 * c["T"] + 1) * n_pad * c["H"] * 2
    mb = (tiles + acts) / 1e6
    l2 = (f"per-step working set ~{mb:.0f} MB (band tiles + activations) > 129 MB L2" if mb > 129
          else f"per-step working set ~{mb:.1f} MB fits the 129 MB L2: repeated steps run "
               "L2-resident (not flushed)")
    return {"workload": name, "graphs": len(graphs), "packed": n_packed, "n_real": n_real,
            "n_pad": n_pad, "K": K, "S": c["S"], "P": c["P"], "H": c["H"], "T": c["T"],
            "l2": l2,
            "parallelism": f"dp{world} (one supergraph per GPU"
                           + (", gradient all-reduce)" if world > 1 else ")")}


def run_reference(args):
    """The reference arm: the fp64 CPU oracle as it stands, on the host cores, each step a bounded
    sample of the same workload; its step time is the sample's measured time."""
    rank, world, _ = _dist()
    if rank != 0:
        return 0
    import oracle
    graphs, c = workload(args.workload, 0, args.S, args.H)
    lay = oracle.layout(graphs, c["P"], c["S"], c["cap"], with_masks=False)
    per_step = max(0.5, min(args.ref_budget, 150.0 / max(1, args.warmup + args.steps)))
    secs, units, last = [], [], None
    for i in range(args.warmup + args.steps):
        v, s = oracle_sample(args.workload, c, budget_s=per_step, graphs=graphs)
        if i >= args.warmup:
            secs.append(s["seconds"])
            units.append(s["nodes"] * c["T"])
            last = s
    value = sum(units) / sum(secs)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "node-steps/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * sum(secs) / len(secs), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": fixed_config(args.workload, graphs, c, world, lay.n_packed, lay.n_real,
                               lay.n_pad, lay.K),
        "cpu_baseline": {"value": value, "unit": "node-steps/s", "cores": 1, "kind": "oracle",
                         "sample": f"per step: {last['text']} (about {per_step:.1f}s); "
                                   f"ms_per_step is the sample's measured time, value the "
                                   f"sample's node-steps over it"},
        "e2e": {"value": value, "unit": "node-steps/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


def run_op(args, st, c):
    """One band propagation call per step (forward or backward) on the workload's supergraph."""
    import torch

    from paper_1906_11786_gb300 import _binding as L
    H = c["H"]
    ws_f = torch.empty(L.workspace_bytes(st.plan, st.dt, H, L.BG_OP_PROPAGATE_FWD),
                       dtype=torch.uint8, device="cuda")
    ws_b = torch.empty(L.workspace_bytes(st.plan, st.dt, H, L.BG_OP_PROPAGATE_BWD),
                       dtype=torch.uint8, device="cuda")

    def one():
        if args.op == "band_fwd":
            L.band_propagate_fwd(st.plan, st.dt, H, st.E0, st.prm["W"], st.prm["b"], st.Y, ws_f)
        else:
            L.band_propagate_bwd(st.plan, st.dt, H, st.E0, st.prm["W"], st.dET, st.dE0,
                                 st.grads["dW"], st.grads["db"], ws_b)

    for _ in range(max(args.warmup, 3)):
        one()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(args.steps):
        one()
    e1.record()
    torch.cuda.synchronize()
    L.check_device()
    ms = e0.elapsed_time(e1) / args.steps
    f = st.plan.flops(H, L.BG_FLOPS_BAND) + st.plan.flops(H, L.BG_FLOPS_XFORM)
    print(json.dumps({"op": args.op, "ms_per_call": ms, "tflops": f / (ms / 1e3) / 1e12,
                      "band_kernels": "tcgen05" if L.band_uses_tensor_cores(st.plan, st.dt, H)
                      else "simt"}))
    return 0


KNAMES = ["band_fwd", "band_bwd", "gru_fwd", "gru_bwd", "dW"]


def roofline(L, st, c, kt, pk, workload_name):
    """Roofline of the dominant band kernel (the one with the larger share of the step): its
    algorithmic FLOPs per launch (band-dense contraction plus the fused edge-type transform chain)
    over its average CUDA-event duration.  Tensor-core kernels against the measured bf16 peak
    (burst; the sustained fraction beside it); the fp32 SIMT path against the fp32 FMA rate of the
    SMs (an ALU bound: 128 lanes x 2 FLOP x SMs x the measured maximum SM clock)."""
    import torch
    H = c["H"]
    fwd_ms, fwd_n = kt[L.BG_KID_BAND_FWD]
    bwd_ms, bwd_n = kt[L.BG_KID_BAND_BWD]
    kern = "band_fwd" if fwd_ms >= bwd_ms else "band_bwd"
    avg_ms = (fwd_ms / max(fwd_n, 1)) if kern == "band_fwd" else (bwd_ms / max(bwd_n, 1))
    flops = st.plan.flops(H, L.BG_FLOPS_BAND) + st.plan.flops(H, L.BG_FLOPS_XFORM)
    achieved = flops / (avg_ms / 1e3) / 1e12 if avg_ms > 0 else 0.0
    tc = L.band_uses_tensor_cores(st.plan, c["dtype"], H)
    if tc:
        bound, peak = "tensor", pk["bf16"]
        peak_src = f"{pk['src']} bf16 burst (kernel timed per launch)"
    else:
        sms = torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count
        bound, peak = "alu", sms * 128 * 2 * pk["sm_max_mhz"] * 1e6 / 1e12
        peak_src = f"fp32 FMA rate: {sms} SMs x 128 lanes x 2 FLOP x {pk['sm_max_mhz']:.0f} MHz"
    traffic = _profiled_traffic(kern.split("_")[1], workload_name) if tc else None
    roof = {"kernel": kern, "bound": bound, "achieved": achieved, "peak": peak,
            "unit": "TFLOP/s", "frac": achieved / peak, "traffic": traffic,
            "traffic_src": "profiles/ ncu capture (dram read+write bytes per launch)"
            if traffic else None, "peak_src": peak_src,
            "kernel_ms": {k: (kt[i][0] / max(kt[i][1], 1)) for i, k in enumerate(KNAMES)},
            "nnz_tflops": st.plan.flops(H, L.BG_FLOPS_NNZ) / (avg_ms / 1e3) / 1e12
            if avg_ms > 0 else 0.0}
    if tc:
        roof["frac_sustained"] = achieved / pk["bf16_sustained"]
    return roof


def measure(L, graphs, c, name, steps, warmup, prof_min_s, e2e_steps, dist=None, rank=0,
            clocks=None):
    """Plans and runs one workload: W warm-up steps, then exactly `steps` timed steps (CUDA events
    on the stream, no per-launch events), then a profiled pass of the same steps with per-kernel
    CUDA events lasting at least prof_min_s, then the end-to-end run with host buffers."""
    import torch
    st = OursStep(graphs, c, seed=rank, dist=dist)
    units = st.n_real * c["T"]

    def barrier():
        if dist is not None:
            dist.barrier()

    for _ in range(max(warmup, 3)):
        st.step()
    torch.cuda.synchronize()
    L.check_device()
    launches0 = L.launch_count()
    stream = torch.cuda.current_stream()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if clocks is not None:
        clocks.mark("timed_start")
    barrier()
    torch.cuda.synchronize()
    ev0.record(stream)
    for _ in range(steps):
        st.step()
    ev1.record(stream)
    torch.cuda.synchronize()
    barrier()
    if clocks is not None:
        clocks.mark("timed_end")
    launches = L.launch_count() - launches0
    ms = ev0.elapsed_time(ev1)
    L.check_device()
    # per-kernel durations: CUDA events around every launch, on its stream
    for k in range(len(KNAMES)):
        L.profile_read(k, reset=True)
    L.profile_enable(True)
    t0, prof_steps = time.perf_counter(), 0
    while prof_steps < min(steps, 20) or time.perf_counter() - t0 < prof_min_s:
        st.step()
        prof_steps += 1
        if prof_steps % 10 == 0:
            torch.cuda.synchronize()
    torch.cuda.synchronize()
    prof_s = time.perf_counter() - t0
    L.profile_enable(False)
    L.check_device()
    kt = {k: L.profile_read(k, reset=True) for k in range(len(KNAMES))}
    ms, total_units = reduce_over_ranks(dist, ms, float(units))
    ms_step = ms / steps
    st.e2e_run(2, stream)
    barrier()
    e_ms, bi, bo = st.e2e_run(e2e_steps, stream)
    e_ms, _ = reduce_over_ranks(dist, e_ms, 0.0)
    return {"st": st, "ms_step": ms_step, "value": total_units / (ms_step / 1e3),
            "units": total_units, "launches": launches, "kt": kt, "prof_steps": prof_steps,
            "prof_s": prof_s, "e2e": {"value": total_units / (e_ms / 1e3), "unit": "node-steps/s",
                                      "h2d_bytes_per_step": bi, "d2h_bytes_per_step": bo}}


# workloads of the sweep beside the headline (the configurations of the workload list that the
# headline does not cover): (name, S, H)
SWEEP = ([("single512", None, None), ("single20k", None, None)] +
         [("sweep131k", s, None) for s in (32, 64, 128, 256, 512)] +
         [("train100k", None, h) for h in (32, 64, 128, 256)])


def sweep_rows(L, args, pk, budget_s):
    """Every other workload of the list at a short fixed length: node-steps/s, end-to-end, the
    band kernel's roofline fraction and the oracle on the host cores (single-threaded, and for the
    three large workloads the multi-threaded variant too)."""
    import torch
    rows = []
    t_all = time.perf_counter()
    for name, S, H in SWEEP:
        if time.perf_counter() - t_all > budget_s:
            rows.append({"workload": name, "S": S, "H": H, "skipped": "sweep time budget spent"})
            continue
        t_row = time.perf_counter()
        graphs, c = workload(name, 0, S, H)
        m = measure(L, graphs, c, name, steps=10, warmup=3, prof_min_s=0.3, e2e_steps=5)
        t_gpu = time.perf_counter() - t_row
        st = m["st"]
        roof = roofline(L, st, c, m["kt"], pk, name)
        row = {"workload": name, "S": c["S"], "H": c["H"], "T": c["T"], "P": c["P"],
               "dtype": c["dtype"], "n_real": st.n_real, "n_pad": st.N, "value": m["value"],
               "ms_per_step": m["ms_step"], "e2e": m["e2e"]["value"],
               "band_kernels": "tcgen05" if L.band_uses_tensor_cores(st.plan, c["dtype"], c["H"])
               else "simt",
               "roofline": {k: roof[k] for k in ("kernel", "bound", "achieved", "peak", "frac")},
               "kernel_ms": roof["kernel_ms"],
               "nnz_over_band_dense": st.plan.flops(c["H"], L.BG_FLOPS_NNZ) /
               max(st.plan.flops(c["H"], L.BG_FLOPS_BAND), 1.0),
               "dropped_edges": st.info["n_dropped"], "kept_edges": st.info["n_kept"]}
        del m, st
        torch.cuda.synchronize()
        torch.cuda.empty_cache()
        wide = c["H"] >= 128 and c["gru"]
        v, s = oracle_sample(name, c, budget_s=2.0, smallest_first=wide, graphs=graphs)
        row["cpu_oracle"] = {"value": v, "cores": 1, "sample": s["text"]}
        if name in ("single20k", "sweep131k", "train100k"):
            v, s = oracle_sample(name, c, budget_s=2.0, parallel=True, smallest_first=wide,
                                 graphs=graphs)
            row["cpu_oracle_parallel"] = {"value": v, "cores": s["threads"], "sample": s["text"]}
        row["seconds"] = {"plan_and_gpu": t_gpu, "total": time.perf_counter() - t_row}
        rows.append(row)
    return rows


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--workload", default="packed64", choices=list(WORKLOAD_NAMES),
                    help="single512: one 512-node graph, S 64, fp32, one propagation; packed64: 64 "
                         "graphs of 200-2000 nodes, S 128, H 64, T 8; single20k: one 20,000-node "
                         "graph, S 256, H 128, T 8; sweep131k: 131,072 packed positions, one "
                         "propagation (set --S); train100k: ~100k nodes, T 8 with readout, loss "
                         "and Adam (set --H)")
    # the position of the workload in the list above, as earlier command lines name it
    ap.add_argument("--config", type=int, default=None, help=argparse.SUPPRESS)
    ap.add_argument("--S", type=int, default=None)
    ap.add_argument("--H", type=int, default=None)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-sweep", action="store_true",
                    help="skip the sweep over the other workloads (run at N = 1 on rank 0 only)")
    ap.add_argument("--sweep-budget", type=float, default=180.0,
                    help="seconds after which the sweep skips its remaining workloads")
    ap.add_argument("--ref-budget", type=float, default=15.0)
    ap.add_argument("--prof-seconds", type=float, default=2.0,
                    help="minimum length of the profiled pass that times every kernel launch")
    ap.add_argument("--op", default="step", choices=["step", "band_fwd", "band_bwd"],
                    help="time one band propagation kernel call instead of the whole step "
                         "(focused profiling of the same workload)")
    args = ap.parse_args()
    if args.config is not None:
        args.workload = WORKLOAD_NAMES[args.config - 1]
    if args.impl == "reference":
        return run_reference(args)

    import torch
    rank, world, local = _dist()
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    import __graft_entry__
    __graft_entry__.build()
    from paper_1906_11786_gb300 import _binding as L

    graphs, c = workload(args.workload, rank, args.S, args.H)
    if args.op != "step":
        return run_op(args, OursStep(graphs, c, seed=rank, dist=dist), c)

    pk = _peaks()
    with Clocks(local) as clk:
        m = measure(L, graphs, c, args.workload, args.steps, args.warmup, args.prof_seconds,
                    args.steps, dist=dist, rank=rank, clocks=clk)
    st = m["st"]
    roof = roofline(L, st, c, m["kt"], pk, args.workload)
    roof["kernel_timing"] = (f"CUDA events around every launch on its stream, in a profiled pass "
                             f"of {m['prof_steps']} steps ({m['prof_s']:.1f}s) right after the "
                             f"timed region")
    line = {
        "metric": METRIC, "value": m["value"], "unit": "node-steps/s", "n_gpus": world,
        "steps": args.steps, "warmup": max(args.warmup, 3), "ms_per_step": m["ms_step"],
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": c["dtype"], "data": "synthetic program-shaped graphs (seeded)",
        "config": fixed_config(args.workload, graphs, c, world, st.info["n_packed"], st.n_real,
                               st.N, st.info["K"]),
        "plan": {"kept_edges": st.info["n_kept"], "dropped_edges": st.info["n_dropped"],
                 "plan_ms": st.plan_ms, "upload_ms": st.upload_ms,
                 "flops_per_pass": _flops(L, st.plan, c["H"]),
                 "band_kernels": "tcgen05" if L.band_uses_tensor_cores(st.plan, c["dtype"], c["H"])
                 else "simt"},
        "e2e": m["e2e"],
        "gpu_launches": m["launches"],
        "roofline": roof,
        "clocks": clk.summary(),
    }
    del m, st
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        v, s = oracle_sample(args.workload, c, graphs=graphs)
        line["cpu_baseline"] = {"value": v, "unit": "node-steps/s", "cores": 1, "kind": "oracle",
                                "sample": s["text"], "host": _host()}
    if rank == 0 and world == 1 and not args.no_sweep:
        torch.cuda.empty_cache()
        line["sweep"] = sweep_rows(L, args, pk, args.sweep_budget)
    if rank == 0:
        print(json.dumps(line))
    if dist is not None:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
