"""The allocation-free forward propagation entry point, for callers that cannot allocate device
memory while they run (no allocator of their own for a workspace, or device allocation forbidden
at that point): its scratch is a fixed array inside the library, so it takes no workspace.
It must give the same result as bg_band_propagate_fwd, on two calls in a row (the array keeps the
previous call's contents), leave the device's free memory unchanged, refuse plans whose scratch
would not fit, and report a device wait that gave up through bg_check_device like every other
entry point.  This file is collected last so that a failure here never hides the rest of the
suite."""
import numpy as np
import pytest
import torch

from paper_1906_11786_gb300 import _binding as L
from paper_1906_11786_gb300 import synth

from gpu_common import TOL, Case, ensure_built, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    ensure_built()


def _both(c: Case, E_dev, b):
    want = torch.empty((c.N, c.H), dtype=torch.float32, device="cuda")
    got = torch.full((c.N, c.H), float("nan"), dtype=torch.float32, device="cuda")
    L.band_propagate_fwd(c.plan, c.dtype, c.H, E_dev, c.dprm["W"], b, want,
                         c.ws(L.BG_OP_PROPAGATE_FWD))
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    L.band_propagate_fwd_noalloc(c.plan, c.dtype, c.H, E_dev, c.dprm["W"], b, got)
    torch.cuda.synchronize()
    free1 = torch.cuda.mem_get_info()[0]
    L.check_device()
    return got.cpu().numpy(), want.cpu().numpy(), free0 - free1


def _rel(a, b):
    return float(np.max(np.abs(a - b)) / max(float(np.max(np.abs(b))), 1e-30))


def _cap_whole_tiles(gs, S):
    n = sum(g.n_nodes for g in gs)
    per_tile = max(1, 128 // S)
    return -(-(-(-n // S)) // per_tile) * per_tile


# (dtype, S, H, P, whole tiles): tensor-core shapes at every H and the S extremes, the fp32 SIMT
# path, and bf16 shapes the tensor-core kernels do not take (H = 96; a ragged last tile), which
# run the SIMT band sums
CASES = [("bf16", 128, 64, 20, 0), ("bf16", 128, 32, 20, 0), ("bf16", 128, 128, 20, 0),
         ("bf16", 128, 256, 8, 0), ("bf16", 32, 64, 20, 1), ("bf16", 512, 64, 20, 0),
         ("bf16", 256, 128, 20, 0), ("f32", 64, 64, 20, 0), ("bf16", 128, 96, 8, 0),
         ("bf16", 32, 64, 8, 0)]


@pytest.mark.parametrize("dtype,S,H,P,whole", CASES)
def test_noalloc_matches_workspace_entry_point_twice(dtype, S, H, P, whole):
    gs = synth.gen_batch(6, 80, 500, P // 2, True, max(8, S // 2), max(8, S // 3), 2.0, 77 + S + H)
    c = Case(gs, P, S, H, dtype, seed=5, cap=_cap_whole_tiles(gs, S) if whole else 0)
    tc = L.band_uses_tensor_cores(c.plan, dtype, H)
    assert tc == (dtype == "bf16" and H != 96 and c.N % 128 == 0)
    got, want, _ = _both(c, c.E_band_dev, c.dprm["b"])
    assert _rel(got, want) < TOL[dtype]
    # second call, different states and no bias: nothing may leak from the first call, and the
    # call leaves the device's free memory as it found it
    E2 = np.random.default_rng(9).standard_normal((c.N, c.H))
    E2[c.n_real:] = 0
    got2, want2, grew = _both(c, to_dev(E2, dtype), None)
    assert _rel(got2, want2) < TOL[dtype]
    assert not np.allclose(got2, got)
    assert grew == 0


def test_noalloc_tensor_core_plan_beyond_the_simt_size():
    """A bf16 tensor-core plan whose SIMT message buffer (P n_pad H 4 bytes = 40 MiB) would not
    fit the array but whose tensor-core scratch (about 1.4 MiB) does: it runs."""
    gs = synth.gen_batch(30, 200, 350, 10, True, 48, 32, 2.0, 3)
    c = Case(gs, 20, 128, 64, "bf16", seed=6, cap=64)
    assert c.N == 8192 and L.band_uses_tensor_cores(c.plan, "bf16", 64)
    assert 20 * c.N * 64 * 4 > 32 << 20
    got, want, _ = _both(c, c.E_band_dev, c.dprm["b"])
    assert _rel(got, want) < TOL["bf16"]


def test_noalloc_rejects_plans_beyond_its_buffer():
    # fp32 path scratch = P * n_pad * H * 4 bytes = 20 * 8192 * 64 * 4 = 40 MiB > 32 MiB
    gs = synth.gen_batch(30, 200, 350, 10, True, 16, 8, 1.0, 3)
    plan = L.band_plan(gs, 20, 32, capacity_blocks=256)
    plan.upload()
    N, H = plan.info()["n_pad"], 64
    E = torch.zeros((N, H), device="cuda")
    W = torch.zeros((20, H, H), device="cuda")
    Y = torch.zeros((N, H), device="cuda")
    with pytest.raises(L.BandGGNNError) as ei:
        L.band_propagate_fwd_noalloc(plan, "f32", H, E, W, None, Y)
    assert ei.value.code == -2 and "static buffer" in str(ei.value)


def test_noalloc_timeouts_reach_bg_check_device():
    """The entry point's bounded waits record a give-up in the library's one status word, so
    bg_check_device sees it: the self test gives up a wait on that word, then a clean no-alloc
    call; the check reports the timeout once, clears it, and the next check is clean."""
    gs = synth.gen_batch(3, 80, 300, 10, True, 48, 32, 2.0, 12)
    c = Case(gs, 20, 128, 64, "bf16", seed=7)
    Y = torch.empty((c.N, c.H), dtype=torch.float32, device="cuda")
    L.selftest_device_wait()
    L.band_propagate_fwd_noalloc(c.plan, c.dtype, c.H, c.E_band_dev, c.dprm["W"], c.dprm["b"], Y)
    with pytest.raises(L.BandGGNNError) as err:
        L.check_device()
    assert "BG_ETIMEOUT" in str(err.value)
    L.band_propagate_fwd_noalloc(c.plan, c.dtype, c.H, c.E_band_dev, c.dprm["W"], c.dprm["b"], Y)
    L.check_device()


def test_noalloc_with_supernodes():
    """A plan with supernodes: their rows and columns are added to Y in place, with no scratch;
    the result equals the workspace entry point's, on two calls in a row."""
    gs = synth.gen_batch(4, 100, 500, 10, True, 48, 32, 2.0, 21)
    g = synth.hub_graph(260, 20, 22, lam=2.0)
    gs.insert(1, g)
    c = Case(gs, 20, 128, 64, "bf16", seed=8, sup=(100, 1))
    assert c.plan.info()["n_super"] == 1
    for E_dev, b in ((c.E_band_dev, c.dprm["b"]), (c.E_band_dev, None)):
        got, want, grew = _both(c, E_dev, b)
        assert _rel(got, want) < TOL["bf16"] and grew == 0
