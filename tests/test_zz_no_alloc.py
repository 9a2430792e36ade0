"""The allocation-free forward propagation entry point, for callers that cannot allocate device
memory while they run: its scratch is a fixed array inside the library, so it takes no workspace.
It must give the same result as bg_band_propagate_fwd, on two calls in a row (the array keeps the
previous call's contents), and refuse plans whose scratch would not fit.  This file is collected
last so that a failure here never hides the rest of the suite."""
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
    L.band_propagate_fwd_noalloc(c.plan, c.dtype, c.H, E_dev, c.dprm["W"], b, got)
    torch.cuda.synchronize()
    return got.cpu().numpy(), want.cpu().numpy()


def _rel(a, b):
    return float(np.max(np.abs(a - b)) / max(float(np.max(np.abs(b))), 1e-30))


@pytest.mark.parametrize("dtype,S,H", [("bf16", 128, 64), ("f32", 64, 64)])
def test_noalloc_matches_workspace_entry_point_twice(dtype, S, H):
    gs = synth.gen_batch(6, 80, 500, 10, True, S // 2, S // 3, 2.0, 77)
    c = Case(gs, 20, S, H, dtype, seed=5)
    got, want = _both(c, c.E_band_dev, c.dprm["b"])
    assert _rel(got, want) < TOL[dtype]
    # second call, different states and no bias: nothing may leak from the first call
    E2 = np.random.default_rng(9).standard_normal((c.N, c.H))
    E2[c.n_real:] = 0
    got2, want2 = _both(c, to_dev(E2, dtype), None)
    assert _rel(got2, want2) < TOL[dtype]
    assert not np.allclose(got2, got)


def test_noalloc_rejects_plans_beyond_its_buffer():
    # fp32 path scratch = P * n_pad * H * 4 bytes = 20 * 8192 * 64 * 4 = 40 MiB > 32 MiB
    gs = synth.gen_batch(30, 200, 350, 10, True, 16, 8, 1.0, 3)
    plan = L.band_plan(gs, 20, 32, capacity_blocks=256)
    plan.upload()
    N, H = plan.info()["n_pad"], 64
    assert L.workspace_bytes(plan, "f32", H, L.BG_OP_PROPAGATE_FWD) > 32 << 20
    E = torch.zeros((N, H), device="cuda")
    W = torch.zeros((20, H, H), device="cuda")
    Y = torch.zeros((N, H), device="cuda")
    with pytest.raises(L.BandGGNNError) as ei:
        L.band_propagate_fwd_noalloc(plan, "f32", H, E, W, None, Y)
    assert ei.value.code == -2 and "static buffer" in str(ei.value)
