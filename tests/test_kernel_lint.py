"""Source checks on the CUDA kernels that need no GPU.

Every mbarrier a kernel signals or waits on must be initialised by that kernel: a commit or
arrive on an uninitialised barrier is undefined on the device.  The kernels keep their barriers
in one shared-memory struct per kernel, reached through a pointer (``bars->name`` /
``b->name``); this test collects, per source file and struct pointer, the barrier fields used by
the mbarrier / TMA / tcgen05 helpers and the fields passed to ``mbar_init``.
"""
from __future__ import annotations

import os
import re

import pytest

CSRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                    "paper_1906_11786_gb300", "csrc")
USERS = ("mbar_wait", "mbar_try", "mbar_arrive", "mbar_expect_tx", "tc_commit", "warp_arrive",
         "drain_mmas", "tma_load_2d", "tma_load_3d", "bulk_load", "settle")


def _barrier_fields(src: str, ptr: str):
    used, init = set(), set()
    for m in re.finditer(r"(\w+)\(([^;]*?)&" + ptr + r"->(\w+)", src):
        fn, field = m.group(1), m.group(3)
        if fn == "mbar_init":
            init.add(field)
        elif fn in USERS:
            used.add(field)
    # ternaries such as `j ? &bars->drain2 : &bars->drain` pass either field to the helper
    for m in re.finditer(r"\?\s*&" + ptr + r"->(\w+)\s*:\s*&" + ptr + r"->(\w+)", src):
        used.update(m.groups())
    return used, init


@pytest.mark.parametrize("fname,ptr", [("band_tc.cu", "bars"), ("gru_tc.cu", "b")])
def test_every_used_barrier_is_initialised(fname, ptr):
    src = open(os.path.join(CSRC, fname)).read()
    used, init = _barrier_fields(src, ptr)
    assert used, "no barrier uses found: the pattern no longer matches the source"
    assert not (used - init), f"{fname}: barriers used but never initialised: {sorted(used - init)}"
