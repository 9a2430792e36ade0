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


def _device_sources():
    return {f: open(os.path.join(CSRC, f)).read() for f in sorted(os.listdir(CSRC))
            if f.endswith((".cu", ".cuh"))}


def _strip_comments(src: str) -> str:
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return re.sub(r"//[^\n]*", "", src)


def test_every_device_wait_is_bounded():
    """No device loop waits without a bound: the only mbarrier polling instruction sits in the
    bounded wait helper (tc_util.cuh, at most kSpinLimit polls, then a status record), and no
    source has an unconditional loop, a trap or a device assert to end a wait."""
    srcs = {f: _strip_comments(s) for f, s in _device_sources().items()}
    assert srcs, "no CUDA sources found"
    for f, s in srcs.items():
        assert not re.search(r"for\s*\(\s*;\s*;\s*\)|while\s*\(\s*(true|1)\s*\)", s), \
            f"{f}: unbounded loop"
        assert "__trap" not in s and not re.search(r"(?<![\w.])assert\s*\(", s), \
            f"{f}: trap or device assert"
        polls = len(re.findall(r"mbarrier\.(try_wait|test_wait)", s))
        if f == "tc_util.cuh":
            assert polls == 1, "the wait helper should hold the one polling instruction"
        else:
            assert polls == 0, f"{f}: mbarrier polled outside the bounded wait helper"
    util = srcs["tc_util.cuh"]
    assert re.search(r"for\s*\(\s*uint32_t\s+\w+\s*=\s*0\s*;\s*\w+\s*<\s*kSpinLimit", util)


def test_no_closed_copy_calls():
    """The batched memcpy entry points are closed on the target machines: no source, header or
    script of the product names them."""
    root = os.path.dirname(os.path.dirname(CSRC))
    names = ("cudaMemcpy" + "BatchAsync", "cudaMemcpy3D" + "BatchAsync", "cuMemcpy" + "BatchAsync",
             "cuMemcpy3D" + "BatchAsync")
    for base, _, files in os.walk(root):
        if any(p in base for p in ("_work", "gpurun_out", ".git", "baseline", "__pycache__")):
            continue
        for f in files:
            if f.endswith((".cu", ".cuh", ".h", ".cpp", ".py", ".sh")):
                txt = open(os.path.join(base, f), errors="ignore").read()
                for n in names:
                    assert n not in txt, f"{os.path.join(base, f)} names {n}"
