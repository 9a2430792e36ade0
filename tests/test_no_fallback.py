"""The product path has no fallback: without the compiled CUDA library every entry point of the
binding raises instead of computing anything (checked on a copy of the package's Python files,
without the library, in a fresh interpreter)."""
import os
import shutil
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_missing_library_raises_on_every_path(tmp_path):
    pkg = tmp_path / "paper_1906_11786_gb300"
    pkg.mkdir()
    for f in ("__init__.py", "_binding.py", "synth.py", "halo.py"):
        shutil.copy(os.path.join(ROOT, "paper_1906_11786_gb300", f), pkg / f)
    code = """
import paper_1906_11786_gb300 as p
from paper_1906_11786_gb300 import lib, synth
assert not __import__("os").path.exists(lib.LIB_PATH)
g = synth.gen_graph(64, 2, True, 8, 8, 1.0, 3)
calls = {
    "load": lambda: lib.load(),
    "band_plan": lambda: lib.band_plan([g], 4, 32),
    "reach_filter": lambda: lib.reach_filter(g, [0], 2),
    "launch_count": lambda: lib.launch_count(),
    "profile_enable": lambda: lib.profile_enable(True),
}
for name, f in calls.items():
    try:
        f()
    except ImportError as e:
        assert "no fallback" in str(e), (name, str(e))
    else:
        raise SystemExit(f"{name} ran without the library")
print("all raised")
"""
    r = subprocess.run([sys.executable, "-c", code], cwd=tmp_path, capture_output=True, text=True,
                       env=dict(os.environ, PYTHONPATH=str(tmp_path), PYTHONDONTWRITEBYTECODE="1"),
                       timeout=300)
    assert r.returncode == 0 and "all raised" in r.stdout, r.stdout[-2000:] + r.stderr[-2000:]
