"""The FRT_DEBUG build: kernels check every derived index against their launch's extents
(an access outside is skipped and FRT_ERR_BOUNDS recorded, never a trap) and every sync
and stream release compares the guard words around the KV cache. Builds the debug
library and runs the small parity suite, the convolution suite (its split tiles' workspace
indices are checked) and the debug-only checks against it in a child process
(FRT_LIBRARY=debug)."""

import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_small_parity_suite_and_bounds_checks_under_the_debug_build():
    from paper_2607_18171_gb300 import _build
    _build.build(debug=True)
    env = dict(os.environ, FRT_LIBRARY="debug")
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q",
                        "tests/test_gpu_10_parity_small.py", "tests/test_gpu_55_state.py",
                        "tests/test_gpu_50_conv.py",
                        "tests/debug_checks.py"],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-4000:] + r.stderr[-2000:]
    assert " passed" in r.stdout and "failed" not in r.stdout
