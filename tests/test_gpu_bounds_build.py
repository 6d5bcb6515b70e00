"""The bounds-checked build (libdkv_debug.so: the same sources with -DDKV_DEBUG)
stands in for a memory checker: its kernels check every index and offset they
read against the ranges the plan gives them, skip an access outside, and set
DKV_DEV_BOUNDS in the plan's status word (no trap, no assert).

This test builds it and runs the parity suites of the map, compaction (out of
place and in place), decode with appends and multi-query in a child pytest
with DKV_LIBRARY pointing at it: every case must match the oracle as before
and end with no bounds bit set (tests/parity.py checks the word when a case
closes). The child also runs tests/test_gpu_bounds_planted.py, which plants a
mistake the host cannot see and expects the checks to catch it."""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

pytestmark = pytest.mark.gpu


def _child(lib, files):
    env = dict(os.environ, DKV_LIBRARY=lib)
    r = subprocess.run([sys.executable, "-m", "pytest", *files, "-x", "-q", "-m", "gpu", "-k", "not full_size",
                        "-p", "no:cacheprovider"], cwd=ROOT, env=env, capture_output=True, text=True, timeout=1200)
    return r.returncode, r.stdout + r.stderr


def test_bounds_checked_build_passes_the_parity_suites(cuda):
    from paper_2609_32663_gb300 import build
    lib = build.build_library(debug=True)
    rc, out = _child(lib, ["tests/test_gpu_parity.py", "tests/test_gpu_multi.py", "tests/test_gpu_inplace.py"])
    assert rc == 0, out[-3000:]
    rc, out = _child(lib, ["tests/test_gpu_bounds_planted.py"])
    assert rc == 0 and "1 passed" in out, out[-3000:]
