"""The checked build of the library (BANDLU_CHECKED=1: every inter-warp hand-off of the
windowed factorisation on mbarriers with bounded waits, so a protocol slip ends the kernel
with an error status instead of a hang) passes the same parity cases as the production
build.  Runs them in a child process, which loads only the checked library."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

SELECT = ("test_gbtrf_matches_oracle or test_gbtrf_zero_pivots or test_gbtrf_forced or test_gbtrf_pivot_ties "
          "or test_gbtrf_garbage or test_gbtrf_nan or test_dispatch_lu_matches or test_gbtrf_tridiagonal")

CHILD = f"""
import os, sys
sys.path.insert(0, {ROOT!r})
from paper_2608_22099_gb300 import bandlu
lib = bandlu.load()
assert os.path.basename(lib._name) == "libbandlu_checked.so", lib._name
import pytest
sys.exit(pytest.main([os.path.join({ROOT!r}, "tests", "test_gpu_parity.py"), "-m", "gpu", "-q", "-x",
                      "-p", "no:cacheprovider", "-k", {SELECT!r}]))
"""


def test_checked_build_passes_the_parity_cases():
    env = dict(os.environ, BANDLU_CHECKED="1")
    r = subprocess.run([sys.executable, "-c", CHILD], cwd=os.path.join(ROOT, "tests"), env=env,
                       capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, (r.stdout[-3000:], r.stderr[-3000:])
    assert " passed" in r.stdout and " failed" not in r.stdout, r.stdout[-2000:]
