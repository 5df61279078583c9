"""The self-checking build (-DFAV_DEBUG_CHECKS) on the GPU (needs a GB300).

That build checks shared-memory addresses, TMA destinations, global indices and, in the D = 128
prefill kernel, every role's unit and key-tile totals; a violation prints, sets device status 6
and skips the access.  The test builds libfav_debug.so next to libfav.so, then runs small
prefill (both head dimensions, capped and default grids, ragged lengths), decode (split and
small-Nq), paged-decode and packed-batch calls through it in a child process: every call must
leave the status at 0 and match the oracle."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))


def test_debug_build_runs_clean():
    from paper_2608_18656_gb300 import build as B
    lib = B.build_debug()
    env = dict(os.environ, FAV_LIBRARY=lib)
    r = subprocess.run([sys.executable, os.path.join(HERE, "debug_build_worker.py")], env=env,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-3000:]
    assert "[fav check]" not in r.stdout + r.stderr, r.stdout[-3000:]
    assert "all cases passed" in r.stdout
