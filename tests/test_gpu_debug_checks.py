"""The debug build (libace_debug.so: index guards in the routing,
compaction, gather and combine kernels, canary words past every device array
of a layer) on small shapes, T in {1, 3, 17, 129, 300} and 20 or 100 experts,
in a child process that loads that library: no guard fires, no canary is
touched, outputs keep replay parity, and a canary overwritten from the host
is reported."""
import os
import subprocess
import sys

import pytest

from paper_2609_05228_gb300 import build

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))


def test_debug_build_runs_clean_on_small_shapes():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    if not os.path.exists(build.DEBUG_LIBPATH):
        build.build()
    env = dict(os.environ, ACE_LIB_VARIANT="debug")
    r = subprocess.run([sys.executable, os.path.join(HERE, "_debug_checks_run.py")], env=env,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-3000:]
    assert "debug checks clean" in r.stdout
