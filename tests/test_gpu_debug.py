"""The bounds-checked debug build (ELBOW_MOE_DEBUG), the stand-in for
compute-sanitizer: its cases (tests/debug_cases.py) run in a child process
that loads the debug library, on small batches T = 1..33, N = 64 / 128,
K = 1..8 and a few prefill batches, with canary-padded outputs."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))


def test_debug_build_cases():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    env = dict(os.environ, ELBOW_MOE_DEBUG="1")
    r = subprocess.run([sys.executable, os.path.join(HERE, "debug_cases.py")], env=env,
                       capture_output=True, text=True, timeout=1200)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
    assert "no bounds violation" in r.stdout
