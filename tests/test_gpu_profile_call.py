"""bench.py --profile-call, the mode every capture in profiles/ runs through:
each kind of call makes its launches on a small workload and exits 0 with a
clean device error word."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.parametrize("what", ["verify", "decode", "draft", "append", "tokens", "magicdec"])
def test_profile_call_runs_and_exits_cleanly(what):
    cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--profile-call", what,
           "--config", "tiny", "--warmup", "1", "--calls", "1"]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-2000:]
    assert ("profile-call %s on tiny" % what) in r.stdout
    assert "device error word 0" in r.stdout
