"""The Python example runs as a user would run it, and succeeds."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_two_replicas_example():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "examples", "two_replicas.py")], cwd=ROOT,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "bit-exact" in r.stdout
