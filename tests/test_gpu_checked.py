"""The checked build on the GPU: the n-gram, word-set and drift-KL parity
suites pass with every device-side bounds check compiled in (ATTT_CHECKED=1
selects libattt_checked.so), so no check fires on valid inputs."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_parity_suites_under_the_checked_build():
    from paper_2607_03441_gb300 import build
    build.build(checked=True)
    env = dict(os.environ, ATTT_CHECKED="1")
    suites = ["tests/test_gpu_ngram.py", "tests/test_gpu_jaccard.py", "tests/test_gpu_kl.py"]
    r = subprocess.run([sys.executable, "-m", "pytest", *suites, "-x", "-q", "-m", "gpu", "-p", "no:cacheprovider"],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=1200)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-2000:]
    # the child really ran the checked library
    probe = ("import paper_2607_03441_gb300.attt as a; "
             "print(a.load_library()._name)")
    name = subprocess.run([sys.executable, "-c", probe], cwd=ROOT, env=env, capture_output=True, text=True,
                          check=True).stdout
    assert "libattt_checked.so" in name
