"""The bounds-checked debug build on the GPU: whole rounds on every workload, the
three search policies, per-row lambda and the N = 512 / 1024 budgets run under
PRESTO_CHECKS=1 (libpresto_checks.so) with the same oracle checks as the release
tests, and no kernel reports PRESTO_DEV_BOUNDS or any other status bit."""

import os
import subprocess
import sys

from gpu_common import GPU

pytestmark = GPU
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_checked_build_passes_the_round_search_and_budget_tests():
    env = dict(os.environ, PRESTO_CHECKS="1")
    r = subprocess.run([sys.executable, "-c",
                        "import paper_2607_22634_gb300 as P; assert P.presto_build_flags() == 1"],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout + r.stderr
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-m", "gpu", "-p", "no:cacheprovider",
                        "tests/test_gpu_round.py", "tests/test_gpu_search.py",
                        "tests/test_gpu_large_budget.py", "tests/test_gpu_mask_accept.py"],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=1800)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-3000:]
