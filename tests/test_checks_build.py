"""The bounds-checked debug build (libpresto_checks.so, -DPRESTO_CHECKS), on the CPU:
the release library reports no build flags; the debug library, loaded in a process
with PRESTO_CHECKS=1, reports BUILD_CHECKS and exports every declared symbol."""

import os
import subprocess
import sys

import paper_2607_22634_gb300 as P

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_release_library_has_no_checks():
    if os.environ.get("PRESTO_CHECKS") == "1":
        return  # this process loads the debug build
    assert P.presto_build_flags() == 0
    assert P.lib_path().endswith("libpresto.so")


def test_debug_library_loads_under_the_environment_switch():
    code = ("import sys; sys.path.insert(0, '.'); sys.path.insert(0, 'tests');"
            "import paper_2607_22634_gb300 as P; from test_abi import declared_functions;"
            "import ctypes;"
            "assert P.presto_build_flags() == P.BUILD_CHECKS, P.presto_build_flags();"
            "assert P.lib_path().endswith('libpresto_checks.so');"
            "lib = ctypes.CDLL(P.lib_path());"
            "missing = [n for n in declared_functions() if not hasattr(lib, n)];"
            "assert not missing, missing; print('ok')")
    env = dict(os.environ, PRESTO_CHECKS="1")
    r = subprocess.run([sys.executable, "-c", code], cwd=ROOT, env=env, capture_output=True,
                       text=True, timeout=900)
    assert r.returncode == 0 and "ok" in r.stdout, r.stdout + r.stderr
