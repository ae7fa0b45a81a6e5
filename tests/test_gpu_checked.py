"""The checked build (-DBP_CHECK) against the normal library.

compute-sanitizer is not available on the GPUs these tests run on, so the
library has a checked build instead: each float32 phase tests that its shared
memory regions fit the launch's dynamic shared memory and that its rows and
TMA tile origins lie inside their buffers, and latches an error bit (reported
by bp_check) instead of touching memory outside them.  This test builds that
variant beside the normal one, runs the same cases through both in fresh
processes and requires clean checks and identical bits: the tests change no
arithmetic.
"""
import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _run(lib):
    r = subprocess.run([sys.executable, os.path.join(ROOT, "tests", "checked_cases.py"), lib],
                       capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-3000:]
    return json.loads(r.stdout.strip().splitlines()[-1])


def test_checked_build_passes_its_checks_and_matches(tmp_path):
    sys.path.insert(0, ROOT)
    from paper_1801_01554_gb300 import build as B
    checked = B.build(extra_flags=["-DBP_CHECK"], lib=str(tmp_path / "libbp_checked.so"),
                      objdir=str(tmp_path / "obj"))
    normal = B.LIB
    assert os.path.exists(normal)
    a, b = _run(checked), _run(normal)
    assert a.keys() == b.keys()
    for k in a:
        assert a[k] == b[k], k
        assert a[k]["agree"] > 0
