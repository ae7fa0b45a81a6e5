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


def _run(lib, script="checked_cases.py", *args):
    r = subprocess.run([sys.executable, os.path.join(ROOT, "tests", script), lib, *args],
                       capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-3000:]
    return json.loads(r.stdout.strip().splitlines()[-1])


@pytest.fixture(scope="module")
def checked_lib(tmp_path_factory):
    sys.path.insert(0, ROOT)
    from paper_1801_01554_gb300 import build as B
    d = tmp_path_factory.mktemp("checked")
    return B.build(extra_flags=["-DBP_CHECK"], lib=str(d / "libbp_checked.so"),
                   objdir=str(d / "obj"))


def test_checked_build_passes_its_checks_and_matches(checked_lib):
    from paper_1801_01554_gb300 import build as B
    checked = checked_lib
    normal = B.LIB
    assert os.path.exists(normal)
    a, b = _run(checked), _run(normal)
    assert a.keys() == b.keys()
    for k in a:
        assert a[k] == b[k], k
        assert a[k]["agree"] > 0


@pytest.mark.parametrize("mode,case", [("barrier", "nettalk120_512"), ("chunk", "nettalk120_512"),
                                       ("chunk", "nettalk60_12288")])
def test_wait_that_runs_out_is_reported_and_recovered(checked_lib, mode, case):
    """Section 8's failure detection without a fault, with a 1 ms limit: either
    the first grid barrier of a training launch waits for a count no CTA
    reaches, or the first chunk copy of every CTA's weight phase never comes
    (whole-tile and balanced weight phases).  The launch latches the timeout
    and stops before any update; bp_check reports BP_ETIMEOUT, clears the latch
    and resets the barrier; the next epoch on the same net matches the oracle
    (float32 bar, per layer)."""
    import numpy as np
    from oracle import bp_oracle as O
    from paper_1801_01554_gb300 import bp, synth
    r = _run(checked_lib, "timeout_case.py", mode, case)
    assert r["status"] == bp.BP_ETIMEOUT
    assert r["weights_unchanged"]
    assert r["seconds"] < 1.0          # the 1 ms limit, not the default 2 s
    sizes, n, mb = {"nettalk120_512": ((203, 120, 26), 2048, 512),
                    "nettalk60_12288": ((203, 60, 26), 24576, 12288)}[case]
    X, T = synth.nettalk_patterns(n, seed=71)
    theta = synth.round_to(synth.init_uniform(sizes, -0.3, 0.3, 71), "f32")
    st = O.State(sizes, theta, lr=0.05, momentum=0.9)
    e_ref = O.train_epoch(st, X, T, mb)
    np.testing.assert_allclose(r["sse"], e_ref, rtol=1e-5)
    offs, _ = synth.param_layout(sizes)
    w, v = np.array(r["w"]), np.array(r["v"])
    for l, (wo, bo) in enumerate(offs, start=1):
        for a, b in ((wo, wo + sizes[l] * sizes[l - 1]), (bo, bo + sizes[l])):
            ref = st.theta[a:b] - theta[a:b]
            assert np.max(np.abs(w[a:b] - theta[a:b] - ref)) <= 1e-5 * np.max(np.abs(ref)), l
            assert np.max(np.abs(v[a:b] - st.V[a:b])) <= 1e-5 * np.max(np.abs(st.V[a:b])), l


def test_wait_test_hook_is_inert_in_the_normal_build():
    from paper_1801_01554_gb300 import bp
    with bp.Net((4, 3, 2), 0.1, 0.9, bp.BP_F32, max_batch=8) as net:
        with pytest.raises(bp.BPError) as e:
            bp.bp_debug_wait_test(net.h, 1000, True)
        assert e.value.status == bp.BP_ESTATE
