"""Failure detection of Section 8 on the host: the diagnostic mode's vote.

The GF11 host compared the total squared error each processor computed alone
on the same training set and approved the processors with the most common
value.  The vote here is host code (bp_vote); its failures are planted in host
arrays, so no GPU is faulted to test it.
"""
import numpy as np
import pytest

from paper_1801_01554_gb300 import bp


@pytest.fixture(scope="module")
def lib():
    try:
        return bp.load()
    except ImportError as e:
        pytest.skip(str(e))


def test_vote_approves_the_most_common_error_sum(lib):
    good = np.float32(123.456)
    vals = np.full(152, good, dtype=np.float32)
    vals[[3, 77]] = np.float32(123.457)        # two faulty units
    vals[150] = np.float32(np.nan)
    mode, agree = bp.bp_vote(vals)
    assert mode == good and agree == 149


def test_vote_is_bit_exact_and_breaks_ties_by_first_value(lib):
    a = np.float32(1.0)
    b = np.nextafter(a, np.float32(2.0))         # one ulp apart: a different answer
    mode, agree = bp.bp_vote(np.array([b, a, a, b], dtype=np.float32))
    assert mode == b and agree == 2
    mode, agree = bp.bp_vote(np.array([a, b, b], dtype=np.float32))
    assert mode == b and agree == 2
    nan = np.array([np.nan, np.nan, 1.0], dtype=np.float32)
    mode, agree = bp.bp_vote(nan)
    assert np.isnan(mode) and agree == 2


def test_vote_rejects_empty_input(lib):
    with pytest.raises(bp.BPError):
        bp.bp_vote(np.zeros(0, dtype=np.float32))
