"""The parity rule for a fused weight-gradient + update against the oracle.

The kernel's fp32 weight gradient differs from the oracle's only in the order
of its fp32 summation; both sides draw the same Philox uniform for each
element.  A code can therefore differ only where that uniform falls between
the two dense targets, and then by exactly one grid step.  The rule: at most
1e-4 of the codes differ (the count is floored: 1e-4 of 14 336 codes allows
one), and every difference is one step.
"""
import numpy as np

MAX_FRACTION = 1e-4


def assert_fused_codes(got, ref, what=""):
    got = np.asarray(got).astype(np.int32).ravel()
    ref = np.asarray(ref).astype(np.int32).ravel()
    assert got.shape == ref.shape
    diff = got != ref
    allowed = int(MAX_FRACTION * diff.size)
    assert int(diff.sum()) <= allowed, (what, int(diff.sum()), allowed, diff.size)
    assert (np.abs(got - ref)[diff] == 1).all(), what
