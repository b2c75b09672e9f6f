"""The oracle still produces the stored tiny-workload values (regression pin).

The stored file is written by ``tests/golden/make_golden.py`` from the oracle
alone; the paper prints no worked numeric example, so these values guard the
oracle against unintended change rather than against the paper.
"""
import os

import numpy as np

from tests.golden.make_golden import read, tiny_values

HERE = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def test_oracle_matches_stored_tiny_values():
    stored = read(os.path.join(HERE, "tiny_fp32_oracle.txt"))
    now = tiny_values()
    assert set(stored) == set(now)
    for k in now:
        np.testing.assert_allclose(np.atleast_2d(now[k]), stored[k], rtol=0, atol=1e-13, err_msg=k)
