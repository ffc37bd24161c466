"""The oracle against its frozen outputs (tests/golden/oracle_*.txt).

The paper prints no worked example, so these files are not paper values: they were
written by tests/golden/make_oracle_golden.py from the pinned oracle and hold its
actions, rewards, dones, returns and episode lengths (exact) and its fp64
log-probabilities and values (to 1e-12, to allow another host's libm) on three small
seeded cases.  A change to the oracle's arithmetic fails here until the files are
regenerated with it."""
import os
import sys

import numpy as np
import pytest

sys.path.insert(0, os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden"))
import make_oracle_golden as G  # noqa: E402


@pytest.mark.parametrize("name", list(G.CASES))
def test_oracle_matches_its_frozen_outputs(name):
    want = G.read(name)
    got = G.compute(name)
    assert set(want) == set(got)
    for k, w in want.items():
        g = np.asarray(got[k])
        assert g.shape == w.shape, k
        if w.dtype == np.float64:
            assert np.allclose(g, w, rtol=1e-12, atol=1e-14), k
        else:
            assert np.array_equal(g.astype(w.dtype), w), k
