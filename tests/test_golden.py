"""The oracle against its stored fixture (tests/golden/oracle_tiny.json,
written by tests/golden/make_golden.py from the oracle alone)."""
import json
import os

import numpy as np

from tests.golden import make_golden

HERE = os.path.dirname(os.path.abspath(__file__))


def test_oracle_matches_stored_fixture():
    with open(os.path.join(HERE, "golden", "oracle_tiny.json")) as f:
        ref = json.load(f)
    now = make_golden.compute()
    assert now["idx"] == ref["idx"]
    assert now["fixed"] == ref["fixed"]
    for key in ("scores", "y", "v_out"):
        np.testing.assert_allclose(np.array(now[key]), np.array(ref[key]), rtol=1e-12, atol=1e-14)
    # converged CG: the stored keys are the linearised ridge solution to ~1e-12
    np.testing.assert_allclose(np.array(now["k_out_key_step"]), np.array(ref["k_out_key_step"]),
                               rtol=0, atol=1e-9)
