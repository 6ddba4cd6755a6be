"""The oracle still reproduces its committed regression fixture (tests/golden/oracle_small.json)."""
import json
import os

import numpy as np

from golden.make_golden import compute

HERE = os.path.dirname(os.path.abspath(__file__))


def test_oracle_matches_committed_fixture():
    with open(os.path.join(HERE, "golden", "oracle_small.json")) as f:
        stored = json.load(f)
    now = compute()
    assert stored["workload"] == json.loads(json.dumps(now["workload"]))
    for a, b in zip(stored["layers"], now["layers"]):
        assert a["out_idx"] == b["out_idx"]
        assert a["htop"] == b["htop"]
        assert a["coverage"] == b["coverage"]
        np.testing.assert_allclose(a["sum_P_O"], b["sum_P_O"], rtol=1e-12)
        np.testing.assert_allclose(a["sum_I"], b["sum_I"], rtol=1e-12)
