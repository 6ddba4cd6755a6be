"""Writes tests/golden/oracle_small.json from the CPU oracle alone.

The K-VEC paper prints no worked numeric example, so this fixture is a
regression guard on the oracle (any change of its arithmetic shows up here and
must be justified); the pins in test_oracle_pins.py are what tie the oracle to
the paper.  Run: python tests/golden/make_golden.py
"""
import json
import os
import sys


ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
from paper_2606_29563_gb300 import synth  # noqa: E402

WORKLOAD = dict(name="golden_small", seqlens=(300, 190), num_q_heads=8, num_kv_heads=2, budget=64,
                layers=3, num_ext_heads=1, lam=1.0, beta=0.25, salient=6, seed=4242)


def compute():
    wl = synth.small_workload(**WORKLOAD)
    p = oracle.OracleParams.from_workload(wl)
    st = oracle.new_state(wl.batch, wl.max_seqlen)
    layers = []
    for x in synth.make_layers(wl, wl.layers):
        r = oracle.select_layer(p, wl.cu_seqlens, x["q_obs"], x["k"], x["v"], st, wl.budget)
        layers.append({
            "out_idx": r["out_idx"].tolist(),
            "htop": r["htop"].tolist(),
            "coverage": r["coverage"].tolist(),
            "sum_P_O": r["P_O"].sum(axis=2).tolist(),
            "sum_I": r["I"].sum(axis=1).tolist(),
        })
    return {"source": "oracle/kvec_oracle.c via tests/golden/make_golden.py", "workload": WORKLOAD,
            "layers": layers}


if __name__ == "__main__":
    out = os.path.join(os.path.dirname(os.path.abspath(__file__)), "oracle_small.json")
    with open(out, "w") as f:
        json.dump(compute(), f, indent=1)
    print("wrote", out)
