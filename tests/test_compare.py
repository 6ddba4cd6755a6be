"""The GPU-versus-oracle comparison (oracle/compare.py) itself, on the CPU: a
result equal to the oracle's (rounded to fp32, as the GPU stores it) passes,
and a planted mistake in any compared score row, P' included, or in the kept
indices is reported."""
import numpy as np
import pytest

import oracle
from oracle import compare
from paper_2606_29563_gb300 import synth


@pytest.fixture(scope="module")
def layer():
    wl = synth.small_workload(seqlens=(300, 200), layers=2, budget=64)
    p = oracle.OracleParams.from_workload(wl)
    st = oracle.new_state(wl.batch, wl.max_seqlen)
    xs = synth.make_layers(wl, 2)
    oracle.select_layer(p, wl.cu_seqlens, xs[0]["q_obs"], xs[0]["k"], xs[0]["v"], st, wl.budget,
                        max_seqlen=wl.max_seqlen)
    r = oracle.select_layer(p, wl.cu_seqlens, xs[1]["q_obs"], xs[1]["k"], xs[1]["v"], st, wl.budget,
                            max_seqlen=wl.max_seqlen)
    Kp = int(np.floor(np.float32(wl.beta) * wl.budget))
    return wl, r, Kp


def _as_gpu(r):
    g = {k: r[k].astype(np.float32) for k in ("P_O", "P_Oext", "I", "sigma", "Pprime")}
    g["htop"] = r["htop"].copy()
    g["out_idx"] = r["out_idx"].copy()
    return g


def _check(wl, r, g, Kp):
    return compare.check_layer(g, r, wl.seqlens, wl.window, wl.budget, Kp, wl.num_ext_heads)


def test_oracle_result_in_fp32_passes(layer):
    wl, r, Kp = layer
    assert _check(wl, r, _as_gpu(r), Kp) == []


@pytest.mark.parametrize("name", ["P_O", "P_Oext", "Pprime"])
def test_planted_score_mistake_is_reported(layer, name):
    wl, r, Kp = layer
    g = _as_gpu(r)
    g[name][0, 1, 17] *= 1.01   # 1 %: five times the tolerance
    errs = _check(wl, r, g, Kp)
    assert any(name in e and "head 1" in e for e in errs), errs


def test_planted_importance_mistake_is_reported(layer):
    wl, r, Kp = layer
    g = _as_gpu(r)
    g["I"][1, 40] *= 0.99
    assert any("I rel err" in e for e in _check(wl, r, g, Kp))


def test_planted_index_mistake_is_reported(layer):
    wl, r, Kp = layer
    g = _as_gpu(r)
    L = wl.seqlens[0]
    key = r["Pprime"][0, 0, :L - wl.window]
    kept = set(g["out_idx"][0, 0].tolist())
    lowest = int(np.argmin(key))   # far outside the tie band
    assert lowest not in kept
    victim = next(t for t in g["out_idx"][0, 0].tolist() if t < L - wl.window and not r["pres"][0, 0, t])
    new = sorted((kept - {victim}) | {lowest})
    g["out_idx"][0, 0, :len(new)] = new
    assert any("outside the tie band" in e for e in _check(wl, r, g, Kp))
