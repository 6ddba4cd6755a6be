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


@pytest.fixture(scope="module")
def ada_layer():
    wl = synth.small_workload(seqlens=(400, 250), num_q_heads=16, num_kv_heads=4, layers=2, budget=96,
                              head_budget=1, ada_floor=0.25)
    p = oracle.OracleParams.from_workload(wl)
    st = oracle.new_state(wl.batch, wl.max_seqlen)
    xs = synth.make_layers(wl, 2)
    for x in xs:
        r = oracle.select_layer(p, wl.cu_seqlens, x["q_obs"], x["k"], x["v"], st, wl.budget, max_seqlen=wl.max_seqlen)
    Kp = int(np.floor(np.float32(wl.beta) * wl.budget))
    f0 = int(np.floor(np.float32(wl.ada_floor) * (wl.budget - wl.window - Kp)))
    return wl, r, Kp, f0


def _check_ada(wl, r, g, Kp, f0):
    return compare.check_layer(g, r, wl.seqlens, wl.window, wl.budget, Kp, wl.num_ext_heads, f0=f0)


def test_adaptive_oracle_result_in_fp32_passes(ada_layer):
    wl, r, Kp, f0 = ada_layer
    counts = (r["out_idx"][0] >= 0).sum(axis=1)
    assert counts.min() < counts.max()   # the fill really moved between heads
    assert _check_ada(wl, r, _as_gpu(r), Kp, f0) == []


def test_adaptive_slot_moved_between_heads_far_from_the_threshold_is_reported(ada_layer):
    """A joint-fill slot taken from the head holding it and given to another
    head's lowest candidate: both lists stay valid and the total is unchanged,
    so only the tie-band check can catch it."""
    wl, r, Kp, f0 = ada_layer
    g = _as_gpu(r)
    L, Lc = wl.seqlens[0], wl.seqlens[0] - wl.window
    counts = (r["out_idx"][0] >= 0).sum(axis=1)
    src, dst = int(counts.argmax()), int(counts.argmin())
    key_s = r["Pprime"][0, src, :Lc]
    kept_s = [t for t in g["out_idx"][0, src].tolist() if 0 <= t < Lc and not r["pres"][0, src, t]]
    victim = max(kept_s, key=lambda t: key_s[t])   # the source head's best fill position
    key_d = r["Pprime"][0, dst, :Lc]
    lowest = int(np.argmin(key_d))
    new_s = sorted(set(g["out_idx"][0, src].tolist()) - {-1, victim})
    new_d = sorted(set(g["out_idx"][0, dst].tolist()) - {-1} | {lowest})
    for h, lst in ((src, new_s), (dst, new_d)):
        g["out_idx"][0, h, :] = -1
        g["out_idx"][0, h, :len(lst)] = lst
    errs = _check_ada(wl, r, g, Kp, f0)
    assert any("outside the tie band" in e for e in errs), errs


def test_adaptive_total_over_heads_is_checked(ada_layer):
    wl, r, Kp, f0 = ada_layer
    g = _as_gpu(r)
    counts = (r["out_idx"][0] >= 0).sum(axis=1)
    h = int(counts.argmax())
    g["out_idx"][0, h, counts[h] - 1] = -1   # drop one kept row
    assert any("kept rows over the heads" in e for e in _check_ada(wl, r, g, Kp, f0))
