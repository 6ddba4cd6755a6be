"""Pins of the fp64 CPU oracle against things other than itself.

* an independent NumPy brute force (full T x T causal attention, full sorts);
* closed forms (all-zero keys give a uniform causal softmax);
* invariants that the K-VEC paper's definitions fix (Eq. 1 mass, Section 4.2
  coverage counting, budget bookkeeping);
* special cases that reduce K-VEC to plain window-score top-B (SnapKV).
"""
import math

import numpy as np
import pytest
import torch

import oracle
from bruteforce import select as bf_select
from paper_2606_29563_gb300 import synth


def _f64(x: torch.Tensor) -> np.ndarray:
    return x.to(torch.float64).numpy()


def _run_oracle(params, q_obs, k, v, state, budget, cu=None, ml=None):
    if cu is None:
        cu = [0, k.shape[0]]
    return oracle.select_layer(params, cu, q_obs, k, v, state, budget, max_seqlen=ml)


TINY_CASES = [
    # (seed, T, Hq, Hkv, d, w, O, O', pool, delta, lam, beta, B)
    (1, 14, 2, 1, 8, 4, 2, 4, 3, 1, 1.0, 0.25, 8),
    (2, 16, 4, 2, 8, 6, 3, 5, 3, 1, 1.0, 0.5, 10),
    (3, 16, 8, 4, 4, 5, 2, 5, 1, 2, 0.5, 0.34, 9),
    (4, 12, 4, 4, 8, 3, 2, 3, 5, 3, 2.0, 0.25, 6),
    (5, 16, 6, 3, 8, 4, 2, 4, 3, 0, 1.0, 0.25, 8),
    (6, 15, 4, 2, 6, 6, 6, 6, 3, 2, 1.0, 1.0, 11),
    (7, 16, 2, 2, 8, 2, 1, 2, 7, 1, 1.0, 0.0, 5),
    (8, 10, 4, 2, 8, 4, 2, 4, 3, 1, 1.0, 0.25, 12),   # L <= B: keep everything
]


@pytest.mark.parametrize("case", TINY_CASES)
def test_oracle_matches_bruteforce_over_layers(case):
    seed, T, Hq, Hkv, d, w, O, Oe, pool, delta, lam, beta, B = case
    params = oracle.OracleParams(num_q_heads=Hq, num_kv_heads=Hkv, head_dim=d, window=w,
                                 obs_window=O, ext_window=Oe, pool_kernel=pool,
                                 num_ext_heads=delta, lam=lam, beta=beta)
    state = oracle.new_state(1, T)
    n_bf = np.zeros(T, np.int64)
    for layer in range(3):
        x = synth.tiny_full_inputs(seed * 100 + layer, T, Hq, Hkv, d)
        q_obs = x["q_full"][T - w:].reshape(1, w, Hq, d)
        r = _run_oracle(params, q_obs, x["k"], x["v"], state, B)
        bf = bf_select(_f64(x["q_full"]), _f64(x["k"]), num_kv_heads=Hkv, window=w, obs_window=O,
                       ext_window=Oe, pool_kernel=pool, num_ext_heads=delta, lam=lam, beta=beta,
                       budget=B, n_counts=n_bf, layers_done=layer)
        Lc = T - w
        np.testing.assert_allclose(r["P_O_raw"][0, :, :T], bf["P_O_raw"], rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(r["P_Oext_raw"][0, :, :T], bf["P_Oext_raw"], rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(r["I_raw"][0, :T], bf["I_raw"], rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(r["P_O"][0, :, :Lc], bf["P_O"], rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(r["P_Oext"][0, :, :Lc], bf["P_Oext"], rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(r["I"][0, :Lc], bf["I"], rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(r["sigma"][0], bf["sigma"], rtol=1e-9, atol=1e-15)
        assert (r["htop"][0].astype(bool) == bf["htop"]).all()
        np.testing.assert_allclose(r["P"][0, :, :Lc], bf["P"], rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(r["Pprime"][0, :, :Lc], bf["Pprime"], rtol=1e-12, atol=1e-15)
        if T > B:
            assert (r["pres"][0, :, :Lc].astype(bool) == bf["pres"]).all()
        assert (r["out_idx"][0] == bf["out_idx"]).all()
        n_bf = bf["n"]
        f = oracle.state_fields(state, T)
        assert (f["n"][0].astype(np.int64) == n_bf).all()
        assert f["layers_done"][0] == layer + 1


def test_softmax_rows_sum_to_one_and_eq1_mass():
    wl = synth.small_workload(seqlens=(257,), num_q_heads=8, num_kv_heads=2)
    x = synth.make_layer(wl, 0)
    p = oracle.OracleParams.from_workload(wl)
    r = oracle.select_layer(p, wl.cu_seqlens, x["q_obs"], x["k"], x["v"], oracle.new_state(1, 257), wl.budget)
    np.testing.assert_allclose(r["row_sums"], 1.0, atol=1e-12)
    # Eq. 1 averages O rows that each sum to 1, summed over the g heads of a group: mass g.
    g = wl.group
    np.testing.assert_allclose(r["P_O_raw"][0].sum(axis=1), g, rtol=1e-12)
    np.testing.assert_allclose(r["P_Oext_raw"][0].sum(axis=1), g, rtol=1e-12)
    # I averages a max over KV heads: between the mean (mass g) and the sum over heads (mass Hq).
    mass_I = r["I_raw"][0].sum()
    assert g - 1e-12 <= mass_I <= wl.num_q_heads + 1e-12


def test_uniform_keys_closed_form_two_layers():
    """K = 0: every visible key gets 1/(p+1); all candidates tie, so lower positions win.

    Layer 0 keeps [0, B-w) plus the window.  At layer 1 those tokens have
    coverage 1/2, so the fill (not the preserved part) moves to [B-w, ...).
    """
    T, Hq, Hkv, d, w, O, Oe, B = 64, 4, 2, 8, 8, 4, 8, 24
    params = oracle.OracleParams(num_q_heads=Hq, num_kv_heads=Hkv, head_dim=d, window=w,
                                 obs_window=O, ext_window=Oe, pool_kernel=3, num_ext_heads=1,
                                 lam=1.0, beta=0.25)
    g = Hq // Hkv
    x = synth.tiny_full_inputs(3, T, Hq, Hkv, d)
    q_obs = x["q_full"][T - w:].reshape(1, w, Hq, d)
    k = torch.zeros(T, Hkv, d, dtype=torch.bfloat16)
    v = x["v"]
    state = oracle.new_state(1, T)
    r = _run_oracle(params, q_obs, k, v, state, B)
    Lc = T - w
    expect_PO = g / O * sum(1.0 / (T - w + q + 1) for q in range(w - O, w))
    expect_POe = g / Oe * sum(1.0 / (T - w + q + 1) for q in range(w - Oe, w))
    expect_I = 1.0 / O * sum(g / (T - w + q + 1) for q in range(w - O, w))
    np.testing.assert_allclose(r["P_O"][0, :, :Lc], expect_PO, rtol=1e-13)
    np.testing.assert_allclose(r["P_Oext"][0, :, :Lc], expect_POe, rtol=1e-13)
    np.testing.assert_allclose(r["I"][0, :Lc], expect_I, rtol=1e-13)
    # Window rows: key t in the window is visible only to rows q with L-w+q >= t.
    t = T - 1
    np.testing.assert_allclose(r["P_O_raw"][0, 0, t], g / O * (1.0 / T), rtol=1e-13)
    assert np.all(r["sigma"][0] < 1e-15) and r["sigma"][0, 0] == r["sigma"][0, 1]
    assert list(r["htop"][0]) == [1, 0]          # equal sigma: the lower head index wins
    Kp = int(math.floor(0.25 * B))
    layer0 = list(range(B - w)) + list(range(T - w, T))
    assert (r["out_idx"][0] == np.array(layer0)).all()
    r1 = _run_oracle(params, q_obs, k, v, state, B)
    layer1 = list(range(Kp)) + list(range(B - w, B - w + (B - w - Kp))) + list(range(T - w, T))
    assert (r1["out_idx"][0] == np.array(sorted(layer1))).all()
    f = oracle.state_fields(state, T)
    expect_n = np.zeros(T, np.int64)
    for sel in (layer0, layer1):
        expect_n[sel] += 1
    assert (f["n"][0] == expect_n).all()
    assert r1["coverage"][0] == np.count_nonzero(expect_n)


def test_lowest_sigma_head_gets_extended_window():
    """A head whose keys are all zero attends uniformly: its sigma is the smallest (Section 4.1)."""
    T, Hq, Hkv, d, w, B = 96, 4, 4, 16, 16, 40
    x = synth.tiny_full_inputs(11, T, Hq, Hkv, d, key_scale=2.0)
    k = x["k"].clone()
    k[:, 2, :] = 0
    params = oracle.OracleParams(num_q_heads=Hq, num_kv_heads=Hkv, head_dim=d, window=w, obs_window=8,
                                 ext_window=16, pool_kernel=3, num_ext_heads=1, lam=0.0, beta=0.25)
    q_obs = x["q_full"][T - w:].reshape(1, w, Hq, d)
    r = _run_oracle(params, q_obs, k, x["v"], oracle.new_state(1, T), B)
    assert int(np.argmin(r["sigma"][0])) == 2
    assert list(r["htop"][0]) == [0, 0, 1, 0]
    Lc = T - w
    np.testing.assert_array_equal(r["P"][0, 2, :Lc], r["P_Oext"][0, 2, :Lc])
    np.testing.assert_array_equal(r["P"][0, 0, :Lc], r["P_O"][0, 0, :Lc])


def _top_positions(score_row, k):
    order = np.lexsort((np.arange(score_row.size), -score_row))
    return np.sort(order[:k])


def _wl_layers(wl, layers):
    return synth.make_layers(wl, layers)


def test_no_coverage_reduces_to_window_score_topB():
    """delta = 0 and lambda = 0: K-VEC is plain top-(B-w) of pooled P_O plus the window."""
    wl = synth.small_workload(seqlens=(400,), num_ext_heads=0, lam=0.0, budget=72)
    p = oracle.OracleParams.from_workload(wl)
    st = oracle.new_state(1, 400)
    Lc = 400 - wl.window
    for layer, x in enumerate(_wl_layers(wl, 2)):
        r = oracle.select_layer(p, wl.cu_seqlens, x["q_obs"], x["k"], x["v"], st, wl.budget)
        for h in range(wl.num_kv_heads):
            expect = np.concatenate([_top_positions(r["P_O"][0, h, :Lc], wl.budget - wl.window),
                                     np.arange(Lc, 400)])
            assert (r["out_idx"][0, h] == expect).all()


def test_equal_windows_disable_cross_head():
    wl = synth.small_workload(seqlens=(350,), ext_window=16, obs_window=16)
    a = oracle.OracleParams.from_workload(wl)
    b = oracle.OracleParams.from_workload(wl, num_ext_heads=0)
    x = synth.make_layer(wl, 0)
    ra = oracle.select_layer(a, wl.cu_seqlens, x["q_obs"], x["k"], x["v"], oracle.new_state(1, 350), wl.budget)
    rb = oracle.select_layer(b, wl.cu_seqlens, x["q_obs"], x["k"], x["v"], oracle.new_state(1, 350), wl.budget)
    assert (ra["out_idx"] == rb["out_idx"]).all()


def test_lambda_zero_makes_preservation_a_no_op():
    wl = synth.small_workload(seqlens=(330,), lam=0.0)
    x = synth.make_layer(wl, 0)
    outs = []
    for beta in (0.0, 0.25, 1.0):
        p = oracle.OracleParams.from_workload(wl, beta=beta)
        outs.append(oracle.select_layer(p, wl.cu_seqlens, x["q_obs"], x["k"], x["v"],
                                        oracle.new_state(1, 330), wl.budget)["out_idx"])
    assert (outs[0] == outs[1]).all() and (outs[1] == outs[2]).all()


def test_full_preservation_ignores_coverage():
    """beta = 1 preserves B - w tokens by P alone: the state has no effect."""
    wl = synth.small_workload(seqlens=(330,), beta=1.0)
    x = synth.make_layer(wl, 0)
    p = oracle.OracleParams.from_workload(wl)
    st = oracle.new_state(1, 330)
    st[0, 16:16 + 330] = 3                       # pretend every token was kept 3 times
    st[0, 0] = 5                                 # ... over 5 layers
    r1 = oracle.select_layer(p, wl.cu_seqlens, x["q_obs"], x["k"], x["v"], st, wl.budget)
    r0 = oracle.select_layer(oracle.OracleParams.from_workload(wl, lam=0.0), wl.cu_seqlens, x["q_obs"],
                             x["k"], x["v"], oracle.new_state(1, 330), wl.budget)
    assert (r1["out_idx"] == r0["out_idx"]).all()


def test_layer0_focus_is_global_importance():
    wl = synth.small_workload(seqlens=(310,), lam=0.5)
    x = synth.make_layer(wl, 0)
    r = oracle.select_layer(oracle.OracleParams.from_workload(wl), wl.cu_seqlens, x["q_obs"], x["k"],
                            x["v"], oracle.new_state(1, 310), wl.budget)
    Lc = 310 - wl.window
    np.testing.assert_allclose(r["Pprime"][0, :, :Lc] - r["P"][0, :, :Lc],
                               np.broadcast_to(0.5 * r["I"][0, :Lc], (wl.num_kv_heads, Lc)),
                               rtol=1e-10, atol=1e-18)


def test_pool_width_one_is_identity():
    wl = synth.small_workload(seqlens=(300,), pool_kernel=1)
    x = synth.make_layer(wl, 0)
    r = oracle.select_layer(oracle.OracleParams.from_workload(wl), wl.cu_seqlens, x["q_obs"], x["k"],
                            x["v"], oracle.new_state(1, 300), wl.budget)
    Lc = 300 - wl.window
    np.testing.assert_array_equal(r["P_O"][0, :, :Lc], r["P_O_raw"][0, :, :Lc])
    np.testing.assert_array_equal(r["I"][0, :Lc], r["I_raw"][0, :Lc])


def test_multilayer_state_and_budget_invariants():
    wl = synth.small_workload(seqlens=(300, 180, 420), budget=64, layers=4)
    p = oracle.OracleParams.from_workload(wl)
    st = oracle.new_state(wl.batch, wl.max_seqlen)
    n_expect = np.zeros((wl.batch, wl.max_seqlen), np.int64)
    cu = wl.cu_seqlens
    for layer, x in enumerate(_wl_layers(wl, 4)):
        r = oracle.select_layer(p, cu, x["q_obs"], x["k"], x["v"], st, wl.budget, max_seqlen=wl.max_seqlen)
        k_np = x["k"].view(torch.int16).numpy().view(np.uint16)
        v_np = x["v"].view(torch.int16).numpy().view(np.uint16)
        f = oracle.state_fields(st, wl.max_seqlen)
        for b, L in enumerate(wl.seqlens):
            union = np.zeros(wl.max_seqlen, bool)
            for h in range(wl.num_kv_heads):
                idx = r["out_idx"][b, h]
                sel = idx[idx >= 0]
                assert sel.size == min(L, wl.budget)
                assert np.all(np.diff(sel) > 0)
                assert set(range(L - wl.window, L)) <= set(sel.tolist())
                pres = np.flatnonzero(r["pres"][b, h])
                assert set(pres.tolist()) <= set(sel.tolist())
                assert pres.size == min(int(math.floor(wl.beta * wl.budget)), wl.budget - wl.window)
                np.testing.assert_array_equal(r["out_k"][b, h, :sel.size], k_np[cu[b] + sel, h])
                np.testing.assert_array_equal(r["out_v"][b, h, :sel.size], v_np[cu[b] + sel, h])
                assert np.all(r["out_k"][b, h, sel.size:] == 0)
                union[sel] = True
            n_expect[b] += union
            bits = np.unpackbits(f["last_union"][b].view(np.uint8), bitorder="little")[:wl.max_seqlen]
            assert (bits.astype(bool) == union).all()
            assert r["coverage"][b] == np.count_nonzero(n_expect[b])
        assert (f["n"].astype(np.int64) == n_expect).all()
        assert (f["layers_done"] == layer + 1).all()
        assert (f["seqlen"] == np.array(wl.seqlens)).all()
        assert np.all(f["n"] <= layer + 1)


def test_keep_all_when_sequence_fits_budget():
    wl = synth.small_workload(seqlens=(50,), budget=64)
    x = synth.make_layer(wl, 0)
    st = oracle.new_state(1, 50)
    r = oracle.select_layer(oracle.OracleParams.from_workload(wl), wl.cu_seqlens, x["q_obs"], x["k"],
                            x["v"], st, wl.budget)
    for h in range(wl.num_kv_heads):
        assert (r["out_idx"][0, h, :50] == np.arange(50)).all()
        assert (r["out_idx"][0, h, 50:] == -1).all()
    assert (oracle.state_fields(st, 50)["n"][0] == 1).all()


def test_cross_layer_coverage_grows_when_layers_repeat():
    """Section 4.2: with the same scores in every layer, SnapKV keeps the same tokens (coverage flat)
    while the (1 - coverage) focus term pushes K-VEC to new tokens (coverage grows)."""
    wl = synth.small_workload(seqlens=(1200,), num_q_heads=8, num_kv_heads=4, budget=96,
                              salient=30, p_share=0.8, num_ext_heads=2, lam=1.0)
    x = synth.make_layer(wl, 0)
    cov = {}
    for name, over in (("kvec", {}), ("snapkv", dict(num_ext_heads=0, lam=0.0))):
        p = oracle.OracleParams.from_workload(wl, **over)
        st = oracle.new_state(1, 1200)
        cov[name] = []
        for _ in range(4):
            r = oracle.select_layer(p, wl.cu_seqlens, x["q_obs"], x["k"], x["v"], st, wl.budget)
            cov[name].append(int(r["coverage"][0]))
    assert cov["snapkv"] == [cov["snapkv"][0]] * 4
    assert cov["kvec"][3] > cov["kvec"][0]
    assert cov["kvec"][3] > cov["snapkv"][3]


@pytest.mark.parametrize("bad", [
    dict(num_kv_heads=3), dict(obs_window=40), dict(pool_kernel=4), dict(num_ext_heads=5),
    dict(beta=1.5), dict(window=0),
])
def test_oracle_rejects_bad_parameters(bad):
    kw = dict(num_q_heads=8, num_kv_heads=4, head_dim=8, window=8, obs_window=4, ext_window=8,
              pool_kernel=3, num_ext_heads=1, lam=1.0, beta=0.25)
    kw.update(bad)
    p = oracle.OracleParams(**kw)
    x = synth.tiny_full_inputs(0, 32, 8, 4, 8)
    with pytest.raises(ValueError):
        oracle.select_layer(p, [0, 32], x["q_full"][24:].reshape(1, 8, 8, 8), x["k"], x["v"],
                            oracle.new_state(1, 32), 16)


# ---- Paper variants: average pooling and the entropy head criterion (Section 5.4
# "Head Selection Criteria"; the average pool of the SnapKV lineage).

VARIANT_CASES = [c for c in TINY_CASES if c[0] in (2, 3, 5, 7)]


@pytest.mark.parametrize("pool_mode,head_criterion", [(1, 0), (0, 1), (1, 1)])
@pytest.mark.parametrize("case", VARIANT_CASES)
def test_oracle_variants_match_bruteforce(case, pool_mode, head_criterion):
    seed, T, Hq, Hkv, d, w, O, Oe, pool, delta, lam, beta, B = case
    params = oracle.OracleParams(num_q_heads=Hq, num_kv_heads=Hkv, head_dim=d, window=w,
                                 obs_window=O, ext_window=Oe, pool_kernel=pool,
                                 num_ext_heads=delta, lam=lam, beta=beta, pool_mode=pool_mode,
                                 head_criterion=head_criterion)
    state = oracle.new_state(1, T)
    n_bf = np.zeros(T, np.int64)
    for layer in range(2):
        x = synth.tiny_full_inputs(seed * 100 + layer, T, Hq, Hkv, d)
        q_obs = x["q_full"][T - w:].reshape(1, w, Hq, d)
        r = _run_oracle(params, q_obs, x["k"], x["v"], state, B)
        bf = bf_select(_f64(x["q_full"]), _f64(x["k"]), num_kv_heads=Hkv, window=w, obs_window=O,
                       ext_window=Oe, pool_kernel=pool, num_ext_heads=delta, lam=lam, beta=beta,
                       budget=B, n_counts=n_bf, layers_done=layer, pool_mode=pool_mode,
                       head_criterion=head_criterion)
        Lc = T - w
        np.testing.assert_allclose(r["P_O"][0, :, :Lc], bf["P_O"], rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(r["P_Oext"][0, :, :Lc], bf["P_Oext"], rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(r["I"][0, :Lc], bf["I"], rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(r["sigma"][0], bf["sigma"], rtol=1e-9, atol=1e-15)
        assert (r["htop"][0].astype(bool) == bf["htop"]).all()
        np.testing.assert_allclose(r["Pprime"][0, :, :Lc], bf["Pprime"], rtol=1e-12, atol=1e-15)
        assert (r["out_idx"][0] == bf["out_idx"]).all()
        n_bf = bf["n"]


def _tiny_layer(seed, T=48, Hq=8, Hkv=4, d=8, w=8):
    x = synth.tiny_full_inputs(seed, T, Hq, Hkv, d)
    return x["q_full"][T - w:].reshape(1, w, Hq, d), x["k"], x["v"]


@pytest.mark.parametrize("delta", [0, 4])
def test_head_criterion_is_moot_when_no_or_every_head_is_extended(delta):
    q, k, v = _tiny_layer(11)
    out = []
    for crit in (0, 1):
        p = oracle.OracleParams(num_q_heads=8, num_kv_heads=4, head_dim=8, window=8, obs_window=4, ext_window=8,
                                pool_kernel=3, num_ext_heads=delta, head_criterion=crit)
        out.append(_run_oracle(p, q, k, v, oracle.new_state(1, 48), 20)["out_idx"])
    assert np.array_equal(out[0], out[1])


def test_average_pool_of_width_one_is_the_identity():
    q, k, v = _tiny_layer(12)
    res = []
    for mode in (0, 1):
        p = oracle.OracleParams(num_q_heads=8, num_kv_heads=4, head_dim=8, window=8, obs_window=4, ext_window=8,
                                pool_kernel=1, num_ext_heads=2, pool_mode=mode)
        res.append(_run_oracle(p, q, k, v, oracle.new_state(1, 48), 20))
    for name in ("P_O", "P_Oext", "I"):
        assert np.array_equal(res[0][name], res[1][name])
    assert np.array_equal(res[0]["out_idx"], res[1]["out_idx"])


def test_uniform_keys_closed_forms_for_the_variants():
    """K = 0: the candidates' raw scores are one constant per row, so the average
    pool returns it unchanged and every head's normalised distribution is uniform:
    entropy ln(Lc), key -ln(Lc)."""
    T, Hq, Hkv, d, w, O, Oe, B = 64, 4, 2, 8, 8, 4, 8, 24
    g = Hq // Hkv
    x = synth.tiny_full_inputs(3, T, Hq, Hkv, d)
    q_obs = x["q_full"][T - w:].reshape(1, w, Hq, d)
    k = torch.zeros(T, Hkv, d, dtype=torch.bfloat16)
    p = oracle.OracleParams(num_q_heads=Hq, num_kv_heads=Hkv, head_dim=d, window=w, obs_window=O, ext_window=Oe,
                            pool_kernel=5, num_ext_heads=1, pool_mode=1, head_criterion=1)
    r = _run_oracle(p, q_obs, k, x["v"], oracle.new_state(1, T), B)
    Lc = T - w
    expect_PO = g / O * sum(1.0 / (T - w + q + 1) for q in range(w - O, w))
    np.testing.assert_allclose(r["P_O"][0, :, :Lc], expect_PO, rtol=1e-13)
    np.testing.assert_allclose(r["sigma"][0], -math.log(Lc), rtol=1e-13)


# Top-B over every position (all_positions = 1): Section 4.1 states the top-B of
# the T input tokens; by default the last w tokens are kept as in SnapKV.

@pytest.mark.parametrize("variant", [dict(), dict(pool_mode=1, head_criterion=1)])
@pytest.mark.parametrize("case", TINY_CASES)
def test_all_positions_matches_bruteforce_over_layers(case, variant):
    seed, T, Hq, Hkv, d, w, O, Oe, pool, delta, lam, beta, B = case
    params = oracle.OracleParams(num_q_heads=Hq, num_kv_heads=Hkv, head_dim=d, window=w,
                                 obs_window=O, ext_window=Oe, pool_kernel=pool,
                                 num_ext_heads=delta, lam=lam, beta=beta, all_positions=1, **variant)
    state = oracle.new_state(1, T)
    n_bf = np.zeros(T, np.int64)
    for layer in range(3):
        x = synth.tiny_full_inputs(seed * 100 + layer + 7, T, Hq, Hkv, d)
        q_obs = x["q_full"][T - w:].reshape(1, w, Hq, d)
        r = _run_oracle(params, q_obs, x["k"], x["v"], state, B)
        bf = bf_select(_f64(x["q_full"]), _f64(x["k"]), num_kv_heads=Hkv, window=w, obs_window=O,
                       ext_window=Oe, pool_kernel=pool, num_ext_heads=delta, lam=lam, beta=beta,
                       budget=B, n_counts=n_bf, layers_done=layer, all_positions=1, **variant)
        np.testing.assert_allclose(r["P_O"][0, :, :T], bf["P_O"], rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(r["P_Oext"][0, :, :T], bf["P_Oext"], rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(r["I"][0, :T], bf["I"], rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(r["sigma"][0], bf["sigma"], rtol=1e-9, atol=1e-15)
        assert (r["htop"][0].astype(bool) == bf["htop"]).all()
        np.testing.assert_allclose(r["Pprime"][0, :, :T], bf["Pprime"], rtol=1e-12, atol=1e-15)
        if T > B:
            assert (r["pres"][0, :, :T].astype(bool) == bf["pres"]).all()
        assert (r["out_idx"][0] == bf["out_idx"]).all()
        n_bf = bf["n"]
        assert (oracle.state_fields(state, T)["n"][0].astype(np.int64) == n_bf).all()


def test_all_positions_uniform_keys_evict_the_window():
    """K = 0: the prefix and the first window positions tie at the highest score and
    the later window positions, seen by fewer window rows, score lower.  The top B
    are then [0, B): nothing of the window stays.  At layer 1 the preserved part
    stays and the fill moves past the covered tokens."""
    T, Hq, Hkv, d, w, O, Oe, B = 64, 4, 2, 8, 8, 4, 8, 24
    params = oracle.OracleParams(num_q_heads=Hq, num_kv_heads=Hkv, head_dim=d, window=w, obs_window=O,
                                 ext_window=Oe, pool_kernel=3, num_ext_heads=1, lam=1.0, beta=0.25,
                                 all_positions=1)
    g = Hq // Hkv
    x = synth.tiny_full_inputs(3, T, Hq, Hkv, d)
    q_obs = x["q_full"][T - w:].reshape(1, w, Hq, d)
    k = torch.zeros(T, Hkv, d, dtype=torch.bfloat16)
    state = oracle.new_state(1, T)
    r = _run_oracle(params, q_obs, k, x["v"], state, B)
    # Raw Eq. 1 score of window position T - w + j: rows q >= max(j, w - O) see it.
    for j in range(w):
        expect = g / O * sum(1.0 / (T - w + q + 1) for q in range(max(j, w - O), w))
        np.testing.assert_allclose(r["P_O_raw"][0, :, T - w + j], expect, rtol=1e-13)
    Kp = int(math.floor(0.25 * B))
    assert (r["out_idx"][0] == np.arange(B)).all()
    r1 = _run_oracle(params, q_obs, k, x["v"], state, B)
    layer1 = list(range(Kp)) + list(range(B, B + (B - Kp)))
    assert (r1["out_idx"][0] == np.array(layer1)).all()
    expect_n = np.zeros(T, np.int64)
    for sel in (list(range(B)), layer1):
        expect_n[sel] += 1
    assert (oracle.state_fields(state, T)["n"][0] == expect_n).all()


def test_all_positions_rejects_nothing_the_default_needs():
    """A budget below the window is refused only when the window is kept."""
    q, k, v = _tiny_layer(5, T=40, w=8)
    base = dict(num_q_heads=8, num_kv_heads=4, head_dim=8, window=8, obs_window=4, ext_window=8, pool_kernel=3,
                num_ext_heads=1)
    with pytest.raises(ValueError):
        _run_oracle(oracle.OracleParams(**base), q, k, v, oracle.new_state(1, 40), 6)
    r = _run_oracle(oracle.OracleParams(all_positions=1, **base), q, k, v, oracle.new_state(1, 40), 6)
    assert (np.diff(r["out_idx"][0], axis=-1) > 0).all() and r["out_idx"].shape[-1] == 6


@pytest.mark.parametrize("beta", [0.0, 0.25, 1.0])
def test_all_positions_without_coverage_is_plain_topB_of_every_position(beta):
    """delta = 0 and lambda = 0: every head keeps the top B of pooled P_O over
    [0, L), whatever beta, with no window kept by rule."""
    wl = synth.small_workload(seqlens=(400,), num_ext_heads=0, lam=0.0, budget=72, all_positions=1, beta=beta)
    p = oracle.OracleParams.from_workload(wl)
    st = oracle.new_state(1, 400)
    for x in _wl_layers(wl, 2):
        r = oracle.select_layer(p, wl.cu_seqlens, x["q_obs"], x["k"], x["v"], st, wl.budget)
        for h in range(wl.num_kv_heads):
            assert (r["out_idx"][0, h] == _top_positions(r["P_O"][0, h, :400], wl.budget)).all()


# ---- head-wise adaptive fill (head_budget = 1) ----

ADA_CASES = [
    # (seed, T, Hq, Hkv, d, w, O, O', pool, delta, lam, beta, B, ada_floor)
    (21, 16, 4, 2, 8, 4, 2, 4, 3, 1, 1.0, 0.25, 8, 0.0),
    (22, 16, 8, 4, 4, 5, 2, 5, 1, 2, 0.5, 0.34, 9, 0.5),
    (23, 15, 6, 3, 8, 4, 2, 4, 3, 1, 1.0, 0.25, 10, 0.2),
    (24, 12, 4, 4, 8, 3, 2, 3, 5, 3, 2.0, 0.0, 7, 0.3),
    (25, 10, 4, 2, 8, 4, 2, 4, 3, 1, 1.0, 0.25, 12, 0.2),   # L <= B: keep everything
]


@pytest.mark.parametrize("case", ADA_CASES)
def test_adaptive_fill_matches_bruteforce_over_layers(case):
    seed, T, Hq, Hkv, d, w, O, Oe, pool, delta, lam, beta, B, a = case
    params = oracle.OracleParams(num_q_heads=Hq, num_kv_heads=Hkv, head_dim=d, window=w, obs_window=O,
                                 ext_window=Oe, pool_kernel=pool, num_ext_heads=delta, lam=lam, beta=beta,
                                 head_budget=1, ada_floor=a)
    state = oracle.new_state(1, T)
    n_bf = np.zeros(T, np.int64)
    for layer in range(3):
        x = synth.tiny_full_inputs(seed * 100 + layer, T, Hq, Hkv, d)
        q_obs = x["q_full"][T - w:].reshape(1, w, Hq, d)
        r = _run_oracle(params, q_obs, x["k"], x["v"], state, B)
        bf = bf_select(_f64(x["q_full"]), _f64(x["k"]), num_kv_heads=Hkv, window=w, obs_window=O,
                       ext_window=Oe, pool_kernel=pool, num_ext_heads=delta, lam=lam, beta=beta,
                       budget=B, n_counts=n_bf, layers_done=layer, head_budget=1, ada_floor=a)
        assert r["out_idx"].shape[2] == bf["out_idx"].shape[1] == oracle.head_capacity(params, B)
        assert (r["out_idx"][0] == bf["out_idx"]).all()
        n_bf = bf["n"]
        assert (oracle.state_fields(state, T)["n"][0].astype(np.int64) == n_bf).all()


@pytest.mark.parametrize("seed", [31, 32])
def test_adaptive_fill_with_floor_one_is_the_uniform_fill(seed):
    wl = synth.small_workload(seqlens=(300, 200), layers=3, budget=64, seed=seed)
    p_u = oracle.OracleParams.from_workload(wl)
    p_a = oracle.OracleParams.from_workload(wl, head_budget=1, ada_floor=1.0)
    assert oracle.head_capacity(p_a, wl.budget) == wl.budget
    su, sa = oracle.new_state(wl.batch, wl.max_seqlen), oracle.new_state(wl.batch, wl.max_seqlen)
    for x in synth.make_layers(wl, 3):
        ru = oracle.select_layer(p_u, wl.cu_seqlens, x["q_obs"], x["k"], x["v"], su, wl.budget, max_seqlen=wl.max_seqlen)
        ra = oracle.select_layer(p_a, wl.cu_seqlens, x["q_obs"], x["k"], x["v"], sa, wl.budget, max_seqlen=wl.max_seqlen)
        assert (ru["out_idx"] == ra["out_idx"]).all()
        assert (su == sa).all()


@pytest.mark.parametrize("a", [0.0, 0.3])
def test_adaptive_fill_of_identical_heads_is_the_uniform_fill(a):
    """Heads with identical rows rank every position the same way: the joint
    ranking takes one position of each head in turn, so every head gets the same
    share and the selection is the uniform one (no pooling and no cross-head
    window, so that the rows are identical and free of ties)."""
    T, Hq, Hkv, d, w, B = 64, 8, 4, 16, 8, 24
    x = synth.tiny_full_inputs(41, T, Hq, Hkv, d)
    k = x["k"].clone()
    k[:] = k[:, :1]                                   # every KV head the same keys
    q = x["q_full"][T - w:].clone().reshape(w, Hkv, Hq // Hkv, d)
    q[:] = q[:, :1]                                   # every group the same queries
    q_obs = q.reshape(1, w, Hq, d)
    common = dict(num_q_heads=Hq, num_kv_heads=Hkv, head_dim=d, window=w, obs_window=4, ext_window=8,
                  pool_kernel=1, num_ext_heads=0, lam=1.0, beta=0.25)
    p_u = oracle.OracleParams(**common)
    p_a = oracle.OracleParams(**common, head_budget=1, ada_floor=a)
    su, sa = oracle.new_state(1, T), oracle.new_state(1, T)
    for _ in range(2):
        ru = _run_oracle(p_u, q_obs, k, x["v"], su, B)
        ra = _run_oracle(p_a, q_obs, k, x["v"], sa, B)
        cap = oracle.head_capacity(p_a, B)
        assert cap > B
        assert (ra["out_idx"][0, :, :B] == ru["out_idx"][0]).all()
        assert (ra["out_idx"][0, :, B:] == -1).all()
        assert (su == sa).all()


def test_adaptive_fill_budget_bookkeeping():
    """Section 4's budget is kept per layer: the heads keep H_kv * B tokens in
    total, each at least its window, preserved tokens and own floor, at most the
    capacity; the preserved tokens and the window are always among them."""
    wl = synth.small_workload(seqlens=(500, 333), layers=2, budget=64, num_kv_heads=4, num_q_heads=16,
                              num_ext_heads=1, head_budget=1, ada_floor=0.25)
    p = oracle.OracleParams.from_workload(wl)
    cap = oracle.head_capacity(p, wl.budget)
    Kp = int(math.floor(np.float32(wl.beta) * wl.budget))
    F = wl.budget - wl.window - Kp
    own = int(math.floor(np.float32(wl.ada_floor) * F))
    assert cap == wl.budget + (wl.num_kv_heads - 1) * (F - own)
    st = oracle.new_state(wl.batch, wl.max_seqlen)
    for x in synth.make_layers(wl, 2):
        r = oracle.select_layer(p, wl.cu_seqlens, x["q_obs"], x["k"], x["v"], st, wl.budget, max_seqlen=wl.max_seqlen)
        for b, L in enumerate(wl.seqlens):
            counts = (r["out_idx"][b] >= 0).sum(axis=1)
            assert counts.sum() == wl.num_kv_heads * wl.budget
            assert (counts >= wl.window + Kp + own).all() and (counts <= cap).all()
            for h in range(wl.num_kv_heads):
                kept = set(r["out_idx"][b, h][r["out_idx"][b, h] >= 0].tolist())
                assert set(range(L - wl.window, L)) <= kept
                assert set(np.flatnonzero(r["pres"][b, h, :L - wl.window]).tolist()) <= kept


def _random_case(i):
    """A random small configuration (shapes, windows, pooling, hyper-parameters and
    the variants), seeded by i; valid for the oracle's parameter checks."""
    rng = np.random.default_rng(9000 + i)
    Hkv = int(rng.choice([1, 2, 4]))
    g = int(rng.choice([1, 2, 3]))
    w = int(rng.integers(2, 9))
    O = int(rng.integers(1, w + 1))
    Oe = int(rng.integers(O, w + 1))
    T = int(rng.integers(w + 1, 25))
    all_positions = int(rng.random() < 0.3)
    B = int(rng.integers(1 if all_positions else w, T + 2))   # B >= T (keep all) now and then
    return dict(seed=9000 + i, T=T, Hq=g * Hkv, Hkv=Hkv, d=int(rng.choice([4, 8])), w=w, O=O, Oe=Oe,
                pool=int(rng.choice([1, 3, 5])), delta=int(rng.integers(0, Hkv + 1)),
                lam=float(rng.choice([0.0, 0.5, 1.0, 2.0])), beta=float(rng.choice([0.0, 0.25, 0.5, 1.0])), B=B,
                pool_mode=int(rng.random() < 0.3), head_criterion=int(rng.random() < 0.3),
                all_positions=all_positions)


@pytest.mark.parametrize("i", range(60))
def test_oracle_matches_bruteforce_on_random_configurations(i):
    """Sixty seeded random configurations (beyond the hand-picked cases above),
    two layers each with the state carried: every score row, sigma, the chosen
    heads, P', the preserved set, the kept indices and n_t equal the brute force."""
    c = _random_case(i)
    T, Hq, Hkv, d, w, B = c["T"], c["Hq"], c["Hkv"], c["d"], c["w"], c["B"]
    variant = dict(pool_mode=c["pool_mode"], head_criterion=c["head_criterion"], all_positions=c["all_positions"])
    params = oracle.OracleParams(num_q_heads=Hq, num_kv_heads=Hkv, head_dim=d, window=w, obs_window=c["O"],
                                 ext_window=c["Oe"], pool_kernel=c["pool"], num_ext_heads=c["delta"],
                                 lam=c["lam"], beta=c["beta"], **variant)
    state = oracle.new_state(1, T)
    n_bf = np.zeros(T, np.int64)
    Lc = T if c["all_positions"] else T - w
    for layer in range(2):
        x = synth.tiny_full_inputs(c["seed"] * 10 + layer, T, Hq, Hkv, d)
        q_obs = x["q_full"][T - w:].reshape(1, w, Hq, d)
        r = _run_oracle(params, q_obs, x["k"], x["v"], state, B)
        bf = bf_select(_f64(x["q_full"]), _f64(x["k"]), num_kv_heads=Hkv, window=w, obs_window=c["O"],
                       ext_window=c["Oe"], pool_kernel=c["pool"], num_ext_heads=c["delta"], lam=c["lam"],
                       beta=c["beta"], budget=B, n_counts=n_bf, layers_done=layer, **variant)
        np.testing.assert_allclose(r["P_O"][0, :, :Lc], bf["P_O"], rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(r["P_Oext"][0, :, :Lc], bf["P_Oext"], rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(r["I"][0, :Lc], bf["I"], rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(r["sigma"][0], bf["sigma"], rtol=1e-9, atol=1e-15)
        assert (r["htop"][0].astype(bool) == bf["htop"]).all(), c
        np.testing.assert_allclose(r["Pprime"][0, :, :Lc], bf["Pprime"], rtol=1e-12, atol=1e-15)
        if T > B:
            assert (r["pres"][0, :, :Lc].astype(bool) == bf["pres"]).all(), c
        assert (r["out_idx"][0] == bf["out_idx"]).all(), c
        n_bf = bf["n"]
        assert (oracle.state_fields(state, T)["n"][0].astype(np.int64) == n_bf).all(), c


@pytest.mark.parametrize("i", range(30))
def test_adaptive_fill_matches_bruteforce_on_random_configurations(i):
    """The head-wise adaptive fill on thirty seeded random configurations (random
    floor α included), two layers each: kept indices, capacity and n_t equal the
    brute force."""
    c = _random_case(1000 + i)
    a = float(np.random.default_rng(7000 + i).choice([0.0, 0.2, 0.5, 0.8, 1.0]))
    T, Hq, Hkv, d, w, B = c["T"], c["Hq"], c["Hkv"], c["d"], c["w"], c["B"]
    variant = dict(pool_mode=c["pool_mode"], head_criterion=c["head_criterion"], all_positions=c["all_positions"])
    params = oracle.OracleParams(num_q_heads=Hq, num_kv_heads=Hkv, head_dim=d, window=w, obs_window=c["O"],
                                 ext_window=c["Oe"], pool_kernel=c["pool"], num_ext_heads=c["delta"],
                                 lam=c["lam"], beta=c["beta"], head_budget=1, ada_floor=a, **variant)
    state = oracle.new_state(1, T)
    n_bf = np.zeros(T, np.int64)
    for layer in range(2):
        x = synth.tiny_full_inputs(c["seed"] * 10 + layer, T, Hq, Hkv, d)
        q_obs = x["q_full"][T - w:].reshape(1, w, Hq, d)
        r = _run_oracle(params, q_obs, x["k"], x["v"], state, B)
        bf = bf_select(_f64(x["q_full"]), _f64(x["k"]), num_kv_heads=Hkv, window=w, obs_window=c["O"],
                       ext_window=c["Oe"], pool_kernel=c["pool"], num_ext_heads=c["delta"], lam=c["lam"],
                       beta=c["beta"], budget=B, n_counts=n_bf, layers_done=layer, head_budget=1, ada_floor=a,
                       **variant)
        assert r["out_idx"].shape[2] == bf["out_idx"].shape[1] == oracle.head_capacity(params, B)
        assert (r["out_idx"][0] == bf["out_idx"]).all(), (c, a)
        n_bf = bf["n"]
        assert (oracle.state_fields(state, T)["n"][0].astype(np.int64) == n_bf).all(), (c, a)
