"""Pins of the fp64 decode-attention oracle against things other than itself.

* closed forms: one cached entry returns its value row; equal keys return the
  mean of the values; two entries give the logistic weight of their logit
  difference (catches a missing or inverted scale, a sign error, a transposed
  operand);
* the query-head to KV-head map of grouped-query attention (h = h_q // g);
* entries past ``lens`` never matter, and ``lens = 0`` gives zeros;
* a pure-Python brute force (math.exp, explicit loops) on tiny inputs.
"""
import math

import numpy as np
import pytest

from oracle.decode import decode_attention


def _rand(rng, *shape):
    return rng.standard_normal(shape)


def test_single_entry_returns_its_value():
    rng = np.random.default_rng(1)
    q, k, v = _rand(rng, 2, 4, 16), _rand(rng, 2, 2, 5, 16), _rand(rng, 2, 2, 5, 16)
    out = decode_attention(q, k, v, [1, 1], 0.25)
    for b in range(2):
        for hq in range(4):
            assert np.array_equal(out[b, hq], v[b, hq // 2, 0])


def test_equal_keys_give_the_mean_value():
    rng = np.random.default_rng(2)
    q = _rand(rng, 1, 6, 8)
    k = np.repeat(_rand(rng, 1, 3, 1, 8), 7, axis=2)
    v = _rand(rng, 1, 3, 7, 8)
    out = decode_attention(q, k, v, [7], 0.5)
    for hq in range(6):
        np.testing.assert_allclose(out[0, hq], v[0, hq // 2].mean(axis=0), rtol=0, atol=1e-14)


def test_two_entries_follow_the_logistic_closed_form():
    d, scale, a = 8, 0.125, 3.0
    q = np.zeros((1, 1, d)); q[0, 0, 0] = 2.0
    k = np.zeros((1, 1, 2, d)); k[0, 0, 0, 0] = a          # s0 = scale * a * 2, s1 = 0
    v = np.zeros((1, 1, 2, d)); v[0, 0, 0, 1] = 1.0; v[0, 0, 1, 2] = 1.0
    out = decode_attention(q, k, v, [2], scale)
    p0 = 1.0 / (1.0 + math.exp(-scale * a * 2.0))
    np.testing.assert_allclose(out[0, 0, :3], [0.0, p0, 1.0 - p0], rtol=0, atol=1e-15)


def test_query_heads_read_their_group_kv_head():
    # Values constant per KV head: the output of query head hq is the constant of hq // g.
    rng = np.random.default_rng(3)
    Hq, Hkv, d = 8, 2, 4
    q, k = _rand(rng, 1, Hq, d), _rand(rng, 1, Hkv, 9, d)
    v = np.zeros((1, Hkv, 9, d))
    v[0, 0] = 10.0
    v[0, 1] = -7.0
    out = decode_attention(q, k, v, [9], 1.0)
    for hq in range(Hq):
        np.testing.assert_allclose(out[0, hq], 10.0 if hq < 4 else -7.0, rtol=0, atol=1e-12)


def test_entries_past_lens_never_matter_and_empty_is_zero():
    rng = np.random.default_rng(4)
    q, k, v = _rand(rng, 3, 2, 8), _rand(rng, 3, 1, 10, 8), _rand(rng, 3, 1, 10, 8)
    lens = [6, 0, 10]
    out = decode_attention(q, k, v, lens, 0.3)
    k2, v2 = k.copy(), v.copy()
    k2[0, :, 6:] = 1e3
    v2[0, :, 6:] = -1e6
    k2[1] = 5.0
    out2 = decode_attention(q, k2, v2, lens, 0.3)
    assert np.array_equal(out, out2)
    assert np.all(out[1] == 0.0)
    # lens beyond the capacity clamp to it
    assert np.array_equal(decode_attention(q, k, v, [6, 0, 99], 0.3), out)


@pytest.mark.parametrize("seed", [5, 6, 7])
def test_matches_pure_python_brute_force(seed):
    rng = np.random.default_rng(seed)
    batch, Hq, Hkv, cap, d = 2, 4, 2, 6, 5
    q, k, v = _rand(rng, batch, Hq, d), _rand(rng, batch, Hkv, cap, d), _rand(rng, batch, Hkv, cap, d)
    lens = [int(rng.integers(1, cap + 1)) for _ in range(batch)]
    scale = 0.7
    out = decode_attention(q, k, v, lens, scale)
    g = Hq // Hkv
    for b in range(batch):
        for hq in range(Hq):
            h = hq // g
            logits = [scale * sum(q[b, hq, i] * k[b, h, j, i] for i in range(d)) for j in range(lens[b])]
            w = [math.exp(x) for x in logits]
            tot = sum(w)
            ref = [sum(w[j] * v[b, h, j, i] for j in range(lens[b])) / tot for i in range(d)]
            np.testing.assert_allclose(out[b, hq], ref, rtol=1e-12, atol=1e-13)
