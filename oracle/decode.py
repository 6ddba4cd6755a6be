"""fp64 decode attention over the compacted KV cache (plain NumPy).

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()``
and the CPU legs of ``bench.py``; the CUDA product path never imports it.

After the selection of Section 4.1, the keys and values of the B kept tokens of
every KV head form the cache that the subsequent decoding steps attend to
(Section 4.1, the sentence after the per-head top-B selection); Section 5.3
(Computational Complexity) measures decoding over that cache.  One decoding
step of query head h_q over the cache of KV head h = h_q // g is the standard
softmax attention

    s_j = scale * <q[h_q], k_j>,   p_j = exp(s_j) / sum_i exp(s_i),
    out[h_q] = sum_j p_j v_j,      j over the first n cached entries,

written here from that definition (the maximum is subtracted before the
exponential, which leaves p unchanged).  A sequence with n = 0 cached entries
gets a zero output, the reading the CUDA path takes.
"""
from __future__ import annotations

import numpy as np


def decode_attention(q: np.ndarray, k_cache: np.ndarray, v_cache: np.ndarray, lens, scale: float) -> np.ndarray:
    """q [batch][Hq][d], k_cache / v_cache [batch][Hkv][cap][d] (any float dtype,
    widened to fp64), lens [batch] valid entries per sequence (clamped to
    [0, cap]).  Returns out [batch][Hq][d] in fp64."""
    q = np.asarray(q, dtype=np.float64)
    k_cache = np.asarray(k_cache, dtype=np.float64)
    v_cache = np.asarray(v_cache, dtype=np.float64)
    batch, Hq, d = q.shape
    Hkv, cap = k_cache.shape[1], k_cache.shape[2]
    g = Hq // Hkv
    out = np.zeros((batch, Hq, d))
    for b in range(batch):
        n = min(max(int(lens[b]), 0), cap)
        if n == 0:
            continue
        for hq in range(Hq):
            h = hq // g
            s = scale * (k_cache[b, h, :n, :] @ q[b, hq, :])
            e = np.exp(s - s.max())
            out[b, hq, :] = (e @ v_cache[b, h, :n, :]) / e.sum()
    return out
