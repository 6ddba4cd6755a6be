"""Brute-force K-VEC selection in NumPy, for tiny inputs only.

An implementation independent of the C oracle, written from the K-VEC paper:
it materialises the full causal attention tensor A[h, q, t] for *every* query
position of a short sequence (Algorithm 1's input), slices the last O / O'
query rows as Eq. 1 states, and resolves every top-k with a full sort.  It is
used only to pin the oracle.
"""
from __future__ import annotations

import math
from typing import Dict

import numpy as np


def causal_attention(q_full: np.ndarray, k: np.ndarray, scale: float) -> np.ndarray:
    """q_full [T][Hq][d], k [T][Hkv][d] (float64) -> A [Hq][T][T] with A[h, i, j] = 0 for j > i."""
    T, Hq, _ = q_full.shape
    Hkv = k.shape[1]
    g = Hq // Hkv
    A = np.zeros((Hq, T, T))
    mask = np.triu(np.ones((T, T), bool), 1)
    for hq in range(Hq):
        s = scale * (q_full[:, hq, :] @ k[:, hq // g, :].T)
        s[mask] = -np.inf
        s = s - s.max(axis=1, keepdims=True)
        e = np.exp(s)
        A[hq] = e / e.sum(axis=1, keepdims=True)
    return A


def _ranked(score: np.ndarray, positions: np.ndarray) -> np.ndarray:
    """positions sorted by descending score, ascending position on ties."""
    order = np.lexsort((positions, -score[positions]))
    return positions[order]


def select(q_full, k, *, num_kv_heads, window, obs_window, ext_window, pool_kernel,
           num_ext_heads, lam, beta, budget, n_counts, layers_done, scale=None, pool_mode=0,
           head_criterion=0, all_positions=0, head_budget=0, ada_floor=1.0) -> Dict[str, np.ndarray]:
    """Algorithm 1 followed by per-head top-B for one sequence of length T = q_full.shape[0]."""
    T, Hq, d = q_full.shape
    Hkv = num_kv_heads
    g = Hq // Hkv
    w, O, Oe = window, obs_window, ext_window
    scale = 1.0 / math.sqrt(d) if scale is None else scale
    A = causal_attention(q_full, k, scale)
    Akv = A.reshape(Hkv, g, T, T).sum(axis=1)               # KV-head attention (GQA group sum)

    # Eq. 1 over the last O (and O') query rows; I: mean over the last O rows of the head-max.
    P_O_raw = Akv[:, T - O:, :].mean(axis=1)
    P_Oe_raw = Akv[:, T - Oe:, :].mean(axis=1)
    I_raw = Akv[:, T - O:, :].max(axis=0).mean(axis=0)

    # Candidates: every position before the kept window tail, or every position
    # when nothing is kept unconditionally (top-B over the T input tokens).
    wk = 0 if all_positions else w
    Lc = T - wk
    r = pool_kernel // 2

    def pool(x):
        if pool_mode == 1:
            return np.array([x[max(0, t - r):min(Lc, t + r + 1)].mean() for t in range(Lc)])
        return np.array([x[max(0, t - r):min(Lc, t + r + 1)].max() for t in range(Lc)])

    PO = np.stack([pool(P_O_raw[h]) for h in range(Hkv)]) if Lc > 0 else np.zeros((Hkv, 0))
    POe = np.stack([pool(P_Oe_raw[h]) for h in range(Hkv)]) if Lc > 0 else np.zeros((Hkv, 0))
    I = pool(I_raw) if Lc > 0 else np.zeros(0)

    if head_criterion == 1:
        # Minus the entropy of each head's pooled scores normalised to a distribution.
        sigma = np.zeros(Hkv)
        for h in range(Hkv):
            tot = PO[h].sum()
            if tot > 0:
                pr = PO[h][PO[h] > 0] / tot
                sigma[h] = float(np.sum(pr * np.log(pr)))
    else:
        sigma = PO.std(axis=1, ddof=1) if Lc >= 2 else np.zeros(Hkv)
    head_order = np.lexsort((np.arange(Hkv), sigma))
    htop = np.zeros(Hkv, bool)
    htop[head_order[:num_ext_heads]] = True
    P = np.where(htop[:, None], POe, PO)

    coverage = n_counts[:Lc].astype(np.float64) / (layers_done + 1)
    Pprime = P + lam * (I * (1.0 - coverage))[None, :]
    Kp = min(int(math.floor(beta * budget)), budget - wk)
    F = budget - wk - Kp
    own = int(math.floor(ada_floor * F)) if head_budget else F   # fill slots ranked within the head
    cap = budget + (Hkv - 1) * (F - own)
    cand = np.arange(Lc)
    keep = np.zeros((Hkv, T), bool)
    pres = np.zeros((Hkv, max(Lc, 0)), bool)
    if T <= budget:
        keep[:] = True
    else:
        for h in range(Hkv):
            top = _ranked(P[h], cand)[:Kp]
            pres[h, top] = True
            rest = cand[~pres[h]]
            fill = _ranked(Pprime[h], rest)[:own]
            keep[h, top] = True
            keep[h, fill] = True
            keep[h, Lc:] = True
        if head_budget:
            # The layer's other fill slots: every head's remaining candidates in one
            # list, higher P' first, then lower head, then lower position.
            pool_ = [(-Pprime[h, t], h, t) for h in range(Hkv) for t in range(Lc) if not keep[h, t]]
            pool_.sort()
            for _, h, t in pool_[:Hkv * (F - own)]:
                keep[h, t] = True
    out_idx = np.full((Hkv, cap), -1, np.int64)
    for h in range(Hkv):
        sel = np.flatnonzero(keep[h])
        out_idx[h, :sel.size] = sel
    union = keep.any(axis=0)
    n_new = n_counts[:T].astype(np.int64) + union
    return dict(A=A, P_O_raw=P_O_raw, P_Oext_raw=P_Oe_raw, I_raw=I_raw, P_O=PO, P_Oext=POe, I=I,
                sigma=sigma, htop=htop, P=P, Pprime=Pprime, pres=pres, out_idx=out_idx,
                union=union, n=n_new)
