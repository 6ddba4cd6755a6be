"""Comparison of a GPU layer result with the oracle's (TEST INFRASTRUCTURE ONLY).

Tolerances (bf16 inputs, fp32 accumulation on the GPU, fp64 in the oracle):
* a score x (P_O, P_O', I and the coverage-adjusted P' of every candidate) passes
  if |x_gpu - x_orc| <= tol * (|x_orc| + mean over candidates of |x_orc|).
  The mean term makes the bound meaningful for tiny scores: at L = 8192 the
  average score is ~1e-4, so a pure 2e-3 absolute bound would accept anything.
* kept-index sets must be identical except for positions whose oracle key lies
  within that tolerance of the selection threshold (the tie band), for the final
  fill and for the preserved set.  A head whose cross-head choice sits on a sigma
  near-tie is compared only for validity.
* with the head-wise adaptive fill (f0 given) a head's fill has two thresholds,
  its own f0-th key and the joint threshold over every head's remaining
  candidates; a near-tie at the joint one can move a slot from one head to
  another, so per-head list lengths are checked against their bounds and the
  total over heads against the oracle's.
* given the GPU's own indices, the gathered K/V rows and the coverage-state
  update must be bit-exact.
"""
from __future__ import annotations

from typing import Dict, List, Optional

import numpy as np

TOL = 2e-3


def rel_err(g: np.ndarray, o: np.ndarray) -> np.ndarray:
    scale = np.abs(o).mean() if o.size else 0.0
    return np.abs(g.astype(np.float64) - o) / (np.abs(o) + scale + 1e-30)


def _threshold_band(key: np.ndarray, cand: np.ndarray, k: int, tol: float):
    """Oracle k-th largest key among `cand` positions and the half-width of its tie band."""
    if k <= 0 or cand.size == 0:
        return None, 0.0
    vals = np.sort(key[cand])[::-1]
    thr = vals[min(k, vals.size) - 1]
    return thr, tol * (abs(thr) + np.abs(key[cand]).mean())


def _joint_band(orc: Dict[str, np.ndarray], b: int, Lc: int, f0: int, extras: int, tol: float):
    """Adaptive fill: the oracle's joint threshold (the extras-th largest key among
    every head's candidates left after its own best f0) and its tie band."""
    pool = []
    for h in range(orc["out_idx"].shape[1]):
        key = orc["Pprime"][b, h, :Lc]
        free = np.sort(key[~orc["pres"][b, h, :Lc].astype(bool)])[::-1]
        pool.append(free[f0:])
    return _threshold_band(np.concatenate(pool), np.arange(sum(x.size for x in pool)), extras, tol)


def check_layer(gpu: Dict[str, np.ndarray], orc: Dict[str, np.ndarray], seqlens, window: int, budget: int,
                Kp: int, num_ext_heads: int, tol: float = TOL, f0: Optional[int] = None) -> List[str]:
    """Returns a list of human-readable mismatches (empty when the layer passes).

    window: the tail kept unconditionally (w, or 0 when every position is a
    candidate); the candidates are [0, L - window).  f0: the fill slots a head
    ranks itself under the head-wise adaptive fill (None for the uniform fill)."""
    errs: List[str] = []
    H = orc["out_idx"].shape[1]
    F = budget - window - Kp
    ada = f0 is not None
    own = f0 if ada else F
    extras = H * (F - own)
    for b, L in enumerate(seqlens):
        Lc = L - window
        if Lc > 0:
            for name in ("P_O", "P_Oext"):
                for h in range(H):
                    e = rel_err(gpu[name][b, h, :Lc], orc[name][b, h, :Lc])
                    if e.max() > tol:
                        errs.append(f"seq {b} head {h}: {name} rel err {e.max():.3g} at t={int(e.argmax())}")
            e = rel_err(gpu["I"][b, :Lc], orc["I"][b, :Lc])
            if e.max() > tol:
                errs.append(f"seq {b}: I rel err {e.max():.3g} at t={int(e.argmax())}")
            # P' = P + lambda * I * (1 - n_t / (l + 1)) (Section 4.2), the key of the
            # final fill; the GPU writes it only when the sequence is evicted (L > B).
            if gpu.get("Pprime") is not None and L > budget:
                for h in range(H):
                    e = rel_err(gpu["Pprime"][b, h, :Lc], orc["Pprime"][b, h, :Lc])
                    if e.max() > tol:
                        errs.append(f"seq {b} head {h}: Pprime rel err {e.max():.3g} at t={int(e.argmax())}")
            e = np.abs(gpu["sigma"][b] - orc["sigma"][b]) / (np.abs(orc["sigma"][b]) + 1e-30)
            if e.max() > tol:
                errs.append(f"seq {b}: sigma rel err {e.max():.3g}")
        # Heads whose sigma lies within tolerance of the delta-th / (delta+1)-th boundary.
        sig = orc["sigma"][b]
        order = np.sort(sig)
        ambiguous = set()
        if 0 < num_ext_heads < H:
            lo, hi = order[num_ext_heads - 1], order[num_ext_heads]
            if hi - lo <= tol * max(abs(hi), 1e-30):
                ambiguous = {h for h in range(H) if abs(sig[h] - lo) <= tol * abs(lo) or abs(sig[h] - hi) <= tol * abs(hi)}
        joint = (None, 0.0)
        if ada and L > budget:
            joint = _joint_band(orc, b, L - window, own, extras, tol)
            g_tot = int((gpu["out_idx"][b] >= 0).sum())
            o_tot = int((orc["out_idx"][b] >= 0).sum())
            if g_tot != o_tot:
                errs.append(f"seq {b}: {g_tot} kept rows over the heads, the oracle keeps {o_tot}")
        for h in range(H):
            gi = gpu["out_idx"][b, h]
            oi = orc["out_idx"][b, h]
            g_sel = gi[gi >= 0]
            o_sel = oi[oi >= 0]
            if ada and L > budget:
                size_ok = budget - F + own <= g_sel.size <= budget - F + own + extras
            else:
                size_ok = g_sel.size == o_sel.size
            if not size_ok or not np.all(np.diff(g_sel) > 0) or np.any(g_sel >= L):
                errs.append(f"seq {b} head {h}: invalid index list (size {g_sel.size} vs {o_sel.size})")
                continue
            if np.any(gi[g_sel.size:] != -1):
                errs.append(f"seq {b} head {h}: padding is not -1")
            if not set(range(max(L - window, 0), L)) <= set(g_sel.tolist()):
                errs.append(f"seq {b} head {h}: observation window not kept")
            if h in ambiguous:
                continue
            if int(gpu["htop"][b, h]) != int(orc["htop"][b, h]):
                errs.append(f"seq {b} head {h}: cross-head choice differs (sigma not near a tie)")
                continue
            if L <= budget:
                if not np.array_equal(g_sel, o_sel):
                    errs.append(f"seq {b} head {h}: keep-all selection differs")
                continue
            diff = set(g_sel.tolist()) ^ set(o_sel.tolist())
            if not diff:
                continue
            cand = np.arange(Lc)
            P = orc["P"][b, h, :Lc]
            pres = orc["pres"][b, h, :Lc].astype(bool)
            thr_p, band_p = _threshold_band(P, cand, Kp, tol)
            key = orc["Pprime"][b, h, :Lc]
            thr_f, band_f = _threshold_band(key, cand[~pres], own, tol)
            thr_j, band_j = joint
            bad = []
            for t in diff:
                if t >= Lc:   # a window position: reported above
                    bad.append(t)
                    continue
                near_fill = thr_f is not None and abs(key[t] - thr_f) <= band_f
                near_joint = thr_j is not None and abs(key[t] - thr_j) <= band_j
                near_pres = thr_p is not None and abs(P[t] - thr_p) <= band_p
                if not (near_fill or near_joint or near_pres):
                    bad.append(t)
            if bad:
                errs.append(f"seq {b} head {h}: {len(bad)} kept positions differ outside the tie band, e.g. {bad[:5]}")
    return errs


def check_state_and_gather(gpu_idx: np.ndarray, gpu_k: np.ndarray, gpu_v: np.ndarray, k_bits: np.ndarray,
                           v_bits: np.ndarray, cu, state_before: Dict[str, np.ndarray],
                           state_after: Dict[str, np.ndarray]) -> List[str]:
    """Bit-exact checks that depend only on the GPU's own indices (uint16 bf16 bit patterns)."""
    errs: List[str] = []
    batch, H, B = gpu_idx.shape
    for b in range(batch):
        L = cu[b + 1] - cu[b]
        union = np.zeros(state_before["n"].shape[1], bool)
        for h in range(H):
            idx = gpu_idx[b, h]
            sel = idx[idx >= 0]
            union[sel] = True
            if not np.array_equal(gpu_k[b, h, :sel.size], k_bits[cu[b] + sel, h]):
                errs.append(f"seq {b} head {h}: gathered K differs")
            if not np.array_equal(gpu_v[b, h, :sel.size], v_bits[cu[b] + sel, h]):
                errs.append(f"seq {b} head {h}: gathered V differs")
            if np.any(gpu_k[b, h, sel.size:] != 0) or np.any(gpu_v[b, h, sel.size:] != 0):
                errs.append(f"seq {b} head {h}: padding rows not zero")
        n_expect = state_before["n"][b].astype(np.int64) + union
        if not np.array_equal(state_after["n"][b].astype(np.int64), n_expect):
            errs.append(f"seq {b}: n_t update differs from the union of kept positions")
        bits = np.unpackbits(state_after["last_union"][b].view(np.uint8), bitorder="little")[:union.size]
        if not np.array_equal(bits.astype(bool), union):
            errs.append(f"seq {b}: last_union bits differ")
        if state_after["layers_done"][b] != state_before["layers_done"][b] + 1:
            errs.append(f"seq {b}: layers_done not incremented")
        if state_after["seqlen"][b] != L:
            errs.append(f"seq {b}: seqlen not recorded")
    return errs
