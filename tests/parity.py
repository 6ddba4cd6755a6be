"""Teacher-forced parity run of the CUDA path against the oracle (TEST INFRASTRUCTURE ONLY).

For every layer: run the GPU layer, copy the GPU's state from *before* that layer
into the oracle, run the oracle on the same inputs, and compare (oracle/compare.py).
Errors therefore never compound across layers.
"""
from __future__ import annotations

import math
from typing import Dict, List, Optional

import numpy as np
import torch

import oracle
from oracle import compare
from paper_2606_29563_gb300 import kvec, synth


def _bits(x: torch.Tensor) -> np.ndarray:
    return x.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def gpu_debug_numpy(sel: kvec.KvecSelector, batch: int, max_seqlen: int) -> Dict[str, np.ndarray]:
    d = {k: v.cpu().numpy() for k, v in sel.debug().items()}
    words = d["pres_bits"][:batch]
    pres = np.unpackbits(words.view(np.uint8), axis=-1, bitorder="little")[..., :max_seqlen]
    return {"P_O": d["P_O"][:batch], "P_Oext": d["P_Oext"][:batch], "I": d["I"][:batch],
            "sigma": d["sigma"][:batch], "htop": d["htop"][:batch], "pres": pres,
            "Pprime": d["Pprime"][:batch], "row_stats": d["row_stats"][:batch]}


def window_lse(wl: synth.Workload, x: Dict[str, torch.Tensor]) -> np.ndarray:
    """fp64 log-sum-exp of every window query row over the keys it sees (the
    prefix and the causal part of the window), [batch][w][H_q]: the input of
    kvec_select_layer_lse, as the caller's prefill attention would give it."""
    w, Hq, Hkv, d = wl.window, wl.num_q_heads, wl.num_kv_heads, wl.head_dim
    g = Hq // Hkv
    scale = 1.0 / math.sqrt(d)
    q = x["q_obs"].float().cpu().numpy().astype(np.float64)
    k = x["k"].float().cpu().numpy().astype(np.float64)
    out = np.empty((wl.batch, w, Hq))
    cu = wl.cu_seqlens
    for s in range(wl.batch):
        L = cu[s + 1] - cu[s]
        visible = np.arange(L)[None, :] <= (L - w + np.arange(w))[:, None]   # [w][L]
        for h in range(Hkv):
            logits = scale * np.einsum("qjd,td->qjt", q[s, :, h * g:(h + 1) * g, :], k[cu[s]:cu[s + 1], h, :])
            logits = np.where(visible[:, None, :], logits, -np.inf)
            m = logits.max(axis=2, keepdims=True)
            out[s, :, h * g:(h + 1) * g] = (m + np.log(np.exp(logits - m).sum(axis=2, keepdims=True)))[..., 0]
    return out


def run_parity(wl: synth.Workload, layers: Optional[int] = None, device: str = "cuda", budget: Optional[int] = None,
               tol: float = compare.TOL, verbose: bool = False, with_lse: bool = False,
               sel: Optional[kvec.KvecSelector] = None) -> List[str]:
    """Returns every mismatch over `layers` layers of `wl` (empty list = parity).
    with_lse: the GPU layers take the window rows' log-sum-exp (window_lse) as input.
    sel: an existing selector made for `wl` (kept open), instead of a new one."""
    layers = layers or wl.layers
    budget = budget or wl.budget
    ML = wl.max_seqlen
    own = sel is None
    if own:
        sel = kvec.KvecSelector(kvec.params_from_workload(wl, max_layers=max(layers, 1)))
    oparams = oracle.OracleParams.from_workload(wl)
    kept_tail = 0 if getattr(wl, "all_positions", 0) else wl.window
    Kp = min(int(math.floor(float(np.float32(wl.beta)) * budget)), budget - kept_tail)
    f0 = None
    if getattr(wl, "head_budget", 0):
        f0 = int(math.floor(float(np.float32(wl.ada_floor)) * (budget - kept_tail - Kp)))
    cu_host = torch.tensor(wl.cu_seqlens, dtype=torch.int32)
    cu_dev = cu_host.to(device)
    state = sel.new_state(wl.batch, device)
    errs: List[str] = []
    inputs = synth.make_layers(wl, layers, device="cpu")
    dev_inputs = [{k: v.to(device) for k, v in x.items()} for x in inputs]
    for l in range(layers):
        before = state.cpu().numpy().copy()
        lse = None
        if with_lse:
            lse = torch.from_numpy(window_lse(wl, inputs[l]).astype(np.float32)).to(device)
        out_idx, out_k, out_v = sel.select_layer(cu_host, cu_dev, dev_inputs[l]["q_obs"], dev_inputs[l]["k"],
                                                 dev_inputs[l]["v"], state, budget, lse=lse)
        torch.cuda.synchronize()
        kvec.kvec_sync_status(sel.handle)
        gdbg = gpu_debug_numpy(sel, wl.batch, ML)
        after = state.cpu().numpy()
        ostate = before.copy()
        r = oracle.select_layer(oparams, wl.cu_seqlens, inputs[l]["q_obs"], inputs[l]["k"], inputs[l]["v"], ostate,
                                budget, max_seqlen=ML)
        g = dict(gdbg)
        g["out_idx"] = out_idx.cpu().numpy()
        layer_errs = compare.check_layer(g, r, wl.seqlens, kept_tail, budget, Kp, wl.num_ext_heads, tol, f0=f0)
        layer_errs += compare.check_state_and_gather(
            g["out_idx"], _bits(out_k), _bits(out_v), _bits(inputs[l]["k"]), _bits(inputs[l]["v"]), wl.cu_seqlens,
            oracle.state_fields(before, ML), oracle.state_fields(after, ML))
        if np.array_equal(g["out_idx"], r["out_idx"]) and not np.array_equal(after, ostate):
            layer_errs.append("same indices as the oracle but a different coverage state")
        errs += [f"layer {l}: {e}" for e in layer_errs]
        if verbose:
            same = np.mean(g["out_idx"] == r["out_idx"])
            print(f"layer {l}: {len(layer_errs)} mismatches, index agreement {same:.5f}")
    if own:
        sel.close()
    return errs
