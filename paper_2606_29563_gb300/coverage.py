"""Token coverage after a prefill's evictions, and its sweep over eviction rates.

Coverage is the paper's measure (Section 3, coverage hypothesis; Section 5.3,
"Coverage of tokens"): the fraction of a sequence's tokens that at least one
(layer, KV head) keeps, C = #{t : n_t > 0} / L, read from the coverage counts
n_t that the selection maintains in the coverage state.  The sweep runs the
selection (the CUDA path, through the C ABI) over every layer at eviction
rates r (budget B = round((1 - r) * L)) for K-VEC and for its SnapKV special
case (no cross-head and no cross-layer step: delta = 0, lambda = 0), and reports
C and the drop C - 1, as the paper's coverage-analysis table does.
"""
from __future__ import annotations

from typing import Dict, Sequence

from . import kvec, synth

# Byte offset of n_t in a sequence's coverage state (layout in kvec.h).
_N_OFFSET = 16


def coverage_of_state(state, seqlens: Sequence[int]):
    """Per-sequence coverage C = #{t < L_s : n_t > 0} / L_s of a coverage-state tensor."""
    out = []
    for b, L in enumerate(seqlens):
        n = state[b, _N_OFFSET:_N_OFFSET + int(L)]
        out.append(float((n > 0).sum().item()) / float(L))
    return out


METHODS = {"kvec": {}, "snapkv": {"num_ext_heads": 0, "lam": 0.0}}


def sweep(wl: synth.Workload, rates: Sequence[float] = (0.25, 0.5, 0.75, 0.9), layers: int = 0,
          device: str = "cuda") -> Dict:
    """Coverage after 1, 2, 4, ... and all `layers` layers (all of the workload's
    by default) for each method of METHODS and eviction rate; one shared set of
    synthetic inputs.  coverage[method][i][k] is the coverage at rates[i] after
    checkpoints[k] layers; drop is coverage - 1 after the last layer."""
    import torch
    layers = layers or wl.layers
    dev = torch.device(device)
    structure = [synth.salient_structure(wl, b, layers) for b in range(wl.batch)]
    xs = [synth.make_layer(wl, l, dev, structure) for l in range(layers)]
    cu_host = torch.tensor(wl.cu_seqlens, dtype=torch.int32).pin_memory()
    cu_dev = cu_host.to(dev)
    L_min = min(wl.seqlens)
    checkpoints = sorted({min(2 ** i, layers) for i in range(layers.bit_length() + 1)})
    result = {"workload": wl.name, "layers": layers, "rates": list(rates), "checkpoints": checkpoints,
              "budgets": [max(wl.window, int(round((1.0 - r) * L_min))) for r in rates], "coverage": {},
              "drop": {}}
    for name, over in METHODS.items():
        per_rate = []
        for B in result["budgets"]:
            w2 = wl.replace(budget=B, **over)
            sel = kvec.KvecSelector(kvec.params_from_workload(w2, max_layers=layers))
            state = sel.new_state(wl.batch, dev)
            outs = sel.alloc_outputs(wl.batch, B, dev)
            stream = torch.cuda.current_stream(dev)
            cov = []
            for l, x in enumerate(xs):
                sel.select_layer(cu_host, cu_dev, x["q_obs"], x["k"], x["v"], state, B, outs, stream)
                if l + 1 in checkpoints:
                    kvec.kvec_sync_status(sel.handle)
                    c = coverage_of_state(state.cpu(), wl.seqlens)
                    cov.append(sum(c) / len(c))
            per_rate.append(cov)
            sel.close()
        result["coverage"][name] = per_rate
        result["drop"][name] = [c[-1] - 1.0 for c in per_rate]
    return result
