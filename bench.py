"""Benchmark of the K-VEC eviction-selection hot path on GB300.

One step = one end-of-prefill eviction pass over every layer of a synthetic
prompt batch: reset the coverage state, then kvec_select_layers over all layers
(window scores, softmax, window sums, pooling, cross-head and cross-layer
coverage, per-KV-head top-B, K/V gather).  The metric is prefix tokens evicted
per second: sum over layers, sequences and KV heads of (L_s - B).

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                       [--workload NAME] [--budget B]
Under torchrun every rank runs its own batch (weak scaling, no collective on the
data path); rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "prefix tokens evicted/sec (all layers, device-timed) and % of HBM roofline"
DEFAULT_WORKLOAD = "llama8b_ragged8_b256"   # the largest single-GPU configuration
FALLBACK_HBM_GBS = 6800.0
KERNEL_SOURCES = {
    "score": "paper_2606_29563_gb300/csrc/score_kernel.cu",
    "window": "paper_2606_29563_gb300/csrc/window_kernel.cu",
    "heads": "paper_2606_29563_gb300/csrc/select_kernels.cu",
    "select": "paper_2606_29563_gb300/csrc/select_kernels.cu",
    "gather": "paper_2606_29563_gb300/csrc/select_kernels.cu",
    "decode": "paper_2606_29563_gb300/csrc/decode_kernel.cu",
}


# ----------------------------------------------------------------------------- distributed plumbing

def dist_env():
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")),
            int(os.environ.get("LOCAL_RANK", "0")))


def init_dist(backend: str):
    import torch.distributed as dist
    rank, world, _ = dist_env()
    if world > 1 and not dist.is_initialized():
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        os.environ.setdefault("MASTER_PORT", "29511")
        dist.init_process_group(backend=backend, rank=rank, world_size=world)
    return rank, world


def barrier():
    import torch.distributed as dist
    if dist.is_initialized():
        dist.barrier()


def max_over_ranks(x: float, device=None) -> float:
    """Largest value of x across ranks (x itself on a single process)."""
    import torch
    import torch.distributed as dist
    if not dist.is_initialized():
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ----------------------------------------------------------------------------- clocks

class ClockSampler:
    """Samples nvidia-smi SM clocks and throttle reasons in the background."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int, interval_ms: int = 50):
        self.samples = []
        self.proc = None
        self.cmd = ["nvidia-smi", "-i", str(gpu_index), f"--query-gpu={self.FIELDS}",
                    "--format=csv,noheader,nounits", f"--loop-ms={interval_ms}"]

    def start(self):
        try:
            self.proc = subprocess.Popen(self.cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            self.proc = None
            return self
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.samples.append((time.perf_counter(), line.strip()))

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.thread.join(timeout=5)

    def summary(self, t0: float, t1: float):
        rows = [s for t, s in self.samples if t0 <= t <= t1]
        window = "timed region"
        if not rows:
            rows = [s for _, s in self.samples]
            window = "whole run (no sample fell inside the timed region)"
        mhz, mx, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for r in rows:
            parts = [p.strip() for p in r.split(",")]
            if len(parts) < 8:
                continue
            try:
                mhz.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for name, val in zip(names, parts[4:8]):
                if val.lower() == "active":
                    reasons.add(name)
        if not mhz:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0, "window": "unavailable"}
        return {"sm_mhz": statistics.median(mhz), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(mhz), "window": window}


# ----------------------------------------------------------------------------- helpers

def measured_hbm_gbs():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            v = float(json.load(f)["hbm_gbs"])
        return v, "measured"
    except (OSError, ValueError, KeyError):
        return FALLBACK_HBM_GBS, "fallback"


def committed_traffic(kernel: str, workload: str):
    """dram read+write bytes per launch from a committed ncu summary, if the kernel is unchanged."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            data = json.load(f)
        entry = data[kernel][workload]
        src = open(os.path.join(ROOT, KERNEL_SOURCES[kernel]), "rb").read()
        if entry.get("source_sha256") != hashlib.sha256(src).hexdigest():
            return None
        return float(entry["bytes_per_launch"])
    except (OSError, ValueError, KeyError, TypeError):
        return None


def committed_step_traffic(wl, layers: int):
    """DRAM bytes (read + written) of one whole step from the committed ncu record of
    every kernel of a layer (profiles/traffic.json, "step"), if no kernel source has
    changed since the capture; else None."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            entry = json.load(f)["step"][wl.name]
        for rel, sha in entry["sources_sha256"].items():
            if hashlib.sha256(open(os.path.join(ROOT, rel), "rb").read()).hexdigest() != sha:
                return None
        return float(entry["bytes_per_layer"]) * layers
    except (OSError, ValueError, KeyError, TypeError):
        return None


E2E_CHUNK = 8            # layers per kvec_select_layers call in the end-to-end step
LAUNCHES_PER_LAYER = 7   # score, row statistics, window, heads pooling, heads top-K, select, gather


def workload_bytes(wl):
    """Algorithmic HBM bytes of one layer (the minimum each step moves) and of one launch of each kernel.

    Per layer: K read once, q_obs read, the kept K/V rows gathered (read + written), the indices written.
    Per kernel (C = candidate positions over the batch, H = KV heads, fp32 score rows):
      score   K + q_obs (+ the (m, Z) row statistics written);
      window  K + q_obs + row statistics read, raw P_O and P_O' rows and raw I written;
      heads   raw rows read, pooled P_O, P_O', I written, the chosen row read again, preserved bits written;
      select  P (chosen row), I, n_t and preserved bits read per head, P' rows and indices written, n_t updated;
      gather  the kept K/V rows read and written, the indices read.
    """
    d, H, Hq, w = wl.head_dim, wl.num_kv_heads, wl.num_q_heads, wl.window
    k_read = wl.total_tokens * H * d * 2
    q_read = wl.batch * w * Hq * d * 2
    C = sum(max(L - w, 0) for L in wl.seqlens)
    kept = sum(min(L, wl.budget) for L in wl.seqlens) * H
    gather_rw = 2 * 2 * kept * d * 2              # K and V rows, read + written
    idx = wl.batch * H * wl.budget * 4
    rowstat = wl.batch * Hq * w * 8
    per_kernel = {
        "score": k_read + q_read + rowstat,
        "window": k_read + q_read + rowstat + (2 * H + 1) * C * 4,
        "heads": (2 * H + 1) * C * 4 * 2 + H * C * 4 + H * C // 8,
        "select": H * C * (4 + 4 + 1) + H * C // 8 + H * C * 4 + idx + 2 * C,
        "gather": gather_rw + idx,
    }
    return {"k_read": k_read, "q_read": q_read, "gather": gather_rw, "idx": idx,
            "layer_total": k_read + q_read + gather_rw + idx, "per_kernel": per_kernel}


def oracle_baseline(wl, budget_s: float = 12.0, max_layers: int = 8, cap_s: float = 30.0):
    """Times the fp64 CPU oracle on a bounded sample of the workload: its first layers,
    repeated from a fresh coverage state until about budget_s of CPU work."""
    import oracle
    from paper_2606_29563_gb300 import synth
    p = oracle.OracleParams.from_workload(wl)
    nl = min(max_layers, wl.layers)
    structure = [synth.salient_structure(wl, b, nl) for b in range(wl.batch)]
    inputs = [synth.make_layer(wl, l, "cpu", structure) for l in range(nl)]
    spent, layers, evicted, passes = 0.0, 0, 0, 0
    while spent < budget_s and spent < cap_s:
        st = oracle.new_state(wl.batch, wl.max_seqlen)
        for x in inputs:
            t0 = time.perf_counter()
            oracle.select_layer(p, wl.cu_seqlens, x["q_obs"], x["k"], x["v"], st, wl.budget,
                                max_seqlen=wl.max_seqlen, debug=False)
            spent += time.perf_counter() - t0
            layers += 1
            evicted += wl.evicted_per_layer()
        passes += 1
    return {"value": evicted / spent, "unit": "tokens/s", "cores": oracle.num_threads(), "kind": "oracle",
            "sample": f"first {nl} of {wl.layers} layers of {wl.name}, {passes} passes from a fresh state "
                      f"(fp64 C oracle, OpenMP), {layers} layers in {spent:.1f} s of CPU work"}


def window_lse_torch(wl, x, dev):
    """Log-sum-exp of every window query row over the keys it sees, [batch][w][H_q]
    fp32: what a caller's prefill attention hands to kvec_select_layers_lse.
    Input preparation for the lse variant (torch, outside the timed region)."""
    import torch
    w, Hq, Hkv, d = wl.window, wl.num_q_heads, wl.num_kv_heads, wl.head_dim
    g, scale = Hq // Hkv, 1.0 / math.sqrt(d)
    out = torch.empty(wl.batch, w, Hq, dtype=torch.float32, device=dev)
    cu = wl.cu_seqlens
    for s in range(wl.batch):
        L = cu[s + 1] - cu[s]
        q = x["q_obs"][s].float()                                        # [w, Hq, d]
        k = x["k"][cu[s]:cu[s + 1]].float().repeat_interleave(g, dim=1)  # [L, Hq, d]
        logits = torch.einsum("qhd,thd->hqt", q, k) * scale              # [Hq, w, L]
        hidden = torch.arange(L, device=dev)[None, :] > (L - w + torch.arange(w, device=dev))[:, None]
        logits.masked_fill_(hidden[None], float("-inf"))
        out[s] = torch.logsumexp(logits, dim=2).transpose(0, 1)
    return out


# ----------------------------------------------------------------------------- our arm

def run_ours(args, wl):
    import torch
    from paper_2606_29563_gb300 import build as kbuild
    from paper_2606_29563_gb300 import kvec, synth

    rank, world = init_dist("nccl" if args.gpus > 1 else "gloo")
    _, _, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    kbuild.build()
    kvec.load()

    L_layers = wl.layers
    params = kvec.params_from_workload(wl)
    sel = kvec.KvecSelector(params)
    cu_host = torch.tensor(wl.cu_seqlens, dtype=torch.int32).pin_memory()
    cu_dev = cu_host.to(dev)
    structure = [synth.salient_structure(wl, b, L_layers) for b in range(wl.batch)]
    # Each rank draws its own batch (seed offset by rank): weak scaling.
    wl_rank = wl.replace(seed=wl.seed + 1000 * rank)
    layers = [synth.make_layer(wl_rank, l, dev, structure) for l in range(L_layers)]
    qs, ks, vs = [x["q_obs"] for x in layers], [x["k"] for x in layers], [x["v"] for x in layers]
    outs = [sel.alloc_outputs(wl.batch, wl.budget, dev) for _ in range(L_layers)]
    state = sel.new_state(wl.batch, dev)
    stream = torch.cuda.current_stream(dev)

    def step():
        kvec.kvec_reset(sel.handle, state.data_ptr(), wl.batch, stream.cuda_stream)
        sel.select_layers(cu_host, cu_dev, qs, ks, vs, state, wl.budget, outs, stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    kvec.kvec_sync_status(sel.handle)

    clocks = ClockSampler(local).start()
    time.sleep(0.3)
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    torch.cuda.synchronize()
    t_host0 = time.perf_counter()
    start.record(stream)
    for _ in range(args.steps):
        step()
    stop.record(stream)
    torch.cuda.synchronize()
    t_host1 = time.perf_counter()
    barrier()
    elapsed_ms = max_over_ranks(start.elapsed_time(stop), dev)
    time.sleep(0.1)
    clocks.stop()
    kvec.kvec_sync_status(sel.handle)

    evicted_per_step = wl.evicted_per_layer() * L_layers
    value = world * evicted_per_step * args.steps / (elapsed_ms / 1e3)
    ms_per_step = elapsed_ms / args.steps

    peak, peak_kind = measured_hbm_gbs()
    by = workload_bytes(wl)
    bytes_step = by["layer_total"] * L_layers
    path_gbs = bytes_step / (ms_per_step / 1e3) / 1e9

    # Clock evidence: when the timed region was too short for the sampler (it
    # polls every 50 ms), the same step keeps running for about a second right
    # after it, and the clocks are read over that run instead.
    clk = clocks.summary(t_host0, t_host1)
    if args.clock_probe and (clk.get("samples", 0) < 3 or clk.get("window") != "timed region"):
        clocks2 = ClockSampler(local).start()
        time.sleep(0.2)
        n_more = max(1, int(1000.0 / max(ms_per_step, 1e-3)))
        t2 = time.perf_counter()
        for _ in range(n_more):
            step()
        torch.cuda.synchronize()
        t3 = time.perf_counter()
        clocks2.stop()
        clk2 = clocks2.summary(t2, t3)
        if clk2.get("sm_mhz") is not None:
            clk2["window"] = (f"{n_more} more steps of the same workload right after the timed region "
                              f"({clk.get('samples', 0)} samples fell inside it)")
            clk = clk2

    # The same step with the window rows' log-sum-exp supplied by the caller
    # (kvec_select_layers_lse, no statistics pass over K); the lse inputs are
    # prepared outside the timed region.
    lse_variant = None
    if args.lse_variant:
        lses = [window_lse_torch(wl_rank, x, dev) for x in layers]

        def step_lse():
            kvec.kvec_reset(sel.handle, state.data_ptr(), wl.batch, stream.cuda_stream)
            sel.select_layers(cu_host, cu_dev, qs, ks, vs, state, wl.budget, outs, stream, lses=lses)

        for _ in range(max(args.warmup, 3)):
            step_lse()
        n_lse = min(args.steps, 500)
        torch.cuda.synchronize()
        start.record(stream)
        for _ in range(n_lse):
            step_lse()
        stop.record(stream)
        torch.cuda.synchronize()
        kvec.kvec_sync_status(sel.handle)
        ms_lse = max_over_ranks(start.elapsed_time(stop), dev) / n_lse
        lse_variant = {"metric": METRIC, "value": world * evicted_per_step / (ms_lse / 1e3), "unit": "tokens/s",
                       "ms_per_step": ms_lse, "steps": n_lse,
                       "api": "kvec_select_layers_lse: window-row log-sum-exp from the caller's prefill attention",
                       "path_roofline_frac": by["layer_total"] * L_layers / (ms_lse / 1e3) / 1e9 / peak}

    def timed_variant(wl_v, api):
        """The same step through a handle made for the variant's parameters (own
        outputs: the adaptive fill has more rows per head)."""
        sel_v = kvec.KvecSelector(kvec.params_from_workload(wl_v))
        state_v = sel_v.new_state(wl.batch, dev)
        outs_v = [sel_v.alloc_outputs(wl.batch, wl.budget, dev) for _ in range(L_layers)]

        def step_v():
            kvec.kvec_reset(sel_v.handle, state_v.data_ptr(), wl.batch, stream.cuda_stream)
            sel_v.select_layers(cu_host, cu_dev, qs, ks, vs, state_v, wl.budget, outs_v, stream)

        for _ in range(max(args.warmup, 3)):
            step_v()
        n_v = min(args.steps, 500)
        torch.cuda.synchronize()
        start.record(stream)
        for _ in range(n_v):
            step_v()
        stop.record(stream)
        torch.cuda.synchronize()
        kvec.kvec_sync_status(sel_v.handle)
        sel_v.close()
        del outs_v, state_v
        ms_v = max_over_ranks(start.elapsed_time(stop), dev) / n_v
        return {"metric": METRIC, "value": world * evicted_per_step / (ms_v / 1e3), "unit": "tokens/s",
                "ms_per_step": ms_v, "steps": n_v, "api": api,
                "path_roofline_frac": by["layer_total"] * L_layers / (ms_v / 1e3) / 1e9 / peak}

    # Every position a candidate (kvec_params.all_positions = 1: Section 4.1's
    # top-B over the T input tokens, no retained window).
    all_positions_variant = None
    if args.all_positions_variant:
        all_positions_variant = timed_variant(
            wl.replace(all_positions=1), "kvec_select_layers with kvec_params.all_positions = 1: top-B over every position")
    # Head-wise adaptive fill (kvec_params.head_budget = 1): each head ranks a
    # fifth of its fill itself, the rest is ranked over the heads of a sequence.
    adaptive_variant = None
    if args.adaptive_variant:
        adaptive_variant = timed_variant(
            wl.replace(head_budget=1, ada_floor=0.2),
            "kvec_select_layers with kvec_params.head_budget = 1, ada_floor = 0.2: head-wise adaptive fill")

    decode = run_decode(args, wl, sel, layers, outs, dev, peak) if args.decode else None

    # End to end through the public API: pinned host inputs copied in, indices and state copied out.
    e2e = run_e2e(args, wl, sel, layers, outs, state, cu_host, cu_dev, dev, stream) if args.e2e else None

    # Per layer: score, row statistics, window, heads pooling, heads top-K, select,
    # gather; per call one finalize launch (the last layer's union into the state).
    gpu_launches = args.steps * (L_layers * LAUNCHES_PER_LAYER + 1)
    sel.close()
    del layers, qs, ks, vs, outs, state
    torch.cuda.empty_cache()
    other = run_other_configs(args, wl, dev, peak) if args.other_configs and world == 1 else None
    result = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": wl.name, "layers": L_layers, "batch": wl.batch, "seqlens": list(wl.seqlens)[:8],
                   "q_heads": wl.num_q_heads, "kv_heads": wl.num_kv_heads, "head_dim": wl.head_dim,
                   "window": wl.window, "budget": wl.budget, "parallelism": f"replicas{world}",
                   "l2": f"inputs larger than L2 ({(by['k_read'] * 2 + by['q_read']) * L_layers / 1e9:.2f} GB per step)",
                   "precision": "bf16 inputs, fp32 accumulation and scores"},
        "roofline": {"bound": "hbm", "kernel": "whole eviction pass: every kernel of one kvec_select_layers call",
                     "achieved": path_gbs, "peak": peak, "unit": "GB/s", "frac": path_gbs / peak,
                     "traffic": committed_step_traffic(wl, L_layers), "peak_source": peak_kind,
                     "bytes_per_step": bytes_step,
                     "bytes": "algorithmic: K read once + q_obs + kept K/V rows read and written + out_idx",
                     "strict_frac": (by["k_read"] + by["gather"] // 2) * L_layers / (ms_per_step / 1e3) / 1e9 / peak},
        "clocks": clk,
        "gpu_launches": gpu_launches,
        "lse_variant": lse_variant,
        "all_positions_variant": all_positions_variant,
        "adaptive_variant": adaptive_variant,
        "decode": decode,
        "e2e": e2e,
        "other_configs": other,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = oracle_baseline(wl)
    return rank, result


def run_other_configs(args, wl_main, dev, peak):
    """The other workloads of the benchmark set, each timed like the main one (one
    step = reset + one kvec_select_layers call over every layer; device time with
    CUDA events on the launching stream, inputs resident in HBM, larger than L2).
    The Qwen2.5-7B-shaped workload runs at every budget of its sweep."""
    import torch
    from paper_2606_29563_gb300 import kvec, synth
    names = [n for n in synth.WORKLOADS if n != wl_main.name]
    runs = []
    for n in names:
        base = synth.WORKLOADS[n]
        if n.startswith("qwen7b"):
            runs += [base.replace(budget=b, name=f"{n.rsplit('_b', 1)[0]}_b{b}") for b in synth.QWEN_BUDGETS]
        else:
            runs.append(base)
    out = {}
    stream = torch.cuda.current_stream(dev)
    for wl in runs:
        if wl.name == wl_main.name:
            continue
        structure = [synth.salient_structure(wl, b, wl.layers) for b in range(wl.batch)]
        xs = [synth.make_layer(wl, l, dev, structure) for l in range(wl.layers)]
        sel = kvec.KvecSelector(kvec.params_from_workload(wl))
        cu_host = torch.tensor(wl.cu_seqlens, dtype=torch.int32).pin_memory()
        cu_dev = cu_host.to(dev)
        outs = [sel.alloc_outputs(wl.batch, wl.budget, dev) for _ in range(wl.layers)]
        state = sel.new_state(wl.batch, dev)
        qs, ks, vs = [x["q_obs"] for x in xs], [x["k"] for x in xs], [x["v"] for x in xs]

        def step():
            kvec.kvec_reset(sel.handle, state.data_ptr(), wl.batch, stream.cuda_stream)
            sel.select_layers(cu_host, cu_dev, qs, ks, vs, state, wl.budget, outs, stream)

        for _ in range(max(args.warmup, 3)):
            step()
        torch.cuda.synchronize()
        n_steps = max(10, min(args.steps, 200))
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(n_steps):
            step()
        b.record(stream)
        torch.cuda.synchronize()
        kvec.kvec_sync_status(sel.handle)
        ms = a.elapsed_time(b) / n_steps
        by = workload_bytes(wl)
        bytes_step = by["layer_total"] * wl.layers
        evicted = wl.evicted_per_layer() * wl.layers
        out[wl.name] = {"ms_per_step": ms, "steps": n_steps, "value": evicted / (ms / 1e3), "unit": "tokens/s",
                        "layers": wl.layers, "batch": wl.batch, "budget": wl.budget,
                        "evicted_per_step": evicted, "bytes_per_step": bytes_step,
                        "path_roofline_frac": bytes_step / (ms / 1e3) / 1e9 / peak}
        sel.close()
        del xs, qs, ks, vs, outs, state
        torch.cuda.empty_cache()
    return out


def run_decode(args, wl, sel, layers, outs, dev, peak):
    """One decoding step (one generated token: every layer) over the compacted
    caches that the selection just wrote, kvec_decode_attention per layer with
    lens = min(L_s, B).  The layer loop is captured in a CUDA graph so that the
    device time is measured, not the host's launch rate.  Roofline bytes per
    call: the kept K and V rows read, the query rows read, the fp32 output
    written."""
    import numpy as np
    import torch
    from paper_2606_29563_gb300 import kvec

    lens = [min(L, wl.budget) for L in wl.seqlens]
    lens_d = torch.tensor(lens, dtype=torch.int32, device=dev)
    dq = [x["q_obs"][:, -1].contiguous() for x in layers]
    dout = [torch.empty((wl.batch, wl.num_q_heads, wl.head_dim), dtype=torch.float32, device=dev) for _ in layers]

    def dstep(st):
        for l in range(len(layers)):
            kvec.kvec_decode_attention(sel.handle, wl.batch, dq[l].data_ptr(), outs[l][1].data_ptr(),
                                       outs[l][2].data_ptr(), lens_d.data_ptr(), wl.budget, dout[l].data_ptr(),
                                       st.cuda_stream)

    side = torch.cuda.Stream(dev)
    side.wait_stream(torch.cuda.current_stream(dev))
    with torch.cuda.stream(side):
        for _ in range(3):
            dstep(side)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        dstep(torch.cuda.current_stream(dev))
    for _ in range(3):
        graph.replay()
    torch.cuda.synchronize()
    n = max(20, min(args.steps, 2000))
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    cur = torch.cuda.current_stream(dev)
    a.record(cur)
    for _ in range(n):
        graph.replay()
    b.record(cur)
    torch.cuda.synchronize()
    ms_token = a.elapsed_time(b) / n
    us_call = ms_token * 1e3 / len(layers)
    bytes_call = (sum(lens) * wl.num_kv_heads * wl.head_dim * 2 * 2 + wl.batch * wl.num_q_heads * wl.head_dim * (2 + 4)
                  + 4 * wl.batch)
    gbs = bytes_call / (us_call / 1e6) / 1e9
    res_cpu = None
    if not args.no_cpu_baseline:
        # CPU baseline leg: the fp64 oracle on the same call (layer 0), host cores.
        from oracle.decode import decode_attention as oracle_decode
        f64 = lambda t: t.float().cpu().numpy().astype(np.float64)
        q0, k0, v0 = f64(dq[0]), f64(outs[0][1]), f64(outs[0][2])
        t0 = time.perf_counter()
        oracle_decode(q0, k0, v0, lens, 1.0 / np.sqrt(wl.head_dim))
        cpu_ms = (time.perf_counter() - t0) * 1e3
        res_cpu = {"value": 1e3 / (cpu_ms * len(layers)), "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
                   "sample": "one layer call of the step (fp64 NumPy; its BLAS may use up to all host threads), scaled to all layers"}
    return {"api": "kvec_decode_attention, one call per layer (one generated token), CUDA graph",
            "ms_per_token": ms_token, "us_per_layer_call": us_call, "tokens_per_s": 1e3 / ms_token,
            "gpu_launches_per_token": len(layers), "bytes_per_call": bytes_call,
            "roofline": {"bound": "hbm", "achieved": gbs, "peak": peak, "unit": "GB/s", "frac": gbs / peak,
                         "traffic": committed_traffic("decode", wl.name)},
            "cache_rows_per_head": lens, "cpu_baseline": res_cpu}


def run_e2e(args, wl, sel, layers, outs, state, cu_host, cu_dev, dev, stream):
    """End to end through the public API.  Every step copies the step's inputs
    (q_obs, K, V of every layer) from pinned host memory and reads the kept
    indices and the coverage state back.  The copies run on their own stream in
    chunks of E2E_CHUNK layers; a chunk's selection (one kvec_select_layers call,
    replayed from the handle's graph cache) starts once its inputs have landed,
    so it overlaps the copy of the next chunks.  Two sets of device input
    buffers alternate between steps, so the next step's copies do not wait for
    this step's last chunk.  The host link (about 210 GB/s measured on this
    machine for pinned copies, by copy engine or by SM loads alike) bounds the
    step."""
    import torch
    from paper_2606_29563_gb300 import kvec
    host = [{k: v.cpu().pin_memory() for k, v in x.items()} for x in layers]
    dev_sets = [[{k: torch.empty_like(v) for k, v in x.items()} for x in layers] for _ in range(2)]
    host_idx = [torch.empty(o[0].shape, dtype=o[0].dtype).pin_memory() for o in outs]
    host_state = torch.empty(state.shape, dtype=state.dtype).pin_memory()
    h2d = sum(t.numel() * t.element_size() for x in host for t in x.values())
    d2h = sum(t.numel() * t.element_size() for t in host_idx) + host_state.numel()
    copy_stream = torch.cuda.Stream(dev)
    chunks = [list(range(c, min(c + E2E_CHUNK, len(layers)))) for c in range(0, len(layers), E2E_CHUNK)]
    landed = [[torch.cuda.Event() for _ in chunks] for _ in range(2)]
    freed = [torch.cuda.Event() for _ in range(2)]
    count = [0]

    def step():
        par = count[0] & 1
        count[0] += 1
        dev_in, land = dev_sets[par], landed[par]
        # The selection of two steps ago must be done with this set of input buffers.
        if count[0] > 2:
            copy_stream.wait_event(freed[par])
        with torch.cuda.stream(copy_stream):
            for c, ls in enumerate(chunks):
                for l in ls:
                    for k in ("q_obs", "k", "v"):
                        dev_in[l][k].copy_(host[l][k], non_blocking=True)
                land[c].record(copy_stream)
        kvec.kvec_reset(sel.handle, state.data_ptr(), wl.batch, stream.cuda_stream)
        for c, ls in enumerate(chunks):
            stream.wait_event(land[c])
            sel.select_layers(cu_host, cu_dev, [dev_in[l]["q_obs"] for l in ls], [dev_in[l]["k"] for l in ls],
                              [dev_in[l]["v"] for l in ls], state, wl.budget, [outs[l] for l in ls], stream)
        freed[par].record(stream)
        for o, h in zip(outs, host_idx):
            h.copy_(o[0], non_blocking=True)
        host_state.copy_(state, non_blocking=True)

    for _ in range(max(1, args.warmup)):
        step()
    torch.cuda.synchronize()
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    # The first copies run on the copy stream: the timed region opens there.
    start.record(copy_stream)
    n = max(1, min(args.steps, 200))
    for _ in range(n):
        step()
    stop.record(stream)
    torch.cuda.synchronize()
    ms = max_over_ranks(start.elapsed_time(stop), dev)
    _, world, _ = dist_env()
    value = world * wl.evicted_per_layer() * wl.layers * n / (ms / 1e3)
    return {"value": value, "unit": "tokens/s", "ms_per_step": ms / n, "steps": n, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h,
            "api": f"kvec_select_layers per chunk of {E2E_CHUNK} layers on the compute stream; pinned copies of "
                   "the next chunks on a copy stream"}


# ----------------------------------------------------------------------------- reference arm (the oracle)

def run_reference(args, wl):
    rank, world, _ = dist_env()
    if rank != 0:
        return rank, None
    import oracle
    from paper_2606_29563_gb300 import synth
    oracle.build()
    p = oracle.OracleParams.from_workload(wl)
    structure = [synth.salient_structure(wl, b, 1) for b in range(wl.batch)]
    x = synth.make_layer(wl, 0, "cpu", structure)
    cu = wl.cu_seqlens
    # A bounded sample per step: layer 0 of one sequence of the batch (the
    # sequences in turn), from a fresh coverage state.
    samples = []
    for b in range(wl.batch):
        wl_b = wl.replace(seqlens=(wl.seqlens[b],))
        samples.append((wl_b, x["q_obs"][b:b + 1], x["k"][cu[b]:cu[b + 1]], x["v"][cu[b]:cu[b + 1]]))
    count = [0]

    def step():
        wl_b, q, k, v = samples[count[0] % len(samples)]
        count[0] += 1
        st = oracle.new_state(1, wl_b.max_seqlen)
        oracle.select_layer(p, wl_b.cu_seqlens, q, k, v, st, wl.budget, max_seqlen=wl_b.max_seqlen, debug=False)
        return wl_b.evicted_per_layer()

    for _ in range(args.warmup):
        step()
    evicted = 0
    t0 = time.perf_counter()
    for _ in range(args.steps):
        evicted += step()
    dt = time.perf_counter() - t0
    value = evicted / dt
    sample = (f"layer 0 of one sequence of {wl.name} per step (the {wl.batch} sequences in turn), fp64 C oracle, "
              f"OpenMP, {oracle.num_threads()} threads")
    return rank, {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3 / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": wl.name, "layers_per_step": 1, "sequences_per_step": 1, "batch": wl.batch,
                   "budget": wl.budget},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": oracle.num_threads(), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1, help="GPUs of one node (N > 1: launched by torch.distributed.run, one replica per GPU)")
    ap.add_argument("--steps", type=int, default=1000, help="timed steps (one step: every layer of one batch)")
    ap.add_argument("--warmup", type=int, default=5, help="untimed steps before the timed ones")
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours",
                    help="reference: time the fp64 oracle on the host cores instead of the CUDA path")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, help="one of synth.WORKLOADS")
    ap.add_argument("--budget", type=int, default=None, help="tokens kept per KV head (default: the workload's)")
    ap.add_argument("--layers", type=int, default=None, help="run only the first N layers (not a bench line)")
    ap.add_argument("--no-e2e", dest="e2e", action="store_false",
                    help="skip the end-to-end measurement with inputs copied from host memory")
    ap.add_argument("--no-cpu-baseline", action="store_true", help="skip timing the fp64 oracle on a sample")
    ap.add_argument("--coverage-sweep", action="store_true",
                    help="print the token coverage of K-VEC and SnapKV at eviction rates 0.25-0.9 and exit")
    ap.add_argument("--no-decode", dest="decode", action="store_false",
                    help="skip the decode-attention measurement over the compacted caches")
    ap.add_argument("--no-lse-variant", dest="lse_variant", action="store_false",
                    help="skip timing the kvec_select_layers_lse variant")
    ap.add_argument("--no-all-positions-variant", dest="all_positions_variant", action="store_false",
                    help="skip timing the top-B-over-every-position variant")
    ap.add_argument("--no-adaptive-variant", dest="adaptive_variant", action="store_false",
                    help="skip timing the head-wise adaptive fill (kvec_params.head_budget = 1)")
    ap.add_argument("--no-clock-probe", dest="clock_probe", action="store_false",
                    help="do not extend a short timed region by a second of steps to read the clocks")
    ap.add_argument("--no-other-configs", dest="other_configs", action="store_false",
                    help="skip timing the other workloads of the benchmark set")
    args = ap.parse_args(argv)
    if args.warmup < 3 and args.impl == "ours":
        args.warmup = 3
    from paper_2606_29563_gb300 import synth
    wl = synth.WORKLOADS[args.workload]
    if args.budget:
        wl = wl.replace(budget=args.budget, name=f"{wl.name.rsplit('_b', 1)[0]}_b{args.budget}")
    if args.layers:
        wl = wl.replace(layers=args.layers)
    if args.coverage_sweep:
        from paper_2606_29563_gb300 import build as kbuild
        from paper_2606_29563_gb300 import coverage
        kbuild.build()
        print(json.dumps({"coverage_sweep": coverage.sweep(wl), "data": "synthetic"}), flush=True)
        return 0
    rank, result = (run_reference if args.impl == "reference" else run_ours)(args, wl)
    if rank == 0 and result is not None:
        print(json.dumps(result), flush=True)


if __name__ == "__main__":
    main()
