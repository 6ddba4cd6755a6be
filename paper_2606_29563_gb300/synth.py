"""Seeded synthetic inputs shaped like long-context prefill for KV-cache eviction.

This module only draws inputs; it holds none of the eviction method's
arithmetic. Both the CUDA path and the CPU oracle consume what it produces.

Recipe (stand-in for LongBench prompts run through Llama-3.1-8B /
Qwen2.5-7B, neither of which is available here):

* q_obs (the last ``w`` query rows of each sequence), K and V are drawn
  N(0, 1) in fp32 and rounded to bf16 (round-to-nearest-even), independently
  for every layer.
* u_h is the unit vector along the mean of the group-h window queries (the
  ``g`` query heads that share KV head h, over all ``w`` window rows).
* Attention sink: K[0, h] += ``sink`` * u_h.
* Planted salient tokens: a per-(sequence, layer) base set of positions in
  [1, L - w).  A fraction ``carry`` of layer l-1's base set is kept for layer
  l, the rest is drawn fresh.  Each KV head keeps every base position with
  probability ``p_share`` and otherwise substitutes a fresh uniform position.
  K[t, h] += m_t * u_h with m_t = ``salient_mag`` (or ``salient_mag`` times a
  LogNormal(0, ``lognormal_sigma``) draw when that sigma is set).

Integer structure (lengths, salient positions) comes from numpy's PCG64 so it
is identical on every platform; Gaussian tensors come from a torch
``Generator`` on the requested device.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional, Sequence

import numpy as np
import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    layers: int
    seqlens: tuple            # prefix length L_s of every sequence in the batch
    num_q_heads: int
    num_kv_heads: int
    head_dim: int = 128
    window: int = 32          # w: observation rows supplied, also the retained tail
    obs_window: int = 16      # O
    ext_window: int = 32      # O'
    pool_kernel: int = 7
    pool_mode: int = 0        # 0 max-pool, 1 average pool (variant)
    head_criterion: int = 0   # 0 standard deviation, 1 entropy (variant)
    all_positions: int = 0    # 0 keep the window tail, 1 every position is a candidate (variant)
    head_budget: int = 0      # 0 uniform fill, 1 head-wise adaptive fill (variant)
    ada_floor: float = 0.2    # adaptive fill: share of a head's fill it keeps by its own ranking
    budget: int = 512         # B per KV head, window included
    num_ext_heads: int = 3    # delta
    lam: float = 1.0          # lambda
    beta: float = 0.25
    salient: int = 0          # salient positions per (sequence, layer)
    salient_frac: float = 0.0 # used when salient == 0: round(frac * L)
    p_share: float = 0.7
    carry: float = 0.0
    salient_mag: float = 3.0
    lognormal_sigma: float = 0.0
    sink: float = 6.0
    seed: int = 20260

    @property
    def batch(self) -> int:
        return len(self.seqlens)

    @property
    def group(self) -> int:
        return self.num_q_heads // self.num_kv_heads

    @property
    def cu_seqlens(self) -> List[int]:
        cu = [0]
        for L in self.seqlens:
            cu.append(cu[-1] + int(L))
        return cu

    @property
    def total_tokens(self) -> int:
        return int(sum(self.seqlens))

    @property
    def max_seqlen(self) -> int:
        return int(max(self.seqlens))

    def salient_count(self, L: int) -> int:
        if self.salient:
            return int(self.salient)
        return int(round(self.salient_frac * L))

    def evicted_per_layer(self) -> int:
        """KV entries freed by one layer: sum over sequences and KV heads of max(L_s - B, 0)."""
        return sum(max(int(L) - self.budget, 0) for L in self.seqlens) * self.num_kv_heads

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


def _ragged_lengths(seed: int, batch: int, lo: int, hi: int) -> tuple:
    rng = np.random.Generator(np.random.PCG64(seed))
    return tuple(int(x) for x in rng.integers(lo, hi + 1, size=batch))


# The five workloads: shapes of the paper's Llama-3.1-8B / Qwen2.5-7B prefill.
WORKLOADS: Dict[str, Workload] = {
    # 1 layer, 8 query heads = 8 KV heads, L=1024, cross-head coverage only.
    "mha8_l1024_b128": Workload(
        name="mha8_l1024_b128", layers=1, seqlens=(1024,), num_q_heads=8, num_kv_heads=8,
        budget=128, num_ext_heads=3, lam=0.0, beta=0.25, salient=40, p_share=0.7,
        carry=0.0, seed=20260),
    # Llama-3.1-8B shaped: 32 layers, 32/8 heads, L=8192, B=512.
    "llama8b_l8192_b512": Workload(
        name="llama8b_l8192_b512", layers=32, seqlens=(8192,), num_q_heads=32, num_kv_heads=8,
        budget=512, salient_frac=0.01, p_share=0.7, carry=0.6, seed=20261),
    # Same shape at L=32768, B=128, heavy-tailed salience at 0.5%.
    "llama8b_l32768_b128": Workload(
        name="llama8b_l32768_b128", layers=32, seqlens=(32768,), num_q_heads=32, num_kv_heads=8,
        budget=128, salient_frac=0.005, p_share=0.7, carry=0.6, lognormal_sigma=0.5, seed=20262),
    # Ragged batch of 8, L ~ U[4096, 16384], B=256.
    "llama8b_ragged8_b256": Workload(
        name="llama8b_ragged8_b256", layers=32, seqlens=_ragged_lengths(20263, 8, 4096, 16384),
        num_q_heads=32, num_kv_heads=8, budget=256, salient_frac=0.01, p_share=0.7, carry=0.6,
        seed=20263),
    # Qwen2.5-7B shaped: 28 layers, 28/4 heads (group 7), L=16384; budget swept.
    "qwen7b_l16384_b512": Workload(
        name="qwen7b_l16384_b512", layers=28, seqlens=(16384,), num_q_heads=28, num_kv_heads=4,
        budget=512, salient_frac=0.01, p_share=0.8, carry=0.6, seed=20264),
}

QWEN_BUDGETS = (64, 128, 256, 512, 1024, 2048)


def salient_structure(wl: Workload, seq: int, layers: int) -> List[List[np.ndarray]]:
    """Per-layer, per-KV-head salient positions for one sequence.

    Returns ``out[layer][h]``: int64 array of positions in [1, L - w).
    """
    L = int(wl.seqlens[seq])
    hi = L - wl.window          # exclusive upper bound of candidate positions
    n = min(wl.salient_count(L), max(hi - 1, 0))
    rng = np.random.Generator(np.random.PCG64([wl.seed, 7, seq]))
    out: List[List[np.ndarray]] = []
    base: Optional[np.ndarray] = None
    for _layer in range(layers):
        if n == 0:
            out.append([np.zeros(0, np.int64) for _ in range(wl.num_kv_heads)])
            continue
        if base is None:
            base = rng.choice(np.arange(1, hi), size=n, replace=False)
        else:
            keep = rng.random(n) < wl.carry
            fresh = rng.integers(1, hi, size=n)
            base = np.where(keep, base, fresh)
        per_head = []
        for _h in range(wl.num_kv_heads):
            share = rng.random(n) < wl.p_share
            fresh = rng.integers(1, hi, size=n)
            per_head.append(np.where(share, base, fresh).astype(np.int64))
        out.append(per_head)
    return out


def salient_magnitudes(wl: Workload, seq: int, layer: int, h: int, count: int) -> np.ndarray:
    if wl.lognormal_sigma <= 0.0:
        return np.full(count, wl.salient_mag, np.float32)
    rng = np.random.Generator(np.random.PCG64([wl.seed, 11, seq, layer, h]))
    return (wl.salient_mag * rng.lognormal(0.0, wl.lognormal_sigma, size=count)).astype(np.float32)


def _gaussians(dev: torch.device, key: tuple):
    """Standard-normal fp32 draws.  On the CPU they come from numpy's PCG64 (identical on x86
    and Arm); on a GPU from a seeded torch generator (fast, same statistics)."""
    if dev.type == "cpu":
        rng = np.random.Generator(np.random.PCG64(list(key)))
        return lambda shape: torch.from_numpy(rng.standard_normal(shape, dtype=np.float32))
    gen = torch.Generator(device=dev)
    gen.manual_seed(key[0] * 1_000_003 + 7919 * key[1] + 17)
    return lambda shape: torch.randn(*shape, generator=gen, device=dev, dtype=torch.float32)


def make_layer(wl: Workload, layer: int, device="cpu",
               structure: Optional[Sequence[List[List[np.ndarray]]]] = None) -> Dict[str, torch.Tensor]:
    """Inputs of one layer: q_obs [batch][w][Hq][d], k and v [total][Hkv][d], all bf16.

    ``structure`` may carry precomputed :func:`salient_structure` results (one per
    sequence, covering at least ``layer + 1`` layers) to avoid recomputation.
    """
    dev = torch.device(device)
    B, w, Hq, Hkv, d = wl.batch, wl.window, wl.num_q_heads, wl.num_kv_heads, wl.head_dim
    T = wl.total_tokens
    draw = _gaussians(dev, (int(wl.seed), int(layer)))
    q = draw((B, w, Hq, d))
    k = draw((T, Hkv, d))
    v = draw((T, Hkv, d))
    # u_h: unit vector along the mean of the group-h window queries.
    qm = q.view(B, w, Hkv, wl.group, d).mean(dim=(1, 3))          # [B][Hkv][d]
    u = qm / qm.norm(dim=-1, keepdim=True).clamp_min(1e-12)
    cu = wl.cu_seqlens
    for b in range(B):
        if wl.sink:
            k[cu[b]] += wl.sink * u[b]
        st = structure[b] if structure is not None else salient_structure(wl, b, layer + 1)
        for h in range(Hkv):
            pos = st[layer][h]
            if pos.size == 0:
                continue
            mag = torch.from_numpy(salient_magnitudes(wl, b, layer, h, pos.size)).to(dev)
            idx = torch.from_numpy(pos + cu[b]).to(dev)
            k[:, h, :].index_add_(0, idx, mag[:, None] * u[b, h][None, :])
    return {
        "q_obs": q.to(torch.bfloat16).contiguous(),
        "k": k.to(torch.bfloat16).contiguous(),
        "v": v.to(torch.bfloat16).contiguous(),
    }


def make_layers(wl: Workload, layers: int, device="cpu") -> List[Dict[str, torch.Tensor]]:
    structure = [salient_structure(wl, b, layers) for b in range(wl.batch)]
    return [make_layer(wl, l, device, structure) for l in range(layers)]


def small_workload(name: str = "tiny", **kw) -> Workload:
    """A small workload for tests: defaults that the oracle finishes in well under a second."""
    base = dict(name=name, layers=2, seqlens=(300,), num_q_heads=8, num_kv_heads=2, head_dim=128,
                window=32, obs_window=16, ext_window=32, pool_kernel=7, budget=64,
                num_ext_heads=1, lam=1.0, beta=0.25, salient=6, p_share=0.7, carry=0.5, seed=99)
    base.update(kw)
    return Workload(**base)


def tiny_full_inputs(seed: int, T: int, num_q_heads: int, num_kv_heads: int, head_dim: int,
                     key_scale: float = 1.0) -> Dict[str, torch.Tensor]:
    """Queries for *every* position of one short sequence plus its K and V (bf16).

    Used to check the oracle against a brute force that materialises the whole
    causal attention matrix; ``q_full[T - w:]`` are the observation rows.
    """
    draw = _gaussians(torch.device("cpu"), (int(seed), 0))
    q = draw((T, num_q_heads, head_dim))
    k = key_scale * draw((T, num_kv_heads, head_dim))
    v = draw((T, num_kv_heads, head_dim))
    return {"q_full": q.to(torch.bfloat16), "k": k.to(torch.bfloat16), "v": v.to(torch.bfloat16)}
